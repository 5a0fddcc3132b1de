"""Seeded synthetic inputs and integer parameters shaped like the paper's models.

This module holds no arithmetic of the method: it only draws integers.  Both the CUDA path and
the CPU oracle consume the arrays it returns, so the two sides always see identical bytes.

Generator: a counter-based SplitMix64 stream per tensor (Steele, Lea, Flood 2014, "Fast
splittable pseudorandom number generators"), keyed by (seed, FNV-1a hash of the tensor name),
so the draw order of tensors never matters and the bytes are identical on every platform.
Bounded integers use the multiply-shift map of the top 32 bits (Lemire 2019); clipped Laplace
values use the inverse CDF in float64.

Shapes follow Table 1 of the paper (Tiny: 6 layers, dim 192; Medium: 10 layers, dim 384; 3
decoder layers; 300 queries) and a 640x640 input with 16x16 patches (1600 tokens).
"""
from __future__ import annotations

import math

import numpy as np

_M64 = (1 << 64) - 1
_GOLD = np.uint64(0x9E3779B97F4A7C15)


def _fnv1a(name: str) -> int:
    h = 0xCBF29CE484222325
    for b in name.encode():
        h ^= b
        h = (h * 0x100000001B3) & _M64
    return h


def _mix(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def raw_u64(seed: int, name: str, n: int) -> np.ndarray:
    """n 64-bit words of the SplitMix64 stream keyed by (seed, name)."""
    key = _mix(np.array([(seed * 0x632BE59BD9B4E019 ^ _fnv1a(name)) & _M64], dtype=np.uint64))[0]
    idx = np.arange(1, n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        state = key + idx * _GOLD
    return _mix(state)


def uniform_int(seed: int, name: str, shape, lo: int, hi: int, dtype=np.int32) -> np.ndarray:
    """Integers uniform in [lo, hi] (inclusive)."""
    n = int(np.prod(shape)) if shape else 1
    span = hi - lo + 1
    assert 0 < span <= (1 << 32)
    u = raw_u64(seed, name, n) >> np.uint64(32)
    v = (u * np.uint64(span)) >> np.uint64(32)
    return (v.astype(np.int64) + lo).astype(dtype).reshape(shape)


def laplace_int(seed: int, name: str, shape, scale: float, clip: int, dtype=np.int8) -> np.ndarray:
    """Laplace(0, scale) draws, rounded half away from zero and clipped to [-clip, clip]."""
    n = int(np.prod(shape))
    u = ((raw_u64(seed, name, n) >> np.uint64(11)).astype(np.float64) + 0.5) / float(1 << 53)
    c = u - 0.5
    v = -scale * np.sign(c) * np.log1p(-2.0 * np.abs(c))
    r = np.sign(v) * np.floor(np.abs(v) + 0.5)
    return np.clip(r, -clip, clip).astype(dtype).reshape(shape)


# ------------------------------------------------------------------------------------------
# Parameter draws.  "calibrated" picks every per-tensor / per-channel shift from the input
# distribution's standard deviation so that outputs use their integer range without mass
# saturation (GEMM shifts stay inside [31, 40]); "literal" draws the GEMM shifts uniformly in
# [31, 40] as stated for the single-block workload.
# ------------------------------------------------------------------------------------------
SIGMA_W = 127.0 / math.sqrt(3.0)  # std of int8 weights uniform in [-127, 127]


def _shift_for(sigma_in: float, target: float, mult_mean: float = 1.5 * 2**30) -> int:
    return int(round(math.log2(mult_mean * sigma_in / target)))


def gemm_params(seed: int, name: str, N: int, K: int, sigma_a: float, target: float,
                mode: str = "calibrated", shift_range=(31, 40)):
    """Weight [N, K] int8, bias [N], per-channel dyadic (mult, shift)."""
    W = uniform_int(seed, name + ".w", (N, K), -127, 127, np.int8)
    b = uniform_int(seed, name + ".b", (N,), -(1 << 15), 1 << 15, np.int32)
    m = uniform_int(seed, name + ".m", (N,), 1 << 30, (1 << 31) - 1, np.int32)
    if mode == "literal":
        s = uniform_int(seed, name + ".s", (N,), shift_range[0], shift_range[1], np.int32)
    else:
        s0 = _shift_for(sigma_a * SIGMA_W * math.sqrt(K), target)
        s0 = min(max(s0, shift_range[0]), shift_range[1])
        s = np.full((N,), s0, dtype=np.int32)
    return W, b, m, s


def ln_params(seed: int, name: str, d: int, target: float = 32.0, mode: str = "calibrated"):
    """I-LayerNorm affine parameters: beta [d], signed mult [d] (|m| in [2^30, 2^31)), shift [d]."""
    beta = uniform_int(seed, name + ".beta", (d,), -(1 << 20), 1 << 20, np.int32)
    mag = uniform_int(seed, name + ".m", (d,), 1 << 30, (1 << 31) - 1, np.int64)
    sign = uniform_int(seed, name + ".sign", (d,), 0, 1, np.int64) * 2 - 1
    mult = (mag * sign).astype(np.int32)
    if mode == "literal":
        shift = uniform_int(seed, name + ".s", (d,), 48, 54, np.int32)
    else:
        # normalised values have std 2^30 / sqrt(d)
        shift = np.full((d,), _shift_for(2**30 / math.sqrt(d), target), dtype=np.int32)
    return beta, mult, shift


def block_params(seed: int, layer: int, d: int, H: int, F: int, win_side: int,
                 mode: str = "calibrated", sigma_x: float = 64.0, ln_iters: int = 10) -> dict:
    """All integer parameters of one encoder block (layer index keys the streams)."""
    p = f"L{layer}."
    bp: dict = {"d": d, "H": H, "F": F, "win_side": win_side, "ln_iters": ln_iters}
    bp["ln1_beta"], bp["ln1_mult"], bp["ln1_shift"] = ln_params(seed, p + "ln1", d, mode=mode)
    bp["ln2_beta"], bp["ln2_mult"], bp["ln2_shift"] = ln_params(seed, p + "ln2", d, mode=mode)
    a_sigma = 32.0  # LN outputs are calibrated to std ~32
    bp["w_qkv"], bp["b_qkv"], bp["m_qkv"], bp["s_qkv"] = gemm_params(
        seed, p + "qkv", 3 * d, d, a_sigma, 40.0, mode)
    # Shiftmax: I0 = round(1/S) of the score scale (scores have std ~ 40^2 * sqrt(dh))
    I0_s = int(uniform_int(seed, p + "smx.I0", (1,), 1 << 12, 1 << 14)[0])
    bp["smx"] = {"I0": I0_s, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
    bp["m_o"] = int(uniform_int(seed, p + "o.m", (1,), 1 << 30, (1 << 31) - 1)[0])
    bp["s_o"] = _shift_for(128.0 * 40.0, 32.0) if mode != "literal" else int(
        uniform_int(seed, p + "o.s", (1,), 31, 40)[0])
    bp["w_proj"], bp["b_proj"], bp["m_proj"], bp["s_proj"] = gemm_params(
        seed, p + "proj", d, d, 32.0, sigma_x / 2, mode)
    bp["m_r1"] = int(uniform_int(seed, p + "r1.m", (1,), 1 << 30, (1 << 31) - 1)[0])
    bp["s_r1"] = 31
    # FC1 output is the GELU input: std ~ 2 I0 so the sigmoid sees real values of a few units
    I0_g = int(uniform_int(seed, p + "gelu.I0", (1,), 1 << 9, 1 << 11)[0])
    bp["w_fc1"], bp["b_fc1"], bp["m_fc1"], bp["s_fc1"] = gemm_params(
        seed, p + "fc1", F, d, a_sigma, 2.0 * I0_g, mode)
    bp["gelu_I0"], bp["gelu_k_inter"], bp["gelu_k_out"] = I0_g, 16, 8
    bp["m_g"] = int(uniform_int(seed, p + "g.m", (1,), 1 << 30, (1 << 31) - 1)[0])
    bp["s_g"] = _shift_for(2.0 * I0_g * 64.0, 32.0) if mode != "literal" else int(
        uniform_int(seed, p + "g.s", (1,), 31, 44)[0])
    bp["w_fc2"], bp["b_fc2"], bp["m_fc2"], bp["s_fc2"] = gemm_params(
        seed, p + "fc2", d, F, 40.0, sigma_x / 2, mode)
    bp["m_r2"] = int(uniform_int(seed, p + "r2.m", (1,), 1 << 30, (1 << 31) - 1)[0])
    bp["s_r2"] = 31
    return bp


def block_input(seed: int, B: int, T: int, d: int, dist: str = "uniform") -> np.ndarray:
    """Block input x (int16 container, int8-valued): uniform [-127,127] or Laplace(20) clip 127."""
    if dist == "laplace":
        return laplace_int(seed, "x", (B * T, d), 20.0, 127, np.int16)
    return uniform_int(seed, "x", (B * T, d), -127, 127, np.int16)


# ------------------------------------------------------------------------------------------
# Workload configurations (sizes of the paper's models, Table 1; 640x640 input, 16x16 patches)
# ------------------------------------------------------------------------------------------
CONFIGS = {
    # single block, batch 1, 256 tokens, dim 192, 3 heads, MLP 768, global attention
    "block_256tok_d192": dict(B=1, T=256, d=192, H=3, F=768, layers=1, global_layers=(0,), mode="literal",
                              dist="uniform"),
    # Tiny-scale backbone: 6 blocks alternating window (2x2 windows of 400 tokens) / global
    "tiny_backbone_b8": dict(B=8, T=1600, d=192, H=3, F=768, layers=6, global_layers=(1, 3, 5),
                             mode="calibrated", dist="uniform"),
    # Medium-scale backbone: 10 blocks, global attention at the output layers 2, 4, 5, 9
    "medium_backbone_b8": dict(B=8, T=1600, d=384, H=6, F=1536, layers=10, global_layers=(2, 4, 5, 9),
                               mode="calibrated", dist="laplace"),
}


# Full integer detector (640x640, batch 16): the Medium backbone with its four output layers
# tapped, a split-convolution projector at strides 8 / 16 / 32 (80x80, 40x40, 20x20 maps of 256
# channels, concatenated as the decoder memory), and 3 decoder layers of 300 queries, dim 256,
# 8 heads, 4 sampling points per level, MLP 1024.
CONFIGS["medium_detector_b16"] = dict(B=16, backbone="medium_backbone_b8", taps=(2, 4, 5, 9), grid=40,
                                      levels=((80, 80), (40, 40), (20, 20)), N=256, Q=300, Hd=8, Fd=1024,
                                      P=4, dec_layers=3)


def _mult(seed: int, name: str) -> int:
    return int(uniform_int(seed, name, (1,), 1 << 30, (1 << 31) - 1)[0])


def projector_params(seed: int, nb: int, K: int, N: int = 256, levels: int = 3,
                     sigma_tap: float = 600.0) -> dict:
    """Tap requantisation (one per-tensor scale per tapped layer, 2^(b) apart so the branches
    really differ) and, per level, one split convolution: branch weights int8 [N, K], per-branch
    dyadic rescale to the largest branch scale (ratio <= 1), bias and per-channel output rq."""
    pp: dict = {"taps": [], "levels": []}
    s_tap = [_shift_for(sigma_tap, 40.0) + b for b in range(nb)]  # branch b: scale 2^b larger
    for b in range(nb):
        pp["taps"].append((_mult(seed, f"prj.t{b}.m"), s_tap[b]))
    s_max = max(s_tap)
    for l in range(levels):
        lv = {"w": [], "m_b": [], "s_b": []}
        for b in range(nb):
            W = uniform_int(seed, f"prj.l{l}.w{b}", (N, K), -127, 127, np.int8)
            lv["w"].append(W)
            lv["m_b"].append(_mult(seed, f"prj.l{l}.mb{b}"))
            lv["s_b"].append(31 + (s_max - s_tap[b]))  # m_b / 2^s_b in [2^-1, 1) * 2^(s_b' - s_max)
        # each branch contributes ~ sqrt(K) * 40 * SIGMA_W, the largest-scale branch fully
        lv["b"] = uniform_int(seed, f"prj.l{l}.b", (N,), -(1 << 15), 1 << 15, np.int32)
        lv["m"] = uniform_int(seed, f"prj.l{l}.m", (N,), 1 << 30, (1 << 31) - 1, np.int32)
        lv["s"] = np.full((N,), _shift_for(40.0 * SIGMA_W * math.sqrt(K) * 1.2, 40.0), dtype=np.int32)
        pp["levels"].append(lv)
    return pp


def decoder_params(seed: int, layer: int, d: int = 256, H: int = 8, F: int = 1024, L: int = 3,
                   P: int = 4, sigma_t: float = 2048.0) -> dict:
    """All integer parameters of one decoder layer (post-norm self-attention, nearest-neighbour
    deformable cross-attention, FFN with SD-ShiftGELU; I-LayerNorm with 20 Newton steps and int16
    outputs of std ~ sigma_t)."""
    p = f"D{layer}."
    dp: dict = {"d": d, "H": H, "F": F, "L": L, "P": P, "ln_iters": 20}
    s_in = _shift_for(sigma_t, 32.0)  # int16 residual stream -> int8 layer input
    for k in ("q1", "q2", "v1", "c1", "c2", "f"):
        dp["m_" + k] = _mult(seed, p + k + ".m")
        dp["s_" + k] = s_in + (1 if k in ("q1", "q2", "c1", "c2") else 0)  # two terms: half each
    dp["w_qk"], dp["b_qk"], dp["m_qk"], dp["s_qk"] = gemm_params(seed, p + "qk", 2 * d, d, 32.0, 40.0)
    dp["w_v"], dp["b_v"], dp["m_v"], dp["s_v"] = gemm_params(seed, p + "v", d, d, 32.0, 40.0)
    I0_s = int(uniform_int(seed, p + "smx.I0", (1,), 1 << 12, 1 << 14)[0])
    dp["smx"] = {"I0": I0_s, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
    dp["m_o"], dp["s_o"] = _mult(seed, p + "o.m"), _shift_for(128.0 * 40.0, 32.0)
    dp["w_o"], dp["b_o"], dp["m_oc"], dp["s_oc"] = gemm_params(seed, p + "out", d, d, 32.0, sigma_t / 2)
    dp["m_r1"], dp["s_r1"] = _mult(seed, p + "r1.m"), 31
    for i in (1, 2, 3):
        dp[f"ln{i}_beta"], dp[f"ln{i}_mult"], dp[f"ln{i}_shift"] = ln_params(seed, p + f"ln{i}", d, target=sigma_t)
    dp["w_val"], dp["b_val"], dp["m_val"], dp["s_val"] = gemm_params(seed, p + "val", d, d, 40.0, 40.0)
    # sampling offsets in Q8 pixels (std ~ 2 pixels) and attention logits (std ~ 2 I0_w)
    dp["w_off"], dp["b_off"], dp["m_off"], dp["s_off"] = gemm_params(seed, p + "off", H * L * P * 2, d, 32.0, 512.0)
    I0_w = int(uniform_int(seed, p + "smxw.I0", (1,), 1 << 6, 1 << 8)[0])
    dp["w_att"], dp["b_att"], dp["m_att"], dp["s_att"] = gemm_params(seed, p + "att", H * L * P, d, 32.0, 2.0 * I0_w)
    dp["smx_w"] = {"I0": I0_w, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
    dp["m_s"], dp["s_s"] = _mult(seed, p + "s.m"), _shift_for(128.0 * 40.0 / 2.0, 32.0)
    dp["w_o2"], dp["b_o2"], dp["m_o2"], dp["s_o2"] = gemm_params(seed, p + "out2", d, d, 32.0, sigma_t / 2)
    dp["m_r2"], dp["s_r2"] = _mult(seed, p + "r2.m"), 31
    I0_g = int(uniform_int(seed, p + "gelu.I0", (1,), 1 << 9, 1 << 11)[0])
    dp["w_fc1"], dp["b_fc1"], dp["m_fc1"], dp["s_fc1"] = gemm_params(seed, p + "fc1", F, d, 32.0, 2.0 * I0_g)
    dp["gelu_I0"], dp["gelu_k_inter"], dp["gelu_k_out"] = I0_g, 16, 8
    dp["m_g"], dp["s_g"] = _mult(seed, p + "g.m"), _shift_for(2.0 * I0_g * 64.0, 32.0)
    dp["w_fc2"], dp["b_fc2"], dp["m_fc2"], dp["s_fc2"] = gemm_params(seed, p + "fc2", d, F, 40.0, sigma_t / 2)
    dp["m_r3"], dp["s_r3"] = _mult(seed, p + "r3.m"), 31
    return dp


def decoder_inputs(seed: int, B: int, Q: int, d: int = 256) -> dict:
    """Initial queries tgt and positional queries pos (int16 [B*Q, d], uniform in +-2^11) and the
    reference points (x, y) in Q16 of the map, fixed across the decoder layers."""
    return {"tgt": uniform_int(seed, "dec.tgt", (B * Q, d), -(1 << 11), 1 << 11, np.int16),
            "pos": uniform_int(seed, "dec.pos", (B * Q, d), -(1 << 11), 1 << 11, np.int16),
            "refs": uniform_int(seed, "dec.refs", (B, Q, 2), 0, (1 << 16) - 1, np.int32)}


def image_input(seed: int, B: int, H: int = 640, W: int = 640) -> np.ndarray:
    """int8 image [B, 3, H, W], uniform in [-127, 127]."""
    return uniform_int(seed, "img", (B, 3, H, W), -127, 127, np.int8)


def patch_embed_params(seed: int, d: int, p: int = 16, T: int = 1600, mode: str = "calibrated",
                       sigma_x: float = 64.0) -> dict:
    """Patch-embedding conv weight [d, 3*p*p], bias, per-channel dyadic pair, position term."""
    W, b, m, s = gemm_params(seed, "pe", d, 3 * p * p, 127.0 / math.sqrt(3.0), sigma_x, mode)
    pos = uniform_int(seed, "pe.pos", (T, d), -64, 64, np.int16)
    return {"p": p, "w": W, "b": b, "m": m, "s": s, "pos": pos, "m_pos": 1 << 30, "s_pos": 31}


def backbone_params(seed: int, cfg: dict) -> list:
    out = []
    for layer in range(cfg["layers"]):
        win = 0 if layer in cfg["global_layers"] else 2
        out.append(block_params(seed, layer, cfg["d"], cfg["H"], cfg["F"], win, cfg["mode"]))
    return out


def head_params(seed: int, d: int = 256, C: int = 80, sigma_in: float = 32.0, k_inter: int = 8) -> dict:
    """Integer parameters of the detection head: class linear layer (raw int32 logits of std ~2/S
    with I0 = 1/S), box MLP d -> d -> d -> 4 (int8 hidden outputs of std ~32), box deltas
    requantised to the reference-logit scale 2^-10 (std ~256, i.e. 0.25 in logit units) and the
    int16 reference logits taken at that scale (identity requantisation)."""
    p = "H."
    hp: dict = {"k_inter": k_inter, "cls_k_out": 8}
    acc_std = sigma_in * 73.3 * math.sqrt(d)  # U[-127, 127] weights: std 73.3
    hp["w_cls"], hp["b_cls"], _, _ = gemm_params(seed, p + "cls", C, d, sigma_in, 1.0)
    hp["cls_I0"] = int(min(acc_std / 2.0, (1 << 15) - 1))
    hp["w_b1"], hp["b_b1"], hp["m_b1"], hp["s_b1"] = gemm_params(seed, p + "b1", d, d, sigma_in, 32.0)
    hp["w_b2"], hp["b_b2"], hp["m_b2"], hp["s_b2"] = gemm_params(seed, p + "b2", d, d, 16.0, 32.0)
    hp["w_b3"], hp["b_b3"], _, _ = gemm_params(seed, p + "b3", 4, d, 16.0, 1.0)
    hp["m_d"] = _mult(seed, p + "d.m")
    hp["s_d"] = _shift_for(16.0 * 73.3 * math.sqrt(d), 256.0)
    hp["m_ref"], hp["s_ref"] = 1 << 30, 30
    hp["box_I0"] = 1024
    # the requantisation of the decoder's int16 output (std ~2^11) to the head's int8 input
    hp["m_in"], hp["s_in"] = _mult(seed, p + "in.m"), _shift_for(2048.0, 32.0)
    return hp


def refine_params(seed: int, layers: int, d: int = 256, sigma_in: float = 32.0, k_inter: int = 8) -> list:
    """Integer parameters of the box refinement between decoder layers (one box branch per layer
    whose output feeds another layer): the decoder output requantised to int8, a box MLP
    d -> d -> d -> 4 with ReLU on its int8 hidden outputs, the deltas requantised to the
    reference-logit scale 2^-10 (std ~256) and added to the current reference logits, the result
    saturated to int16 and passed through the integer sigmoid (scale 2^-16).  Same recipe as the
    detection head's box branch, drawn per layer."""
    out = []
    acc_std = sigma_in * 73.3 * math.sqrt(d)
    for l in range(layers):
        p = f"RB{l}."
        rp: dict = {"k_inter": k_inter}
        rp["w_b1"], rp["b_b1"], rp["m_b1"], rp["s_b1"] = gemm_params(seed, p + "b1", d, d, sigma_in, 32.0)
        rp["w_b2"], rp["b_b2"], rp["m_b2"], rp["s_b2"] = gemm_params(seed, p + "b2", d, d, 16.0, 32.0)
        rp["w_b3"], rp["b_b3"], _, _ = gemm_params(seed, p + "b3", 4, d, 16.0, 1.0)
        rp["m_d"] = _mult(seed, p + "d.m")
        rp["s_d"] = _shift_for(16.0 * 73.3 * math.sqrt(d), 256.0)
        rp["m_ref"], rp["s_ref"] = 1 << 30, 30
        rp["box_I0"] = 1024
        rp["m_in"], rp["s_in"] = _mult(seed, p + "in.m"), _shift_for(2048.0, 32.0)
        assert acc_std > 0
        out.append(rp)
    return out


def anchor_logits(levels=((80, 80), (40, 40), (20, 20)), scale: float = 1024.0) -> np.ndarray:
    """Anchor boxes of every memory token as int16 logits at scale 1/`scale`: token (y, x) of
    level l has cx = (x + 0.5) / W_l, cy = (y + 0.5) / H_l, w = h = 0.05 * 2^l; logit(p) =
    log(p / (1 - p)), rounded half away from zero and clipped to int16 (host-side input
    preparation, as the projector's anchors are fixed per resolution)."""
    rows = []
    for l, (H, W) in enumerate(levels):
        ys, xs = np.meshgrid(np.arange(H), np.arange(W), indexing="ij")
        cx = (xs.reshape(-1) + 0.5) / W
        cy = (ys.reshape(-1) + 0.5) / H
        wh = np.full(H * W, 0.05 * 2.0 ** l)
        rows.append(np.stack([cx, cy, wh, wh], axis=1))
    pr = np.concatenate(rows, axis=0)
    lg = np.log(pr / (1.0 - pr)) * scale
    lg = np.sign(lg) * np.floor(np.abs(lg) + 0.5)
    return np.clip(lg, -32767, 32767).astype(np.int16)


def two_stage_params(seed: int, d: int = 256, C: int = 80, levels=((80, 80), (40, 40), (20, 20)),
                     sigma_in: float = 40.0, k_inter: int = 8) -> dict:
    """Integer parameters of the two-stage query selection: encoder class linear layer (raw int32
    logits), proposal MLP d -> d -> 4 with deltas requantised to the anchor-logit scale 2^-10, the
    anchors (``anchor_logits``) and the sigmoid constants of the reference boxes."""
    p = "TS."
    tp: dict = {"k_inter": k_inter, "ref_I0": 1024}
    tp["w_enc"], tp["b_enc"], _, _ = gemm_params(seed, p + "enc", C, d, sigma_in, 1.0)
    tp["w_p1"], tp["b_p1"], tp["m_p1"], tp["s_p1"] = gemm_params(seed, p + "p1", d, d, sigma_in, 32.0)
    tp["w_p2"], tp["b_p2"], _, _ = gemm_params(seed, p + "p2", 4, d, 16.0, 1.0)
    tp["m_d"] = _mult(seed, p + "d.m")
    tp["s_d"] = _shift_for(16.0 * 73.3 * math.sqrt(d), 256.0)
    tp["anchor16"] = anchor_logits(levels)
    tp["m_a"], tp["s_a"] = 1 << 30, 30
    return tp


def query_pos_params(seed: int, d: int = 256, hidden: int = 256, sigma_pos: float = 2048.0) -> dict:
    """Integer parameters of the learnable positional-query projection (Sec. 3.1.2: linear layers
    on the reference-box coordinates in place of the sinusoidal encoding): the Q16 box (cx, cy, w,
    h) requantised to int8 (box / 512, in [0, 128]), a linear layer 4 -> hidden with ReLU on its
    int8 outputs (std ~32), a linear layer hidden -> d to the decoder's int16 positional query
    (std ~sigma_pos)."""
    p = "QP."
    pq: dict = {"m_box": 1 << 30, "s_box": 39}
    pq["w_q1"], pq["b_q1"], pq["m_q1"], pq["s_q1"] = gemm_params(seed, p + "q1", hidden, 4, 40.0, 32.0)
    pq["w_q2"], pq["b_q2"], pq["m_q2"], pq["s_q2"] = gemm_params(seed, p + "q2", d, hidden, 16.0, sigma_pos)
    return pq
