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
    "block_c0": dict(B=1, T=256, d=192, H=3, F=768, layers=1, global_layers=(0,), mode="literal",
                     dist="uniform"),
    # Tiny-scale backbone: 6 blocks alternating window (2x2 windows of 400 tokens) / global
    "tiny_c1": dict(B=8, T=1600, d=192, H=3, F=768, layers=6, global_layers=(1, 3, 5),
                    mode="calibrated", dist="uniform"),
    # Medium-scale backbone: 10 blocks, global attention at the output layers 2, 4, 5, 9
    "medium_c2": dict(B=8, T=1600, d=384, H=6, F=1536, layers=10, global_layers=(2, 4, 5, 9),
                      mode="calibrated", dist="laplace"),
}


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
