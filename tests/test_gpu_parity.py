"""Bit-exact parity of every CUDA entry point with the CPU oracle, element by element, on seeded
inputs that span several tiles plus ragged tails, and on the edge cases of each operator.
The whole path is integer, so the tolerance is zero everywhere."""
import numpy as np
import pytest

from paper_2607_24981_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def ilw():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_24981_gb300 as m
    from paper_2607_24981_gb300 import build

    build.build()
    m.lib()
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def assert_same(got, want, what=""):
    got = np.asarray(got)
    want = np.asarray(want).astype(got.dtype)
    if not np.array_equal(got, want):
        bad = np.argwhere(got != want)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} mismatches, first at {i}: gpu={got[i]} oracle={want[i]}")


# ------------------------------------------------------------------------------ GEMM
@pytest.mark.parametrize("M,N,K", [(1, 1, 16), (37, 29, 64), (130, 200, 384), (257, 129, 80),
                                   (300, 1152, 384), (128, 384, 1536)])
@pytest.mark.parametrize("out_bits,mode", [(8, "calibrated"), (8, "literal"), (16, "calibrated"), (32, "literal"),
                                           (108, "calibrated")])
def test_gemm_requant(ilw, orc, M, N, K, out_bits, mode):
    """out_bits 108 (ILW_I8_IN_F16): the out_bits 8 result carried as float16."""
    A = synth.uniform_int(1, f"A{M}{K}", (M, K), -127, 127, np.int8)
    W, b, m, s = synth.gemm_params(1, f"W{N}{K}", N, K, 73.0, 40.0, mode)
    Wp = ilw.pack_weight(dev(W))
    got = ilw.gemm_requant(dev(A), Wp, N, dev(b), dev(m), dev(s), out_bits)
    want = orc.gemm_requant(A, W, b, m, s, 8 if out_bits == ilw.I8_IN_F16 else out_bits)
    if out_bits == ilw.I8_IN_F16:
        assert got.dtype == torch.float16
    assert_same(host(got), want, "gemm")


def test_gemm_extremes_and_residual(ilw, orc):
    """All-(+127) and all-(-127) operands reach the largest accumulators; the residual term
    broadcasts rows (row % rows) as the patch embedding's position term does."""
    M, N, K = 200, 96, 1536
    A = np.full((M, K), 127, np.int8)
    A[::2] = -127
    W = np.full((N, K), 127, np.int8)
    W[:, ::3] = -127
    _, b, m, s = synth.gemm_params(2, "Wx", N, K, 73.0, 40.0, "literal")
    res = synth.uniform_int(2, "res", (50, N), -32767, 32767, np.int16)
    Wp = ilw.pack_weight(dev(W))
    got = ilw.gemm_requant(dev(A), Wp, N, dev(b), dev(m), dev(s), 16, res=dev(res), m_r=3 << 29, s_r=31)
    want = orc.gemm_requant(A, W, b, m, s, 16, res, 3 << 29, 31)
    assert_same(host(got), want, "gemm+res")
    got32 = ilw.gemm_requant(dev(A), Wp, N, dev(b), None, None, 32)
    assert_same(host(got32), orc.gemm_requant(A, W, b, m, s, 32), "gemm raw")


@pytest.mark.parametrize("M,N,K,I0", [(100, 96, 64, 300), (513, 768, 192, 1 << 10), (64, 1536, 384, 2047)])
def test_gemm_gelu(ilw, orc, M, N, K, I0):
    A = synth.uniform_int(3, "Ag", (M, K), -127, 127, np.int8)
    W, b, m, s = synth.gemm_params(3, "Wg", N, K, 73.0, 2.0 * I0, "calibrated")
    Wp = ilw.pack_weight(dev(W))
    m_g, s_g = 3 << 29, 40
    got = ilw.gemm_gelu(dev(A), Wp, N, dev(b), dev(m), dev(s), {"I0": I0}, m_g, s_g)
    g = orc.gemm_requant(A, W, b, m, s, 16)
    gi = orc.sdshiftgelu(g, I0).astype(np.int64)
    want = np.array([[orc.sat(orc.rq(int(v), m_g, s_g), 8) for v in row] for row in gi], np.int8)
    assert_same(host(got), want, "gemm_gelu")


# fp16-carried int8 A (ilwdetr_gemm a_form ILW_I8_IN_F16): resident-weight tiles of 192 (N % 192 == 0)
# and 128 columns, streamed weights for K > 1024, ragged M / N, every epilogue form
@pytest.mark.parametrize("M,N,K", [(1, 1, 16), (37, 29, 64), (300, 1152, 384), (257, 384, 1024), (130, 200, 384),
                                   (128, 96, 256), (12800, 1536, 384), (333, 384, 1536), (64, 192, 1040)])
@pytest.mark.parametrize("kind", ["rq8", "rq16res", "f16", "raw32", "gelu8", "gelu_f16"])
def test_gemm_f16_operand(ilw, orc, M, N, K, kind):
    if M * N * K > 1e9 and kind not in ("f16", "gelu_f16", "rq16res"):
        pytest.skip("the large case runs the encoder's forms only")
    A = synth.uniform_int(11, f"Af{M}{K}", (M, K), -127, 127, np.int8)
    I0 = 700
    W, b, m, s = synth.gemm_params(11, f"Wf{N}{K}", N, K, 73.0, 2.0 * I0 if kind.startswith("gelu") else 40.0)
    Wp = ilw.pack_weight(dev(W))
    Ad = dev(A.astype(np.float16))
    F16 = ilw.I8_IN_F16
    if kind.startswith("gelu"):
        m_g, s_g = 3 << 29, 40
        got = ilw.gemm(Ad, Wp, N, dev(b), dev(m), dev(s), F16 if kind == "gelu_f16" else 8, gelu={"I0": I0},
                       m_g=m_g, s_g=s_g)
        gi = orc.sdshiftgelu(orc.gemm_requant(A, W, b, m, s, 16), I0).astype(np.int64)
        want = np.array([[orc.sat(orc.rq(int(v), m_g, s_g), 8) for v in row] for row in gi], np.int8) \
            if M * N <= 1 << 20 else orc.requant(gi.astype(np.int32), m_g, s_g, out_bits=8)
    elif kind == "rq16res":
        res = synth.uniform_int(12, "resf", (M, N), -32767, 32767, np.int16)
        got = ilw.gemm(Ad, Wp, N, dev(b), dev(m), dev(s), 16, res=dev(res), m_r=3 << 29, s_r=31)
        want = orc.gemm_requant(A, W, b, m, s, 16, res, 3 << 29, 31)
    else:
        ob = {"rq8": 8, "f16": F16, "raw32": 32}[kind]
        got = ilw.gemm(Ad, Wp, N, dev(b), dev(m), dev(s), ob)
        want = orc.gemm_requant(A, W, b, m, s, 8 if ob == F16 else ob)
    if kind in ("f16", "gelu_f16"):
        assert got.dtype == torch.float16
    assert_same(host(got), want, f"gemm fp16-A {kind}")


# ------------------------------------------------------------------------------ Shiftmax rows
@pytest.mark.parametrize("L", [1, 3, 4, 63, 64, 65, 128, 400, 1600, 1664, 2048, 2100])
def test_shiftmax_rows(ilw, orc, L):
    rows = 257
    X = synth.uniform_int(4, f"smx{L}", (rows, L), -(1 << 15), 1 << 15)
    for I0, sd in ((1 << 11, -1), (1 << 13, -1), (3000, 0), (5000, 7)):
        got = ilw.shiftmax_rows(dev(X), {"I0": I0, "s_d": sd})
        P, *_ = orc.shiftmax_rows(X, I0, s_d=sd)
        assert_same(host(got), P, f"shiftmax L={L} I0={I0} s_d={sd}")


def test_shiftmax_rows_edge_values(ilw, orc):
    """Full-int32 scores (differences far below the ShiftExp clamp), constant rows, a strided
    (non-contiguous) layout and the largest I0."""
    X = synth.uniform_int(5, "smxe", (64, 100), -(1 << 31), (1 << 31) - 1)
    X[3] = 7
    X[4, ::2] = 2**31 - 1
    X[4, 1::2] = -(2**31)
    for I0 in (1, 2, (1 << 15) - 1):
        got = ilw.shiftmax_rows(dev(X), {"I0": I0})
        assert_same(host(got), orc.shiftmax_rows(X, I0)[0], f"edge I0={I0}")
    Xs = dev(synth.uniform_int(5, "smxs", (40, 130), -5000, 5000))
    sub = Xs[:, 3:124]  # ld 130, len 121, unaligned start
    got = ilw.shiftmax_rows(sub, {"I0": 999})
    assert_same(host(got), orc.shiftmax_rows(host(sub), 999)[0], "strided")


# ------------------------------------------------------------------------------ SD-ShiftGELU
@pytest.mark.parametrize("I0", [1, 7, 256, 1 << 10, 2047, (1 << 14) - 1])
def test_sdshiftgelu_all_int16(ilw, orc, I0):
    """Every int16 value (covers every int8 value), plus large-magnitude values."""
    x = np.arange(-(1 << 15), 1 << 15, dtype=np.int32)
    x = np.concatenate([x, np.array([1 << 23, -(1 << 23), (1 << 24) - 1, -(1 << 24) + 1, 3], np.int32)])
    got = ilw.sdshiftgelu(dev(x), {"I0": I0})
    assert_same(host(got), orc.sdshiftgelu(x, I0), f"gelu I0={I0}")


@pytest.mark.parametrize("I0", [1, 300, 1 << 10, 2047, 4000])
def test_sdshiftgelu_large_input(ilw, orc, I0):
    """Large inputs take the tabulated path (I_div(x) in shared memory for |x| <= T, constant
    beyond): every int16 value four times over, plus magnitudes far past the table's range."""
    x = np.tile(np.arange(-(1 << 15), 1 << 15, dtype=np.int32), 4)
    x = np.concatenate([x, np.array([1 << 20, -(1 << 20), (1 << 24) - 1, -(1 << 24) + 1, 40000, -40000], np.int32)])
    x = np.concatenate([x, np.zeros((-len(x)) % 4, np.int32)])
    got = ilw.sdshiftgelu(dev(x), {"I0": I0})
    assert_same(host(got), orc.sdshiftgelu(x, I0), f"gelu table I0={I0}")


def test_sdshiftgelu_unaligned_tail(ilw, orc):
    x = synth.uniform_int(6, "gt", (1003,), -4096, 4096)
    xd = dev(np.concatenate([np.zeros(1, np.int32), x]))[1:]  # 4-byte but not 16-byte aligned
    got = ilw.sdshiftgelu(xd, {"I0": 500})
    assert_same(host(got), orc.sdshiftgelu(x, 500), "gelu tail")


# ------------------------------------------------------------------------------ I-LayerNorm
@pytest.mark.parametrize("C", [1, 7, 64, 192, 384, 500, 1000, 4096])
@pytest.mark.parametrize("in_bits,out_bits,iters", [(16, 8, 10), (32, 8, 10), (32, 16, 20), (16, 16, 20)])
def test_int_layernorm(ilw, orc, C, in_bits, out_bits, iters):
    rows = 77
    lim = (1 << 14) if in_bits == 32 else 32767
    X = synth.uniform_int(7, f"ln{C}", (rows, C), -lim, lim, np.int32 if in_bits == 32 else np.int16)
    X[5] = 123  # constant row: V = 0
    X[6, :] = 0
    X[6, 0] = lim  # one dominant element
    beta, mult, shift = synth.ln_params(7, f"lnp{C}", C)
    if out_bits == 16:
        shift = shift - 7
    got = ilw.int_layernorm(dev(X), dev(beta), dev(mult), dev(shift), iters, out_bits)
    want = orc.int_layernorm(X, beta, mult, shift, iters, out_bits)
    assert_same(host(got), want, f"ln C={C}")


@pytest.mark.parametrize("C,in_bits", [(384, 16), (192, 32), (100, 16), (1000, 32)])
def test_int_layernorm_f16_out(ilw, orc, C, in_bits):
    """out_bits ILW_I8_IN_F16: the int8 outputs carried in float16 (the encoder's form)."""
    rows = 1000
    lim = (1 << 14) if in_bits == 32 else 32767
    X = synth.uniform_int(9, f"lnf{C}", (rows, C), -lim, lim, np.int32 if in_bits == 32 else np.int16)
    beta, mult, shift = synth.ln_params(9, f"lnpf{C}", C)
    got = ilw.int_layernorm(dev(X), dev(beta), dev(mult), dev(shift), 10, ilw.I8_IN_F16)
    assert got.dtype == torch.float16
    assert_same(host(got), orc.int_layernorm(X, beta, mult, shift, 10, 8), f"ln f16 C={C}")


# ------------------------------------------------------------------------------ attention
@pytest.mark.parametrize("B,T,H,dh,win", [(1, 17, 1, 64, 0), (2, 64, 2, 64, 0), (1, 256, 3, 64, 0),
                                          (1, 300, 2, 32, 0), (2, 100, 2, 64, 2), (1, 1600, 1, 64, 2),
                                          (1, 144, 2, 32, 3), (1, 400, 1, 64, 0)])
@pytest.mark.parametrize("form", ["int8", "f16"])
def test_attention(ilw, orc, B, T, H, dh, win, form):
    """form f16: q|k|v handed over as float16 holding the int8 values (ILW_I8_IN_F16)."""
    d = H * dh
    qkv = synth.uniform_int(8, f"qkv{T}{dh}", (B * T, 3 * d), -127, 127, np.int8)
    q_dev = dev(qkv) if form == "int8" else dev(qkv.astype(np.float16))
    for I0, sd in ((1 << 13, -1), (1 << 12, -1), (20000, 3)):
        smx = {"I0": I0, "k_inter": 16, "k_out": 8, "s_d": sd, "m_p": 4, "M_hw": 31}
        got = ilw.shiftmax_attn(q_dev, B, T, H, dh, win, smx, 3 << 29, 36)
        want = orc.attention(qkv, B, T, H, dh, win, smx, 3 << 29, 36)
        assert_same(host(got), want, f"attn T={T} win={win} I0={I0} {form}")


@pytest.mark.parametrize("B,T,H,dh,win", [(2, 1600, 2, 64, 0), (2, 1600, 2, 64, 2), (1, 300, 8, 32, 0)])
def test_attention_f16_output(ilw, orc, B, T, H, dh, win):
    """o_form ILW_I8_IN_F16 with float16 q|k|v: the encoder block's launch form."""
    d = H * dh
    qkv = synth.uniform_int(13, f"qkvo{T}{dh}", (B * T, 3 * d), -127, 127, np.int8)
    smx = {"I0": 6000, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
    got = ilw.shiftmax_attn(dev(qkv.astype(np.float16)), B, T, H, dh, win, smx, 3 << 29, 36, o_f16=True)
    assert got.dtype == torch.float16
    assert_same(host(got), orc.attention(qkv, B, T, H, dh, win, smx, 3 << 29, 36), f"attn f16 out T={T}")


@pytest.mark.parametrize("B,T,H,dh,win", [(1, 128, 2, 64, 0), (1, 129, 1, 64, 0), (2, 257, 2, 64, 0),
                                          (1, 130, 8, 64, 0), (3, 900, 3, 64, 0), (1, 196, 1, 64, 2),
                                          (1, 1296, 1, 64, 3), (2, 6400, 1, 64, 2)])
@pytest.mark.parametrize("o_f16", [False, True])
def test_attention_tensor_memory_shapes(ilw, orc, B, T, H, dh, win, o_f16):
    """Shapes at the tensor-memory kernel's block edges with fp16-carried q|k|v: a group of exactly
    one query tile, one query past it (a tile whose warps but one have no query), several images,
    8 heads, window sides 7 (one key block of 49), 12 (two blocks of 120 keys) and 40 (14 blocks;
    the last key box reaches past the window and, for the last image, past the matrix).  Global
    groups whose last tile has at most 64 queries put two (image, head) units' last tiles in one
    CTA: T = 129, 257, 130 and 900 run that form, 3 x 3 units at T = 900 with pairs that span two
    images and a last CTA with one unit."""
    d = H * dh
    qkv = synth.uniform_int(14, f"qkvtc{T}{H}{win}", (B * T, 3 * d), -127, 127, np.int8)
    smx = {"I0": 5000, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
    got = ilw.shiftmax_attn(dev(qkv.astype(np.float16)), B, T, H, dh, win, smx, 3 << 29, 36, o_f16=o_f16)
    want = orc.attention(qkv, B, T, H, dh, win, smx, 3 << 29, 36)
    assert_same(host(got), want, f"attn tc T={T} win={win} o_f16={o_f16}")


@pytest.mark.parametrize("I0", [1, 16, 200])
def test_attention_small_sums(ilw, orc, I0):
    """Small I0 gives row sums below 2^23, so F >= 2^(sh0) for some rows and the tensor-memory
    kernel's pass 3 takes the P form without the high-word product (every warp whose rows all allow
    it takes the other); global and windowed, fp16-carried q|k|v."""
    for B, T, H, win in ((1, 300, 2, 0), (1, 400, 1, 2)):
        d = H * 64
        qkv = synth.uniform_int(15, f"qkvsm{T}{I0}", (B * T, 3 * d), -40, 40, np.int8)
        smx = {"I0": I0, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
        got = ilw.shiftmax_attn(dev(qkv.astype(np.float16)), B, T, H, 64, win, smx, 3 << 29, 36)
        assert_same(host(got), orc.attention(qkv, B, T, H, 64, win, smx, 3 << 29, 36), f"attn small I0={I0} T={T}")


def test_attention_extreme_scores(ilw, orc):
    """All q, k = +127 (largest scores, every row uniform) and alternating signs."""
    B, T, H, dh = 1, 130, 2, 64
    d = H * dh
    qkv = np.full((B * T, 3 * d), 127, np.int8)
    qkv[::2, d:2 * d] = -127
    smx = {"I0": 1 << 14, "k_inter": 16, "k_out": 8, "s_d": -1, "m_p": 4, "M_hw": 31}
    got = ilw.shiftmax_attn(dev(qkv), B, T, H, dh, 0, smx, 1 << 30, 33)
    assert_same(host(got), orc.attention(qkv, B, T, H, dh, 0, smx, 1 << 30, 33), "attn extreme")


# ------------------------------------------------------------------------------ split conv
def test_split_conv(ilw, orc):
    M, N, Ks = 333, 256, (384, 384, 384, 384)
    Xs = [synth.uniform_int(9, f"sx{i}", (M, k), -127, 127, np.int8) for i, k in enumerate(Ks)]
    Ws = [synth.uniform_int(9, f"sw{i}", (N, k), -127, 127, np.int8) for i, k in enumerate(Ks)]
    bias = synth.uniform_int(9, "sb", (N,), -(1 << 15), 1 << 15)
    mult = synth.uniform_int(9, "sm", (N,), 1 << 30, (1 << 31) - 1)
    shift = np.full(N, 40, np.int32)
    m_b = [1 << 30, 3 << 28, 1 << 29, 1 << 30]
    s_b = [30, 31, 31, 32]
    got = ilw.split_conv([dev(x) for x in Xs], [ilw.pack_weight(dev(w)) for w in Ws], N, m_b, s_b,
                         dev(bias), dev(mult), dev(shift))
    want = orc.split_conv(Xs, Ws, m_b, s_b, bias, mult, shift)
    assert_same(host(got), want, "split conv")


# ------------------------------------------------------------------------------ deformable sampling
def test_deform_attn(ilw, orc):
    B, Q, H, L, P, dh = 2, 300, 8, 3, 4, 32
    hw = [(80, 80), (40, 40), (20, 20)]
    S = sum(h * w for h, w in hw)
    value = synth.uniform_int(10, "dv", (B, S, H * dh), -127, 127, np.int8)
    ref = synth.uniform_int(10, "dr", (B, Q, 2), 0, 65535)
    off = synth.uniform_int(10, "do", (B, Q, H, L, P, 2), -(8 << 8), 8 << 8)
    off[0, 0] = -(1 << 20)  # every sample of one query far outside
    w = synth.uniform_int(10, "dw", (B, Q, H, L * P), 0, 40, np.uint8)
    got = ilw.deform_attn(dev(value), hw, dev(ref), dev(off), dev(w), 3 << 29, 36)
    want = orc.deform_attn(value, hw, ref, off, w, 3 << 29, 36)
    assert_same(host(got), want, "deform")


# ------------------------------------------------------------------------------ block
@pytest.mark.parametrize("cfg", ["block256_literal", "block256_calibrated", "small_window"])
def test_block_forward(ilw, orc, cfg):
    if cfg.startswith("block256"):
        B, T, d, H, F, win, mode = 1, 256, 192, 3, 768, 0, cfg.split("_")[1]
    else:
        B, T, d, H, F, win, mode = 2, 400, 128, 2, 256, 2, "calibrated"
    bp = synth.block_params(0, 0, d, H, F, win, mode)
    x = synth.block_input(0, B, T, d)
    bw = ilw.BlockWeights(bp)
    ws = torch.empty(ilw.block_workspace_bytes(B, T, d, F), dtype=torch.uint8, device="cuda")
    y = ilw.block_forward(bw, dev(x), B, T, ws)
    y_ref, taps = orc.block_forward(bp, x, B, T, taps=True)
    assert_same(host(y), y_ref, f"block {cfg}")
    # every intermediate, through the op-level entry points
    t = bw.t
    a1 = ilw.int_layernorm(dev(x), t["ln1_beta"], t["ln1_mult"], t["ln1_shift"], 10, 8)
    assert_same(host(a1), taps["a1"], "a1")
    qkv = ilw.gemm_requant(a1, t["w_qkv_p"], 3 * d, t["b_qkv"], t["m_qkv"], t["s_qkv"], 8)
    assert_same(host(qkv), taps["qkv"], "qkv")
    o = ilw.shiftmax_attn(qkv, B, T, H, d // H, win, bp["smx"], bp["m_o"], bp["s_o"])
    assert_same(host(o), taps["o"], "attention")
    x1 = ilw.gemm_requant(o, t["w_proj_p"], d, t["b_proj"], t["m_proj"], t["s_proj"], 16, res=dev(x),
                          m_r=bp["m_r1"], s_r=bp["s_r1"])
    assert_same(host(x1), taps["x1"], "x1")
    a2 = ilw.int_layernorm(x1, t["ln2_beta"], t["ln2_mult"], t["ln2_shift"], 10, 8)
    assert_same(host(a2), taps["a2"], "a2")
    h = ilw.gemm_gelu(a2, t["w_fc1_p"], F, t["b_fc1"], t["m_fc1"], t["s_fc1"],
                      {"I0": bp["gelu_I0"]}, bp["m_g"], bp["s_g"])
    assert_same(host(h), taps["h"], "h")
    y2 = ilw.gemm_requant(h, t["w_fc2_p"], d, t["b_fc2"], t["m_fc2"], t["s_fc2"], 16, res=x1,
                          m_r=bp["m_r2"], s_r=bp["s_r2"])
    assert_same(host(y2), y_ref, "y via ops")
    ilw.device_status()
