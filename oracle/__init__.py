"""Python access to the plain CPU oracle (``oracle/ilw_oracle.cpp``).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline / reference arm may import this package.  It never imports the product package
and the product package never imports it.

Every function takes and returns numpy arrays; the integer semantics are those of the C++
oracle (see ``ilw_oracle.h``): Algorithm 1 (ShiftExp, SD-ShiftGELU), Algorithm 2
(CalibrateShift, Constrained Shiftmax), Sec. 3.2 (integer linear layers, split convolution),
Sec. 3.3 (I-LayerNorm) and Sec. 3.1.1 (nearest-neighbour deformable sampling).

Parity status of the compositions written here in Python from the pinned C++ operators:
``projector``, ``decoder_layer``, ``detection_head``, ``refine_references``, ``decoder_stack``,
``two_stage`` and ``query_pos`` follow a reading of the paper, which does not state their
structure; tests/test_oracle_pins.py pins them by reductions to closed forms (the decoder layer
with constant branches, uniform self-attention scores, or one sampling point at pixel centres; the
projector with identity scales; the head and the refinement with a zero last box layer; the
plain 4-column query projection) and by invariants (query-permutation equivariance, image
independence, selection of the best tokens, row-wise application).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ilw_oracle.cpp")
_LIB_PATH = os.path.join(_HERE, "libilw_oracle.so")
_lib = None

i8p = C.POINTER(C.c_int8)
u8p = C.POINTER(C.c_uint8)
i16p = C.POINTER(C.c_int16)
i32p = C.POINTER(C.c_int32)
i64p = C.POINTER(C.c_int64)


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (C++20, -O2) into ``oracle/libilw_oracle.so``."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "ilw_oracle.h"))
    ):
        tmp = _LIB_PATH + ".tmp%d" % os.getpid()
        subprocess.check_call(
            ["g++", "-std=c++20", "-O2", "-fPIC", "-shared", "-Wall", "-o", tmp, _SRC]
        )
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class ShiftmaxParams(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("I0", "k_inter", "k_out", "s_d", "m_p", "M_hw")]


class BlockParams(C.Structure):
    _fields_ = [
        ("d", C.c_int32), ("H", C.c_int32), ("F", C.c_int32), ("win_side", C.c_int32),
        ("ln_iters", C.c_int32),
        ("ln1_beta", i32p), ("ln1_mult", i32p), ("ln1_shift", i32p),
        ("ln2_beta", i32p), ("ln2_mult", i32p), ("ln2_shift", i32p),
        ("w_qkv", i8p), ("b_qkv", i32p), ("m_qkv", i32p), ("s_qkv", i32p),
        ("smx", ShiftmaxParams),
        ("m_o", C.c_int32), ("s_o", C.c_int32),
        ("w_proj", i8p), ("b_proj", i32p), ("m_proj", i32p), ("s_proj", i32p),
        ("m_r1", C.c_int32), ("s_r1", C.c_int32),
        ("w_fc1", i8p), ("b_fc1", i32p), ("m_fc1", i32p), ("s_fc1", i32p),
        ("gelu_I0", C.c_int32), ("gelu_k_inter", C.c_int32), ("gelu_k_out", C.c_int32),
        ("m_g", C.c_int32), ("s_g", C.c_int32),
        ("w_fc2", i8p), ("b_fc2", i32p), ("m_fc2", i32p), ("s_fc2", i32p),
        ("m_r2", C.c_int32), ("s_r2", C.c_int32),
    ]


class BlockTaps(C.Structure):
    _fields_ = [("a1", i8p), ("qkv", i8p), ("o", i8p), ("x1", i16p), ("a2", i8p),
                ("g", i16p), ("h", i8p)]


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(_LIB_PATH)
        L.orc_rq.restype = C.c_int64
        L.orc_rq.argtypes = [C.c_int64, C.c_int32, C.c_int32]
        L.orc_sat.restype = C.c_int64
        L.orc_sat.argtypes = [C.c_int64, C.c_int32]
        L.orc_shiftexp.restype = C.c_int64
        L.orc_shiftexp.argtypes = [C.c_int64, C.c_int64, C.c_int32]
        L.orc_calibrate_shift.restype = C.c_int32
        L.orc_calibrate_shift.argtypes = [C.c_int64, C.c_int32, C.c_int32]
        L.orc_sdshiftgelu_idiv.restype = C.c_int64
        L.orc_sdshiftgelu_idiv.argtypes = [C.c_int64, C.c_int32, C.c_int32, C.c_int32]
        L.orc_newton_isqrt.restype = C.c_int64
        L.orc_newton_isqrt.argtypes = [C.c_int64, C.c_int32]
        L.orc_shiftexp_vec.restype = None
        L.orc_shiftexp_vec.argtypes = [i32p, C.c_int64, C.c_int32, C.c_int32, i64p]
        L.orc_shiftmax_rows.restype = C.c_int
        L.orc_shiftmax_rows.argtypes = [i32p, C.c_int64, C.c_int64, C.c_int64,
                                        C.POINTER(ShiftmaxParams), u8p, C.c_int64, i64p, i32p, i64p]
        L.orc_sdshiftgelu.restype = C.c_int
        L.orc_sdshiftgelu.argtypes = [i32p, i32p, C.c_int64, C.c_int32, C.c_int32, C.c_int32]
        L.orc_int_layernorm.restype = C.c_int
        L.orc_int_layernorm.argtypes = [i32p, C.c_int64, C.c_int64, C.c_int64, i32p, i32p, i32p,
                                        C.c_int32, C.c_int32, i32p, C.c_int64]
        L.orc_gemm_requant.restype = C.c_int
        L.orc_gemm_requant.argtypes = [i8p, C.c_int64, i8p, C.c_int64, i32p, i32p, i32p,
                                       C.c_int64, C.c_int64, C.c_int64, C.c_int32,
                                       i16p, C.c_int64, C.c_int64, C.c_int32, C.c_int32,
                                       i32p, C.c_int64]
        L.orc_patch_embed.restype = C.c_int
        L.orc_patch_embed.argtypes = [i8p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int32,
                                      i8p, i32p, i32p, i32p, C.c_int32, i16p, C.c_int32,
                                      C.c_int32, i16p]
        L.orc_attention.restype = C.c_int
        L.orc_attention.argtypes = [i8p, i8p, i8p, C.c_int64, C.c_int32, C.c_int32, C.c_int32,
                                    C.c_int32, C.c_int32, C.POINTER(ShiftmaxParams), C.c_int32,
                                    C.c_int32, i8p, C.c_int64]
        L.orc_block_forward.restype = C.c_int
        L.orc_block_forward.argtypes = [C.POINTER(BlockParams), i16p, i16p, C.c_int32, C.c_int32,
                                        C.POINTER(BlockTaps)]
        L.orc_split_conv.restype = C.c_int
        L.orc_split_conv.argtypes = [C.POINTER(i8p), i64p, C.c_int32, C.c_int64, i32p,
                                     C.POINTER(i8p), i32p, i32p, i32p, i32p, i32p, C.c_int64,
                                     i8p, C.c_int64]
        L.orc_deform_attn.restype = C.c_int
        L.orc_deform_attn.argtypes = [i8p, i32p, C.c_int32, i32p, i32p, u8p, C.c_int32,
                                      C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int64,
                                      C.c_int32, C.c_int32, i8p]
        L.orc_requant.restype = C.c_int
        L.orc_requant.argtypes = [i32p, C.c_int64, C.c_int64, C.c_int64, C.c_int32, C.c_int32,
                                  i32p, C.c_int64, C.c_int64, C.c_int32, C.c_int32, C.c_int32,
                                  i32p, C.c_int64]
        L.orc_resample_nearest.restype = C.c_int
        L.orc_resample_nearest.argtypes = [i8p, C.c_int64, C.c_int32, C.c_int32, C.c_int32,
                                           C.c_int32, i8p, C.c_int64, C.c_int32, C.c_int32]
        L.orc_int_sigmoid1.restype = C.c_int64
        L.orc_int_sigmoid1.argtypes = [C.c_int64, C.c_int32, C.c_int32, C.c_int32]
        L.orc_int_sigmoid.restype = C.c_int
        L.orc_int_sigmoid.argtypes = [i32p, i32p, C.c_int64, C.c_int32, C.c_int32, C.c_int32]
        L.orc_topk.restype = C.c_int
        L.orc_topk.argtypes = [i32p, C.c_int64, C.c_int32, C.c_int32, C.c_int32, i32p, i32p]
        L.orc_ivit_shiftgelu.restype = C.c_int
        L.orc_ivit_shiftgelu.argtypes = [i32p, C.c_int64, C.c_int64, C.c_int64, C.c_int32, C.c_int32,
                                         C.c_int32, i32p, C.c_int64]
        L.orc_gather_rows.restype = C.c_int
        L.orc_gather_rows.argtypes = [u8p, C.c_int64, C.c_int64, i32p, C.c_int64, C.c_int64, u8p,
                                      C.c_int64]
        _lib = L
    return _lib


def _p(a: np.ndarray, ptype):
    assert a.flags["C_CONTIGUOUS"], "oracle wants C-contiguous arrays"
    return a.ctypes.data_as(ptype)


def _check(rc: int, what: str) -> None:
    if rc != 0:
        raise ValueError(f"oracle {what} rejected its arguments (rc={rc})")


# ---------------------------------------------------------------- scalar building blocks
def rq(v: int, m: int, s: int) -> int:
    return int(lib().orc_rq(int(v), int(m), int(s)))


def sat(v: int, bits: int) -> int:
    return int(lib().orc_sat(int(v), int(bits)))


def shiftexp(I: int, I0: int, k_inter: int = 16) -> int:
    return int(lib().orc_shiftexp(int(I), int(I0), int(k_inter)))


def calibrate_shift(S_sum: int, m_p: int = 4, M_hw: int = 31) -> int:
    return int(lib().orc_calibrate_shift(int(S_sum), int(m_p), int(M_hw)))


def sdshiftgelu_idiv(x: int, I0: int, k_inter: int = 16, k_out: int = 8) -> int:
    return int(lib().orc_sdshiftgelu_idiv(int(x), int(I0), int(k_inter), int(k_out)))


def newton_isqrt(V: int, iters: int) -> int:
    return int(lib().orc_newton_isqrt(int(V), int(iters)))


# ---------------------------------------------------------------- tensor operators
def shiftexp_vec(I: np.ndarray, I0: int, k_inter: int = 16) -> np.ndarray:
    I = np.ascontiguousarray(I, dtype=np.int32)
    out = np.empty(I.shape, dtype=np.int64)
    lib().orc_shiftexp_vec(_p(I, i32p), I.size, I0, k_inter, _p(out, i64p))
    return out


def shiftmax_rows(X: np.ndarray, I0: int, k_inter: int = 16, k_out: int = 8, s_d: int = -1,
                  m_p: int = 4, M_hw: int = 31):
    """Constrained Shiftmax (Algorithm 2) on every row of a 2-D int32 array.

    Returns (P u8 [rows, len], S_sum int64 [rows], s_d int32 [rows], S_R int64 [rows])."""
    X = np.ascontiguousarray(X, dtype=np.int32)
    rows, n = X.shape
    P = np.zeros((rows, n), dtype=np.uint8)
    S = np.zeros(rows, dtype=np.int64)
    sd = np.zeros(rows, dtype=np.int32)
    SR = np.zeros(rows, dtype=np.int64)
    prm = ShiftmaxParams(I0, k_inter, k_out, s_d, m_p, M_hw)
    _check(lib().orc_shiftmax_rows(_p(X, i32p), n, rows, n, C.byref(prm), _p(P, u8p), n,
                                   _p(S, i64p), _p(sd, i32p), _p(SR, i64p)), "shiftmax_rows")
    return P, S, sd, SR


def sdshiftgelu(X: np.ndarray, I0: int, k_inter: int = 16, k_out: int = 8) -> np.ndarray:
    """SD-ShiftGELU (Algorithm 1): returns I_out = x * I_div as int32 (scale S_x 2^-(k_out-1))."""
    X = np.ascontiguousarray(X, dtype=np.int32)
    Y = np.empty_like(X)
    _check(lib().orc_sdshiftgelu(_p(X, i32p), _p(Y, i32p), X.size, I0, k_inter, k_out),
           "sdshiftgelu")
    return Y


def int_layernorm(X: np.ndarray, beta, mult, shift, iters: int = 10, out_bits: int = 8):
    """I-LayerNorm over the last axis of a 2-D integer array; returns int32 values."""
    X = np.ascontiguousarray(X, dtype=np.int32)
    rows, Cn = X.shape
    beta = np.ascontiguousarray(beta, dtype=np.int32)
    mult = np.ascontiguousarray(mult, dtype=np.int32)
    shift = np.ascontiguousarray(shift, dtype=np.int32)
    Y = np.empty((rows, Cn), dtype=np.int32)
    _check(lib().orc_int_layernorm(_p(X, i32p), Cn, rows, Cn, _p(beta, i32p), _p(mult, i32p),
                                   _p(shift, i32p), iters, out_bits, _p(Y, i32p), Cn),
           "int_layernorm")
    return Y


def gemm_requant(A: np.ndarray, W: np.ndarray, bias, mult, shift, out_bits: int = 8,
                 res: np.ndarray | None = None, m_r: int = 0, s_r: int = 0) -> np.ndarray:
    """Integer linear layer: A int8 [M,K], W int8 [N,K] -> int32 [M,N] holding the result."""
    A = np.ascontiguousarray(A, dtype=np.int8)
    W = np.ascontiguousarray(W, dtype=np.int8)
    M, K = A.shape
    N = W.shape[0]
    assert W.shape[1] == K
    bias = None if bias is None else np.ascontiguousarray(bias, dtype=np.int32)
    mult = np.ascontiguousarray(mult if mult is not None else np.zeros(N), dtype=np.int32)
    shift = np.ascontiguousarray(shift if shift is not None else np.zeros(N), dtype=np.int32)
    Cm = np.empty((M, N), dtype=np.int32)
    if res is not None:
        res = np.ascontiguousarray(res, dtype=np.int16)
        rp, ldr, rrows = _p(res, i16p), res.shape[1], res.shape[0]
    else:
        rp, ldr, rrows = None, 0, 1
    _check(lib().orc_gemm_requant(_p(A, i8p), K, _p(W, i8p), K,
                                  None if bias is None else _p(bias, i32p), _p(mult, i32p),
                                  _p(shift, i32p), M, N, K, out_bits, rp, ldr, rrows, m_r, s_r,
                                  _p(Cm, i32p), N), "gemm_requant")
    return Cm


def patch_embed(img: np.ndarray, p: int, W: np.ndarray, bias, mult, shift,
                pos: np.ndarray | None = None, m_pos: int = 0, s_pos: int = 0) -> np.ndarray:
    """p x p stride-p integer convolution of int8 img [B, C, H, W] -> int16 [B*T, d]."""
    img = np.ascontiguousarray(img, dtype=np.int8)
    B, Cin, Hh, Ww = img.shape
    W = np.ascontiguousarray(W, dtype=np.int8)
    d = W.shape[0]
    bias = np.ascontiguousarray(bias, dtype=np.int32)
    mult = np.ascontiguousarray(mult, dtype=np.int32)
    shift = np.ascontiguousarray(shift, dtype=np.int32)
    T = (Hh // p) * (Ww // p)
    x0 = np.empty((B * T, d), dtype=np.int16)
    pp = None
    if pos is not None:
        pos = np.ascontiguousarray(pos, dtype=np.int16)
        pp = _p(pos, i16p)
    _check(lib().orc_patch_embed(_p(img, i8p), B, Cin, Hh, Ww, p, _p(W, i8p), _p(bias, i32p),
                                 _p(mult, i32p), _p(shift, i32p), d, pp, m_pos, s_pos,
                                 _p(x0, i16p)), "patch_embed")
    return x0


def attention(qkv: np.ndarray, B: int, T: int, H: int, dh: int, win_side: int, smx: dict,
              m_o: int, s_o: int) -> np.ndarray:
    """Attention over a token-major [B*T, 3*H*dh] int8 q|k|v buffer -> int8 O [B*T, H*dh]."""
    qkv = np.ascontiguousarray(qkv, dtype=np.int8)
    d = H * dh
    ld = qkv.shape[1]
    O = np.zeros((B * T, d), dtype=np.int8)
    prm = ShiftmaxParams(smx["I0"], smx.get("k_inter", 16), smx.get("k_out", 8),
                         smx.get("s_d", -1), smx.get("m_p", 4), smx.get("M_hw", 31))
    base = qkv.ctypes.data
    _check(lib().orc_attention(C.cast(base, i8p), C.cast(base + d, i8p), C.cast(base + 2 * d, i8p),
                               ld, B, T, H, dh, win_side, C.byref(prm), m_o, s_o, _p(O, i8p), d),
           "attention")
    return O


def _block_struct(bp: dict, keep: list) -> BlockParams:
    def arr(name, dt):
        a = np.ascontiguousarray(bp[name], dtype=dt)
        keep.append(a)
        return _p(a, i8p if dt == np.int8 else i32p)

    s = bp["smx"]
    return BlockParams(
        bp["d"], bp["H"], bp["F"], bp["win_side"], bp["ln_iters"],
        arr("ln1_beta", np.int32), arr("ln1_mult", np.int32), arr("ln1_shift", np.int32),
        arr("ln2_beta", np.int32), arr("ln2_mult", np.int32), arr("ln2_shift", np.int32),
        arr("w_qkv", np.int8), arr("b_qkv", np.int32), arr("m_qkv", np.int32), arr("s_qkv", np.int32),
        ShiftmaxParams(s["I0"], s["k_inter"], s["k_out"], s["s_d"], s["m_p"], s["M_hw"]),
        bp["m_o"], bp["s_o"],
        arr("w_proj", np.int8), arr("b_proj", np.int32), arr("m_proj", np.int32), arr("s_proj", np.int32),
        bp["m_r1"], bp["s_r1"],
        arr("w_fc1", np.int8), arr("b_fc1", np.int32), arr("m_fc1", np.int32), arr("s_fc1", np.int32),
        bp["gelu_I0"], bp["gelu_k_inter"], bp["gelu_k_out"], bp["m_g"], bp["s_g"],
        arr("w_fc2", np.int8), arr("b_fc2", np.int32), arr("m_fc2", np.int32), arr("s_fc2", np.int32),
        bp["m_r2"], bp["s_r2"],
    )


def block_forward(bp: dict, x: np.ndarray, B: int, T: int, taps: bool = False):
    """One integer encoder block on int16 x [B*T, d]; returns y (and a dict of taps)."""
    keep: list = []
    st = _block_struct(bp, keep)
    x = np.ascontiguousarray(x, dtype=np.int16)
    y = np.empty_like(x)
    d, F = bp["d"], bp["F"]
    M = B * T
    tp = None
    out = {}
    if taps:
        out = {"a1": np.empty((M, d), np.int8), "qkv": np.empty((M, 3 * d), np.int8),
               "o": np.empty((M, d), np.int8), "x1": np.empty((M, d), np.int16),
               "a2": np.empty((M, d), np.int8), "g": np.empty((M, F), np.int16),
               "h": np.empty((M, F), np.int8)}
        tp = BlockTaps(*[_p(out[k], i16p if out[k].dtype == np.int16 else i8p)
                         for k in ("a1", "qkv", "o", "x1", "a2", "g", "h")])
    _check(lib().orc_block_forward(C.byref(st), _p(x, i16p), _p(y, i16p), B, T,
                                   None if tp is None else C.byref(tp)), "block_forward")
    return (y, out) if taps else y


def split_conv(Xs: list, Ws: list, m_b, s_b, bias, mult, shift) -> np.ndarray:
    """Scale-preserving split convolution (Sec. 3.2.2) over nb branches of int8 [M, K_b]."""
    nb = len(Xs)
    Xs = [np.ascontiguousarray(x, dtype=np.int8) for x in Xs]
    Ws = [np.ascontiguousarray(w, dtype=np.int8) for w in Ws]
    M = Xs[0].shape[0]
    N = Ws[0].shape[0]
    Kb = np.array([x.shape[1] for x in Xs], dtype=np.int32)
    ldx = np.array([x.shape[1] for x in Xs], dtype=np.int64)
    xp = (i8p * nb)(*[_p(x, i8p) for x in Xs])
    wp = (i8p * nb)(*[_p(w, i8p) for w in Ws])
    m_b = np.ascontiguousarray(m_b, dtype=np.int32)
    s_b = np.ascontiguousarray(s_b, dtype=np.int32)
    bias = np.ascontiguousarray(bias, dtype=np.int32)
    mult = np.ascontiguousarray(mult, dtype=np.int32)
    shift = np.ascontiguousarray(shift, dtype=np.int32)
    Y = np.empty((M, N), dtype=np.int8)
    _check(lib().orc_split_conv(xp, _p(ldx, i64p), nb, M, _p(Kb, i32p), wp, _p(m_b, i32p),
                                _p(s_b, i32p), _p(bias, i32p), _p(mult, i32p), _p(shift, i32p),
                                N, _p(Y, i8p), N), "split_conv")
    return Y


def deform_attn(value: np.ndarray, level_hw, ref_q16: np.ndarray, off_q8: np.ndarray,
                w: np.ndarray, m: int, s: int) -> np.ndarray:
    """Nearest-neighbour deformable sampling: value int8 [B, S, H*dh]; ref [B,Q,2];
    off [B,Q,H,L,P,2]; w u8 [B,Q,H,L*P] -> int8 [B, Q, H*dh]."""
    value = np.ascontiguousarray(value, dtype=np.int8)
    lhw = np.ascontiguousarray(level_hw, dtype=np.int32).reshape(-1, 2)
    ref_q16 = np.ascontiguousarray(ref_q16, dtype=np.int32)
    off_q8 = np.ascontiguousarray(off_q8, dtype=np.int32)
    w = np.ascontiguousarray(w, dtype=np.uint8)
    B, S, Dm = value.shape
    _, Q, H, L, P, _ = off_q8.shape
    dh = Dm // H
    out = np.empty((B, Q, Dm), dtype=np.int8)
    _check(lib().orc_deform_attn(_p(value, i8p), _p(lhw, i32p), L, _p(ref_q16, i32p),
                                 _p(off_q8, i32p), _p(w, u8p), B, Q, H, P, dh, S, m, s,
                                 _p(out, i8p)), "deform_attn")
    return out


# ---------------------------------------------------------------- detector: projector, decoder
_OUT_DT = {8: np.int8, 16: np.int16, 32: np.int32}


def requant(X: np.ndarray, m1: int, s1: int, Z: np.ndarray | None = None, m2: int = 0, s2: int = 1,
            out_bits: int = 8) -> np.ndarray:
    """sat_{out_bits}(rq(X; m1, s1) + rq(Z[r mod z_rows]; m2, s2)) elementwise over a 2-D X."""
    X32 = np.ascontiguousarray(X, dtype=np.int32)
    rows, Cn = X32.shape
    Y = np.empty((rows, Cn), dtype=np.int32)
    if Z is not None:
        Z32 = np.ascontiguousarray(Z, dtype=np.int32)
        zp, zr, zl = _p(Z32, i32p), Z32.shape[0], Z32.shape[1]
    else:
        zp, zr, zl = None, 1, Cn
    _check(lib().orc_requant(_p(X32, i32p), Cn, rows, Cn, m1, s1, zp, zl, zr, m2, s2, out_bits,
                             _p(Y, i32p), Cn), "requant")
    return Y.astype(_OUT_DT[out_bits])


def resample_nearest(X: np.ndarray, B: int, Hi: int, Wi: int, Ho: int, Wo: int) -> np.ndarray:
    """B maps [Hi*Wi, C] int8 (stacked as [B*Hi*Wi, C]) -> [B*Ho*Wo, C] by nearest resampling."""
    X = np.ascontiguousarray(X, dtype=np.int8)
    Cn = X.shape[1]
    Y = np.empty((B * Ho * Wo, Cn), dtype=np.int8)
    _check(lib().orc_resample_nearest(_p(X, i8p), Hi * Wi, B, Hi, Wi, Cn, _p(Y, i8p), Ho * Wo, Ho, Wo),
           "resample_nearest")
    return Y


def projector(pp: dict, taps: list, B: int, grid: int, levels) -> np.ndarray:
    """Multi-scale projector (Sec. 3.2.2 split convolution; strides read as nearest resampling):
    each tapped layer x_b (int16 [B*grid*grid, K]) is requantised to int8 with its own scale; per
    level, one split convolution over the branches gives [B*grid*grid, N] int8, resampled by
    nearest neighbour to the level's H_l x W_l (a 1x1 convolution commutes with it); the levels
    are concatenated per image into the decoder memory [B*S, N], S = sum H_l W_l."""
    t = [requant(x, m, s_, out_bits=8) for x, (m, s_) in zip(taps, pp["taps"])]
    outs = []
    for lv, (Hl, Wl) in zip(pp["levels"], levels):
        y = split_conv(t, lv["w"], lv["m_b"], lv["s_b"], lv["b"], lv["m"], lv["s"])
        outs.append(resample_nearest(y, B, grid, grid, Hl, Wl).reshape(B, Hl * Wl, -1))
    return np.concatenate(outs, axis=1).reshape(B * sum(h * w for h, w in levels), -1)


def decoder_layer(dp: dict, tgt: np.ndarray, pos: np.ndarray, memory: np.ndarray, level_hw,
                  refs: np.ndarray, B: int, Q: int) -> np.ndarray:
    """One integer decoder layer (post-norm, Deformable-DETR order), every step one of the pinned
    operators above:
      self-attention: q = k from sat8(rq(tgt) + rq(pos)), v from sat8(rq(tgt)); global
        attention over the Q queries; output projection + residual tgt -> sat16; I-LayerNorm
        (20 Newton steps, int16 out);
      deformable cross-attention: query sat8(rq(t1) + rq(pos)); value = rq8(memory W_val);
        Q8 offsets and logits = rq16 of two linear layers of the query; weights = Constrained
        Shiftmax over the L*P logits of each head; nearest-neighbour sampling; output
        projection + residual t1; I-LayerNorm;
      FFN: sat8(rq(t2)) -> FC1 + SD-ShiftGELU -> FC2 + residual t2; I-LayerNorm."""
    d, H, F, L, P = dp["d"], dp["H"], dp["F"], dp["L"], dp["P"]
    dh = d // H
    M = B * Q
    lhw = np.asarray(level_hw, dtype=np.int32).reshape(-1, 2)
    it = dp["ln_iters"]
    # self-attention
    qk_in = requant(tgt, dp["m_q1"], dp["s_q1"], pos, dp["m_q2"], dp["s_q2"], 8)
    v_in = requant(tgt, dp["m_v1"], dp["s_v1"], out_bits=8)
    qk = gemm_requant(qk_in, dp["w_qk"], dp["b_qk"], dp["m_qk"], dp["s_qk"], 8).astype(np.int8)
    v = gemm_requant(v_in, dp["w_v"], dp["b_v"], dp["m_v"], dp["s_v"], 8).astype(np.int8)
    o = attention(np.concatenate([qk, v], axis=1), B, Q, H, dh, 0, dp["smx"], dp["m_o"], dp["s_o"])
    x1 = gemm_requant(o, dp["w_o"], dp["b_o"], dp["m_oc"], dp["s_oc"], 16, tgt, dp["m_r1"], dp["s_r1"])
    t1 = int_layernorm(x1, dp["ln1_beta"], dp["ln1_mult"], dp["ln1_shift"], it, 16).astype(np.int16)
    # deformable cross-attention
    qc = requant(t1, dp["m_c1"], dp["s_c1"], pos, dp["m_c2"], dp["s_c2"], 8)
    value = gemm_requant(memory, dp["w_val"], dp["b_val"], dp["m_val"], dp["s_val"], 8).astype(np.int8)
    off = gemm_requant(qc, dp["w_off"], dp["b_off"], dp["m_off"], dp["s_off"], 16)
    att = gemm_requant(qc, dp["w_att"], dp["b_att"], dp["m_att"], dp["s_att"], 16)
    sw = dp["smx_w"]
    w, *_ = shiftmax_rows(att.reshape(M * H, L * P), sw["I0"], sw["k_inter"], sw["k_out"], sw["s_d"],
                          sw["m_p"], sw["M_hw"])
    S = memory.shape[0] // B
    samp = deform_attn(value.reshape(B, S, d), lhw, refs, off.reshape(B, Q, H, L, P, 2),
                       w.reshape(B, Q, H, L * P), dp["m_s"], dp["s_s"]).reshape(M, d)
    x2 = gemm_requant(samp, dp["w_o2"], dp["b_o2"], dp["m_o2"], dp["s_o2"], 16, t1, dp["m_r2"], dp["s_r2"])
    t2 = int_layernorm(x2, dp["ln2_beta"], dp["ln2_mult"], dp["ln2_shift"], it, 16).astype(np.int16)
    # FFN
    fin = requant(t2, dp["m_f"], dp["s_f"], out_bits=8)
    g = gemm_requant(fin, dp["w_fc1"], dp["b_fc1"], dp["m_fc1"], dp["s_fc1"], 16)
    gi = sdshiftgelu(g, dp["gelu_I0"], dp["gelu_k_inter"], dp["gelu_k_out"])  # g * I_div(g), int32
    h = requant(gi, dp["m_g"], dp["s_g"], out_bits=8)
    x3 = gemm_requant(h, dp["w_fc2"], dp["b_fc2"], dp["m_fc2"], dp["s_fc2"], 16, t2, dp["m_r3"], dp["s_r3"])
    return int_layernorm(x3, dp["ln3_beta"], dp["ln3_mult"], dp["ln3_shift"], it, 16).astype(np.int16)


# ---------------------------------------------------------------- detection head, two-stage selection
def int_sigmoid1(x: int, I0: int, k_inter: int = 16, k_out: int = 8) -> int:
    return int(lib().orc_int_sigmoid1(int(x), int(I0), int(k_inter), int(k_out)))


def int_sigmoid(X: np.ndarray, I0: int, k_inter: int = 16, k_out: int = 8) -> np.ndarray:
    """Integer sigmoid (Table 5's ShiftExp in the detection head, in SD-ShiftGELU's sign-dependent
    form): int32 logits -> int32 outputs at scale 2^-(k_out-1), same shape."""
    X32 = np.ascontiguousarray(X, dtype=np.int32)
    Y = np.empty_like(X32)
    _check(lib().orc_int_sigmoid(_p(X32, i32p), _p(Y, i32p), X32.size, I0, k_inter, k_out), "int_sigmoid")
    return Y


def topk(S: np.ndarray, K: int):
    """Per row of the 2-D int32 S: the K largest values in decreasing order, equal values by
    increasing index -> (values int32 [rows, K], indices int32 [rows, K])."""
    S32 = np.ascontiguousarray(S, dtype=np.int32)
    rows, N = S32.shape
    vals = np.empty((rows, K), dtype=np.int32)
    idx = np.empty((rows, K), dtype=np.int32)
    _check(lib().orc_topk(_p(S32, i32p), N, rows, N, K, _p(vals, i32p), _p(idx, i32p)), "topk")
    return vals, idx


def gather_rows(X: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Rows idx of the 2-D X (any integer type)."""
    X = np.ascontiguousarray(X)
    idx = np.ascontiguousarray(idx, dtype=np.int32).reshape(-1)
    rb = X.shape[1] * X.itemsize
    Y = np.empty((idx.size, X.shape[1]), dtype=X.dtype)
    _check(lib().orc_gather_rows(X.view(np.uint8).ctypes.data_as(u8p), rb, X.shape[0], _p(idx, i32p),
                                 idx.size, rb, Y.view(np.uint8).ctypes.data_as(u8p), rb), "gather_rows")
    return Y


def relu(X: np.ndarray) -> np.ndarray:
    return np.maximum(X, 0).astype(X.dtype)


def detection_head(hp: dict, out: np.ndarray, ref16: np.ndarray):
    """Detection head on the decoder output (Table 5: QuantLinear and ShiftExp; the box refinement in the logit domain is a reading, as the paper gives no integer inverse sigmoid):
      class scores = IntSigmoid(Linear_cls(out))               (raw int32 logits, k_out = cls_k_out)
      box logits   z = rq(Linear_3(ReLU(Linear_2(ReLU(Linear_1(out))))); m_d, s_d) + rq(ref16; m_ref, s_ref)
      boxes        = IntSigmoid(z) with k_out = 17             (cx, cy, w, h at scale 2^-16)
    ReLU acts on the int8 outputs of the hidden layers.  Returns (scores, boxes, z)."""
    logits = gemm_requant(out, hp["w_cls"], hp["b_cls"], None, None, 32)
    scores = int_sigmoid(logits, hp["cls_I0"], hp["k_inter"], hp["cls_k_out"])
    h1 = relu(gemm_requant(out, hp["w_b1"], hp["b_b1"], hp["m_b1"], hp["s_b1"], 8).astype(np.int8))
    h2 = relu(gemm_requant(h1, hp["w_b2"], hp["b_b2"], hp["m_b2"], hp["s_b2"], 8).astype(np.int8))
    d = gemm_requant(h2, hp["w_b3"], hp["b_b3"], None, None, 32)
    z = requant(d, hp["m_d"], hp["s_d"], ref16, hp["m_ref"], hp["s_ref"], out_bits=32)
    boxes = int_sigmoid(z, hp["box_I0"], hp["k_inter"], 17)
    return scores, boxes, z


def refine_references(rp: dict, t: np.ndarray, ref16: np.ndarray):
    """Box refinement after a decoder layer (the two-stage pipeline's references refined layer by
    layer, Sec. 3.1.2; the head rows of Table 5; the logit-domain update is a reading, as the paper
    gives no integer inverse sigmoid):
      a      = sat8(rq(t; m_in, s_in))                              (decoder output, int16 -> int8)
      d      = Linear_3(ReLU(Linear_2(ReLU(Linear_1(a)))))          (raw int32 deltas)
      ref16' = sat16(rq(d; m_d, s_d) + rq(ref16; m_ref, s_ref))     (new reference logits, scale 2^-10)
      boxes  = IntSigmoid(ref16') with k_out = 17                   (cx, cy, w, h at scale 2^-16)
    Returns (ref16' int16 [M, 4], boxes int32 [M, 4])."""
    a = requant(t, rp["m_in"], rp["s_in"], out_bits=8).astype(np.int8)
    h1 = relu(gemm_requant(a, rp["w_b1"], rp["b_b1"], rp["m_b1"], rp["s_b1"], 8).astype(np.int8))
    h2 = relu(gemm_requant(h1, rp["w_b2"], rp["b_b2"], rp["m_b2"], rp["s_b2"], 8).astype(np.int8))
    d = gemm_requant(h2, rp["w_b3"], rp["b_b3"], None, None, 32)
    ref = requant(d, rp["m_d"], rp["s_d"], ref16, rp["m_ref"], rp["s_ref"], out_bits=16).astype(np.int16)
    boxes = int_sigmoid(ref.astype(np.int32), rp["box_I0"], rp["k_inter"], 17)
    return ref, boxes


def decoder_stack(dps: list, tgt: np.ndarray, memory: np.ndarray, level_hw, ref16: np.ndarray,
                  boxes: np.ndarray, B: int, Q: int, pq: dict | None = None, pos: np.ndarray | None = None,
                  rps: list | None = None):
    """The decoder layers with the references refined between them: layer l samples at the (cx, cy)
    of the current boxes with positional queries from the learnable projection of those boxes (pq),
    or the fixed `pos`; after every layer but the last, the box branch rps[l] gives the next
    references (refine_references).  Without rps the references stay fixed.  Returns (decoder output
    int16 [B*Q, d], the last layer's input reference logits int16 [B*Q, 4])."""
    t = tgt
    for l, dp in enumerate(dps):
        refs = np.ascontiguousarray(boxes[:, :2]).reshape(B, Q, 2).astype(np.int32)
        p = query_pos(pq, boxes) if pq is not None else pos
        t = decoder_layer(dp, t, p, memory, level_hw, refs, B, Q)
        if rps is not None and l + 1 < len(dps):
            ref16, boxes = refine_references(rps[l], t, ref16)
    return t, ref16


def two_stage(tp: dict, memory: np.ndarray, B: int, S: int, K: int):
    """Two-stage query selection (a reading of the two-stage pipeline of Sec. 3.1.2): encoder class logits of every memory token,
    the token's best class logit (top-1 over classes), the K best tokens of each image
    (top-K, ties to the lower index), and their reference-box logits
      ref16 = sat16(rq(Linear_2(ReLU(Linear_1(memory[token]))); m_d, s_d) + rq(anchor16[token]; m_a, s_a))
    and the reference boxes IntSigmoid(ref16) (cx, cy, w, h at scale 2^-16; the decoder samples at
    (cx, cy)).  Returns (values [B, K], token indices [B, K], ref16 [B*K, 4], boxes [B*K, 4])."""
    enc = gemm_requant(memory, tp["w_enc"], tp["b_enc"], None, None, 32)
    best, _ = topk(enc, 1)
    vals, idx = topk(best.reshape(B, S), K)
    rows = (idx + (np.arange(B, dtype=np.int32) * S)[:, None]).reshape(-1)
    sel = gather_rows(memory, rows)
    anc = gather_rows(tp["anchor16"], idx.reshape(-1))
    h1 = relu(gemm_requant(sel, tp["w_p1"], tp["b_p1"], tp["m_p1"], tp["s_p1"], 8).astype(np.int8))
    d = gemm_requant(h1, tp["w_p2"], tp["b_p2"], None, None, 32)
    ref16 = requant(d, tp["m_d"], tp["s_d"], anc, tp["m_a"], tp["s_a"], out_bits=16)
    boxes = int_sigmoid(ref16, tp["ref_I0"], tp["k_inter"], 17)
    return vals, idx, ref16, boxes


def query_pos(pq: dict, boxes: np.ndarray) -> np.ndarray:
    """Learnable positional-query projection (Sec. 3.1.2; the layer sizes and the int8 box input are a reading): int16 query_pos [M, d] =
    sat16(rq(Linear_2(ReLU(sat8(rq(Linear_1(b))))))) with b = sat8(rq(box; m_box, s_box)), the Q16
    box [M, 4] requantised to int8; Linear_1 is a 4 -> hidden layer."""
    b8 = requant(boxes, pq["m_box"], pq["s_box"], out_bits=8).astype(np.int8)
    h = relu(gemm_requant(b8, pq["w_q1"], pq["b_q1"], pq["m_q1"], pq["s_q1"], 8).astype(np.int8))
    return gemm_requant(h, pq["w_q2"], pq["b_q2"], pq["m_q2"], pq["s_q2"], 16).astype(np.int16)


def ivit_shiftgelu(X: np.ndarray, I0: int, k_inter: int = 16, k_out: int = 8) -> np.ndarray:
    """I-ViT's ShiftGELU over the rows of the 2-D int32 X (row-maximum subtraction; Sec. 3.3.1's
    baseline; the row maximum is clamped at 0) -> int32 I_x * I_div."""
    X32 = np.ascontiguousarray(X, dtype=np.int32)
    rows, L = X32.shape
    Y = np.empty_like(X32)
    _check(lib().orc_ivit_shiftgelu(_p(X32, i32p), L, rows, L, I0, k_inter, k_out, _p(Y, i32p), L),
           "ivit_shiftgelu")
    return Y
