"""GB300 (sm_103a) integer-only I-LW-DETR forward path.

Python names mirror the C-ABI of ``include/ilwdetr.h`` (``libilwdetr.so`` in this directory).
This module only marshals arguments: torch tensors provide device memory and the current CUDA
stream; every step of the computation runs in the library's CUDA kernels.  There is no CPU
fallback: if the library is missing or cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os

__all__ = [
    "lib", "IlwError", "I8_IN_F16", "version", "pack_weight", "gemm_requant", "gemm_gelu", "gemm", "split_conv",
    "shiftmax_rows", "sdshiftgelu", "int_layernorm", "shiftmax_attn", "deform_attn",
    "BlockWeights", "block_forward", "block_workspace_bytes", "device_status",
    "patch_embed", "patch_embed_workspace_bytes", "Backbone", "Graphed",
    "requant", "resample_nearest", "DecoderWeights", "decoder_workspace_bytes", "decoder_layer_forward",
    "Projector", "Detector", "int_sigmoid", "relu_i8", "topk", "gather_rows", "DetectionHead", "TwoStage",
    "QueryPos", "BoxRefine", "ivit_shiftgelu",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libilwdetr.so")
_lib = None


class IlwError(RuntimeError):
    pass


# ILW_I8_IN_F16: int8-range integers carried as fp16 (an out_bits value of gemm_requant and the
# float16 q|k|v form of shiftmax_attn)
I8_IN_F16 = 108


class ShiftmaxT(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("I0", "k_inter", "k_out", "s_d", "m_p", "M_hw")]


class GeluT(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("I0", "k_inter", "k_out")]


class ResidualT(C.Structure):
    _fields_ = [("x", C.c_void_p), ("ldx", C.c_int64), ("rows", C.c_int64),
                ("mult", C.c_int32), ("shift", C.c_int32)]


class BlockParamsT(C.Structure):
    _fields_ = [
        ("struct_size", C.c_uint32),
        ("d", C.c_int32), ("H", C.c_int32), ("F", C.c_int32), ("win_side", C.c_int32),
        ("ln_iters", C.c_int32),
        ("ln1_beta", C.c_void_p), ("ln1_mult", C.c_void_p), ("ln1_shift", C.c_void_p),
        ("ln2_beta", C.c_void_p), ("ln2_mult", C.c_void_p), ("ln2_shift", C.c_void_p),
        ("w_qkv", C.c_void_p), ("b_qkv", C.c_void_p), ("m_qkv", C.c_void_p), ("s_qkv", C.c_void_p),
        ("smx", ShiftmaxT), ("m_o", C.c_int32), ("s_o", C.c_int32),
        ("w_proj", C.c_void_p), ("b_proj", C.c_void_p), ("m_proj", C.c_void_p), ("s_proj", C.c_void_p),
        ("m_r1", C.c_int32), ("s_r1", C.c_int32),
        ("w_fc1", C.c_void_p), ("b_fc1", C.c_void_p), ("m_fc1", C.c_void_p), ("s_fc1", C.c_void_p),
        ("gelu", GeluT), ("m_g", C.c_int32), ("s_g", C.c_int32),
        ("w_fc2", C.c_void_p), ("b_fc2", C.c_void_p), ("m_fc2", C.c_void_p), ("s_fc2", C.c_void_p),
        ("m_r2", C.c_int32), ("s_r2", C.c_int32),
    ]


class GemmT(C.Structure):
    _fields_ = [("struct_size", C.c_uint32), ("A", C.c_void_p), ("a_form", C.c_int32), ("lda", C.c_int64),
                ("Wp", C.c_void_p), ("bias", C.c_void_p), ("mult", C.c_void_p), ("shift", C.c_void_p),
                ("M", C.c_int32), ("N", C.c_int32), ("K", C.c_int32), ("epilogue", C.c_int32),
                ("out_bits", C.c_int32), ("C", C.c_void_p), ("ldc", C.c_int64),
                ("res", C.POINTER(ResidualT)), ("gelu", C.POINTER(GeluT)), ("m_g", C.c_int32), ("s_g", C.c_int32)]


EPI_REQUANT, EPI_GELU = 0, 1


class SigmoidT(C.Structure):
    _fields_ = [("I0", C.c_int32), ("k_inter", C.c_int32), ("k_out", C.c_int32)]


class DecoderParamsT(C.Structure):
    _fields_ = [
        ("struct_size", C.c_uint32),
        ("d", C.c_int32), ("H", C.c_int32), ("F", C.c_int32), ("L", C.c_int32), ("P", C.c_int32),
        ("ln_iters", C.c_int32),
        ("m_q1", C.c_int32), ("s_q1", C.c_int32), ("m_q2", C.c_int32), ("s_q2", C.c_int32),
        ("m_v1", C.c_int32), ("s_v1", C.c_int32),
        ("w_qk", C.c_void_p), ("b_qk", C.c_void_p), ("m_qk", C.c_void_p), ("s_qk", C.c_void_p),
        ("w_v", C.c_void_p), ("b_v", C.c_void_p), ("m_v", C.c_void_p), ("s_v", C.c_void_p),
        ("smx", ShiftmaxT), ("m_o", C.c_int32), ("s_o", C.c_int32),
        ("w_o", C.c_void_p), ("b_o", C.c_void_p), ("m_oc", C.c_void_p), ("s_oc", C.c_void_p),
        ("m_r1", C.c_int32), ("s_r1", C.c_int32),
        ("ln1_beta", C.c_void_p), ("ln1_mult", C.c_void_p), ("ln1_shift", C.c_void_p),
        ("m_c1", C.c_int32), ("s_c1", C.c_int32), ("m_c2", C.c_int32), ("s_c2", C.c_int32),
        ("w_val", C.c_void_p), ("b_val", C.c_void_p), ("m_val", C.c_void_p), ("s_val", C.c_void_p),
        ("w_off", C.c_void_p), ("b_off", C.c_void_p), ("m_off", C.c_void_p), ("s_off", C.c_void_p),
        ("w_att", C.c_void_p), ("b_att", C.c_void_p), ("m_att", C.c_void_p), ("s_att", C.c_void_p),
        ("smx_w", ShiftmaxT), ("m_s", C.c_int32), ("s_s", C.c_int32),
        ("w_o2", C.c_void_p), ("b_o2", C.c_void_p), ("m_o2", C.c_void_p), ("s_o2", C.c_void_p),
        ("m_r2", C.c_int32), ("s_r2", C.c_int32),
        ("ln2_beta", C.c_void_p), ("ln2_mult", C.c_void_p), ("ln2_shift", C.c_void_p),
        ("m_f", C.c_int32), ("s_f", C.c_int32),
        ("w_fc1", C.c_void_p), ("b_fc1", C.c_void_p), ("m_fc1", C.c_void_p), ("s_fc1", C.c_void_p),
        ("gelu", GeluT), ("m_g", C.c_int32), ("s_g", C.c_int32),
        ("w_fc2", C.c_void_p), ("b_fc2", C.c_void_p), ("m_fc2", C.c_void_p), ("s_fc2", C.c_void_p),
        ("m_r3", C.c_int32), ("s_r3", C.c_int32),
        ("ln3_beta", C.c_void_p), ("ln3_mult", C.c_void_p), ("ln3_shift", C.c_void_p),
    ]


# C signatures (argtypes, restype) of every export declared in include/ilwdetr.h
_VP, _I32, _I64 = C.c_void_p, C.c_int32, C.c_int64
SIGNATURES = {
    "ilwdetr_version": ([], C.c_char_p),
    "ilwdetr_last_error": ([], C.c_char_p),
    "ilwdetr_device_status": ([_VP], C.c_int),
    "ilwdetr_validate_only": ([_I32], C.c_int),
    "ilwdetr_debug_gemm_wait": ([_I32, C.c_int64], C.c_int),
    "ilwdetr_packed_weight_bytes": ([_I32, _I32], C.c_size_t),
    "ilwdetr_pack_weight": ([_VP, _I32, _I32, _VP, _VP], C.c_int),
    "ilwdetr_gemm_requant": ([_VP, _I64, _VP, _VP, _VP, _VP, _I32, _I32, _I32, _I32, _VP, _I64,
                              C.POINTER(ResidualT), _VP], C.c_int),
    "ilwdetr_gemm_gelu": ([_VP, _I64, _VP, _VP, _VP, _VP, _I32, _I32, _I32, C.POINTER(GeluT),
                           _I32, _I32, _VP, _I64, _VP], C.c_int),
    "ilwdetr_split_conv": ([C.POINTER(_VP), C.POINTER(_I64), _I32, _I32, C.POINTER(_I32),
                            C.POINTER(_VP), C.POINTER(_I32), C.POINTER(_I32), _VP, _VP, _VP, _I32,
                            _VP, _I64, _VP], C.c_int),
    "ilwdetr_shiftmax_rows": ([_VP, _I64, _I64, _I32, C.POINTER(ShiftmaxT), _VP, _I64, _VP], C.c_int),
    "ilwdetr_sdshiftgelu": ([_VP, _VP, _I64, C.POINTER(GeluT), _VP], C.c_int),
    "ilwdetr_int_layernorm": ([_VP, _I32, _I64, _I64, _I32, _VP, _VP, _VP, _I32, _VP, _I32, _I64,
                               _VP], C.c_int),
    "ilwdetr_shiftmax_attn": ([_VP, _VP, _VP, _I64, _I32, _I32, _I32, _I32, _I32, _I32,
                               C.POINTER(ShiftmaxT), _I32, _I32, _VP, _I32, _I64, _VP], C.c_int),
    "ilwdetr_gemm": ([C.POINTER(GemmT), _VP], C.c_int),
    "ilwdetr_deform_attn": ([_VP, C.POINTER(_I32), _I32, _VP, _VP, _VP, _I32, _I32, _I32, _I32,
                             _I32, _I32, _I32, _VP, _VP], C.c_int),
    "ilwdetr_patch_embed_workspace_bytes": ([_I32, _I32, _I32, _I32, _I32], C.c_size_t),
    "ilwdetr_patch_embed": ([_VP, _I32, _I32, _I32, _I32, _I32, _VP, _VP, _VP, _VP, _I32, _VP, _I32,
                             _I32, _VP, _VP, C.c_size_t, _VP], C.c_int),
    "ilwdetr_patch_embed_noalloc_max_bytes": ([], C.c_size_t),
    "ilwdetr_patch_embed_noalloc": ([_VP, _I32, _I32, _I32, _I32, _I32, _VP, _VP, _VP, _VP, _I32, _VP,
                                     _I32, _I32, _VP, _VP], C.c_int),
    "ilwdetr_block_workspace_bytes": ([_I32, _I32, _I32, _I32], C.c_size_t),
    "ilwdetr_block_forward": ([C.POINTER(BlockParamsT), _VP, _VP, _I32, _I32, _VP, C.c_size_t, _VP],
                              C.c_int),
    "ilwdetr_requant": ([_VP, _I32, _I64, _I64, _I32, _I32, _I32, _VP, _I64, _I64, _I32, _I32, _I32, _VP,
                         _I64, _VP], C.c_int),
    "ilwdetr_resample_nearest": ([_VP, _I64, _I32, _I32, _I32, _I32, _VP, _I64, _I32, _I32, _VP], C.c_int),
    "ilwdetr_int_sigmoid": ([_VP, _VP, _I64, C.POINTER(SigmoidT), _VP], C.c_int),
    "ilwdetr_relu_i8": ([_VP, _VP, _I64, _VP], C.c_int),
    "ilwdetr_ivit_shiftgelu": ([_VP, _I64, _I64, _I32, _VP, _I64, C.POINTER(GeluT), _VP], C.c_int),
    "ilwdetr_topk": ([_VP, _I64, _I32, _I32, _I32, _VP, _VP, _VP], C.c_int),
    "ilwdetr_gather_rows": ([_VP, _I64, _I64, _VP, _I64, _I64, _VP, _I64, _VP], C.c_int),
    "ilwdetr_decoder_workspace_bytes": ([_I32, _I32, _I64, _I32, _I32, _I32, _I32, _I32], C.c_size_t),
    "ilwdetr_decoder_layer_forward": ([C.POINTER(DecoderParamsT), _VP, _VP, _VP, C.POINTER(_I32), _I32, _VP,
                                       _I32, _I32, _VP, _VP, C.c_size_t, _VP], C.c_int),
}


def lib():
    """Load libilwdetr.so (raises IlwError if it is missing: there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise IlwError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        for name, (args, res) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _check(rc: int, what: str) -> None:
    if rc != 0:
        msg = lib().ilwdetr_last_error().decode()
        raise IlwError(f"{what} failed ({rc}): {msg}")


def _stream():
    import torch

    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _dev(t, dtype):
    import torch

    assert isinstance(t, torch.Tensor) and t.is_cuda and t.dtype == dtype, (t.dtype, dtype)
    return t


def version() -> str:
    return lib().ilwdetr_version().decode()


def device_status() -> None:
    _check(lib().ilwdetr_device_status(_stream()), "device_status")


# ---------------------------------------------------------------------------- linear layers
def pack_weight(W):
    """Pack an int8 [N, K] CUDA weight once (ilwdetr_pack_weight)."""
    import torch

    _dev(W, torch.int8)
    N, K = W.shape
    W = W.contiguous()
    nbytes = lib().ilwdetr_packed_weight_bytes(N, K)
    out = torch.empty(nbytes, dtype=torch.uint8, device=W.device)
    _check(lib().ilwdetr_pack_weight(_ptr(W), N, K, _ptr(out), _stream()), "pack_weight")
    return out


def gemm_requant(A, Wp, N, bias, mult, shift, out_bits=8, res=None, m_r=0, s_r=0, out=None):
    """ilwdetr_gemm_requant: A int8 [M, K] x packed W [N, K] -> int8/int16/int32 [M, N], or, with
    out_bits I8_IN_F16, the int8 values as float16."""
    import torch

    M, K = A.shape
    dt = {8: torch.int8, 16: torch.int16, 32: torch.int32, I8_IN_F16: torch.float16}[out_bits]
    if out is None:
        out = torch.empty((M, N), dtype=dt, device=A.device)
    r = None
    if res is not None:
        r = ResidualT(res.data_ptr(), res.stride(0), res.shape[0], m_r, s_r)
    _check(lib().ilwdetr_gemm_requant(_ptr(A), A.stride(0), _ptr(Wp), _ptr(bias), _ptr(mult),
                                      _ptr(shift), M, N, K, out_bits, _ptr(out), out.stride(0),
                                      None if r is None else C.byref(r), _stream()), "gemm_requant")
    return out


def gemm(A, Wp, N, bias, mult, shift, out_bits=8, res=None, m_r=0, s_r=0, gelu: dict | None = None, m_g=0, s_g=1,
         out=None):
    """ilwdetr_gemm: A int8 or float16 (the int8 values) [M, K] x packed W [N, K]; epilogue
    requantisation (with optional residual) or, with ``gelu``, SD-ShiftGELU; out_bits 8 / 16 / 32 /
    I8_IN_F16."""
    import torch

    M, K = A.shape
    dt = {8: torch.int8, 16: torch.int16, 32: torch.int32, I8_IN_F16: torch.float16}[out_bits]
    if out is None:
        out = torch.empty((M, N), dtype=dt, device=A.device)
    r = None if res is None else ResidualT(res.data_ptr(), res.stride(0), res.shape[0], m_r, s_r)
    g = None if gelu is None else GeluT(gelu["I0"], gelu.get("k_inter", 16), gelu.get("k_out", 8))
    a_form = I8_IN_F16 if A.dtype == torch.float16 else 8
    desc = GemmT(C.sizeof(GemmT), A.data_ptr(), a_form, A.stride(0), Wp.data_ptr(), _ptr(bias), _ptr(mult), _ptr(shift),
                 M, N, K, EPI_GELU if gelu is not None else EPI_REQUANT, out_bits, out.data_ptr(), out.stride(0),
                 None if r is None else C.pointer(r), None if g is None else C.pointer(g), m_g, s_g)
    _check(lib().ilwdetr_gemm(C.byref(desc), _stream()), "gemm")
    return out


def gemm_gelu(A, Wp, N, bias, mult, shift, gelu: dict, m_g, s_g, out=None):
    """ilwdetr_gemm_gelu: linear + SD-ShiftGELU epilogue -> int8 [M, N]."""
    import torch

    M, K = A.shape
    if out is None:
        out = torch.empty((M, N), dtype=torch.int8, device=A.device)
    g = GeluT(gelu["I0"], gelu.get("k_inter", 16), gelu.get("k_out", 8))
    _check(lib().ilwdetr_gemm_gelu(_ptr(A), A.stride(0), _ptr(Wp), _ptr(bias), _ptr(mult),
                                   _ptr(shift), M, N, K, C.byref(g), m_g, s_g, _ptr(out),
                                   out.stride(0), _stream()), "gemm_gelu")
    return out


def split_conv(Xs, Wps, N, m_b, s_b, bias, mult, shift, out=None):
    """ilwdetr_split_conv over nb branches of int8 [M, K_b] with packed weights [N, K_b]."""
    import torch

    nb = len(Xs)
    M = Xs[0].shape[0]
    if out is None:
        out = torch.empty((M, N), dtype=torch.int8, device=Xs[0].device)
    xp = (C.c_void_p * nb)(*[x.data_ptr() for x in Xs])
    ld = (C.c_int64 * nb)(*[x.stride(0) for x in Xs])
    kb = (C.c_int32 * nb)(*[x.shape[1] for x in Xs])
    wp = (C.c_void_p * nb)(*[w.data_ptr() for w in Wps])
    mb = (C.c_int32 * nb)(*[int(v) for v in m_b])
    sb = (C.c_int32 * nb)(*[int(v) for v in s_b])
    _check(lib().ilwdetr_split_conv(xp, ld, nb, M, kb, wp, mb, sb, _ptr(bias), _ptr(mult),
                                    _ptr(shift), N, _ptr(out), out.stride(0), _stream()),
           "split_conv")
    return out


# ---------------------------------------------------------------------------- nonlinear ops
def _smx(p: dict) -> ShiftmaxT:
    return ShiftmaxT(p["I0"], p.get("k_inter", 16), p.get("k_out", 8), p.get("s_d", -1),
                     p.get("m_p", 4), p.get("M_hw", 31))


def shiftmax_rows(X, smx: dict, out=None):
    """ilwdetr_shiftmax_rows: int32 [rows, len] -> u8 [rows, len]."""
    import torch

    rows, n = X.shape
    if out is None:
        out = torch.empty((rows, n), dtype=torch.uint8, device=X.device)
    p = _smx(smx)
    _check(lib().ilwdetr_shiftmax_rows(_ptr(X), X.stride(0), rows, n, C.byref(p), _ptr(out),
                                       out.stride(0), _stream()), "shiftmax_rows")
    return out


def sdshiftgelu(X, gelu: dict, out=None):
    """ilwdetr_sdshiftgelu: int32 -> int32 (x * I_div)."""
    import torch

    if out is None:
        out = torch.empty_like(X)
    g = GeluT(gelu["I0"], gelu.get("k_inter", 16), gelu.get("k_out", 8))
    _check(lib().ilwdetr_sdshiftgelu(_ptr(X), _ptr(out), X.numel(), C.byref(g), _stream()),
           "sdshiftgelu")
    return out


def int_layernorm(X, beta, mult, shift, iters=10, out_bits=8, out=None):
    """ilwdetr_int_layernorm: int16/int32 [rows, C] -> int8/int16 [rows, C]."""
    import torch

    rows, Cn = X.shape
    in_bits = {torch.int16: 16, torch.int32: 32}[X.dtype]
    if out is None:
        out = torch.empty((rows, Cn), dtype={8: torch.int8, 16: torch.int16, I8_IN_F16: torch.float16}[out_bits],
                          device=X.device)
    _check(lib().ilwdetr_int_layernorm(_ptr(X), in_bits, X.stride(0), rows, Cn, _ptr(beta),
                                       _ptr(mult), _ptr(shift), iters, _ptr(out), out_bits,
                                       out.stride(0), _stream()), "int_layernorm")
    return out


def shiftmax_attn(qkv, B, T, H, dh, win_side, smx: dict, m_o, s_o, out=None, o_f16=False):
    """ilwdetr_shiftmax_attn on a token-major [B*T, 3*H*dh] q|k|v buffer (int8, or float16
    holding the int8 values) -> int8 [B*T, H*dh] (float16 holding them with ``o_f16``)."""
    import torch

    d = H * dh
    if out is None:
        out = torch.empty((B * T, d), dtype=torch.float16 if o_f16 else torch.int8, device=qkv.device)
    form = I8_IN_F16 if qkv.dtype == torch.float16 else 8
    o_form = I8_IN_F16 if out.dtype == torch.float16 else 8
    base, es = qkv.data_ptr(), qkv.element_size()
    p = _smx(smx)
    _check(lib().ilwdetr_shiftmax_attn(C.c_void_p(base), C.c_void_p(base + d * es), C.c_void_p(base + 2 * d * es),
                                       qkv.stride(0), form, B, T, H, dh, win_side, C.byref(p), m_o, s_o,
                                       _ptr(out), o_form, out.stride(0), _stream()), "shiftmax_attn")
    return out


def deform_attn(value, level_hw, ref_q16, off_q8, w, m, s, out=None):
    """ilwdetr_deform_attn: value int8 [B,S,H*dh]; ref int32 [B,Q,2]; off int32 [B,Q,H,L,P,2];
    w u8 [B,Q,H,L*P] -> int8 [B,Q,H*dh]."""
    import torch

    B, S, Dm = value.shape
    _, Q, H, L, P, _ = off_q8.shape
    dh = Dm // H
    if out is None:
        out = torch.empty((B, Q, Dm), dtype=torch.int8, device=value.device)
    hw = [int(v) for pair in level_hw for v in pair]
    arr = (C.c_int32 * len(hw))(*hw)
    _check(lib().ilwdetr_deform_attn(_ptr(value), arr, L, _ptr(ref_q16), _ptr(off_q8), _ptr(w), B,
                                     Q, H, P, dh, m, s, _ptr(out), _stream()), "deform_attn")
    return out


# ---------------------------------------------------------------------------- encoder block
class BlockWeights:
    """Device copies of one block's integer parameters (from a dict of numpy arrays / ints, as
    produced by ``synth.block_params``) plus its ilw_block_params_t."""

    def __init__(self, bp: dict, device="cuda"):
        import numpy as np
        import torch

        self.bp = bp
        self.t = {}
        for k, v in bp.items():
            if isinstance(v, np.ndarray):
                self.t[k] = torch.from_numpy(np.ascontiguousarray(v)).to(device)
        for k in ("w_qkv", "w_proj", "w_fc1", "w_fc2"):
            self.t[k + "_p"] = pack_weight(self.t[k])
        s, T = bp["smx"], self.t
        self.params = BlockParamsT(
            C.sizeof(BlockParamsT), bp["d"], bp["H"], bp["F"], bp["win_side"], bp["ln_iters"],
            T["ln1_beta"].data_ptr(), T["ln1_mult"].data_ptr(), T["ln1_shift"].data_ptr(),
            T["ln2_beta"].data_ptr(), T["ln2_mult"].data_ptr(), T["ln2_shift"].data_ptr(),
            T["w_qkv_p"].data_ptr(), T["b_qkv"].data_ptr(), T["m_qkv"].data_ptr(), T["s_qkv"].data_ptr(),
            ShiftmaxT(s["I0"], s["k_inter"], s["k_out"], s["s_d"], s["m_p"], s["M_hw"]),
            bp["m_o"], bp["s_o"],
            T["w_proj_p"].data_ptr(), T["b_proj"].data_ptr(), T["m_proj"].data_ptr(), T["s_proj"].data_ptr(),
            bp["m_r1"], bp["s_r1"],
            T["w_fc1_p"].data_ptr(), T["b_fc1"].data_ptr(), T["m_fc1"].data_ptr(), T["s_fc1"].data_ptr(),
            GeluT(bp["gelu_I0"], bp["gelu_k_inter"], bp["gelu_k_out"]), bp["m_g"], bp["s_g"],
            T["w_fc2_p"].data_ptr(), T["b_fc2"].data_ptr(), T["m_fc2"].data_ptr(), T["s_fc2"].data_ptr(),
            bp["m_r2"], bp["s_r2"],
        )


def block_workspace_bytes(B, T, d, F) -> int:
    return int(lib().ilwdetr_block_workspace_bytes(B, T, d, F))


def block_forward(bw: BlockWeights, x, B, T, workspace, out=None):
    """ilwdetr_block_forward: int16 [B*T, d] -> int16 [B*T, d]."""
    import torch

    if out is None:
        out = torch.empty_like(x)
    _check(lib().ilwdetr_block_forward(C.byref(bw.params), _ptr(x), _ptr(out), B, T,
                                       _ptr(workspace), workspace.numel() * workspace.element_size(),
                                       _stream()), "block_forward")
    return out


# ---------------------------------------------------------------------------- patch embedding
def patch_embed_workspace_bytes(B, Cin, Hh, Ww, p) -> int:
    return int(lib().ilwdetr_patch_embed_workspace_bytes(B, Cin, Hh, Ww, p))


def patch_embed(img, p, Wp, d, bias, mult, shift, pos=None, m_pos=0, s_pos=0, workspace=None, out=None):
    """ilwdetr_patch_embed: int8 image [B, C, H, W] -> int16 x0 [B*T, d]."""
    import torch

    B, Cin, Hh, Ww = img.shape
    T = (Hh // p) * (Ww // p)
    if workspace is None:
        workspace = torch.empty(patch_embed_workspace_bytes(B, Cin, Hh, Ww, p), dtype=torch.uint8,
                                device=img.device)
    if out is None:
        out = torch.empty((B * T, d), dtype=torch.int16, device=img.device)
    _check(lib().ilwdetr_patch_embed(_ptr(img), B, Cin, Hh, Ww, p, _ptr(Wp), _ptr(bias), _ptr(mult),
                                     _ptr(shift), d, _ptr(pos), m_pos, s_pos, _ptr(out),
                                     _ptr(workspace), workspace.numel(), _stream()), "patch_embed")
    return out


class Backbone:
    """The integer ViT encoder of one configuration on the device: patch embedding followed by
    ``len(blocks)`` encoder blocks (each an ilwdetr_block_forward call), with its buffers."""

    def __init__(self, pe: dict, blocks: list, B: int, img_hw=(640, 640), device="cuda"):
        import numpy as np
        import torch

        self.B, self.p, self.hw = B, pe["p"], img_hw
        self.d, self.F = blocks[0]["d"], blocks[0]["F"]
        self.T = (img_hw[0] // self.p) * (img_hw[1] // self.p)
        self.pe = {k: torch.from_numpy(np.ascontiguousarray(v)).to(device)
                   for k, v in pe.items() if isinstance(v, np.ndarray)}
        self.pe_s = pe
        self.pe["w_p"] = pack_weight(self.pe["w"])
        self.blocks = [BlockWeights(bp, device) for bp in blocks]
        M = B * self.T
        self.ws_pe = torch.empty(patch_embed_workspace_bytes(B, 3, img_hw[0], img_hw[1], self.p),
                                 dtype=torch.uint8, device=device)
        self.ws_blk = torch.empty(block_workspace_bytes(B, self.T, self.d, self.F), dtype=torch.uint8,
                                  device=device)
        self.x = [torch.empty((M, self.d), dtype=torch.int16, device=device) for _ in range(2)]

    def forward(self, img, taps: dict | None = None):
        """img int8 [B, 3, H, W] (device) -> x_L int16 [B*T, d] (a buffer owned by the backbone).
        ``taps`` maps block indices to int16 [B*T, d] buffers that receive those blocks' outputs."""
        pe = self.pe
        x = patch_embed(img, self.p, pe["w_p"], self.d, pe["b"], pe["m"], pe["s"], pe["pos"],
                        self.pe_s["m_pos"], self.pe_s["s_pos"], self.ws_pe, self.x[0])
        for i, bw in enumerate(self.blocks):
            # a tapped block writes straight into its tap buffer; the others ping-pong
            out = taps[i] if taps and i in taps else (self.x[1] if x is self.x[0] else self.x[0])
            x = block_forward(bw, x, self.B, self.T, self.ws_blk, out=out)
        return x

    def capture(self, img) -> "Graphed":
        """The forward of ``img`` recorded as one CUDA graph: ``replay()`` re-runs the patch
        embedding and every block on the current contents of ``img`` (a fixed device buffer) and
        returns the backbone's output buffer."""
        return Graphed(lambda: self.forward(img))


class Graphed:
    """A CUDA graph of one sequence of library calls on fixed buffers.  The calls run once on a
    side stream (so every lazily built table and tensor map exists), are then recorded, and each
    ``replay()`` launches the recorded kernels on the current stream in one graph launch."""

    def __init__(self, fn, warmup: int = 1):
        import torch

        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for _ in range(warmup):
                fn()
        torch.cuda.current_stream().wait_stream(side)
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self.out = fn()

    def replay(self):
        self.graph.replay()
        return self.out


# ---------------------------------------------------------------------------- detector
def requant(X, m1, s1, Z=None, m2=0, s2=1, out_bits=8, out=None):
    """ilwdetr_requant: sat(rq(X; m1, s1) + rq(Z[r mod z_rows]; m2, s2)), X int16/int32 [rows, C],
    Z int16 or None -> int8/int16/int32 [rows, C]."""
    import torch

    rows, Cn = X.shape
    in_bits = {torch.int16: 16, torch.int32: 32}[X.dtype]
    if out is None:
        out = torch.empty((rows, Cn), dtype={8: torch.int8, 16: torch.int16, 32: torch.int32}[out_bits],
                          device=X.device)
    zp, ldz, zr = (None, 0, 1) if Z is None else (_ptr(Z), Z.stride(0), Z.shape[0])
    _check(lib().ilwdetr_requant(_ptr(X), in_bits, X.stride(0), rows, Cn, m1, s1, zp, ldz, zr, m2, s2, out_bits,
                                 _ptr(out), out.stride(0), _stream()), "requant")
    return out


def resample_nearest(X, B, Hi, Wi, Ho, Wo, out=None, x_bstride=None, y_bstride=None):
    """ilwdetr_resample_nearest over B maps of int8 [Hi*Wi, C] rows -> [B*Ho*Wo, C] (or into `out`
    with its own batch stride in rows)."""
    import torch

    Cn = X.shape[-1]
    if out is None:
        out = torch.empty((B * Ho * Wo, Cn), dtype=torch.int8, device=X.device)
    xs = Hi * Wi if x_bstride is None else x_bstride
    ys = Ho * Wo if y_bstride is None else y_bstride
    _check(lib().ilwdetr_resample_nearest(_ptr(X), xs, B, Hi, Wi, Cn, _ptr(out), ys, Ho, Wo, _stream()),
           "resample_nearest")
    return out


class DecoderWeights:
    """Device copies of one decoder layer's integer parameters (``synth.decoder_params``) and its
    ilw_decoder_params_t."""

    _W = ("w_qk", "w_v", "w_o", "w_val", "w_off", "w_att", "w_o2", "w_fc1", "w_fc2")

    def __init__(self, dp: dict, device="cuda"):
        import numpy as np
        import torch

        self.dp = dp
        T = self.t = {k: torch.from_numpy(np.ascontiguousarray(v)).to(device)
                      for k, v in dp.items() if isinstance(v, np.ndarray)}
        for k in self._W:
            T[k + "_p"] = pack_weight(T[k])
        a = lambda k: T[k].data_ptr()  # noqa: E731
        self.params = DecoderParamsT(
            C.sizeof(DecoderParamsT), dp["d"], dp["H"], dp["F"], dp["L"], dp["P"], dp["ln_iters"],
            dp["m_q1"], dp["s_q1"], dp["m_q2"], dp["s_q2"], dp["m_v1"], dp["s_v1"],
            a("w_qk_p"), a("b_qk"), a("m_qk"), a("s_qk"), a("w_v_p"), a("b_v"), a("m_v"), a("s_v"),
            _smx(dp["smx"]), dp["m_o"], dp["s_o"],
            a("w_o_p"), a("b_o"), a("m_oc"), a("s_oc"), dp["m_r1"], dp["s_r1"],
            a("ln1_beta"), a("ln1_mult"), a("ln1_shift"),
            dp["m_c1"], dp["s_c1"], dp["m_c2"], dp["s_c2"],
            a("w_val_p"), a("b_val"), a("m_val"), a("s_val"),
            a("w_off_p"), a("b_off"), a("m_off"), a("s_off"),
            a("w_att_p"), a("b_att"), a("m_att"), a("s_att"),
            _smx(dp["smx_w"]), dp["m_s"], dp["s_s"],
            a("w_o2_p"), a("b_o2"), a("m_o2"), a("s_o2"), dp["m_r2"], dp["s_r2"],
            a("ln2_beta"), a("ln2_mult"), a("ln2_shift"),
            dp["m_f"], dp["s_f"],
            a("w_fc1_p"), a("b_fc1"), a("m_fc1"), a("s_fc1"),
            GeluT(dp["gelu_I0"], dp["gelu_k_inter"], dp["gelu_k_out"]), dp["m_g"], dp["s_g"],
            a("w_fc2_p"), a("b_fc2"), a("m_fc2"), a("s_fc2"), dp["m_r3"], dp["s_r3"],
            a("ln3_beta"), a("ln3_mult"), a("ln3_shift"),
        )


def decoder_workspace_bytes(B, Q, S_total, d, F, H, L, P) -> int:
    return int(lib().ilwdetr_decoder_workspace_bytes(B, Q, S_total, d, F, H, L, P))


def decoder_layer_forward(dw: DecoderWeights, tgt, pos, memory, level_hw, refs, B, Q, workspace, out=None):
    """ilwdetr_decoder_layer_forward: tgt, pos int16 [B*Q, d], memory int8 [B*S, d], refs int32
    [B, Q, 2] -> int16 [B*Q, d]."""
    import torch

    if out is None:
        out = torch.empty_like(tgt)
    L = len(level_hw)
    lhw = (C.c_int32 * (2 * L))(*[int(v) for hw in level_hw for v in hw])
    _check(lib().ilwdetr_decoder_layer_forward(C.byref(dw.params), _ptr(tgt), _ptr(pos), _ptr(memory), lhw, L,
                                               _ptr(refs), B, Q, _ptr(out), _ptr(workspace),
                                               workspace.numel() * workspace.element_size(), _stream()),
           "decoder_layer_forward")
    return out


class Projector:
    """The split-convolution projector on the device: the tapped encoder layers requantised to int8
    (one scale each), one ilwdetr_split_conv per level on the stride-16 grid, and the levels
    resampled by nearest neighbour into one concatenated decoder memory [B*S, N]."""

    def __init__(self, pp: dict, B: int, grid: int, levels, K: int, device="cuda"):
        import numpy as np
        import torch

        self.pp, self.B, self.grid, self.levels = pp, B, grid, [tuple(x) for x in levels]
        self.N = pp["levels"][0]["w"][0].shape[0]
        self.S = sum(h * w for h, w in self.levels)
        dv = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.lv = []
        for lv in pp["levels"]:
            self.lv.append({"w_p": [pack_weight(dv(w)) for w in lv["w"]], "b": dv(lv["b"]), "m": dv(lv["m"]),
                            "s": dv(lv["s"]), "m_b": list(lv["m_b"]), "s_b": list(lv["s_b"])})
        M = B * grid * grid
        self.t = [torch.empty((M, K), dtype=torch.int8, device=device) for _ in pp["taps"]]
        self.y = torch.empty((M, self.N), dtype=torch.int8, device=device)
        self.memory = torch.empty((B * self.S, self.N), dtype=torch.int8, device=device)

    def forward(self, taps):
        for x, (m, s), t in zip(taps, self.pp["taps"], self.t):
            requant(x, m, s, out_bits=8, out=t)
        start = 0
        for lv, (Hl, Wl) in zip(self.lv, self.levels):
            split_conv(self.t, lv["w_p"], self.N, lv["m_b"], lv["s_b"], lv["b"], lv["m"], lv["s"], out=self.y)
            resample_nearest(self.y, self.B, self.grid, self.grid, Hl, Wl, out=self.memory[start:],
                             y_bstride=self.S)
            start += Hl * Wl
        return self.memory


class Detector:
    """The full integer detector forward: Backbone (with its output layers tapped) -> Projector ->
    decoder layers (ilwdetr_decoder_layer_forward), all on fixed device buffers.  With two-stage
    parameters (``synth.two_stage_params``) the decoder's reference points come from the two-stage
    query selection over the memory, and with positional-query parameters as well
    (``synth.query_pos_params``) so do its positional queries (the learnable projection of the
    selected boxes); with refinement parameters (``synth.refine_params``) the references are
    refined after every layer but the last (BoxRefine), and each layer samples at, and projects, the
    current boxes; with head parameters (``synth.head_params``) the decoder output is requantised
    to int8 and the detection head gives class scores and boxes."""

    def __init__(self, pe: dict, blocks: list, taps, pp: dict, dps: list, B: int, Q: int, levels, grid: int = 40,
                 tsp: dict | None = None, hp: dict | None = None, pq: dict | None = None, rps: list | None = None,
                 device="cuda"):
        import torch

        self.backbone = Backbone(pe, blocks, B, device=device)
        self.taps = tuple(taps)
        self.proj = Projector(pp, B, grid, levels, self.backbone.d, device)
        self.dec = [DecoderWeights(dp, device) for dp in dps]
        self.B, self.Q, self.levels = B, Q, [tuple(x) for x in levels]
        d, dp0 = dps[0]["d"], dps[0]
        self.d = d
        M = B * self.backbone.T
        self.tap_buf = [torch.empty((M, self.backbone.d), dtype=torch.int16, device=device) for _ in self.taps]
        self.ws = torch.empty(decoder_workspace_bytes(B, Q, self.proj.S, d, dp0["F"], dp0["H"], dp0["L"], dp0["P"]),
                              dtype=torch.uint8, device=device)
        self.t = [torch.empty((B * Q, d), dtype=torch.int16, device=device) for _ in range(2)]
        self.ts = TwoStage(tsp, device) if tsp is not None else None
        self.head = DetectionHead(hp, device) if hp is not None else None
        if self.ts is not None:
            # (cx, cy) of each selected box: a gather of the first 8 bytes of every box row
            self.ident = torch.arange(B * Q, dtype=torch.int32, device=device)
            self.refs_buf = torch.empty((B, Q, 2), dtype=torch.int32, device=device)
        self.qp = QueryPos(pq, B * Q, device) if (pq is not None and self.ts is not None) else None
        if rps is not None and self.ts is None:
            raise ValueError("Detector: box refinement needs the two-stage references (tsp)")
        self.refine = [BoxRefine(rp, device) for rp in rps[: len(dps) - 1]] if rps is not None else None
        if self.qp is not None:
            self.pos_buf = torch.empty((B * Q, d), dtype=torch.int16, device=device)

    def forward(self, img, tgt, pos=None, refs=None, ref16=None):
        """img int8 [B, 3, H, W]; tgt, pos int16 [B*Q, d] (pos ignored with the positional-query
        projection); refs int32 [B, Q, 2] (Q16 sampling points; ignored with two-stage selection)
        -> int16 [B*Q, d], or, with a detection head, (that output, class scores int32 [B*Q, C],
        boxes int32 [B*Q, 4]); ref16: int16 [B*Q, 4] reference logits for the head when there is
        no two-stage selection."""
        self.backbone.forward(img, taps=dict(zip(self.taps, self.tap_buf)))
        memory = self.proj.forward(self.tap_buf)
        boxes = None
        if self.ts is not None:
            _, _, ref16, boxes = self.ts.forward(memory, self.B, self.proj.S, self.Q)
        x = tgt
        for i, dw in enumerate(self.dec):
            if boxes is not None:  # this layer's sampling points and positional queries from the current boxes
                gather_rows(boxes[:, :2], self.ident, out=self.refs_buf.view(self.B * self.Q, 2))
                refs = self.refs_buf
                if self.qp is not None:
                    pos = self.qp.forward(boxes, out=self.pos_buf)
            if pos is None or refs is None:
                raise ValueError("Detector.forward: pos and refs are needed unless the two-stage selection "
                                 "(and, for pos, the positional-query projection) provides them")
            x = decoder_layer_forward(dw, x, pos, memory, self.levels, refs, self.B, self.Q, self.ws,
                                      out=self.t[i % 2])
            if self.refine is not None and i + 1 < len(self.dec):
                ref16, boxes = self.refine[i].forward(x, ref16)
        if self.head is None:
            return x
        hp = self.head.hp
        a = requant(x, hp["m_in"], hp["s_in"], out_bits=8)
        scores, boxes, _ = self.head.forward(a, ref16)
        return x, scores, boxes


# ---------------------------------------------------------------- detection head, two-stage selection
def int_sigmoid(X, sig: dict, out=None):
    """ilwdetr_int_sigmoid: int32 logits -> int32 sigmoid at scale 2^-(k_out-1) (same shape)."""
    import torch

    if out is None:
        out = torch.empty_like(X)
    p = SigmoidT(sig["I0"], sig.get("k_inter", 8), sig.get("k_out", 8))
    _check(lib().ilwdetr_int_sigmoid(_ptr(X), _ptr(out), X.numel(), C.byref(p), _stream()), "int_sigmoid")
    return out


def relu_i8(X, out=None):
    """ilwdetr_relu_i8: max(X, 0) on int8 (in place when out is X)."""
    import torch

    if out is None:
        out = torch.empty_like(X)
    _check(lib().ilwdetr_relu_i8(_ptr(X), _ptr(out), X.numel(), _stream()), "relu_i8")
    return out


def topk(S, K, vals=None, idx=None):
    """ilwdetr_topk over the rows of the 2-D int32 S -> (values int32 [rows, K], indices int32 [rows, K])."""
    import torch

    rows, N = S.shape
    if vals is None:
        vals = torch.empty((rows, K), dtype=torch.int32, device=S.device)
    if idx is None:
        idx = torch.empty((rows, K), dtype=torch.int32, device=S.device)
    _check(lib().ilwdetr_topk(_ptr(S), S.stride(0), rows, N, K, _ptr(vals), _ptr(idx), _stream()), "topk")
    return vals, idx


def gather_rows(X, idx, out=None):
    """ilwdetr_gather_rows: rows idx (int32, any shape) of the 2-D X -> [idx.numel(), X.shape[1]]."""
    import torch

    n = idx.numel()
    rb = X.shape[1] * X.element_size()
    if out is None:
        out = torch.empty((n, X.shape[1]), dtype=X.dtype, device=X.device)
    _check(lib().ilwdetr_gather_rows(_ptr(X), X.stride(0) * X.element_size(), X.shape[0], _ptr(idx), n, rb,
                                     _ptr(out), out.stride(0) * out.element_size(), _stream()), "gather_rows")
    return out


class DetectionHead:
    """The detection head on the decoder output (``synth.head_params``): class scores by the integer
    sigmoid of a linear layer's raw logits; box logits from a 3-layer integer MLP (ReLU on the int8
    hidden outputs) added to the reference logits at one scale, and boxes (cx, cy, w, h at scale
    2^-16) by the integer sigmoid.  Every step is an ilwdetr_* call."""

    def __init__(self, hp: dict, device="cuda"):
        import numpy as np
        import torch

        self.hp = hp
        dv = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.t = {k: dv(v) for k, v in hp.items() if isinstance(v, np.ndarray)}
        for k in ("w_cls", "w_b1", "w_b2", "w_b3"):
            self.t[k + "_p"] = pack_weight(self.t[k])
        self.C = hp["w_cls"].shape[0]

    def forward(self, out, ref16):
        """out int8 [M, d] (decoder output), ref16 int16 [M, 4] (reference logits) ->
        (scores int32 [M, C], boxes int32 [M, 4], box logits z int32 [M, 4])."""
        hp, t = self.hp, self.t
        d = out.shape[1]
        logits = gemm_requant(out, t["w_cls_p"], self.C, t["b_cls"], None, None, 32)
        scores = int_sigmoid(logits, {"I0": hp["cls_I0"], "k_inter": hp["k_inter"], "k_out": hp["cls_k_out"]})
        h1 = gemm_requant(out, t["w_b1_p"], d, t["b_b1"], t["m_b1"], t["s_b1"], 8)
        relu_i8(h1, out=h1)
        h2 = gemm_requant(h1, t["w_b2_p"], d, t["b_b2"], t["m_b2"], t["s_b2"], 8)
        relu_i8(h2, out=h2)
        dlt = gemm_requant(h2, t["w_b3_p"], 4, t["b_b3"], None, None, 32)
        z = requant(dlt, hp["m_d"], hp["s_d"], ref16, hp["m_ref"], hp["s_ref"], out_bits=32)
        boxes = int_sigmoid(z, {"I0": hp["box_I0"], "k_inter": hp["k_inter"], "k_out": 17})
        return scores, boxes, z


class BoxRefine:
    """The box refinement after a decoder layer (``synth.refine_params``, one per layer): the decoder
    output requantised to int8, a 3-layer integer MLP (ReLU on the int8 hidden outputs), the deltas
    requantised to the reference-logit scale and added to the current reference logits (saturated
    to int16), and the new boxes by the integer sigmoid (scale 2^-16).  Every step is an ilwdetr_*
    call."""

    def __init__(self, rp: dict, device="cuda"):
        import numpy as np
        import torch

        self.rp = rp
        dv = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.t = {k: dv(v) for k, v in rp.items() if isinstance(v, np.ndarray)}
        for k in ("w_b1", "w_b2", "w_b3"):
            self.t[k + "_p"] = pack_weight(self.t[k])

    def forward(self, x, ref16):
        """x int16 [M, d] (decoder output), ref16 int16 [M, 4] -> (new ref16 int16 [M, 4], boxes int32 [M, 4])."""
        rp, t = self.rp, self.t
        d = x.shape[1]
        a = requant(x, rp["m_in"], rp["s_in"], out_bits=8)
        h1 = gemm_requant(a, t["w_b1_p"], d, t["b_b1"], t["m_b1"], t["s_b1"], 8)
        relu_i8(h1, out=h1)
        h2 = gemm_requant(h1, t["w_b2_p"], d, t["b_b2"], t["m_b2"], t["s_b2"], 8)
        relu_i8(h2, out=h2)
        dlt = gemm_requant(h2, t["w_b3_p"], 4, t["b_b3"], None, None, 32)
        ref = requant(dlt, rp["m_d"], rp["s_d"], ref16, rp["m_ref"], rp["s_ref"], out_bits=16)
        ref32 = requant(ref, 1 << 30, 30, out_bits=32)
        boxes = int_sigmoid(ref32, {"I0": rp["box_I0"], "k_inter": rp["k_inter"], "k_out": 17})
        return ref, boxes


class TwoStage:
    """Two-stage query selection (``synth.two_stage_params``): encoder class logits of every
    memory token, its best class logit (top-1), the K best tokens per image (top-K, ties to the
    lower index), and their reference logits sat16(rq(MLP(memory[token])) + rq(anchor[token])) and
    boxes (integer sigmoid, scale 2^-16).  Every step is an ilwdetr_* call."""

    def __init__(self, tp: dict, device="cuda"):
        import numpy as np
        import torch

        self.tp = tp
        dv = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.t = {k: dv(v) for k, v in tp.items() if isinstance(v, np.ndarray)}
        for k in ("w_enc", "w_p1", "w_p2"):
            self.t[k + "_p"] = pack_weight(self.t[k])

    def forward(self, memory, B, S, K):
        """memory int8 [B*S, d] -> (values [B, K], token indices [B, K], ref16 int16 [B*K, 4],
        boxes int32 [B*K, 4])."""
        import torch

        tp, t = self.tp, self.t
        d = memory.shape[1]
        Cn = tp["w_enc"].shape[0]
        enc = gemm_requant(memory, t["w_enc_p"], Cn, t["b_enc"], None, None, 32)
        best, _ = topk(enc, 1)
        vals, idx = topk(best.view(B, S), K)
        # the selected tokens' memory rows and anchors, image by image (views of the batch)
        sel = torch.empty((B * K, d), dtype=torch.int8, device=memory.device)
        for b in range(B):
            gather_rows(memory[b * S:(b + 1) * S], idx[b], out=sel[b * K:(b + 1) * K])
        anc = gather_rows(t["anchor16"], idx.view(-1))
        h1 = gemm_requant(sel, t["w_p1_p"], d, t["b_p1"], t["m_p1"], t["s_p1"], 8)
        relu_i8(h1, out=h1)
        dlt = gemm_requant(h1, t["w_p2_p"], 4, t["b_p2"], None, None, 32)
        ref16 = requant(dlt, tp["m_d"], tp["s_d"], anc, tp["m_a"], tp["s_a"], out_bits=16)
        ref32 = requant(ref16, 1 << 30, 30, out_bits=32)
        boxes = int_sigmoid(ref32, {"I0": tp["ref_I0"], "k_inter": tp["k_inter"], "k_out": 17})
        return vals, idx, ref16, boxes


class QueryPos:
    """The learnable positional-query projection (``synth.query_pos_params``): Q16 boxes [M, 4] ->
    int8 (requantised) -> linear 4 -> hidden, ReLU -> linear hidden -> d -> int16 positional queries
    [M, d].  Every step is an ilwdetr_* call.  The GEMM takes K in multiples of 16, so the 4-column
    layer runs as a 16-column one: the int8 boxes sit in columns 0..3 of a zeroed [M, 16] buffer and
    the packed weight has zero columns 4..15 (zero products, the same integers)."""

    def __init__(self, pq: dict, M: int, device="cuda"):
        import numpy as np
        import torch

        self.pq, self.M = pq, M
        dv = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)  # noqa: E731
        self.t = {k: dv(v) for k, v in pq.items() if isinstance(v, np.ndarray)}
        w1 = pq["w_q1"]
        w1p = np.zeros((w1.shape[0], 16), dtype=np.int8)
        w1p[:, :w1.shape[1]] = w1
        self.t["w_q1_p"] = pack_weight(dv(w1p))
        self.t["w_q2_p"] = pack_weight(self.t["w_q2"])
        self.hidden, self.d = pq["w_q1"].shape[0], pq["w_q2"].shape[0]
        self.b8 = torch.zeros((M, 16), dtype=torch.int8, device=device)  # columns 4..15 stay zero

    def forward(self, boxes, out=None):
        pq, t = self.pq, self.t
        requant(boxes, pq["m_box"], pq["s_box"], out_bits=8, out=self.b8[:, :4])
        h = gemm_requant(self.b8, t["w_q1_p"], self.hidden, t["b_q1"], t["m_q1"], t["s_q1"], 8)
        relu_i8(h, out=h)
        return gemm_requant(h, t["w_q2_p"], self.d, t["b_q2"], t["m_q2"], t["s_q2"], 16, out=out)


def ivit_shiftgelu(X, gelu: dict, out=None):
    """ilwdetr_ivit_shiftgelu: I-ViT's ShiftGELU (row-maximum subtraction) over the rows of the 2-D
    int32 X -> int32 x * I_div (the ablation baseline of SD-ShiftGELU)."""
    import torch

    rows, L = X.shape
    if out is None:
        out = torch.empty_like(X)
    g = GeluT(gelu["I0"], gelu.get("k_inter", 16), gelu.get("k_out", 8))
    _check(lib().ilwdetr_ivit_shiftgelu(_ptr(X), X.stride(0), rows, L, _ptr(out), out.stride(0), C.byref(g), _stream()),
           "ivit_shiftgelu")
    return out
