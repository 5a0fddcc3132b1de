"""The C-ABI library builds, loads without a GPU and exports every entry point declared in
include/ilwdetr.h; the Python binding covers the same names.  No kernel runs here: argument checks
are exercised up to the first CUDA call, which fails on a machine without a device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "ilwdetr.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ilwdetr_\w+)\s*\(", src)))


@pytest.fixture(scope="module")
def built_lib():
    from paper_2607_24981_gb300 import build

    path = build.build()
    return path


@pytest.fixture
def validate_only(built_lib):
    """Validate-only mode for the calling thread during one test: the argument checks run as usual
    and nothing can be launched, so the fake addresses these tests pass are never used."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    assert L.ilwdetr_validate_only(1) == 0
    yield L
    L.ilwdetr_validate_only(0)


def test_header_declares_the_paths_entry_points():
    syms = declared_symbols()
    for name in ("ilwdetr_gemm_requant", "ilwdetr_shiftmax_attn", "ilwdetr_sdshiftgelu",
                 "ilwdetr_int_layernorm", "ilwdetr_split_conv", "ilwdetr_deform_attn",
                 "ilwdetr_block_forward", "ilwdetr_shiftmax_rows", "ilwdetr_requant",
                 "ilwdetr_resample_nearest", "ilwdetr_decoder_layer_forward"):
        assert name in syms


def test_library_exports_every_declared_symbol(built_lib):
    L = ctypes.CDLL(built_lib)
    missing = [s for s in declared_symbols() if not hasattr(L, s)]
    assert not missing, missing


def test_binding_signatures_cover_the_header(built_lib):
    import paper_2607_24981_gb300 as ilw

    assert set(ilw.SIGNATURES) == set(declared_symbols())
    hdr = open(os.path.join(ROOT, "include", "ilwdetr.h")).read()
    assert int(re.search(r"#define ILW_I8_IN_F16 (\d+)", hdr).group(1)) == ilw.I8_IN_F16
    ilw.lib()
    assert ilw.version().startswith("ilwdetr")


def test_host_side_validation_without_gpu(validate_only):
    """Argument errors are reported before any launch, so they work with no device at all."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    bad = ilw.ShiftmaxT(0, 16, 8, -1, 4, 31)  # I0 = 0 is outside the domain of ShiftExp
    rc = L.ilwdetr_shiftmax_rows(ctypes.c_void_p(16), 4, 1, 4, ctypes.byref(bad), ctypes.c_void_p(16), 4, None)
    assert rc == -1 and b"I0" in L.ilwdetr_last_error()
    g = ilw.GeluT(1 << 14, 16, 8)  # I0 * 2^(k+1) = 2^31: overflows
    rc = L.ilwdetr_sdshiftgelu(ctypes.c_void_p(16), ctypes.c_void_p(16), 4, ctypes.byref(g), None)
    assert rc == -1
    smx = ilw.ShiftmaxT(100, 16, 8, -1, 4, 31)
    rc = L.ilwdetr_shiftmax_attn(ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16), 48, 8, 1, 64, 1, 48,
                                 0, ctypes.byref(smx), 1 << 30, 30, ctypes.c_void_p(16), 8, 48, None)
    assert rc == -2  # dh = 48 unsupported
    rc = L.ilwdetr_shiftmax_attn(ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16), 64, 16, 1, 64, 1, 64,
                                 0, ctypes.byref(smx), 1 << 30, 30, ctypes.c_void_p(16), 8, 64, None)
    assert rc == -1 and b"qkv_form" in L.ilwdetr_last_error()  # neither int8 nor ILW_I8_IN_F16
    rc = L.ilwdetr_shiftmax_attn(ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16), 68, ilw.I8_IN_F16, 1,
                                 64, 1, 64, 0, ctypes.byref(smx), 1 << 30, 30, ctypes.c_void_p(16), 8, 64, None)
    assert rc == -1  # fp16 rows of 68 elements are not 16-byte aligned
    rc = L.ilwdetr_gemm_requant(ctypes.c_void_p(16), 24, ctypes.c_void_p(256), None, None, None, 4, 4, 24, 8,
                                ctypes.c_void_p(16), 4, None, None)
    assert rc == -2  # K % 16 != 0
    assert L.ilwdetr_packed_weight_bytes(3, 32) > 0
    assert L.ilwdetr_block_workspace_bytes(8, 1600, 384, 1536) > 8 * 1600 * 384 * 8
    assert L.ilwdetr_decoder_workspace_bytes(16, 300, 8400, 256, 1024, 8, 3, 4) > 16 * 8400 * 256
    rc = L.ilwdetr_requant(ctypes.c_void_p(16), 16, 12, 4, 10, 1 << 30, 30, None, 0, 1, 0, 1, 8,
                           ctypes.c_void_p(16), 12, None)
    assert rc == -2  # C % 4 != 0
    rc = L.ilwdetr_resample_nearest(ctypes.c_void_p(16), 100, 1, 10, 10, 24, ctypes.c_void_p(16), 400, 20, 20, None)
    assert rc == -2  # C % 16 != 0


def test_detection_entry_points_validate_without_gpu(validate_only):
    """The detection-head and selection entry points reject bad arguments before any launch."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    p = ilw.SigmoidT(1 << 14, 16, 8)  # I0 * 2^(k+1) = 2^31: overflows the IntDiv denominator
    assert L.ilwdetr_int_sigmoid(ctypes.c_void_p(16), ctypes.c_void_p(16), 4, ctypes.byref(p), None) == -1
    p = ilw.SigmoidT(1024, 8, 25)  # k_out above 24: the output no longer fits int32
    assert L.ilwdetr_int_sigmoid(ctypes.c_void_p(16), ctypes.c_void_p(16), 4, ctypes.byref(p), None) == -1
    p = ilw.SigmoidT(1024, 8, 17)
    assert L.ilwdetr_int_sigmoid(ctypes.c_void_p(20), ctypes.c_void_p(16), 4, ctypes.byref(p), None) == -1  # not 16 B
    assert L.ilwdetr_topk(ctypes.c_void_p(16), 10, 2, 10, 11, ctypes.c_void_p(16), ctypes.c_void_p(16), None) == -1
    assert L.ilwdetr_topk(ctypes.c_void_p(16), 20000, 1, 20000, 5, ctypes.c_void_p(16), ctypes.c_void_p(16),
                          None) == -2  # past the shared-memory sort's 16384 keys
    assert b"16384" in L.ilwdetr_last_error()
    assert L.ilwdetr_gather_rows(ctypes.c_void_p(16), 12, 5, ctypes.c_void_p(16), 3, 6, ctypes.c_void_p(16), 12,
                                 None) == -1  # 6-byte rows
    assert L.ilwdetr_relu_i8(ctypes.c_void_p(17), ctypes.c_void_p(16), 8, None) == -1  # misaligned
    g = ilw.GeluT(600, 16, 8)
    assert L.ilwdetr_ivit_shiftgelu(ctypes.c_void_p(16), 4, 3, 8, ctypes.c_void_p(16), 8, ctypes.byref(g), None) == -1
    assert L.ilwdetr_topk(ctypes.c_void_p(16), 10, 0, 10, 3, ctypes.c_void_p(16), ctypes.c_void_p(16), None) == 0


def test_layernorm_and_noalloc_validate_without_gpu(validate_only):
    """I-LayerNorm and the allocation-free patch embedding reject bad arguments before any CUDA
    call (so with no device at all): the no-alloc entry checks its weights and its scratch bound
    before it looks up the scratch array or launches the gather."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    v = ctypes.c_void_p(256)

    def ln(in_bits=16, rows=4, C=64, beta=v, iters=10, out_bits=8):
        return L.ilwdetr_int_layernorm(v, in_bits, C, rows, C, beta, v, v, iters, v, out_bits, C, None)

    assert ln(in_bits=8) == -1
    assert ln(out_bits=12) == -1
    assert ln(C=5000) == -2 and b"4096" in L.ilwdetr_last_error()
    assert ln(iters=65) == -1
    assert ln(beta=None) == -1
    assert ln(rows=0) == 0  # nothing to do, nothing launched

    def pe(img=v, B=1, Cin=3, H=640, W=640, p=16, Wp=v, mult=v, pos=None, s_pos=10):
        return L.ilwdetr_patch_embed_noalloc(img, B, Cin, H, W, p, Wp, v, mult, v, 384, pos, 1 << 30, s_pos, v, None)

    assert pe(p=15) == -2  # the patch must be a multiple of 16
    assert pe(H=632) == -2  # p must divide H
    assert pe(img=ctypes.c_void_p(257)) == -1  # misaligned image
    assert pe(Wp=None) == -1 and b"weight" in L.ilwdetr_last_error()
    assert pe(Wp=ctypes.c_void_p(272)) == -1  # packed weight not 256-byte aligned
    assert pe(mult=None) == -1
    assert pe(pos=v, s_pos=63) == -1  # position-term shift outside [1, 62]
    assert pe(B=0) == 0
    # 7 images of 3 x 640 x 640 gather 8.6 MB of patches: more than the fixed scratch
    assert 6 * 3 * 640 * 640 <= L.ilwdetr_patch_embed_noalloc_max_bytes() < 7 * 3 * 640 * 640
    assert pe(B=7) == -2 and b"8 MiB" in L.ilwdetr_last_error()


# Fake device addresses: only ever passed to calls that fail their argument checks or run in
# validate-only mode (ilwdetr_validate_only), so nothing is launched on them on any machine.
def _fake_ptrs(struct, base):
    """Every pointer field of a ctypes struct set to a distinct 256-byte aligned fake address."""
    k = 0
    for name, typ in struct._fields_:
        if typ is ctypes.c_void_p:
            setattr(struct, name, base + 0x10000 * k)
            k += 1


def test_composite_entry_points_check_every_step_before_launching(built_lib):
    """The encoder block, the decoder layer and the patch embedding check the arguments of all
    their steps (the pass a real call makes before its first launch): a bad parameter of a late step
    (the attention's Shiftmax, the FFN's GELU, a residual shift, the deformable weights' Shiftmax) is
    an argument error, and valid arguments pass every step.  Run in validate-only mode, so nothing is
    launched whether or not a device is present."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    assert L.ilwdetr_validate_only(1) == 0
    try:
        _composite_checks(ilw, L)
    finally:
        L.ilwdetr_validate_only(0)


def _composite_checks(ilw, L):
    B, T, d, H, F = 2, 1600, 384, 6, 1536

    def block(**over):
        bp = ilw.BlockParamsT()
        _fake_ptrs(bp, 0x7000000)
        bp.struct_size = ctypes.sizeof(ilw.BlockParamsT)
        bp.d, bp.H, bp.F, bp.win_side, bp.ln_iters = d, H, F, 2, 10
        bp.smx = ilw.ShiftmaxT(3000, 16, 8, -1, 4, 31)
        bp.gelu = ilw.GeluT(600, 16, 8)
        bp.m_o, bp.s_o, bp.m_r1, bp.s_r1, bp.m_g, bp.s_g, bp.m_r2, bp.s_r2 = (1 << 30, 34) * 4
        for k, val in over.items():
            setattr(bp, k, val)
        ws = L.ilwdetr_block_workspace_bytes(B, T, d, F)
        return L.ilwdetr_block_forward(ctypes.byref(bp), ctypes.c_void_p(0x100000), ctypes.c_void_p(0x200000),
                                       B, T, ctypes.c_void_p(0x300000), ws, None)

    assert block() == 0  # every step's arguments pass
    assert block(smx=ilw.ShiftmaxT(0, 16, 8, -1, 4, 31)) == -1 and b"I0" in L.ilwdetr_last_error()
    assert block(gelu=ilw.GeluT(1 << 15, 16, 8)) == -1
    assert block(s_r2=63) == -1 and b"residual" in L.ilwdetr_last_error()
    assert block(s_g=0) == -1
    assert block(win_side=7) == -1 and b"window" in L.ilwdetr_last_error()  # 40 x 40 grid, 7 does not divide 40

    lvl = (ctypes.c_int32 * 6)(80, 80, 40, 40, 20, 20)
    Bd, Q, dd, Hd, Fd, Ld, Pd = 2, 300, 256, 8, 1024, 3, 4

    def decoder(**over):
        dp = ilw.DecoderParamsT()
        _fake_ptrs(dp, 0x9000000)
        dp.struct_size = ctypes.sizeof(ilw.DecoderParamsT)
        dp.d, dp.H, dp.F, dp.L, dp.P, dp.ln_iters = dd, Hd, Fd, Ld, Pd, 20
        for name, typ in ilw.DecoderParamsT._fields_:
            if typ is ctypes.c_int32 and name.startswith("s_"):
                setattr(dp, name, 34)
            elif typ is ctypes.c_int32 and name.startswith("m_"):
                setattr(dp, name, 1 << 30)
        dp.smx = ilw.ShiftmaxT(3000, 16, 8, -1, 4, 31)
        dp.smx_w = ilw.ShiftmaxT(3000, 16, 8, -1, 4, 31)
        dp.gelu = ilw.GeluT(600, 16, 8)
        for k, val in over.items():
            setattr(dp, k, val)
        ws = L.ilwdetr_decoder_workspace_bytes(Bd, Q, 8400, dd, Fd, Hd, Ld, Pd)
        return L.ilwdetr_decoder_layer_forward(ctypes.byref(dp), ctypes.c_void_p(0x100000), ctypes.c_void_p(0x200000),
                                               ctypes.c_void_p(0x300000), lvl, Ld, ctypes.c_void_p(0x400000), Bd, Q,
                                               ctypes.c_void_p(0x500000), ctypes.c_void_p(0x600000), ws, None)

    assert decoder() == 0
    assert decoder(smx_w=ilw.ShiftmaxT(0, 16, 8, -1, 4, 31)) == -1  # the deformable weights, late in the layer
    assert decoder(s_s=0) == -1 and b"deform" in L.ilwdetr_last_error()
    assert decoder(gelu=ilw.GeluT(1 << 15, 16, 8)) == -1
    assert decoder(s_r3=63) == -1

    def patch(Wp=0x200000, s_pos=10):
        ws = L.ilwdetr_patch_embed_workspace_bytes(2, 3, 640, 640, 16)
        return L.ilwdetr_patch_embed(ctypes.c_void_p(0x100000), 2, 3, 640, 640, 16, ctypes.c_void_p(Wp),
                                     ctypes.c_void_p(0x300000), ctypes.c_void_p(0x400000), ctypes.c_void_p(0x500000),
                                     384, ctypes.c_void_p(0x600000), 1 << 30, s_pos, ctypes.c_void_p(0x700000),
                                     ctypes.c_void_p(0x800000), ws, None)

    assert patch() == 0
    assert patch(Wp=0x200010) == -1 and b"256-byte" in L.ilwdetr_last_error()  # the GEMM's check, before the gather
    assert patch(s_pos=63) == -1 and b"residual" in L.ilwdetr_last_error()


def test_int8_tcgen05_mma_is_not_available_on_sm103a(tmp_path):
    """The reason the integer GEMMs and attention run on kind::f16 (int8 values carried exactly in
    fp16, fp32 accumulation kept below 2^24): ptxas of this toolkit rejects the int8 tensor-core
    MMA for sm_103a while accepting the fp16 form.  Compiles a one-instruction kernel of each kind."""
    from paper_2607_24981_gb300 import build

    def compile_kind(kind):
        src = tmp_path / f"probe_{kind}.cu"
        src.write_text(
            "#include <cstdint>\n"
            "__global__ void k(uint32_t d, uint64_t a, uint64_t b, uint32_t i) {\n"
            "  asm volatile(\"{\\n .reg .pred p;\\n setp.ne.b32 p, %4, 0;\\n"
            f" tcgen05.mma.cta_group::1.kind::{kind} [%0], %1, %2, %3, p;\\n}}\\n\""
            " :: \"r\"(d), \"l\"(a), \"l\"(b), \"r\"(i), \"r\"(1u) : \"memory\");\n}\n")
        import subprocess

        r = subprocess.run([build.nvcc()] + build.ARCH + ["-c", str(src), "-o", str(tmp_path / f"{kind}.o")],
                           capture_output=True, text=True)
        return r.returncode, r.stdout + r.stderr

    rc16, _ = compile_kind("f16")
    rc8, msg = compile_kind("i8")
    assert rc16 == 0
    assert rc8 != 0 and "kind::i8" in msg and "sm_103a" in msg, msg


def test_empty_extents_return_ok_without_a_launch(built_lib):
    """A call whose batch, row, token or element count is 0 checks its scalar parameters and
    returns ILW_OK without launching anything (its tensor pointers may be NULL), so it also
    succeeds on a machine without a device."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    smx = ctypes.byref(ilw.ShiftmaxT(100, 16, 8, -1, 4, 31))
    g = ctypes.byref(ilw.GeluT(600, 16, 8))
    calls = {
        "gemm_requant M=0": lambda: L.ilwdetr_gemm_requant(None, 16, None, None, None, None, 0, 4, 16, 8, None, 4, None, None),
        "gemm_requant N=0": lambda: L.ilwdetr_gemm_requant(None, 16, None, None, None, None, 4, 0, 16, 8, None, 4, None, None),
        "gemm_gelu M=0": lambda: L.ilwdetr_gemm_gelu(None, 16, None, None, None, None, 0, 4, 16, g, 1 << 30, 31, None, 4, None),
        "shiftmax_rows rows=0": lambda: L.ilwdetr_shiftmax_rows(None, 4, 0, 4, smx, None, 4, None),
        "shiftmax_rows len=0": lambda: L.ilwdetr_shiftmax_rows(None, 4, 4, 0, smx, None, 4, None),
        "sdshiftgelu n=0": lambda: L.ilwdetr_sdshiftgelu(None, None, 0, g, None),
        "int_layernorm rows=0": lambda: L.ilwdetr_int_layernorm(None, 16, 64, 0, 64, None, None, None, 10, None, 8, 64, None),
        "shiftmax_attn B=0": lambda: L.ilwdetr_shiftmax_attn(None, None, None, 192, 8, 0, 64, 3, 64, 0, smx, 1 << 30, 31,
                                                             None, 8, 192, None),
        "shiftmax_attn T=0": lambda: L.ilwdetr_shiftmax_attn(None, None, None, 192, 8, 1, 0, 3, 64, 0, smx, 1 << 30, 31,
                                                             None, 8, 192, None),
        "int_sigmoid n=0": lambda: L.ilwdetr_int_sigmoid(None, None, 0, ctypes.byref(ilw.SigmoidT(1024, 8, 17)), None),
        "relu_i8 n=0": lambda: L.ilwdetr_relu_i8(None, None, 0, None),
        "topk rows=0": lambda: L.ilwdetr_topk(None, 10, 0, 10, 3, None, None, None),
        "gather_rows n=0": lambda: L.ilwdetr_gather_rows(None, 16, 5, None, 0, 16, None, 16, None),
        "requant rows=0": lambda: L.ilwdetr_requant(None, 16, 16, 0, 16, 1 << 30, 30, None, 0, 1, 0, 1, 8, None, 16, None),
        "resample_nearest B=0": lambda: L.ilwdetr_resample_nearest(None, 100, 0, 10, 10, 16, None, 400, 20, 20, None),
        "ivit_shiftgelu rows=0": lambda: L.ilwdetr_ivit_shiftgelu(None, 8, 0, 8, None, 8, g, None),
        "patch_embed B=0": lambda: L.ilwdetr_patch_embed(None, 0, 3, 640, 640, 16, None, None, None, None, 384, None,
                                                         1 << 30, 31, None, None, 0, None),
        "patch_embed_noalloc B=0": lambda: L.ilwdetr_patch_embed_noalloc(None, 0, 3, 640, 640, 16, None, None, None, None,
                                                                         384, None, 1 << 30, 31, None, None),
        "pack_weight N=0": lambda: L.ilwdetr_pack_weight(None, 0, 16, None, None),
    }
    for name, call in calls.items():
        assert call() == 0, (name, L.ilwdetr_last_error())


def test_product_fails_loudly_without_the_library(monkeypatch):
    """With libilwdetr.so absent the binding raises instead of computing anything elsewhere: there
    is no CPU fallback."""
    import paper_2607_24981_gb300 as ilw

    monkeypatch.setattr(ilw, "_lib", None)
    monkeypatch.setattr(ilw, "LIB_PATH", os.path.join(os.path.dirname(ilw.LIB_PATH), "absent", "libilwdetr.so"))
    with pytest.raises(ilw.IlwError, match="missing"):
        ilw.lib()


def test_product_sources_never_reach_the_oracle():
    """The product package and the C-ABI header neither import, link nor name the oracle."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    pkg = os.path.join(root, "paper_2607_24981_gb300")
    files = [os.path.join(dp, f) for dp, _, fs in os.walk(pkg) for f in fs if f.endswith((".py", ".cu", ".cuh", ".h"))]
    files.append(os.path.join(root, "include", "ilwdetr.h"))
    assert len(files) > 10
    for path in files:
        text = open(path).read()
        for needle in ("import oracle", "from oracle", "ilw_oracle", "libilw_oracle"):
            assert needle not in text, (path, needle)


def test_oracle_sources_never_reach_the_product():
    """The oracle (Python wrapper and C++ source) neither imports nor links the product package or
    its CUDA library; tests hand it the same seeded arrays they hand the GPU path."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    odir = os.path.join(root, "oracle")
    files = [os.path.join(odir, f) for f in os.listdir(odir) if f.endswith((".py", ".cpp", ".h"))]
    assert len(files) >= 3
    for path in files:
        text = open(path).read()
        for needle in ("paper_2607_24981_gb300", "libilwdetr", "ilwdetr.h", "cuda"):
            assert needle not in text, (path, needle)


def test_validate_only_mode_checks_without_launching(built_lib):
    """In validate-only mode every launching entry point runs its usual checks and returns ILW_OK
    (or the error found) without launching: valid calls on fake, aligned addresses succeed and bad
    ones still fail, on any machine."""
    import paper_2607_24981_gb300 as ilw

    L = ilw.lib()
    v, w = ctypes.c_void_p(0x100000), ctypes.c_void_p(0x200000)
    smx = ctypes.byref(ilw.ShiftmaxT(3000, 16, 8, -1, 4, 31))
    g = ctypes.byref(ilw.GeluT(600, 16, 8))
    sg = ctypes.byref(ilw.SigmoidT(1024, 8, 17))
    assert L.ilwdetr_validate_only(1) == 0
    try:
        ok = {
            "pack_weight": L.ilwdetr_pack_weight(v, 64, 64, w, None),
            "gemm_requant": L.ilwdetr_gemm_requant(v, 64, w, v, v, v, 100, 64, 64, 8, v, 64, None, None),
            "gemm_gelu": L.ilwdetr_gemm_gelu(v, 64, w, v, v, v, 100, 64, 64, g, 1 << 30, 35, v, 64, None),
            "shiftmax_rows": L.ilwdetr_shiftmax_rows(v, 400, 10, 400, smx, w, 400, None),
            "sdshiftgelu": L.ilwdetr_sdshiftgelu(v, w, 1000, g, None),
            "int_layernorm": L.ilwdetr_int_layernorm(v, 16, 384, 10, 384, v, v, v, 10, w, 8, 384, None),
            "shiftmax_attn": L.ilwdetr_shiftmax_attn(v, v, v, 192, 8, 1, 64, 3, 64, 0, smx, 1 << 30, 35, w, 8, 192, None),
            "requant": L.ilwdetr_requant(v, 16, 64, 10, 64, 1 << 30, 30, None, 0, 1, 0, 1, 8, w, 64, None),
            "resample": L.ilwdetr_resample_nearest(v, 100, 1, 10, 10, 16, w, 400, 20, 20, None),
            "int_sigmoid": L.ilwdetr_int_sigmoid(v, w, 100, sg, None),
            "relu_i8": L.ilwdetr_relu_i8(v, w, 100, None),
            "topk": L.ilwdetr_topk(v, 100, 2, 100, 10, w, v, None),
            "gather_rows": L.ilwdetr_gather_rows(v, 16, 10, w, 5, 16, v, 16, None),
            "ivit_shiftgelu": L.ilwdetr_ivit_shiftgelu(v, 64, 4, 64, w, 64, g, None),
            "patch_embed_noalloc": L.ilwdetr_patch_embed_noalloc(v, 2, 3, 640, 640, 16, w, v, v, v, 384, None,
                                                                 1 << 30, 31, ctypes.c_void_p(0x300000), None),
        }
        assert all(rc == 0 for rc in ok.values()), ok
        # the checks themselves still run
        assert L.ilwdetr_gemm_requant(v, 24, w, v, v, v, 100, 64, 24, 8, v, 64, None, None) == -2  # K % 16
        assert L.ilwdetr_topk(v, 100, 2, 100, 101, w, v, None) == -1  # K > N
        assert L.ilwdetr_patch_embed_noalloc(v, 7, 3, 640, 640, 16, w, v, v, v, 384, None, 1 << 30, 31,
                                             ctypes.c_void_p(0x300000), None) == -2  # beyond the 8 MiB scratch
    finally:
        L.ilwdetr_validate_only(0)
