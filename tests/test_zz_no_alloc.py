"""ilwdetr_patch_embed_noalloc: the patch embedding for callers that cannot give the library any
device memory (a host runtime owning the whole memory budget, or a loop that cannot afford
cudaMalloc's synchronisation).  It keeps its scratch in a fixed array inside the library.

Called through the C-ABI on two calls in a row with different images (a stale scratch array from
the first call would show up in the second), and compared with the CPU oracle's patch embedding
and with ilwdetr_patch_embed (which takes a workspace).  This file is collected last on purpose."""
import ctypes

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


def _noalloc(ilw, img, p, Wp, d, pe, pos, out):
    B, Cin, Hh, Ww = img.shape
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return ilw.lib().ilwdetr_patch_embed_noalloc(
        ctypes.c_void_p(img.data_ptr()), B, Cin, Hh, Ww, p, ctypes.c_void_p(Wp.data_ptr()),
        ctypes.c_void_p(pe["b"].data_ptr()), ctypes.c_void_p(pe["m"].data_ptr()),
        ctypes.c_void_p(pe["s"].data_ptr()), d, ctypes.c_void_p(pos.data_ptr()), 1 << 30, 31,
        ctypes.c_void_p(out.data_ptr()), stream)


def test_noalloc_patch_embed_matches_oracle_and_workspace_version(ilw):
    import oracle

    d, p = 384, 16
    pe_h = synth.patch_embed_params(40, d)
    pe = {k: torch.from_numpy(np.ascontiguousarray(pe_h[k])).cuda() for k in ("w", "b", "m", "s", "pos")}
    Wp = ilw.pack_weight(pe["w"])
    for call, (seed, B) in enumerate(((41, 2), (42, 3))):
        img_h = synth.image_input(seed, B)
        img = torch.from_numpy(img_h).cuda()
        want = ilw.patch_embed(img, p, Wp, d, pe["b"], pe["m"], pe["s"], pe["pos"], 1 << 30, 31)
        got = torch.full_like(want, 12345)
        rc = _noalloc(ilw, img, p, Wp, d, pe, pe["pos"], got)
        assert rc == 0, ilw.lib().ilwdetr_last_error()
        torch.cuda.synchronize()
        ref = oracle.patch_embed(img_h, p, pe_h["w"], pe_h["b"], pe_h["m"], pe_h["s"], pe_h["pos"], 1 << 30, 31)
        got_h = got.cpu().numpy()
        assert np.array_equal(got_h, ref), f"call {call}: {(got_h != ref).sum()} mismatches against the oracle"
        assert torch.equal(got, want), f"call {call}: {(got != want).sum().item()} mismatches"


def test_noalloc_checks_arguments_before_launching(ilw):
    d, p = 64, 16
    w = torch.zeros((d, 768), dtype=torch.int8, device="cuda")
    Wp = ilw.pack_weight(w)
    pe = {k: torch.zeros(d, dtype=torch.int32, device="cuda") for k in ("b", "m", "s")}
    pos = torch.zeros((1600, d), dtype=torch.int16, device="cuda")
    img = torch.zeros((1, 3, 640, 640), dtype=torch.int8, device="cuda")
    out = torch.zeros((1600, d), dtype=torch.int16, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    L = ilw.lib()
    rc = L.ilwdetr_patch_embed_noalloc(ctypes.c_void_p(img.data_ptr()), 1, 3, 640, 640, p, None,
                                       ctypes.c_void_p(pe["b"].data_ptr()), ctypes.c_void_p(pe["m"].data_ptr()),
                                       ctypes.c_void_p(pe["s"].data_ptr()), d, ctypes.c_void_p(pos.data_ptr()),
                                       1 << 30, 31, ctypes.c_void_p(out.data_ptr()), stream)
    assert rc == -1 and b"packed weight" in L.ilwdetr_last_error()
    rc = L.ilwdetr_patch_embed_noalloc(ctypes.c_void_p(img.data_ptr()), 1, 3, 640, 640, p,
                                       ctypes.c_void_p(Wp.data_ptr()), ctypes.c_void_p(pe["b"].data_ptr()), None,
                                       ctypes.c_void_p(pe["s"].data_ptr()), d, ctypes.c_void_p(pos.data_ptr()),
                                       1 << 30, 31, ctypes.c_void_p(out.data_ptr()), stream)
    assert rc == -1 and b"mult/shift" in L.ilwdetr_last_error()
    torch.cuda.synchronize()
    assert int(out.abs().sum()) == 0  # nothing ran


def test_noalloc_rejects_batches_beyond_its_scratch(ilw):
    d, p = 64, 16
    limit = int(ilw.lib().ilwdetr_patch_embed_noalloc_max_bytes())
    assert limit == 8 << 20
    B = limit // (1600 * 3 * 256) + 1  # one image more than fits
    w = torch.zeros((d, 768), dtype=torch.int8, device="cuda")
    Wp = ilw.pack_weight(w)
    pe = {k: torch.zeros(d, dtype=torch.int32, device="cuda") for k in ("b", "m", "s")}
    pos = torch.zeros((1600, d), dtype=torch.int16, device="cuda")
    img = torch.zeros((B, 3, 640, 640), dtype=torch.int8, device="cuda")
    out = torch.empty((B * 1600, d), dtype=torch.int16, device="cuda")
    rc = _noalloc(ilw, img, p, Wp, d, pe, pos, out)
    assert rc == -2 and b"8 MiB" in ilw.lib().ilwdetr_last_error()
