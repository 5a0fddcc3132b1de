"""The bounded-wait path of the kernels, exercised without a fault: with the test hook
ilwdetr_debug_gemm_wait the GEMM producer skips one operand load, so the MMA warp's wait for it
never completes; the wait runs out after about a millisecond, the kernel latches the device status
word, drains what it issued, frees its tensor memory and returns.  ilwdetr_device_status must report
ILW_ERR_TIMEOUT, and the next call (hook off) must be bit-exact against the oracle."""
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


@pytest.mark.parametrize("a_form", ["int8", "fp16"])
def test_gemm_wait_runs_out_then_recovers(ilw, orc, a_form):
    M, N, K = 256, 256, 256
    A = synth.uniform_int(90, "to.A", (M, K), -127, 127, np.int8)
    W, b, m, s = synth.gemm_params(90, "to.W", N, K, 40.0, 40.0)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()  # noqa: E731
    Ad = dev(A.astype(np.float16)) if a_form == "fp16" else dev(A)
    Wp = ilw.pack_weight(dev(W))
    bd, md, sd = dev(b), dev(m), dev(s)
    L = ilw.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert L.ilwdetr_device_status(stream) == 0
    assert L.ilwdetr_debug_gemm_wait(0, 2_000_000) == 0  # skip K block 0 of the first tile, ~1 ms bound
    try:
        ilw.gemm(Ad, Wp, N, bd, md, sd, 8)  # the launch itself succeeds
        rc = L.ilwdetr_device_status(stream)
        assert rc == -4, (rc, L.ilwdetr_last_error())
        assert b"bounded wait" in L.ilwdetr_last_error()
    finally:
        assert L.ilwdetr_debug_gemm_wait(-1, 0) == 0
    # the context is usable and the next call is exact
    got = ilw.gemm(Ad, Wp, N, bd, md, sd, 8)
    assert L.ilwdetr_device_status(stream) == 0
    want = orc.gemm_requant(A, W, b, m, s, 8)
    assert np.array_equal(got.cpu().numpy().astype(np.int32), want)
