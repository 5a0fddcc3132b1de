"""Bit-exact parity of the detection head and the two-stage query selection with the CPU oracle:
the integer sigmoid over the whole int32 range, ReLU on int8, per-row top-K (ties, extremes,
K = N, the encoder's 8400 tokens), row gather (and its out-of-range report), and the two
compositions at the detector's sizes (300 queries per image, 8400 memory tokens, 80 classes)."""
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


def same(got, want, what):
    got, want = np.asarray(got), np.asarray(want).astype(np.asarray(got).dtype)
    bad = np.argwhere(got != want)
    assert len(bad) == 0, f"{what}: {len(bad)} mismatches, first {tuple(bad[0])}"


@pytest.mark.parametrize("I0,k_inter,k_out", [(1024, 8, 17), (18764, 8, 8), (3, 16, 24), (32767, 0, 1)])
def test_int_sigmoid(ilw, orc, I0, k_inter, k_out):
    n = 100003  # a ragged tail after the 4-wide vectors
    X = synth.uniform_int(70, f"sig{I0}", (n,), -(1 << 31), (1 << 31) - 1)
    X[:9] = [0, 1, -1, np.iinfo(np.int32).min, np.iinfo(np.int32).max, I0, -I0, 1 << 30, -(1 << 30)]
    X[9:40009] = synth.uniform_int(71, f"sigs{I0}", (40000,), -20 * I0, 20 * I0)  # the informative range
    got = ilw.int_sigmoid(dev(X), {"I0": I0, "k_inter": k_inter, "k_out": k_out})
    same(host(got), orc.int_sigmoid(X, I0, k_inter, k_out), f"int_sigmoid I0={I0}")


def test_relu_i8(ilw):
    X = synth.uniform_int(72, "relu", (4099,), -128, 127, np.int8)
    X[:3] = [-128, 0, 127]
    same(host(ilw.relu_i8(dev(X))), np.maximum(X, 0), "relu")
    t = dev(X)
    ilw.relu_i8(t, out=t)  # in place
    same(host(t), np.maximum(X, 0), "relu in place")


@pytest.mark.parametrize("rows,N,K,lo,hi", [(3, 1, 1, -5, 5), (700, 80, 1, -(1 << 20), 1 << 20),
                                            (2, 8400, 300, -(1 << 24), 1 << 24), (4, 1000, 1000, -3, 3),
                                            (1, 16384, 16384, -(1 << 31), (1 << 31) - 1), (5, 333, 17, -2, 2)])
def test_topk(ilw, orc, rows, N, K, lo, hi):
    S = synth.uniform_int(73, f"topk{rows}.{N}", (rows, N), lo, hi)
    if N >= 4:
        S[0, :4] = [np.iinfo(np.int32).min, np.iinfo(np.int32).max, np.iinfo(np.int32).max, 0]
    v, i = ilw.topk(dev(S), K)
    wv, wi = orc.topk(S, K)
    same(host(i), wi, f"topk idx {rows}x{N} K={K}")
    same(host(v), wv, f"topk values {rows}x{N} K={K}")


def test_gather_rows(ilw, orc):
    X = synth.uniform_int(74, "gather", (1000, 6), -(1 << 30), 1 << 30)
    idx = synth.uniform_int(75, "gather.i", (777,), 0, 999)
    same(host(ilw.gather_rows(dev(X), dev(idx))), orc.gather_rows(X, idx), "gather")
    ilw.device_status()  # raises if the kernel latched an out-of-range index


def test_gather_rows_reports_an_index_past_the_source(ilw):
    """The kernel's own bounds check: a zero row, and the next device_status says so."""
    X = dev(np.arange(40, dtype=np.int32).reshape(10, 4))
    idx = dev(np.array([3, 10, -1, 9], dtype=np.int32))
    got = host(ilw.gather_rows(X, idx))
    assert np.array_equal(got[[0, 3]], np.arange(40).reshape(10, 4)[[3, 9]])
    assert not got[[1, 2]].any()
    import ctypes

    rc = ilw.lib().ilwdetr_device_status(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == -1 and b"gather index" in ilw.lib().ilwdetr_last_error()
    ilw.device_status()  # read and cleared: raises if anything is still latched


def test_detection_head(ilw, orc):
    B, Q, d = 2, 300, 256
    hp = synth.head_params(8, d=d, C=80)
    out = synth.uniform_int(8, "dh.out", (B * Q, d), -127, 127, np.int8)
    ref = synth.uniform_int(8, "dh.ref", (B * Q, 4), -6000, 6000, np.int16)
    head = ilw.DetectionHead(hp)
    scores, boxes, z = head.forward(dev(out), dev(ref))
    ws, wb, wz = orc.detection_head(hp, out, ref)
    same(host(z), wz, "box logits")
    same(host(boxes), wb, "boxes")
    same(host(scores), ws, "scores")


def test_two_stage(ilw, orc):
    B, K, d = 2, 300, 256
    levels = ((80, 80), (40, 40), (20, 20))
    S = sum(h * w for h, w in levels)
    tp = synth.two_stage_params(9, d=d, C=80, levels=levels)
    mem = synth.uniform_int(9, "ts.mem", (B * S, d), -127, 127, np.int8)
    ts = ilw.TwoStage(tp)
    vals, idx, ref16, boxes = ts.forward(dev(mem), B, S, K)
    wv, wi, wr, wb = orc.two_stage(tp, mem, B, S, K)
    same(host(idx), wi, "selected tokens")
    same(host(vals), wv, "selected values")
    same(host(ref16), wr, "reference logits")
    same(host(boxes), wb, "reference boxes")


@pytest.mark.parametrize("rows,L,I0,k_inter", [(300, 1536, 600, 16), (7, 1000, 1000, 8), (1, 5, 3, 16),
                                               (64, 64, 20000, 0)])
def test_ivit_shiftgelu(ilw, orc, rows, L, I0, k_inter):
    X = synth.uniform_int(76, f"ivit{L}", (rows, L), -4 * I0, 4 * I0)
    X[0, 0] = 40 * I0  # an outlier that drives the row maximum
    if L >= 4:
        X[-1, :4] = [(1 << 24) - 1, -(1 << 24) + 1, 0, -1]  # the domain's extremes (k_out 8)
    got = ilw.ivit_shiftgelu(dev(X), {"I0": I0, "k_inter": k_inter, "k_out": 8})
    same(host(got), orc.ivit_shiftgelu(X, I0, k_inter, 8), f"ivit shiftgelu {rows}x{L}")
