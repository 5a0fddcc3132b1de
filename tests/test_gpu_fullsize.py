"""Parity at the workloads' full sizes, in the launch configuration bench.py times.

The GPU runs the whole batch / tensor; the oracle checks sampled outputs it can compute one by
one: whole images (images are independent through the encoder) and sampled rows / elements of
the nonlinearity sweep.  Bit-exact everywhere."""
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


def same(got, want, what):
    got, want = np.asarray(got), np.asarray(want).astype(np.asarray(got).dtype)
    bad = np.argwhere(got != want)
    assert len(bad) == 0, f"{what}: {len(bad)} mismatches, first {tuple(bad[0])}"


@pytest.mark.parametrize("workload", ["medium_backbone_b8", "tiny_backbone_b8"])
def test_backbone_full_batch_sampled_images(ilw, orc, workload):
    """Full batch of 8 images through the whole backbone on the GPU (Backbone.forward, the call
    bench.py times); the oracle recomputes one sampled image end to end."""
    cfg = synth.CONFIGS[workload]
    B, T, d = cfg["B"], cfg["T"], cfg["d"]
    blocks = synth.backbone_params(0, cfg)
    pe = synth.patch_embed_params(0, d, mode=cfg["mode"])
    img = synth.image_input(0, B)
    bb = ilw.Backbone(pe, blocks, B)
    dimg = dev(img)
    y = bb.forward(dimg)
    torch.cuda.synchronize()
    ilw.device_status()
    yh = y.cpu().numpy().reshape(B, T, d)
    # the same forward recorded as a CUDA graph (Backbone.capture, the step bench.py replays):
    # identical bytes, on a fresh input too
    g = bb.capture(dimg)
    same(g.replay().cpu().numpy().reshape(B, T, d), yh, f"{workload} graph replay")
    img2 = synth.image_input(1, B)
    dimg.copy_(dev(img2))
    y2g = g.replay().cpu().numpy()
    y2 = bb.forward(dimg).cpu().numpy()
    same(y2g, y2, f"{workload} graph replay, second input")
    assert not np.array_equal(y2, yh.reshape(y2.shape))
    pick = 5 if workload == "medium_backbone_b8" else 2
    x = orc.patch_embed(img[pick:pick + 1], pe["p"], pe["w"], pe["b"], pe["m"], pe["s"], pe["pos"],
                        pe["m_pos"], pe["s_pos"])
    for bp in blocks:
        x = orc.block_forward(bp, x, 1, T)
    same(yh[pick], x, f"{workload} image {pick}")
    # the activations stay in range (no collapse to saturation or to zero)
    assert 10 < float(np.abs(yh).mean()) < 20000


def test_patch_embed_full_batch(ilw, orc):
    B, d = 16, 384
    pe = synth.patch_embed_params(1, d)
    img = synth.image_input(1, B)
    Wp = ilw.pack_weight(dev(pe["w"]))
    x0 = ilw.patch_embed(dev(img), 16, Wp, d, dev(pe["b"]), dev(pe["m"]), dev(pe["s"]), dev(pe["pos"]),
                         pe["m_pos"], pe["s_pos"]).cpu().numpy().reshape(B, 1600, d)
    for i in (0, 11):
        want = orc.patch_embed(img[i:i + 1], 16, pe["w"], pe["b"], pe["m"], pe["s"], pe["pos"], pe["m_pos"], pe["s_pos"])
        same(x0[i], want, f"patch embed image {i}")


@pytest.mark.parametrize("L", [64, 400, 1600])
def test_shiftmax_rows_sweep_sampled(ilw, orc, L):
    """2^27 int32 scores uniform in [-2^15, 2^15] as rows of length L; 4096 rows checked."""
    rows = (1 << 27) // L
    X = synth.uniform_int(30, f"c3smx{L}", (rows, L), -(1 << 15), 1 << 15)
    I0 = int(synth.uniform_int(30, f"c3I0{L}", (1,), 1 << 11, 1 << 13)[0])
    P = ilw.shiftmax_rows(dev(X), {"I0": I0}).cpu().numpy()
    idx = np.unique(synth.uniform_int(31, f"pick{L}", (4096,), 0, rows - 1))
    idx = np.concatenate([idx, [0, rows - 1]])
    want, *_ = orc.shiftmax_rows(X[idx], I0)
    same(P[idx], want, f"shiftmax L={L}")


def test_sdshiftgelu_sweep_sampled(ilw, orc):
    """2^28 int32 values uniform in [-2^12, 2^12]; 2^20 sampled elements checked."""
    n = 1 << 28
    X = synth.uniform_int(32, "c3gelu", (n,), -(1 << 12), 1 << 12)
    I0 = int(synth.uniform_int(32, "c3gI0", (1,), 1 << 8, 1 << 10)[0])
    Y = ilw.sdshiftgelu(dev(X), {"I0": I0}).cpu().numpy()
    idx = synth.uniform_int(33, "gpick", (1 << 20,), 0, n - 1).astype(np.int64)
    same(Y[idx], orc.sdshiftgelu(X[idx], I0), "gelu c3")
    same(Y[-1000:], orc.sdshiftgelu(X[-1000:], I0), "gelu c3 tail")


@pytest.mark.parametrize("C", [192, 384])
def test_layernorm_sweep_sampled(ilw, orc, C):
    """2^20 rows of dim C, int32 uniform in [-2^14, 2^14]; 2048 rows checked."""
    rows = 1 << 20
    X = synth.uniform_int(34, f"c3ln{C}", (rows, C), -(1 << 14), 1 << 14)
    beta, mult, shift = synth.ln_params(34, f"c3lnp{C}", C)
    Y = ilw.int_layernorm(dev(X), dev(beta), dev(mult), dev(shift), 10, 8).cpu().numpy()
    idx = np.unique(synth.uniform_int(35, f"lpick{C}", (2048,), 0, rows - 1))
    same(Y[idx], orc.int_layernorm(X[idx], beta, mult, shift, 10, 8), f"ln C={C}")
