"""Bit-exact parity of the detector path (projector and decoder) with the CPU oracle: the
requantisation and resampling entry points element by element, the projector and one decoder
layer at the full detector's level sizes, and the whole detector forward (640x640, batch 16:
backbone, projector, 3 decoder layers) on the GPU with one sampled image recomputed by the
oracle end to end."""
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


@pytest.mark.parametrize("in_bits,out_bits,with_z", [(16, 8, True), (16, 8, False), (16, 16, False),
                                                      (16, 32, False), (32, 8, True), (32, 16, True)])
def test_requant(ilw, orc, in_bits, out_bits, with_z):
    rows, C = 333, 264
    lo, hi = (-32767, 32767) if in_bits == 16 else (-(1 << 24), 1 << 24)
    X = synth.uniform_int(60, f"rq.x{in_bits}", (rows, C), lo, hi, np.int16 if in_bits == 16 else np.int32)
    X[0, :8] = [lo, hi, 0, 1, -1, lo + 1, hi - 1, 2]
    Z = synth.uniform_int(61, "rq.z", (3, C), -32767, 32767, np.int16) if with_z else None
    m1, s1, m2, s2 = 1987654321, 38 if out_bits != 32 else 31, 1234567890, 40
    got = ilw.requant(dev(X), m1, s1, None if Z is None else dev(Z), m2, s2, out_bits)
    want = orc.requant(X, m1, s1, Z, m2, s2, out_bits)
    same(host(got), want, f"requant {in_bits}->{out_bits}")


def test_resample_nearest(ilw, orc):
    B, g, C = 3, 40, 256
    X = synth.uniform_int(62, "rs.x", (B * g * g, C), -127, 127, np.int8)
    for Ho, Wo in ((80, 80), (40, 40), (20, 20), (13, 27)):
        same(host(ilw.resample_nearest(dev(X), B, g, g, Ho, Wo)), orc.resample_nearest(X, B, g, g, Ho, Wo),
             f"resample {Ho}x{Wo}")


def test_projector(ilw, orc):
    cfg = synth.CONFIGS["medium_detector_b16"]
    B, g, K = 2, cfg["grid"], 384
    pp = synth.projector_params(0, 4, K)
    taps = [synth.uniform_int(63 + i, "pj.tap", (B * g * g, K), -3000, 3000, np.int16) for i in range(4)]
    proj = ilw.Projector(pp, B, g, cfg["levels"], K)
    got = host(proj.forward([dev(t) for t in taps]))
    want = orc.projector(pp, taps, B, g, cfg["levels"])
    same(got, want, "projector memory")


@pytest.mark.parametrize("B,Q", [(2, 300), (1, 37)])
def test_decoder_layer(ilw, orc, B, Q):
    cfg = synth.CONFIGS["medium_detector_b16"]
    levels = cfg["levels"]
    S = sum(h * w for h, w in levels)
    dp = synth.decoder_params(0, 1)
    inp = synth.decoder_inputs(0, B, Q)
    mem = synth.laplace_int(0, "dec.mem", (B * S, 256), 20.0, 127, np.int8)
    dw = ilw.DecoderWeights(dp)
    ws = torch.empty(ilw.decoder_workspace_bytes(B, Q, S, 256, dp["F"], dp["H"], dp["L"], dp["P"]),
                     dtype=torch.uint8, device="cuda")
    got = ilw.decoder_layer_forward(dw, dev(inp["tgt"]), dev(inp["pos"]), dev(mem), levels, dev(inp["refs"]), B, Q,
                                    ws)
    want = orc.decoder_layer(dp, inp["tgt"], inp["pos"], mem, levels, inp["refs"], B, Q)
    same(host(got), want, f"decoder layer B={B} Q={Q}")
    ilw.device_status()


def test_detector_full_batch_sampled_image(ilw, orc):
    """The full integer detector forward at its workload size (batch 16) on the GPU; the oracle
    recomputes one image end to end (patch embedding, 10 blocks, the four taps, projector, three
    decoder layers)."""
    cfg = synth.CONFIGS["medium_detector_b16"]
    bb = synth.CONFIGS[cfg["backbone"]]
    B, Q, g = cfg["B"], cfg["Q"], cfg["grid"]
    blocks = synth.backbone_params(0, bb)
    pe = synth.patch_embed_params(0, bb["d"], mode=bb["mode"])
    pp = synth.projector_params(0, len(cfg["taps"]), bb["d"], cfg["N"])
    dps = [synth.decoder_params(0, i) for i in range(cfg["dec_layers"])]
    inp = synth.decoder_inputs(0, B, Q)
    img = synth.image_input(0, B)
    det = ilw.Detector(pe, blocks, cfg["taps"], pp, dps, B, Q, cfg["levels"], g)
    out = host(det.forward(dev(img), dev(inp["tgt"]), dev(inp["pos"]), dev(inp["refs"])))
    ilw.device_status()
    pick = 11
    x = orc.patch_embed(img[pick:pick + 1], pe["p"], pe["w"], pe["b"], pe["m"], pe["s"], pe["pos"], pe["m_pos"],
                        pe["s_pos"])
    taps = {}
    for i, bp in enumerate(blocks):
        x = orc.block_forward(bp, x, 1, bb["T"])
        if i in cfg["taps"]:
            taps[i] = x
    mem = orc.projector(pp, [taps[i] for i in cfg["taps"]], 1, g, cfg["levels"])
    r = slice(pick * Q, (pick + 1) * Q)
    t = inp["tgt"][r]
    for dp in dps:
        t = orc.decoder_layer(dp, t, inp["pos"][r], mem, cfg["levels"], inp["refs"][pick:pick + 1], 1, Q)
    same(out[r], t, f"detector image {pick}")
    assert 10 < float(np.abs(out.astype(np.int64)).mean()) < 30000


def test_detector_two_stage_refinement_and_head_sampled_image(ilw, orc):
    """The detector with two-stage query selection (the decoder's reference points from the top-300
    memory tokens, its positional queries by the learnable projection of their boxes), the reference
    boxes refined after each decoder layer but the last, and the detection head (class scores,
    boxes) at batch 2; the oracle recomputes one image end to end (backbone, projector, two-stage
    selection, three decoder layers with refinement and positional queries, head)."""
    cfg = synth.CONFIGS["medium_detector_b16"]
    bb = synth.CONFIGS[cfg["backbone"]]
    B, Q, g = 2, cfg["Q"], cfg["grid"]
    blocks = synth.backbone_params(0, bb)
    pe = synth.patch_embed_params(0, bb["d"], mode=bb["mode"])
    pp = synth.projector_params(0, len(cfg["taps"]), bb["d"], cfg["N"])
    dps = [synth.decoder_params(0, i) for i in range(cfg["dec_layers"])]
    tsp = synth.two_stage_params(3, d=cfg["N"], C=80, levels=cfg["levels"])
    hp = synth.head_params(3, d=cfg["N"], C=80)
    pq = synth.query_pos_params(3, d=cfg["N"])
    rps = synth.refine_params(3, cfg["dec_layers"] - 1, d=cfg["N"])
    inp = synth.decoder_inputs(1, B, Q)
    img = synth.image_input(1, B)
    det = ilw.Detector(pe, blocks, cfg["taps"], pp, dps, B, Q, cfg["levels"], g, tsp=tsp, hp=hp, pq=pq, rps=rps)
    x, scores, boxes = det.forward(dev(img), dev(inp["tgt"]))
    x, scores, boxes = host(x), host(scores), host(boxes)
    ilw.device_status()
    pick = 1
    xo = orc.patch_embed(img[pick:pick + 1], pe["p"], pe["w"], pe["b"], pe["m"], pe["s"], pe["pos"], pe["m_pos"],
                         pe["s_pos"])
    taps = {}
    for i, bp in enumerate(blocks):
        xo = orc.block_forward(bp, xo, 1, bb["T"])
        if i in cfg["taps"]:
            taps[i] = xo
    mem = orc.projector(pp, [taps[i] for i in cfg["taps"]], 1, g, cfg["levels"])
    S = mem.shape[0]
    _, _, ref16, bx = orc.two_stage(tsp, mem, 1, S, Q)
    r = slice(pick * Q, (pick + 1) * Q)
    t, ref_last = orc.decoder_stack(dps, inp["tgt"][r], mem, cfg["levels"], ref16, bx, 1, Q, pq=pq, rps=rps)
    same(x[r], t, f"decoder output image {pick}")
    assert not np.array_equal(ref_last, ref16)  # the references did move
    a = orc.requant(t, hp["m_in"], hp["s_in"], out_bits=8)
    ws, wb, _ = orc.detection_head(hp, a, ref_last)
    same(scores[r], ws, f"scores image {pick}")
    same(boxes[r], wb, f"boxes image {pick}")


def test_query_pos(ilw, orc):
    M = 600
    pq = synth.query_pos_params(5)
    boxes = synth.uniform_int(5, "qp.box", (M, 4), 0, 1 << 16)
    boxes[:3] = [[0, 0, 0, 0], [1 << 16, 1 << 16, 1 << 16, 1 << 16], [32768, 1, 65535, 2]]
    qp = ilw.QueryPos(pq, M)
    same(host(qp.forward(dev(boxes))), orc.query_pos(pq, boxes), "query pos")
