"""Single-kernel workloads of the path, for timing and for profiler captures.

  python -m paper_2607_24981_gb300.cases <case> [--reps N] [--graph]

Each case builds its seeded inputs (shapes of the paper's Medium model and of the nonlinearity
sweep), runs the entry point `reps` times after 3 warm-up calls, each launch timed with CUDA
events, and prints the median (and minimum) device time with the case's algorithmic work; with
--graph the case is recorded as a CUDA graph and `reps` replays run back to back between one pair
of events (the mean per launch, free of the host's per-call marshalling, which otherwise shows in
launches of a few tens of microseconds).  Cases:
  attn_global   attention, 2 images x 1600 tokens, 6 heads, dh 64, global (fp16-carried q|k|v);
                --batch 8 gives the encoder's launch
  attn_window   attention, 8 images x 1600 tokens, 6 heads, 2x2 windows of 400
  heads         detection head (class sigmoid, 3-layer box MLP, box sigmoid), 16 x 300 queries
  two_stage     two-stage query selection, 16 images x 8400 memory tokens, top 300
  gemm_qkv / gemm_proj / gemm_fc1_gelu / gemm_fc2
                the block GEMMs at 12800 tokens, d 384, MLP 1536
  ln_encoder    I-LayerNorm on the int16 residual stream, 12800 x 384
  smx_64 / smx_400 / smx_1600
                Constrained Shiftmax over 2^27 int32 scores in rows of 64 / 400 / 1600
  gelu_2p28     SD-ShiftGELU over 2^28 int32 values
  ln_192 / ln_384
                I-LayerNorm over 2^20 int32 rows of dim 192 / 384
"""
from __future__ import annotations

import argparse
import json

import numpy as np

from . import synth


def _dev(a):
    import torch

    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def build(case: str, batch: int = 0):
    """Returns (fn, work dict) for a case; fn() launches the entry point once.  ``batch`` > 0
    overrides the number of images of the attention cases."""
    import torch

    import paper_2607_24981_gb300 as ilw

    ilw.lib()
    if case.startswith("attn"):
        B, T, H, dh = (2, 1600, 6, 64) if case == "attn_global" else (8, 1600, 6, 64)
        B = batch or B
        win = 0 if case == "attn_global" else 2
        # q|k|v as the QKV GEMM hands them over: the int8 values carried in float16
        qkv = _dev(synth.uniform_int(0, "case.qkv", (B * T, 3 * H * dh), -127, 127, np.int8).astype(np.float16))
        out = torch.empty((B * T, H * dh), dtype=torch.float16, device="cuda")  # the encoder's O form
        scores = B * H * (T * T if win == 0 else 4 * (T // 4) ** 2)
        return (lambda: ilw.shiftmax_attn(qkv, B, T, H, dh, win, {"I0": 6000}, 3 << 29, 36, out=out),
                {"scores": scores})
    if case.startswith("gemm"):
        M, d, F = 12800, 384, 1536
        N, K = {"gemm_qkv": (3 * d, d), "gemm_proj": (d, d), "gemm_fc1_gelu": (F, d), "gemm_fc2": (d, F),
                "gemm_fc2_i8": (d, F), "gemm_fc1_gelu_i8": (F, d)}[case]
        # the activations as the encoder hands them over: int8 values carried in fp16 (the _i8 cases:
        # plain int8, converted to the fp16 operand inside the GEMM)
        A8 = synth.uniform_int(1, "case.A", (M, K), -127, 127, np.int8)
        A = _dev(A8) if case.endswith("_i8") else _dev(A8.astype(np.float16))
        W, b, m, s = synth.gemm_params(1, "case.W", N, K, 40.0, 40.0)
        Wp = ilw.pack_weight(_dev(W))
        b, m, s = _dev(b), _dev(m), _dev(s)
        if case == "gemm_fc1_gelu":  # h written as fp16-carried int8, as the encoder block does
            out = torch.empty((M, N), dtype=torch.float16, device="cuda")
            fn = lambda: ilw.gemm(A, Wp, N, b, m, s, ilw.I8_IN_F16, gelu={"I0": 1000}, m_g=3 << 29, s_g=40, out=out)
        elif case == "gemm_fc1_gelu_i8":  # int8 a2 in, int8 h out
            out = torch.empty((M, N), dtype=torch.int8, device="cuda")
            fn = lambda: ilw.gemm(A, Wp, N, b, m, s, 8, gelu={"I0": 1000}, m_g=3 << 29, s_g=40, out=out)
        elif case == "gemm_qkv":  # q|k|v written as fp16-carried int8
            out = torch.empty((M, N), dtype=torch.float16, device="cuda")
            fn = lambda: ilw.gemm(A, Wp, N, b, m, s, ilw.I8_IN_F16, out=out)
        else:
            res = _dev(synth.uniform_int(1, "case.res", (M, N), -3000, 3000, np.int16))
            out = torch.empty((M, N), dtype=torch.int16, device="cuda")
            fn = lambda: ilw.gemm(A, Wp, N, b, m, s, 16, res=res, m_r=1 << 30, s_r=31, out=out)
        return fn, {"flops": 2.0 * M * N * K}
    if case.startswith("smx"):
        L = int(case.split("_")[1])
        X = _dev(synth.uniform_int(30, f"c3smx{L}", ((1 << 27) // L, L), -(1 << 15), 1 << 15))
        P = torch.empty(X.shape, dtype=torch.uint8, device="cuda")
        return (lambda: ilw.shiftmax_rows(X, {"I0": 3000}, out=P)), {"bytes": 5.0 * X.numel()}
    if case == "gelu_2p28":
        X = _dev(synth.uniform_int(32, "c3gelu", (1 << 28,), -(1 << 12), 1 << 12))
        Y = torch.empty_like(X)
        return (lambda: ilw.sdshiftgelu(X, {"I0": 600}, out=Y)), {"bytes": 8.0 * X.numel()}
    if case.startswith("ln"):
        if case == "ln_encoder":
            X = _dev(synth.uniform_int(34, "case.ln", (12800, 384), -3000, 3000, np.int16))
            per = 3.0  # int16 in, int8 out (carried in fp16, the encoder's form)
        else:
            C = int(case.split("_")[1])
            X = _dev(synth.uniform_int(34, f"c3ln{C}", (1 << 20, C), -(1 << 14), 1 << 14))
            per = 5.0
        C = X.shape[1]
        beta, mult, shift = (_dev(a) for a in synth.ln_params(34, f"c3lnp{C}", C))
        ob = ilw.I8_IN_F16 if case == "ln_encoder" else 8
        Y = torch.empty(X.shape, dtype=torch.float16 if case == "ln_encoder" else torch.int8, device="cuda")
        return (lambda: ilw.int_layernorm(X, beta, mult, shift, 10, ob, out=Y)), {"bytes": per * X.numel()}
    if case == "heads":  # detection head on 16 images x 300 decoder queries, 80 classes
        B, Q, d = batch or 16, 300, 256
        head = ilw.DetectionHead(synth.head_params(8, d=d, C=80))
        out = _dev(synth.uniform_int(8, "case.dh.out", (B * Q, d), -127, 127, np.int8))
        ref = _dev(synth.uniform_int(8, "case.dh.ref", (B * Q, 4), -6000, 6000, np.int16))
        return (lambda: head.forward(out, ref)), {"queries": B * Q}
    if case == "two_stage":  # two-stage selection over 16 images x 8400 memory tokens, top 300
        B, K, d = batch or 16, 300, 256
        S = 8400
        ts = ilw.TwoStage(synth.two_stage_params(9, d=d, C=80))
        mem = _dev(synth.uniform_int(9, "case.ts.mem", (B * S, d), -127, 127, np.int8))
        return (lambda: ts.forward(mem, B, S, K)), {"tokens": B * S}
    raise SystemExit(f"unknown case {case}")


def main(argv=None):
    import torch

    ap = argparse.ArgumentParser()
    ap.add_argument("case")
    ap.add_argument("--reps", type=int, default=20)
    ap.add_argument("--batch", type=int, default=0, help="images of the attention cases")
    ap.add_argument("--graph", action="store_true",
                    help="record the case as a CUDA graph and time `reps` replays back to back between one pair "
                         "of events (mean per launch): the host's argument marshalling stays out of the device time")
    a = ap.parse_args(argv)
    fn, work = build(a.case, a.batch)
    if a.graph:
        import paper_2607_24981_gb300 as ilw

        fn = ilw.Graphed(fn, warmup=2).replay
    for _ in range(3):
        fn()
    torch.cuda.synchronize()
    # every launch timed on its own (events on the launching stream), median reported; the SM clock
    # and throttle reasons are sampled over the timed launches
    from .clocks import ClockSampler

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(max(a.reps, 1))]
    with ClockSampler(torch.cuda.current_device()) as clk:
        if a.graph:
            e0, e1 = ev[0]
            e0.record()
            for _ in range(max(a.reps, 1)):
                fn()
            e1.record()
        else:
            for e0, e1 in ev:
                e0.record()
                fn()
                e1.record()
        torch.cuda.synchronize()
    if a.graph:
        ms = ev[0][0].elapsed_time(ev[0][1]) / max(a.reps, 1)
        times = [ms]
    else:
        times = sorted(e0.elapsed_time(e1) for e0, e1 in ev)
        ms = times[len(times) // 2]
    out = {"case": a.case, "us": ms * 1000.0, "us_min": times[0] * 1000.0, "graph": bool(a.graph),
           "timing": "mean of back-to-back graph replays" if a.graph else "median of per-launch events",
           "clocks": clk.summary()}
    if "flops" in work:
        out["tflops"] = work["flops"] / (ms / 1000.0) / 1e12
    if "bytes" in work:
        out["gbs"] = work["bytes"] / (ms / 1000.0) / 1e9
    if "scores" in work:
        out["gscores_s"] = work["scores"] / (ms / 1000.0) / 1e9
    if "queries" in work:
        out["mqueries_s"] = work["queries"] / (ms / 1000.0) / 1e6
    if "tokens" in work:
        out["mtokens_s"] = work["tokens"] / (ms / 1000.0) / 1e6
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
