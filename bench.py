#!/usr/bin/env python
"""Throughput of the integer-only I-LW-DETR encoder on GB300.

Default workload (N=1): the Medium-scale integer ViT backbone of the paper's Table 1 -- patch
embedding of a 640x640 int8 image (1600 tokens of dim 384) followed by 10 encoder blocks (6
heads, MLP 1536; global attention at layers 2, 4, 5, 9, 2x2-window attention elsewhere), batch
8, seeded synthetic int8 inputs and weights.  One step = one backbone forward of the batch.
The metric counts encoder-block tokens: value = blocks * B * T / step time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Under torchrun (N > 1) every rank runs its own replica on its own batch (no data-path
collective: the path shards by image); the step time is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "int-only encoder block tokens/s (1600 tok, d=384)"
UNIT = "block-tokens/s"
WORKLOAD = "medium_backbone_b8"
SEED = 0
# cpu baseline sample: each image through blocks 0..4 (3 window + 2 global, the backbone's 6:4
# window/global ratio); the reference arm instead cycles over all 10 blocks, one block per step
CPU_SAMPLE_BLOCKS = 5


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ilw", choices=["ilw", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-legs", action="store_true", help="skip the block-variant, sweep and detector legs")
    return ap.parse_args(argv)


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def max_over_ranks(value: float, world: int) -> float:
    """Max of a per-rank float over the process group (identity for one process)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist

    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int) -> None:
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


# ------------------------------------------------------------------------------ workload
def workload_cfg():
    from paper_2607_24981_gb300 import synth

    return dict(synth.CONFIGS[WORKLOAD])


def workload_config(cfg, world):
    """The `config` of the bench line: the workload both arms report on (the reference arm times a
    bounded sample of it, described in its cpu_baseline)."""
    return {"workload": "medium_backbone_b8: Medium integer ViT backbone (patch embed + 10 blocks)",
            "B": cfg["B"], "T": cfg["T"], "d": cfg["d"], "H": cfg["H"], "F": cfg["F"], "blocks": cfg["layers"],
            "global_layers": list(cfg["global_layers"]), "window": "2x2 windows of 400 tokens",
            "image": "640x640 int8, 16x16 patches", "per_gpu_batch": cfg["B"],
            "units": "block-tokens = blocks x images x tokens per step",
            "l2": "flushed between timed steps (256 MB write)", "parallelism": f"replicas x{world}"}


def build_host_params():
    from paper_2607_24981_gb300 import synth

    cfg = workload_cfg()
    blocks = synth.backbone_params(SEED, cfg)
    pe = synth.patch_embed_params(SEED, cfg["d"], mode=cfg["mode"])
    return cfg, pe, blocks


class Instrumented:
    """The backbone forward issued as the same sequence of ABI calls that ilwdetr_patch_embed and
    ilwdetr_block_forward make, with CUDA events around each call so every kernel class gets its
    own device time.  With ``external`` events the sequence can be recorded into a CUDA graph: the
    events become graph nodes, so one replay times every kernel without host launch gaps."""

    def __init__(self, bb, torch, external=False):
        self.bb, self.torch, self.external = bb, torch, external
        M, d, F = bb.B * bb.T, bb.d, bb.F
        dev = bb.x[0].device
        # every int8 activation between kernels is carried in fp16 (the tensor cores' operand form)
        f16 = torch.float16
        self.a1 = torch.empty((M, d), dtype=f16, device=dev)
        self.qkv = torch.empty((M, 3 * d), dtype=f16, device=dev)
        self.o = torch.empty((M, d), dtype=f16, device=dev)
        self.x1 = torch.empty((M, d), dtype=torch.int16, device=dev)
        self.a2 = torch.empty((M, d), dtype=f16, device=dev)
        self.h = torch.empty((M, F), dtype=f16, device=dev)
        self.xs = [torch.empty((M, d), dtype=torch.int16, device=dev) for _ in range(2)]
        self.records = []  # (kernel class, start event, end event, launches)

    def _ev(self):
        e = (self.torch.cuda.Event(enable_timing=True, external=True) if self.external
             else self.torch.cuda.Event(enable_timing=True))
        e.record()
        return e

    def _rec(self, name, fn, launches=1):
        s = self._ev()
        out = fn()
        self.records.append((name, s, self._ev(), launches))
        return out

    def forward(self, img):
        import paper_2607_24981_gb300 as ilw

        bb, pe = self.bb, self.bb.pe
        B, T, d, F = bb.B, bb.T, bb.d, bb.F
        M = B * T
        x = self._rec("patch_embed", lambda: ilw.patch_embed(
            img, bb.p, pe["w_p"], d, pe["b"], pe["m"], pe["s"], pe["pos"], bb.pe_s["m_pos"],
            bb.pe_s["s_pos"], bb.ws_pe, self.xs[0]), launches=2)
        for i, bw in enumerate(bb.blocks):
            t, p = bw.t, bw.bp
            y = self.xs[(i + 1) % 2]
            F16 = ilw.I8_IN_F16
            self._rec("layernorm", lambda: ilw.int_layernorm(x, t["ln1_beta"], t["ln1_mult"], t["ln1_shift"],
                                                             p["ln_iters"], F16, out=self.a1))
            self._rec("gemm_qkv", lambda: ilw.gemm(self.a1, t["w_qkv_p"], 3 * d, t["b_qkv"], t["m_qkv"],
                                                   t["s_qkv"], F16, out=self.qkv))
            kind = "attention_global" if p["win_side"] <= 1 else "attention_window"
            self._rec(kind, lambda: ilw.shiftmax_attn(self.qkv, B, T, p["H"], d // p["H"], p["win_side"], p["smx"],
                                                      p["m_o"], p["s_o"], out=self.o))
            self._rec("gemm_proj", lambda: ilw.gemm(self.o, t["w_proj_p"], d, t["b_proj"], t["m_proj"],
                                                    t["s_proj"], 16, res=x, m_r=p["m_r1"], s_r=p["s_r1"],
                                                    out=self.x1))
            self._rec("layernorm", lambda: ilw.int_layernorm(self.x1, t["ln2_beta"], t["ln2_mult"], t["ln2_shift"],
                                                             p["ln_iters"], F16, out=self.a2))
            self._rec("gemm_fc1_gelu", lambda: ilw.gemm(self.a2, t["w_fc1_p"], F, t["b_fc1"], t["m_fc1"],
                                                        t["s_fc1"], F16, gelu={"I0": p["gelu_I0"]}, m_g=p["m_g"],
                                                        s_g=p["s_g"], out=self.h))
            self._rec("gemm_fc2", lambda: ilw.gemm(self.h, t["w_fc2_p"], d, t["b_fc2"], t["m_fc2"], t["s_fc2"],
                                                   16, res=self.x1, m_r=p["m_r2"], s_r=p["s_r2"], out=y))
            x = y
        # empty event pairs: the cost of the timing nodes themselves, subtracted from every class
        for _ in range(8):
            self._rec(EVENT_PAIR, lambda: None, launches=0)
        return x


EVENT_PAIR = "_event_pair"


def kernel_work(cfg, B):
    """Algorithmic work per launch of each kernel class (one backbone step)."""
    T, d, F, H = cfg["T"], cfg["d"], cfg["F"], cfg["H"]
    M = B * T
    dh = d // H
    Tw = T // 4  # 2x2 windows
    return {
        # tensor classes: 2*M*N*K integer multiply-adds per launch
        "gemm_qkv": ("tensor", 2.0 * M * 3 * d * d),
        "gemm_proj": ("tensor", 2.0 * M * d * d),
        "gemm_fc1_gelu": ("tensor", 2.0 * M * F * d),
        "gemm_fc2": ("tensor", 2.0 * M * d * F),
        "patch_embed": ("tensor", 2.0 * M * d * 768),
        # attention: scores per launch (q.k^T, Shiftmax, P.V), see the ALU roofline
        "attention_global": ("alu", float(B * H * T * T)),
        "attention_window": ("alu", float(B * H * 4 * Tw * Tw)),
        # I-LayerNorm: int16 in (2 B) + int8 out (1 B, carried in a 2-byte fp16) per element
        "layernorm": ("hbm", 3.0 * M * d),
    }


def host_cpu() -> dict:
    """The host's usable cores and CPU model (lscpu's model name, when lscpu answers)."""
    import subprocess

    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    model = "unknown"
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.TimeoutExpired):
        pass
    return {"cores": cores, "model": model}


def _oracle_image(job):
    """One image through the given encoder blocks in the oracle (a spawned worker process);
    returns the seconds the blocks took."""
    seed, pe, blocks, T = job
    import oracle
    from paper_2607_24981_gb300 import synth

    img = synth.image_input(seed, 1)
    x = oracle.patch_embed(img, pe["p"], pe["w"], pe["b"], pe["m"], pe["s"], pe["pos"], pe["m_pos"], pe["s_pos"])
    t0 = time.perf_counter()
    for bp in blocks:
        x = oracle.block_forward(bp, x, 1, T)
    return time.perf_counter() - t0


def oracle_pool(n):
    """A pool of n spawned processes for the oracle (spawn: safe after the CUDA context exists)."""
    import multiprocessing as mp

    import oracle

    oracle.build()  # built once here, so the workers only load it
    return mp.get_context("spawn").Pool(n)


def run_cpu_sample(cfg, pe, blocks) -> dict:
    """The oracle as it stands, timed on the host's cores: single-threaded (one image through
    blocks 0..CPU_SAMPLE_BLOCKS-1), then on every core (one image per core, in separate processes,
    each through the same blocks; the loops of the oracle stay plain)."""
    host = host_cpu()
    sub = blocks[:CPU_SAMPLE_BLOCKS]
    with oracle_pool(host["cores"]) as pool:
        t1 = pool.apply(_oracle_image, ((SEED, pe, sub, cfg["T"]),))
        t0 = time.perf_counter()
        pool.map(_oracle_image, [(SEED + 1 + i, pe, sub, cfg["T"]) for i in range(host["cores"])], chunksize=1)
        tall = time.perf_counter() - t0
    units = CPU_SAMPLE_BLOCKS * cfg["T"]
    blocks_desc = f"encoder blocks 0-{CPU_SAMPLE_BLOCKS - 1} (3 window + 2 global)"
    return {"value": host["cores"] * units / tall, "unit": UNIT, "cores": host["cores"], "kind": "oracle",
            "cpu": host["model"],
            "sample": f"{host['cores']} images (one per core, separate processes) x {blocks_desc}: "
                      f"{host['cores'] * units} block-tokens in {tall:.1f} s wall; C++ oracle (g++ -O2)",
            "single_thread": {"value": units / t1, "unit": UNIT, "cores": 1,
                              "sample": f"1 image x {blocks_desc}, {units} block-tokens, {t1:.1f} s"}}


# ------------------------------------------------------------------------------ further legs
def _time_launches(torch, fn, reps, flush=None):
    """Median and minimum device time (ms) of `reps` calls of fn, each bracketed by CUDA events on
    the current stream; `flush` (a buffer larger than L2) is rewritten before each call."""
    ts = []
    for _ in range(reps):
        if flush is not None:
            flush.fill_(1)
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        fn()
        e.record()
        e.synchronize()
        ts.append(s.elapsed_time(e))
    ts.sort()
    return ts[len(ts) // 2], ts[0]


def _time_graph_back_to_back(ilw, torch, fn, reps):
    """Mean device time (ms) of one call of fn: fn recorded once as a CUDA graph, the graph replayed
    `reps` times back to back between two CUDA events, so the GPU never waits for the host between
    launches.  For working sets larger than L2, where one launch leaves nothing for the next."""
    g = ilw.Graphed(fn)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    s = torch.cuda.Event(enable_timing=True)
    e = torch.cuda.Event(enable_timing=True)
    s.record()
    for _ in range(reps):
        g.replay()
    e.record()
    e.synchronize()
    return s.elapsed_time(e) / reps


def leg_blocks(ilw, torch, bb, img, reps, flush):
    """One global-attention block and one window block of the backbone, each a CUDA graph of one
    ilwdetr_block_forward on the patch embedding of the batch; block tokens/s = B T / block time."""
    pe = bb.pe
    x0 = torch.empty((bb.B * bb.T, bb.d), dtype=torch.int16, device=img.device)
    ilw.patch_embed(img, bb.p, pe["w_p"], bb.d, pe["b"], pe["m"], pe["s"], pe["pos"], bb.pe_s["m_pos"],
                    bb.pe_s["s_pos"], bb.ws_pe, x0)
    out = torch.empty_like(x0)
    res = {}
    for kind in ("global", "window"):
        i = next(j for j, bw in enumerate(bb.blocks) if (bw.bp["win_side"] <= 1) == (kind == "global"))
        bw = bb.blocks[i]
        g = ilw.Graphed(lambda: ilw.block_forward(bw, x0, bb.B, bb.T, bb.ws_blk, out=out))
        med, best = _time_launches(torch, g.replay, reps, flush)
        res[kind] = {"block": i, "ms": med, "ms_best": best, "tokens_per_s": bb.B * bb.T / (med / 1000.0)}
    return res


def leg_sweep(ilw, torch, dev, reps):
    """The nonlinearity sweep at its workload sizes: Constrained Shiftmax over 2^27 int32 scores in
    rows of 64 / 400 / 1600, SD-ShiftGELU over 2^28 int32 values, I-LayerNorm over 2^20 int32 rows
    of 192 / 384.  Inputs drawn on the device from a seeded generator with the workload's ranges;
    every working set is larger than L2, so no flush is needed, and each kernel is timed as `reps`
    back-to-back replays of a one-launch CUDA graph (the host's argument marshalling stays out of the
    device time).  GB/s counts the algorithmic bytes (4 B in + 1 B out per Shiftmax or LayerNorm
    element, 4 B + 4 B per GELU element)."""
    from paper_2607_24981_gb300 import synth

    gen = torch.Generator(device=dev)
    gen.manual_seed(SEED)
    res = {}

    def draw(shape, lo, hi):
        return torch.randint(lo, hi + 1, shape, generator=gen, device=dev, dtype=torch.int32)

    for L in (64, 400, 1600):
        X = draw(((1 << 27) // L, L), -(1 << 15), 1 << 15)
        P = torch.empty(X.shape, dtype=torch.uint8, device=dev)
        med = _time_graph_back_to_back(ilw, torch, lambda: ilw.shiftmax_rows(X, {"I0": 3000}, out=P), reps)
        res[f"shiftmax_{L}"] = {"ms": med, "gbs": 5.0 * X.numel() / (med / 1000.0) / 1e9}
        del X, P
    X = draw((1 << 28,), -(1 << 12), 1 << 12)
    Y = torch.empty_like(X)
    med = _time_graph_back_to_back(ilw, torch, lambda: ilw.sdshiftgelu(X, {"I0": 600}, out=Y), reps)
    res["sdshiftgelu"] = {"ms": med, "gbs": 8.0 * X.numel() / (med / 1000.0) / 1e9}
    del X, Y
    for C in (192, 384):
        X = draw((1 << 20, C), -(1 << 14), 1 << 14)
        beta, mult, shift = (torch.from_numpy(a).to(dev) for a in synth.ln_params(34, f"c3lnp{C}", C))
        Y = torch.empty(X.shape, dtype=torch.int8, device=dev)
        med = _time_graph_back_to_back(ilw, torch, lambda: ilw.int_layernorm(X, beta, mult, shift, 10, 8, out=Y), reps)
        res[f"layernorm_{C}"] = {"ms": med, "gbs": 5.0 * X.numel() / (med / 1000.0) / 1e9}
        del X, Y
    return res


def leg_detector(ilw, torch, dev, reps, flush):
    """The full integer detector forward at batch 16 (Medium backbone with its four output layers
    tapped, split-convolution projector, two-stage query selection with the positional-query
    projection, three decoder layers, detection head), one CUDA graph per forward."""
    from paper_2607_24981_gb300 import synth

    cfg = synth.CONFIGS["medium_detector_b16"]
    bbc = synth.CONFIGS[cfg["backbone"]]
    B, Q, g = cfg["B"], cfg["Q"], cfg["grid"]
    det = ilw.Detector(synth.patch_embed_params(SEED, bbc["d"], mode=bbc["mode"]), synth.backbone_params(SEED, bbc),
                       cfg["taps"], synth.projector_params(SEED, len(cfg["taps"]), bbc["d"], cfg["N"]),
                       [synth.decoder_params(SEED, i) for i in range(cfg["dec_layers"])], B, Q, cfg["levels"], g,
                       tsp=synth.two_stage_params(SEED, d=cfg["N"], C=80, levels=cfg["levels"]),
                       hp=synth.head_params(SEED, d=cfg["N"], C=80), pq=synth.query_pos_params(SEED, d=cfg["N"]),
                       rps=synth.refine_params(SEED, cfg["dec_layers"] - 1, d=cfg["N"]), device=dev)
    img = torch.from_numpy(synth.image_input(SEED, B)).to(dev)
    tgt = torch.from_numpy(synth.decoder_inputs(SEED, B, Q)["tgt"]).to(dev)
    graph = ilw.Graphed(lambda: det.forward(img, tgt))
    med, best = _time_launches(torch, graph.replay, reps, flush)
    return {"B": B, "queries": Q, "ms": med, "ms_best": best, "images_per_s": B / (med / 1000.0),
            "stages": "patch embed + 10 blocks, projector (3 levels), two-stage top-300 with positional "
                      "queries, 3 decoder layers with the reference boxes refined between them, detection "
                      "head (80 classes)"}


# ------------------------------------------------------------------------------ reference arm
def run_reference(args) -> None:
    """The oracle as it stands on the host's cores: each step runs one image per core (separate
    processes) through one encoder block, cycling over the backbone's 10 blocks step by step."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    cfg, pe, blocks = build_host_params()
    host = host_cpu()
    n = host["cores"]
    times = []
    with oracle_pool(n) as pool:
        for step in range(args.warmup + args.steps):
            bp = blocks[step % len(blocks)]
            t0 = time.perf_counter()
            pool.map(_oracle_image, [(SEED + i, pe, [bp], cfg["T"]) for i in range(n)], chunksize=1)
            if step >= args.warmup:
                times.append(time.perf_counter() - t0)
    ms = 1000.0 * statistics.mean(times)
    value = n * cfg["T"] / (ms / 1000.0)
    sample = (f"per step: {n} images (one per core, separate processes, 1600 tokens each) through one "
              f"encoder block, cycling over the 10 blocks (6 window, 4 global) step by step; the patch "
              f"embedding is outside the timed region; C++ oracle (g++ -O2)")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": workload_config(cfg, world),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": n, "kind": "oracle", "cpu": host["model"],
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------ main arm
def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    rank, world, local = dist_env()
    import torch

    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    import numpy as np

    import paper_2607_24981_gb300 as ilw
    from paper_2607_24981_gb300 import synth

    ilw.lib()
    cfg, pe, blocks = build_host_params()
    B, T, L = cfg["B"], cfg["T"], cfg["layers"]
    units_per_step = L * B * T
    dev = torch.device("cuda", local)
    bb = ilw.Backbone(pe, blocks, B, device=dev)
    img_h = synth.image_input(SEED + rank, B)
    img = torch.from_numpy(img_h).to(dev)
    # the instrumented sequence and the public Backbone.forward must agree bit for bit
    ref_out = bb.forward(img).clone()
    chk = Instrumented(bb, torch)
    out = chk.forward(img)
    torch.cuda.synchronize()
    assert torch.equal(ref_out, out), "instrumented launch sequence differs from the public API path"

    # one step = one replay of the public forward recorded as a CUDA graph (Backbone.capture); the
    # instrumented sequence is recorded too, with its events inside the graph, for the per-kernel
    # device times (fallback without graph events: the instrumented calls issued eagerly)
    step = bb.capture(img)
    try:
        inst = Instrumented(bb, torch, external=True)
        # records are reset at each call, so after capture they hold the graph's own events
        inst_graph = ilw.Graphed(lambda: (inst.records.clear(), inst.forward(img))[1])
        replay_inst = inst_graph.replay
    except TypeError:  # a torch without external (graph-node) events
        inst = Instrumented(bb, torch)
        replay_inst = lambda: inst.forward(img)
    torch.cuda.synchronize()
    assert torch.equal(step.replay(), ref_out), "graph replay differs from the eager forward"
    inst_out = replay_inst()
    torch.cuda.synchronize()
    assert torch.equal(inst_out, ref_out), "instrumented replay differs from the eager forward"

    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # > 129 MB L2

    for _ in range(args.warmup):
        step.replay()
        if not inst.external:
            inst.records.clear()
        replay_inst()
    torch.cuda.synchronize()

    step_ms = []
    per = {}  # kernel class -> (total ms, records, launches)

    def collect():
        for name, s_, e_, n in inst.records:
            tot, cnt, ln = per.get(name, (0.0, 0, 0))
            per[name] = (tot + s_.elapsed_time(e_), cnt + 1, ln + n)

    barrier(world)
    from paper_2607_24981_gb300.clocks import ClockSampler

    with ClockSampler(local) as clk:
        for _ in range(args.steps):
            flush.fill_(1)  # evict L2 before every timed step
            s = torch.cuda.Event(enable_timing=True)
            e = torch.cuda.Event(enable_timing=True)
            s.record()
            step.replay()
            e.record()
            e.synchronize()
            step_ms.append(s.elapsed_time(e))
            # the same step once more, instrumented: per-kernel durations
            flush.fill_(1)
            if not inst.external:
                inst.records.clear()
            replay_inst()
            torch.cuda.synchronize()
            collect()
            if not inst.external:
                inst.records.clear()
        torch.cuda.synchronize()
    barrier(world)
    ilw.device_status()
    ms_local = statistics.mean(step_ms)
    ms = max_over_ranks(ms_local, world)
    value = world * units_per_step / (ms / 1000.0)

    # per-kernel device times (average launch duration per class, over the timed steps), less the
    # duration of an empty pair of timing events recorded the same way
    ev_tot, ev_cnt, _ = per.pop(EVENT_PAIR, (0.0, 0, 0))
    event_pair_ms = ev_tot / ev_cnt if ev_cnt else 0.0
    launches_per_step = sum(v[2] for v in per.values()) // args.steps
    step_total = sum(v[0] - v[1] * event_pair_ms for v in per.values())
    work = kernel_work(cfg, B)
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))) if os.path.exists(
        os.path.join(ROOT, "MEASURED_PEAKS.json")) else {}
    clocks = clk.summary()
    kernels = {}
    for name, (tot, cnt, _) in per.items():
        avg_ms = max(tot / cnt - event_pair_ms, 1e-6)
        bound, w = work[name]
        kernels[name] = {"share": avg_ms * cnt / step_total, "avg_ms": avg_ms, "avg_ms_with_events": tot / cnt,
                         "launches_per_step": cnt // args.steps, "bound": bound}
        if bound == "tensor":
            kernels[name]["tops"] = w / (avg_ms / 1000.0) / 1e12
        elif bound == "hbm":
            kernels[name]["gbs"] = w / (avg_ms / 1000.0) / 1e9
        else:
            kernels[name]["gscores_s"] = w / (avg_ms / 1000.0) / 1e9
    dom = max(per, key=lambda k: per[k][0])
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    roofline = roofline_entry(dom, kernels[dom], work[dom], peaks, clocks, sms)

    # end to end through the public API: pinned host image -> device, backbone, result -> host
    pin_in = torch.from_numpy(img_h).pin_memory()
    pin_out = torch.empty((B * T, cfg["d"]), dtype=torch.int16).pin_memory()
    dimg = torch.empty_like(img)
    dimg.copy_(img)
    e2e_step = bb.capture(dimg)
    e2e_ms = []
    for i in range(args.warmup + args.steps):
        flush.fill_(1)
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        dimg.copy_(pin_in, non_blocking=True)
        y = e2e_step.replay()
        pin_out.copy_(y, non_blocking=True)
        e.record()
        e.synchronize()
        if i >= args.warmup:
            e2e_ms.append(s.elapsed_time(e))
    assert np.array_equal(pin_out.numpy(), ref_out.cpu().numpy())
    e2e_t = max_over_ranks(statistics.mean(e2e_ms), world)
    e2e = {"value": world * units_per_step / (e2e_t / 1000.0), "unit": UNIT,
           "h2d_bytes_per_step": int(pin_in.numel()), "d2h_bytes_per_step": int(pin_out.numel() * 2)}

    # further legs, timed in this run under their own clock record: the two block variants of the
    # headline metric, the nonlinearity sweep and the full detector
    legs = None
    if not args.no_legs:
        reps = max(args.steps, 10)
        with ClockSampler(local) as clk2:
            legs = {"blocks": leg_blocks(ilw, torch, bb, img, reps, flush)}
            del bb, step, inst, e2e_step
            torch.cuda.empty_cache()
            legs["nonlinearity_sweep"] = leg_sweep(ilw, torch, dev, reps)
            legs["detector"] = leg_detector(ilw, torch, dev, reps, flush)
            torch.cuda.synchronize()
        legs["clocks"] = clk2.summary()
        hbm = peaks.get("hbm_gbs") or 6800.0
        for v in legs["nonlinearity_sweep"].values():
            v["frac_of_measured_hbm"] = v["gbs"] / hbm
            v["frac_of_8tbs"] = v["gbs"] / 8000.0
        ilw.device_status()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = run_cpu_sample(cfg, pe, blocks)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int8", "data": "synthetic",
            "config": workload_config(cfg, world),
            "clocks": clocks, "e2e": e2e, "gpu_launches": launches_per_step * args.steps,
            "roofline": roofline, "kernels": kernels, "kernel_timing": {
                "method": "CUDA events around each call inside a graph replay of the step, L2 flushed; "
                          "an empty event pair recorded the same way is subtracted",
                "event_pair_us": event_pair_ms * 1000.0},
            "legs": legs, "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one ncu capture of the
# kernel at this launch size, for the kernels whose code has not changed since that capture
# (the global attention's capture, 29.61 MB per launch, predates its current CTA order: none listed)
NCU_TRAFFIC = {}


def roofline_entry(name, k, work, peaks, clocks, sms):
    bound, w = work
    avg_s = k["avg_ms"] / 1000.0
    if bound == "hbm":
        peak = peaks.get("hbm_gbs")
        src = "measured" if peak else "fallback"
        peak = peak or 6800.0
        a = w / avg_s / 1e9
        return {"kernel": name, "bound": "hbm", "achieved": a, "peak": peak, "unit": "GB/s", "frac": a / peak,
                "traffic": NCU_TRAFFIC.get(name), "peak_source": src}
    if bound == "tensor":
        peak = peaks.get("bf16_tflops_sustained")
        src = "measured bf16 sustained (same rate as fp16 kind::f16)" if peak else "fallback"
        peak = peak or 1700.0
        a = w / avg_s / 1e12
        return {"kernel": name, "bound": "tensor", "achieved": a, "peak": peak, "unit": "TFLOP/s",
                "frac": a / peak, "traffic": NCU_TRAFFIC.get(name), "peak_source": src}
    # ALU: integer operations per score of the exact three-pass method (row maximum; ShiftExp and the
    # int64 sum; ShiftExp again, the normalising multiply and shift, the fp16 P), the midpoint of the
    # 30-40 that the method needs, against SMs x 128 lanes x the median SM clock; the figure at 16
    # operations (ShiftExp counted once per score) is reported beside it
    ops_per_score = 35.0
    mhz = clocks.get("sm_mhz") or 1500.0
    peak = sms * 128 * mhz * 1e6 / 1e12
    a = w * ops_per_score / avg_s / 1e12
    return {"kernel": name, "bound": "alu", "achieved": a, "peak": peak, "unit": "Tops/s", "frac": a / peak,
            "traffic": NCU_TRAFFIC.get(name),
            "peak_source": f"derived: {sms} SMs (read from the device) x 128 int32 lanes x {mhz:.0f} MHz (median SM clock)",
            "ops_per_score": ops_per_score, "frac_at_16_ops_per_score": a / peak * 16.0 / ops_per_score}


if __name__ == "__main__":
    main()
