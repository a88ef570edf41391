#!/usr/bin/env python
"""Benchmark of the retrieve-and-verify step (FastCoder, arXiv 2502.17139).

Workload (the full step loop): a general datastore of 100M tokens (Zipf 1.1)
and a project datastore of 5M tokens (Zipf 1.3 + 20,000 planted 8-64-token
repeats), vocab 32256; 32 sequences whose 128-token contexts end with spans
copied from the project store (50%), the general store (25%) or pure Zipf
draws (25%); retrieval n 16 -> 2, top-64 drafts of 10 tokens per source,
alpha = beta = 1; draft trees of at most 128 nodes; tree attention with 32
query / 8 KV heads, head dim 128, KV cache 16384 tokens (bf16); greedy
acceptance against the synthetic target model; cache append; a context-keyed
replay cache with a seeded 50% hit pattern.  One step = one pass of all of
that over the batch.  The datastores are built once (offline, Section IV-A)
before timing; their build time is reported separately.

Arms:
  default           the CUDA path (libfastcoder.so through its C ABI)
  --impl reference  the CPU oracle, timed on the host cores, each timed step
                    one full, unsampled step of all 32 sequences

Under torchrun every rank runs an independent batch of 32 sequences on its
own GPU against replicated datastores (no data-path collective); the timed
region is bracketed by barriers and the slowest rank's time is used.
"""
from __future__ import annotations

import argparse
import contextlib
import gc
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "retrieve+verify steps/s"
PAD_TOKEN = 0xFFFFFFFF
UNIT = "steps/s"
# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of the tree-attention
# launch the roofline times (all 32 sequences on one stream), as a ratio to the
# launch's algorithmic bytes, from one ncu capture of three launches:
#   ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum,gpu__time_duration.sum
#       --clock-control none -k regex:k_tree_attn -s 10 -c 3 --csv
#       python bench.py --steps 4 --warmup 3 --split 1 --no-e2e --no-cpu-baseline --no-graph
# (one pass per launch; the recording pass's 7 launches and the 3 warm-up launches are
# skipped, so the captured launches are timed steps 3-5 of the trajectory, the first
# three launches of the bench's single-stream pass, whose algorithmic bytes that run
# prints as roofline.algorithmic_bytes_first_launches).  The bench reports traffic =
# ratio x the algorithmic bytes per launch of its own launches.  The ratio is valid
# only for the kernel sources it was taken on (their SHA-256 below); otherwise the
# bench reports traffic as null until it is measured again.
ATTN_TRAFFIC = {"ratio": 1.0624,
                "sources": ["paper_2502_17139_gb300/csrc/tree_attn.cu", "paper_2502_17139_gb300/csrc/fc_common.cuh"],
                "sha256": "43b044e94f2cc97452818a22d11aa8bcea7db9717ac19c720f55fd3e5c941192"}

WORKLOAD = ("full step loop: two-source datastore 100M (Zipf 1.1) + 5M (Zipf 1.3, 20k planted repeats) tokens, "
            "vocab 32256, batch 32, ctx 128, n 16->2, top-64 x 10 tokens per source, tree <=128 nodes, "
            "GQA 32/8 heads, head_dim 128, KV 16384 bf16, 50% replay-cache hits")


def src_weights(args):
    w = [int(x) for x in args.weights.split(",")]
    if len(w) != 2 or min(w) < 0 or max(w) > 65535:
        raise SystemExit("--weights takes two integers in 0..65535")
    return w


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--scale", type=float, default=1.0,
                    help="shrink the datastores and KV length (tests only; 1.0 is the benchmark workload)")
    ap.add_argument("--batch", type=int, default=32)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mode", choices=["step", "attn", "argmax", "configs", "retrieve", "algorithm1", "cache", "gemm", "build",
                                       "small",
                                       "decoder"],
                    default="step",
                    help="step: the full step loop (the benchmark); attn: tree attention alone on the step loop's "
                         "attention shape with seeded trees (a small profiling / sweep target); argmax: greedy "
                         "verification from bf16 logits (fc_argmax_accept) on the step loop's tree shape; configs: "
                         "every stage of the five benchmark configurations timed once each (a report, not the "
                         "benchmark line); retrieve: two-source retrieval alone for --batch queries (batch sweeps); "
                         "small: the step's small kernels (tree build, predictions, acceptance, KV append, "
                         "replay-cache lookup) over the batches of --batches")
    ap.add_argument("--batches", default="32,256,2048,16384", help="small mode: comma-separated batch sizes")
    ap.add_argument("--nodes", type=int, default=128, help="attn mode: tree nodes per sequence")
    ap.add_argument("--kv", type=int, default=16384, help="attn mode: KV cache length")
    ap.add_argument("--no-graph", action="store_true",
                    help="step mode: skip timing the same steps replayed from CUDA graphs (two steps per graph)")
    ap.add_argument("--split", type=int, default=4,
                    help="step and algorithm1 modes: sub-batches of the sequences, each on CUDA streams of its own, issued by the "
                         "native step executor (1: the single-stream StepLoop)")
    ap.add_argument("--all-occ", action="store_true",
                    help="retrieve mode: also time the all-occurrence trie (fc_retrieve_all + fc_build_tree_all)")
    ap.add_argument("--rev", action="store_true",
                    help="retrieve mode: also time the reversed-corpus variant (fc_retrieve_rev) on the same queries")
    ap.add_argument("--rope", action="store_true",
                    help="attn mode: unrotated queries, rotated in the kernel by node position (fc_tree_attn_rope)")
    ap.add_argument("--weights", type=str, default="1,1",
                    help="Eq. 3 source weights alpha,beta (project store, general store) for the step loop")
    ap.add_argument("--fill", type=int, default=None,
                    help="algorithm1 / cache modes: steps that fill the CACHE first (default 100 / 450)")
    ap.add_argument("--skip-1b", action="store_true", help="configs mode: leave out the 1B-token configuration")
    ap.add_argument("--tokens", type=int, default=100_000_000, help="build mode: corpus tokens (Zipf 1.1)")
    ap.add_argument("--traffic-bytes", type=float, default=None,
                    help="ncu dram read+write bytes of one single-stream tree-attention launch of this workload")
    return ap.parse_args(argv)


# ---------------------------------------------------------------- helpers
def attn_traffic(args, algorithmic_bytes_per_launch):
    """DRAM bytes per attention launch: the measured ratio to the algorithmic
    bytes times this run's algorithmic bytes per launch, or None when the
    kernel changed since the ratio was measured."""
    if args.traffic_bytes is not None:
        return args.traffic_bytes
    if ATTN_TRAFFIC["ratio"] is None or ATTN_TRAFFIC["sha256"] is None:
        return None
    import hashlib
    h = hashlib.sha256()
    for f in ATTN_TRAFFIC["sources"]:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    if h.hexdigest() != ATTN_TRAFFIC["sha256"]:
        return None
    return ATTN_TRAFFIC["ratio"] * algorithmic_bytes_per_launch


def step_status(fc, loop):
    """The device errors of a step loop: fc_get_error() and, for the pipelined
    loop, every sub-batch's own error word (the most severe first found)."""
    sts = [fc.fc_get_error()] + (loop.errors() if hasattr(loop, "errors") else [])
    bad = [x for x in sts if x != "FC_OK"]
    return bad[0] if bad else "FC_OK"


@contextlib.contextmanager
def no_gc():
    """The Python garbage collector off inside a timed region: a collection
    pause on the host would land in a wall-clock (e2e) number."""
    was = gc.isenabled()
    gc.disable()
    try:
        yield
    finally:
        if was:
            gc.enable()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), tc_burst=float(p["bf16_tflops"]),
                    tc_sustained=float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), source="measured")
    return dict(hbm=6800.0, tc_burst=1900.0, tc_sustained=1700.0, source="fallback")


class ClockSampler:
    """nvidia-smi clock/throttle samples during the timed region."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 20):
        self.proc = None
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={gpu_index}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", str(interval_ms)],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.proc = None

    def wait_first(self, timeout_s: float = 3.0):
        """Block until the sampler has written its first sample (nvidia-smi takes a
        moment to start), so that the samples cover the region that follows."""
        self.skip = 0
        t0 = time.perf_counter()
        while self.proc is not None and time.perf_counter() - t0 < timeout_s:
            if os.path.getsize(self.file.name) > 0:
                with open(self.file.name) as f:  # samples taken so far precede the region
                    self.skip = sum(1 for r in f if r.strip())
                return
            time.sleep(0.01)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        with open(self.file.name) as f:
            rows = [r.strip().split(", ") for r in f if r.strip()]
        os.unlink(self.file.name)
        rows = rows[getattr(self, "skip", 0):] or rows[-1:]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except (ValueError, IndexError):
                continue
            for k, nm in enumerate(names):
                if len(r) > 5 + k and r[5 + k].strip().lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(gpus: int):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return rank, ws, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def weak_value(steps_per_rank: int, ws: int, t_max_ms: float) -> float:
    """Whole-job throughput: every rank runs its own batch for `steps_per_rank`
    steps; the job takes as long as its slowest rank."""
    return ws * steps_per_rank / (t_max_ms * 1e-3)


def max_over_ranks(x: float, ws: int) -> float:
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------- workload
def workload_spec(scale: float, batch: int):
    import paper_2502_17139_gb300.synth as synth
    cfg = dict(synth.WORKLOADS[5])
    c2 = synth.WORKLOADS[2]
    corpora = [synth.scaled_corpus_spec(s, scale) for s in c2["corpus"]]
    kv = max(256, int(cfg["kv_len"] * scale))
    return cfg, corpora, kv, batch


def make_inputs(scale: float, batch: int, rank: int, steps_total: int):
    """Host-side seeded inputs; rank r gets its own batch of sequences."""
    import paper_2502_17139_gb300.synth as synth
    cfg, corp_specs, kv0, B = workload_spec(scale, batch)
    rng = synth.rng_for(2)                      # datastores: identical on every rank
    corpora = []
    import torch
    gen_dev = "cuda" if torch.cuda.is_available() else None
    for spec in corp_specs:
        T, _ = synth.build_corpus(rng, spec, device=gen_dev)
        corpora.append(T)
    Tr, Tc = corpora                            # project store first (alpha), general second (beta)
    rr = synth.rng_for(5, 1 + rank)             # per-rank sequences
    n_pad, d = cfg["n_pad"], cfg["draft_len"]
    stride = cfg["ctx_len"] + (steps_total + 1) * (d + 1)
    ctx, cl, _ = synth.make_contexts(rr, B, cfg["ctx_len"], cfg["n_copy"], [Tr, Tc, None], cfg["probs"], 1.1,
                                     ctx_stride=stride)
    hits = synth.cache_hit_pattern(rr, steps_total, B, cfg["hit_p"])
    plen = np.empty((steps_total, B), np.int32)
    rtok = np.empty((steps_total, B, n_pad), np.uint32)
    for s in range(steps_total):
        plen[s], rtok[s] = synth.argmax_draws(rr, B, n_pad)
    return dict(cfg=cfg, corpora=corpora, kv0=kv0, B=B, ctx=ctx, cl=cl, hits=hits, plen=plen, rtok=rtok,
                stride=stride, seed=1000 * (rank + 1))


# ---------------------------------------------------------------- our arm
def run_ours(args, rank, ws, local):
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    K, W = args.steps, args.warmup
    total = K + W + 1
    inp = make_inputs(args.scale, args.batch, rank, total)
    cfg, B = inp["cfg"], inp["B"]
    H, Hkv, D, n_pad, d = cfg["H"], cfg["Hkv"], cfg["D"], cfg["n_pad"], cfg["draft_len"]
    kv0 = inp["kv0"]
    cap = kv0 + total * (d + 1) + 8
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)

    t0 = time.perf_counter()
    sources = [fc.fc_datastore_build(to_dev(T), synth.VOCAB) for T in inp["corpora"]]
    torch.cuda.synchronize()
    build_s = time.perf_counter() - t0
    build_tokens = sum(len(T) for T in inp["corpora"])

    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], d, 4096)
    kc = torch.empty((B, Hkv, cap, D), dtype=torch.bfloat16, device=dev)
    vc = torch.empty_like(kc)
    g = torch.Generator(device=dev)
    g.manual_seed(inp["seed"])
    kc[:, :, :kv0].normal_(generator=g)
    vc[:, :, :kv0].normal_(generator=g)
    kc[:, :, kv0:].zero_()
    vc[:, :, kv0:].zero_()

    weights = src_weights(args)

    nsub = max(1, min(args.split, B))

    def new_loop():
        if nsub > 1:
            return PipelinedStepLoop(nsub, sources, inp["ctx"], inp["cl"], p, cfg["node_budget"], n_pad, weights, H,
                                     Hkv, D, cap, kv0, synth.VOCAB, cache_capacity=1 << 14, device=dev, k_cache=kc,
                                     v_cache=vc)
        return StepLoop(sources, inp["ctx"], inp["cl"], p, cfg["node_budget"], n_pad, weights, H, Hkv, D, cap, kv0,
                        synth.VOCAB, cache_capacity=1 << 14, device=dev, k_cache=kc, v_cache=vc)

    def join(lp):
        if nsub > 1:
            lp.join()

    # device-resident per-step inputs (a pool of distinct activations, cycled)
    P = min(16, K + W)
    q_pool = torch.randn((P, B, n_pad, H, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    kt_pool = torch.randn((P, B, Hkv, n_pad, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    vt_pool = torch.randn((P, B, Hkv, n_pad, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    hits_d, plen_d, rtok_d = to_dev(inp["hits"]), to_dev(inp["plen"]), to_dev(inp["rtok"])

    loop = new_loop()
    no_hit = torch.zeros(B, dtype=torch.int32, device=dev)
    for s in range(W + K):  # recording pass: fills the replay cache along the trajectory
        loop.step(q_pool[s % P], kt_pool[s % P], vt_pool[s % P], no_hit, plen_d[s], rtok_d[s])
    loop.reset()
    stream = torch.cuda.current_stream()
    mk = lambda: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    # stage events per timed step and sub-batch (recorded on the sub-batch's stream)
    stage_ev = [[dict(attn=mk(), retrieve=mk(), tree=mk(), tail=mk()) for _ in range(nsub)] for _ in range(K)]
    for per_step in stage_ev:  # torch creates an event at its first record: do that before the timed region
        for d in per_step:
            for a, b in d.values():
                a.record()
                b.record()

    def do_step(s, timed_idx=None):
        j = s % P
        evs = None if timed_idx is None else (stage_ev[timed_idx] if nsub > 1 else stage_ev[timed_idx][0])
        loop.step(q_pool[j], kt_pool[j], vt_pool[j], hits_d[s], plen_d[s], rtok_d[s], events=evs)

    for s in range(W):
        do_step(s)
    join(loop)
    assert step_status(fc, loop) == "FC_OK"
    barrier(ws)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.wait_first()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with no_gc():
        start.record(stream)
        for i in range(K):
            do_step(W + i, i)
        join(loop)
        end.record(stream)
        torch.cuda.synchronize()
    clock_rec = clocks.stop()
    barrier(ws)
    t_ms = start.elapsed_time(end)
    status = step_status(fc, loop)
    assert status == "FC_OK", status
    t_max = max_over_ranks(t_ms, ws)
    graph_rec = None
    if not args.no_graph:
        try:
            graph_rec = run_graph_pass(loop, q_pool, kt_pool, vt_pool, hits_d, plen_d, rtok_d, P, W, K)
            assert step_status(fc, loop) == "FC_OK"
        except Exception as e:  # reported, not fatal: the eager line stands
            graph_rec = {"error": f"{type(e).__name__}: {e}"[:200]}
    stage_ms = {k: [[a.elapsed_time(b) for a, b in (stage_ev[i][h][k] for h in range(nsub))] for i in range(K)]
                for k in ("attn", "retrieve", "tree", "tail")}  # [K][nsub] per stage
    attn_ms = stage_ms["attn"]

    # replay the same (deterministic) trajectory untimed to count the
    # attention work of every timed launch
    flops_seq, bytes_seq, nodes_hist, acc_hist, hits_used = replay_counts(inp, sources, p, cfg, cap, kv0, dev, W, K,
                                                                          weights, nsub)
    peaks = load_peaks()
    # the attention kernel's own roofline: the same trajectory on one stream
    # (32 sequences a launch), where each launch shares the GPU with nothing,
    # so its event time is the kernel's own duration
    ss = single_stream_attn(sources, inp, p, cfg, cap, kv0, dev, weights, kc, vc, q_pool, kt_pool, vt_pool, hits_d,
                            plen_d, rtok_d, P, W, min(K, 64), flops_seq, bytes_seq)
    roof = attn_roofline(ss["flops"], ss["bytes"], ss["seconds"], ss["launches"], peaks)
    roof["traffic"] = (attn_traffic(args, roof["algorithmic_bytes_per_launch"]) if args.scale == 1.0
                       else args.traffic_bytes)
    roof["traffic_ratio_to_algorithmic"] = ATTN_TRAFFIC["ratio"] if roof["traffic"] is not None else None
    roof["algorithmic_bytes_first_launches"] = ss["bytes_by_launch"][:3]
    roof["launch"] = (f"k_tree_attn over all {B} sequences on one stream (the step loop's trajectory, "
                      f"first {ss['launches']} timed steps), CUDA events on its stream")
    # the pipelined step's own launches (16 sequences each): their event times
    # include the other sub-batch's kernels running beside them
    piped_f = sum(float(flops_seq[i].sum()) for i in range(K))
    piped_t = sum(attn_ms[i][h] for i in range(K) for h in range(nsub)) * 1e-3
    piped = {"launches": K * nsub, "mean_launch_us": 1e6 * piped_t / (K * nsub),
             "tflops_per_launch_time": piped_f / piped_t / 1e12,
             "note": "per sub-batch launch; the two sub-batches' kernels overlap, so a launch's event time "
                     "includes time shared with the other sub-batch" if nsub > 1 else "the timed loop itself"}

    out = {
        "metric": METRIC, "value": weak_value(K, ws, t_max), "unit": UNIT, "n_gpus": ws, "steps": K, "warmup": W,
        "ms_per_step": t_max / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16 attention (fp32 accumulate) + u32 retrieval", "data": "synthetic",
        **({"graph": graph_rec} if graph_rec else {}),
        "config": {"workload": (WORKLOAD if args.scale == 1.0 else WORKLOAD + f" (scaled x{args.scale})")
                   + ("" if weights == [1, 1] else f", source weights alpha={weights[0]} beta={weights[1]}"),
                   "batch_per_gpu": B, "global_batch": B * ws, "kv_len0": kv0, "n_pad": n_pad,
                   "l2": "inputs larger than L2 (KV cache %.1f GB per GPU)" % (2 * kc.numel() * 2 / 1e9),
                   "parallelism": f"replicas x{ws}",
                   "streams": (f"{nsub} sub-batches of {B // nsub}-{-(-B // nsub)} sequences issued by the native "
                               "step executor, each on a chain stream and an attention stream" if nsub > 1
                               else "one stream")},
        "roofline": roof,
        # per sub-batch step: cached retrieval, insert, tree, attention, predictions, accept, append
        "gpu_launches": 7 * K * nsub,
        "clocks": clock_rec,
        # each stage's mean time per sub-batch launch; with sub-batches on separate
        # streams the stages of different sub-batches overlap, so they do not add up to "all"
        "sub_batches": nsub,
        "stages_ms_per_step": {"tree_attn": mean2(attn_ms), "retrieve": mean2(stage_ms["retrieve"]),
                               "build_tree": mean2(stage_ms["tree"]),
                               "argmax_accept_append": mean2(stage_ms["tail"]), "all": t_ms / K},
        "queries_per_s": ws * B * K / (t_max * 1e-3),
        "retrievals_per_s": ws * (2 * (B * K - hits_used)) / (t_max * 1e-3),
        "tree_attn_tflops": roof["achieved_tflops"],
        "attn_in_timed_step": piped,
        "avg_acceptance_length": float(np.mean([a.mean() + 1 for a in acc_hist])),
        "avg_tree_nodes": float(np.mean([n.mean() for n in nodes_hist])),
        # trees by node count in 32-node bins (1-32, 33-64, 65-96, 97-128): with four
        # query heads per kv head, the number of 128-row tiles a group needs
        "tree_nodes_bins": np.bincount((np.concatenate(nodes_hist) - 1) // 32, minlength=n_pad // 32).tolist(),
        "datastore_build": {"tokens": build_tokens, "seconds": build_s, "tokens_per_s": build_tokens / build_s},
    }
    if not args.no_e2e:
        loop.reset()
        out["e2e"] = run_e2e(loop, inp, dev, W, K, P, q_pool, kt_pool, vt_pool, ws)
    if not args.no_cpu_baseline and rank == 0 and ws == 1:
        out["cpu_baseline"] = cpu_baseline(inp, cfg, kv0, out["avg_tree_nodes"], B)
    return out


def run_graph_pass(loop, q_pool, kt_pool, vt_pool, hits_d, plen_d, rtok_d, P, W, K):
    """The same trajectory again, from the start: the W warm-up steps eager
    (one more when W is odd, since a graph starts at an even step: its
    lengths ping-pong between two buffers), then the timed steps replayed
    from CUDA graphs of G steps each (G = 8, 4 or 2, the largest that divides
    the pool size and the number of timed steps).  The timed steps are the K
    steps after the warm-up, or K - 1 when the odd warm-up took one of them
    (K - 1 is then rounded down to a multiple of 2).
    A pipelined loop: every window of G timed steps has, per sub-batch, a
    graph of its own captured by the step executor (kernels at the eager
    streams' priorities, uploaded at capture), reading that window's inputs
    where the eager loop reads them; each sub-batch launches its graphs into
    a stream of its own, so the sub-batches never join.  One stream: one graph
    per pool offset, reading the pooled activations directly, with a step's
    small draws copied into the graph's input buffers before each replay."""
    import torch
    W2 = W + (W % 2)
    K2 = K - (W2 - W)
    G = next((g for g in (8, 4, 2) if K2 % g == 0 and P % g == 0), None)
    if G is None:
        K2 -= K2 % 2
        G = 2 if P % 2 == 0 and K2 >= 2 else None
    if G is None:
        return {"skipped": "needs an even pool size and at least 2 steps after the warm-up"}
    loop.reset()
    for s in range(W2):  # eager warm-up; it also makes workspaces and kernel attributes
        loop.step(q_pool[s % P], kt_pool[s % P], vt_pool[s % P], hits_d[s], plen_d[s], rtok_d[s])
    parts = hasattr(loop, "capture_native")  # a pipelined loop: graphs per sub-batch, never joined
    slices = loop.slices if parts else [slice(None)]
    small = [(torch.empty_like(hits_d[0]), torch.empty_like(plen_d[0]), torch.empty_like(rtok_d[0])) for _ in range(G)]
    graphs = {}
    if parts:
        for s0 in range(W2, W2 + K2, G):
            ins = [(q_pool[(s0 + t) % P], kt_pool[(s0 + t) % P], vt_pool[(s0 + t) % P], hits_d[s0 + t], plen_d[s0 + t],
                    rtok_d[s0 + t]) for t in range(G)]
            graphs[s0] = loop.capture_native(ins)
    else:
        for i in range(P // G):
            s0 = W2 + i * G
            ins = [(q_pool[(s0 + t) % P], kt_pool[(s0 + t) % P], vt_pool[(s0 + t) % P]) + small[t] for t in range(G)]
            graphs[s0 % P] = [loop.capture(ins)]
    main = torch.cuda.current_stream()
    streams = [torch.cuda.Stream() for _ in slices] if parts else [main]

    def block(s):
        if parts:  # each sub-batch launches its graph of this window on its own stream
            for h, st in enumerate(streams):
                with torch.cuda.stream(st):
                    graphs[s][h].launch()
            return
        for t in range(G):  # one stream: the step's small draws into the graph's buffers, then the replay
            small[t][0].copy_(hits_d[s + t])
            small[t][1].copy_(plen_d[s + t])
            small[t][2].copy_(rtok_d[s + t])
        graphs[s % P][0].replay()

    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record()
    for st in streams:
        st.wait_stream(main)
    for i in range(0, K2, G):
        block(W2 + i)
    for st in streams:
        main.wait_stream(st)
    end.record()
    torch.cuda.synchronize()
    ms = start.elapsed_time(end) / K2
    return {"ms_per_step": ms, "steps_per_s": 1e3 / ms, "steps": K2, "eager_warmup_steps": W2,
            "graphs": sum(len(g) for g in graphs.values()), "steps_per_graph": G,
            "note": f"the timed steps from graphs of {G} steps"
                    + (", per window of steps and sub-batch, captured by the step executor (kernel nodes at their "
                       "streams' priorities, uploaded at capture) and reading the window's inputs where the eager "
                       "loop reads them; each sub-batch launches its graphs into a stream of its own (the "
                       "sub-batches never join)" if parts else
                       " (first replays include the graphs' upload); the step's small draws copied in before "
                       "each replay")}


def single_stream_attn(sources, inp, p, cfg, cap, kv0, dev, weights, kc, vc, q_pool, kt_pool, vt_pool, hits_d, plen_d,
                       rtok_d, P, W, K2, flops_seq, bytes_seq):
    """The attention launches of the first K2 timed steps, run on one stream
    (the step loop over the whole batch, from the same starting state, the
    same trajectory), each timed with CUDA events on its stream.  Returns the
    launches' total algorithmic FLOPs and bytes and their total time."""
    import torch

    import paper_2502_17139_gb300.synth as synth
    from paper_2502_17139_gb300.step import StepLoop
    kc[:, :, kv0:].zero_()
    vc[:, :, kv0:].zero_()
    lp = StepLoop(sources, inp["ctx"], inp["cl"], p, cfg["node_budget"], cfg["n_pad"], weights, cfg["H"], cfg["Hkv"],
                  cfg["D"], cap, kv0, synth.VOCAB, cache_capacity=1 << 14, device=dev, k_cache=kc, v_cache=vc)
    mk = lambda: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    no_hit = torch.zeros_like(hits_d[0])
    for s in range(W + K2):  # recording pass, as in the timed run
        lp.step(q_pool[s % P], kt_pool[s % P], vt_pool[s % P], no_hit, plen_d[s], rtok_d[s])
    lp.reset()
    evs = []
    for s in range(W + K2):
        e = dict(attn=mk()) if s >= W else None
        lp.step(q_pool[s % P], kt_pool[s % P], vt_pool[s % P], hits_d[s], plen_d[s], rtok_d[s], events=e)
        if e:
            evs.append(e["attn"])
    torch.cuda.synchronize()
    t = sum(a.elapsed_time(b) for a, b in evs) * 1e-3
    f = sum(float(flops_seq[i].sum()) for i in range(K2))
    by = sum(float(bytes_seq[i].sum()) for i in range(K2))
    return {"launches": K2, "seconds": t, "flops": f, "bytes": by,
            "bytes_by_launch": [float(bytes_seq[i].sum()) for i in range(K2)]}


def attn_roofline(flops, nbytes, seconds, launches, peaks):
    """The roofline object of the attention kernel from its launches' total
    algorithmic FLOPs and bytes and their total event time.  The kernel is
    timed in a region of milliseconds, so the tensor peak is the burst one.
    The bound is whichever floor (tensor time or HBM time) is larger; the
    other side's fraction is reported beside it."""
    ach_tf = flops / seconds / 1e12
    ach_gb = nbytes / seconds / 1e9
    tensor_frac = ach_tf / peaks["tc_burst"]
    hbm_frac = ach_gb / peaks["hbm"]
    tensor_bound = flops / (peaks["tc_burst"] * 1e12) >= nbytes / (peaks["hbm"] * 1e9)
    roof = dict(bound="tensor" if tensor_bound else "hbm", achieved=ach_tf if tensor_bound else ach_gb,
                peak=peaks["tc_burst"] if tensor_bound else peaks["hbm"], unit="TFLOP/s" if tensor_bound else "GB/s")
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["peak_source"] = peaks["source"] + (" burst bf16 (bf16_tflops)" if tensor_bound else " hbm copy (hbm_gbs)")
    roof.update(kernel="k_tree_attn", launches=launches, mean_launch_us=1e6 * seconds / launches,
                algorithmic_flops_per_launch=flops / launches, algorithmic_bytes_per_launch=nbytes / launches,
                achieved_tflops=ach_tf, tensor_frac=tensor_frac, achieved_gbs=ach_gb, hbm_frac=hbm_frac,
                tensor_frac_of_sustained=ach_tf / peaks["tc_sustained"])
    return roof


def mean2(rows):
    return float(np.mean(np.asarray(rows, np.float64)))


def replay_counts(inp, sources, p, cfg, cap, kv0, dev, W, K, weights=(1, 1), nsub=1):
    """Re-run the loop (untimed, fresh state, the same sub-batches) and count
    the attention work of every timed step per sequence: FLOPs over unmasked
    (q, k) pairs and algorithmic HBM bytes ([K] arrays over the batch)."""
    import torch

    import paper_2502_17139_gb300.synth as synth
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    B, H, Hkv, D, n_pad = inp["B"], cfg["H"], cfg["Hkv"], cfg["D"], cfg["n_pad"]
    kc = torch.zeros((B, Hkv, cap, D), dtype=torch.bfloat16, device=dev)
    largs = (sources, inp["ctx"], inp["cl"], p, cfg["node_budget"], n_pad, list(weights), H, Hkv, D, cap, kv0,
             synth.VOCAB)
    lkw = dict(cache_capacity=1 << 14, device=dev, k_cache=kc, v_cache=kc)
    loop = PipelinedStepLoop(nsub, *largs, **lkw) if nsub > 1 else StepLoop(*largs, **lkw)
    join = loop.join if nsub > 1 else (lambda: None)
    q = torch.zeros((B, n_pad, H, D), dtype=torch.bfloat16, device=dev)
    kt = torch.zeros((B, Hkv, n_pad, D), dtype=torch.bfloat16, device=dev)
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
    flops, bytes_, nodes_hist, acc_hist = [], [], [], []
    hits_used = 0
    zero = to_dev(np.zeros(B, np.int32))
    for s in range(W + K):  # recording pass, as in the timed run
        loop.step(q, kt, kt, zero, to_dev(inp["plen"][s]), to_dev(inp["rtok"][s]), attention=False)
    loop.reset()
    for s in range(W + K):
        join()
        kvl = loop.kv_len_now.cpu().numpy().astype(np.int64)
        loop.step(q, kt, kt, to_dev(inp["hits"][s]), to_dev(inp["plen"][s]), to_dev(inp["rtok"][s]), attention=False)
        join()
        if s < W:
            continue
        nn = loop.tree["n_nodes"].cpu().numpy().astype(np.int64)
        dep = loop.tree["depth"].cpu().numpy().astype(np.int64)
        pairs = np.array([H * (nn[b] * kvl[b] + int((dep[b, :nn[b]] + 1).sum())) for b in range(B)], np.float64)
        flops.append(4.0 * D * pairs)
        by = (2 * Hkv * kvl * D * 2          # K and V cache rows
              + 2 * Hkv * nn * D * 2         # tree K and V
              + 2 * nn * H * D * 2           # Q in, O out
              + nn * (n_pad // 64) * 8)      # mask rows
        bytes_.append(by.astype(np.float64))
        nodes_hist.append(nn)
        acc_hist.append(loop.acc["acc_len"].cpu().numpy())
        hits_used += int(loop.skip.sum().item())
    return flops, bytes_, nodes_hist, acc_hist, hits_used


def run_e2e(loop, inp, dev, W, K, P, q_pool, kt_pool, vt_pool, ws):
    """Same metric through the public API with host buffers: each step copies
    its inputs host->device from pinned memory and reads its result
    (accepted lengths and bonus tokens) back to the host.  The copies run on
    a second stream into two alternating input sets, so step s + 1's inputs
    travel while step s computes (copy of s + 1 waits until step s - 1 has
    finished reading that set)."""
    import torch
    R = min(4, P)
    hq = [q_pool[j].cpu().pin_memory() for j in range(R)]
    hk = [kt_pool[j].cpu().pin_memory() for j in range(R)]
    hv = [vt_pool[j].cpu().pin_memory() for j in range(R)]
    B = inp["B"]
    hh = torch.from_numpy(inp["hits"].view(np.int32)).pin_memory()
    hp = torch.from_numpy(inp["plen"].view(np.int32)).pin_memory()
    hr = torch.from_numpy(np.ascontiguousarray(inp["rtok"]).view(np.int32)).pin_memory()
    sets = [dict(q=torch.empty_like(q_pool[0]), k=torch.empty_like(kt_pool[0]), v=torch.empty_like(vt_pool[0]),
                 h=torch.empty(B, dtype=torch.int32, device=dev), p=torch.empty(B, dtype=torch.int32, device=dev),
                 r=torch.empty(inp["rtok"].shape[1:], dtype=torch.int32, device=dev)) for _ in range(2)]
    main = torch.cuda.current_stream()
    cs = torch.cuda.Stream()
    # (loop, sequences, stream) per sub-batch: a pipelined loop's sub-batches
    # read the inputs and write the results on their own streams, each into its
    # own pinned buffer (a copy into a slice of one buffer at an odd offset is
    # not asynchronous)
    subs = list(zip(loop.loops, loop.slices, loop.streams)) if hasattr(loop, "loops") else [(loop, slice(0, B), main)]
    res = [torch.empty((2, sl.stop - sl.start), dtype=torch.int32).pin_memory() for _, sl, _ in subs]
    copied = [torch.cuda.Event() for _ in range(2)]
    consumed = [[torch.cuda.Event() for _ in subs] for _ in range(2)]
    for evs in consumed:
        for e in evs:
            e.record(main)

    def copy_in(s):
        slot, j = s % 2, s % R
        d = sets[slot]
        with torch.cuda.stream(cs):
            for e in consumed[slot]:
                cs.wait_event(e)
            d["q"].copy_(hq[j], non_blocking=True)
            d["k"].copy_(hk[j], non_blocking=True)
            d["v"].copy_(hv[j], non_blocking=True)
            d["h"].copy_(hh[s], non_blocking=True)
            d["p"].copy_(hp[s], non_blocking=True)
            d["r"].copy_(hr[s], non_blocking=True)
            copied[slot].record(cs)

    def run(first, count):
        copy_in(first)
        for s in range(first, first + count):
            if s + 1 < first + count:
                copy_in(s + 1)
            slot = s % 2
            d = sets[slot]
            main.wait_event(copied[slot])
            loop.step(d["q"], d["k"], d["v"], d["h"], d["p"], d["r"])
            for h, (lp, sl, st) in enumerate(subs):
                with torch.cuda.stream(st):
                    consumed[slot][h].record(st)
                    res[h][0].copy_(lp.acc["acc_len"], non_blocking=True)
                    res[h][1].copy_(lp.acc["bonus"], non_blocking=True)

    run(0, W)
    torch.cuda.synchronize()
    barrier(ws)
    with no_gc():
        t0 = time.perf_counter()
        run(W, K)
        torch.cuda.synchronize()
        t1 = time.perf_counter()
    import paper_2502_17139_gb300.fastcoder as fc
    status = step_status(fc, loop)
    assert status == "FC_OK", status
    t = max_over_ranks(t1 - t0, ws)
    d = sets[0]
    h2d = d["q"].numel() * 2 + d["k"].numel() * 2 + d["v"].numel() * 2 + 4 * (2 * B + d["r"].numel())
    return {"value": weak_value(K, ws, t * 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(sum(r.numel() for r in res) * 4),
            "note": "host->device copies on a second stream, double-buffered: step s + 1's inputs travel while "
                    "step s computes"}


# ------------------------------------------------------------ CPU oracle
def cpu_baseline(inp, cfg, kv0, avg_nodes, B, budget_s=20.0):
    """The oracle (as it stands) on a bounded sample of one step, scaled to a
    full step: retrieval for a few queries on both sources, a tree and an
    acceptance walk for them, and attention for one (sequence, kv head)
    group; each stage's time per unit times the units of one full step."""
    import paper_2502_17139_gb300.synth as synth
    from oracle import oracle as orc
    rng = synth.rng_for(5, 777)
    nq = 2
    qs = np.arange(nq)
    t0 = time.perf_counter()
    res = [orc.retrieve(T, inp["ctx"][qs], inp["cl"][qs], cfg["n_max"], cfg["n_min"], cfg["top_k"],
                        cfg["draft_len"], 4096) for T in inp["corpora"]]
    t_ret = (time.perf_counter() - t0) / (nq * len(inp["corpora"]))
    root = inp["ctx"][qs, inp["cl"][qs] - 1]
    t0 = time.perf_counter()
    tr = orc.build_tree(res, [1, 1], root, np.full(nq, kv0, np.int32), cfg["node_budget"], cfg["n_pad"])
    am = orc.synth_argmax(tr["tok"], tr["parent"], tr["n_nodes"], inp["plen"][0][qs], inp["rtok"][0][qs], synth.VOCAB)
    orc.accept(tr["tok"], tr["parent"], tr["n_nodes"], am, cfg["draft_len"] + 2)
    t_tree = (time.perf_counter() - t0) / nq
    # attention for one (sequence, kv group): G query heads x its nodes
    H, Hkv, D, n_pad = cfg["H"], cfg["Hkv"], cfg["D"], cfg["n_pad"]
    G = H // Hkv
    n = max(1, int(round(avg_nodes)))
    bits = lambda a: (a.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = bits(rng.standard_normal((1, n_pad, H, D), dtype=np.float32))
    kc = bits(rng.standard_normal((1, Hkv, kv0, D), dtype=np.float32))
    kt = bits(rng.standard_normal((1, Hkv, n_pad, D), dtype=np.float32))
    par = np.full((1, n_pad), -1, np.int32)
    _, pp = synth.random_tree(rng, n, 10, 4, 1000)
    par[0, :n] = pp
    mask = orc.tree_mask(par, np.array([n], np.int32), np.array([kv0], np.int32), n_pad)["mask"]
    rows = np.array([(0, i, h) for i in range(n) for h in range(G)], np.int32)
    t0 = time.perf_counter()
    orc.tree_attn(q, kc, kc, np.array([kv0], np.int32), kt, kt, mask, np.array([n], np.int32), rows=rows)
    t_attn_group = time.perf_counter() - t0
    hit_rate = float(inp["hits"].mean())  # the replay cache holds every key of the trajectory
    step_s = (t_ret * B * len(inp["corpora"]) * (1 - hit_rate) + t_tree * B + t_attn_group * B * Hkv)
    cores = orc.hardware_threads()
    return {"value": 1.0 / step_s, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": (f"{nq} queries x {len(inp['corpora'])} sources retrieval (linear corpus scans), their trees "
                       f"and acceptance, attention for 1 (sequence, kv-head) group ({G} heads x {n} nodes x "
                       f"{kv0} keys, fp64); per-unit times scaled to one step of {B} sequences"),
            "stage_seconds_per_unit": {"retrieve": t_ret, "tree_accept": t_tree, "attn_group": t_attn_group}}


def run_reference(args, rank, ws):
    """CPU oracle arm: the step loop through the oracle on the host cores.

    Every timed step is a full, unsampled step of all B sequences: the
    replay-cache lookup and the retrievals it does not serve (both sources,
    linear corpus scans), the trees, the tree attention of every (sequence,
    node, query head) row in fp64 against the whole KV cache, the synthetic
    target model, acceptance and the cache append.  As in the GPU arm, a
    recording pass first fills the replay cache along the trajectory (no
    hits, no attention), and the W warm-up steps advance the trajectory
    before the timed ones; they skip the attention, which does not steer the
    trajectory."""
    if rank != 0:
        return None
    import paper_2502_17139_gb300.synth as synth
    from oracle import oracle as orc
    K, W = args.steps, args.warmup
    inp = make_inputs(args.scale, args.batch, 0, K + W + 1)
    cfg, B, kv0 = inp["cfg"], inp["B"], inp["kv0"]
    H, Hkv, D, n_pad, d = cfg["H"], cfg["Hkv"], cfg["D"], cfg["n_pad"], cfg["draft_len"]
    cap = kv0 + (K + W + 1) * (d + 1) + 8
    rng = synth.rng_for(5, 999)
    block = (rng.standard_normal(1 << 22, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)
    tile = lambda shape, off: np.resize(np.roll(block, off), shape)  # bf16 N(0,1) bit patterns
    kc, vc = tile((B, Hkv, cap, D), 0), tile((B, Hkv, cap, D), 12345)
    q, kt, vt = tile((B, n_pad, H, D), 777), tile((B, Hkv, n_pad, D), 999), tile((B, Hkv, n_pad, D), 4242)
    po = dict(n_max=cfg["n_max"], n_min=cfg["n_min"], top_k=cfg["top_k"], max_occ=4096)
    weights = src_weights(args)
    cache = {}

    def run(hits, timed_from, attention):
        ctx, cl = inp["ctx"].copy(), inp["cl"].copy()
        kvl = np.full(B, kv0, np.int32)
        times = []
        for s in range(W + K):
            t0 = time.perf_counter()
            keys = [orc.cache_key(ctx[b], cl[b], po["n_max"]) for b in range(B)]
            served = [bool(hits[s, b]) and keys[b] in cache for b in range(B)]
            todo = np.array([b for b in range(B) if not served[b]], np.int64)
            res = [dict(drafts=np.full((B, po["top_k"], d), PAD_TOKEN, np.uint32),
                        draft_len=np.zeros((B, po["top_k"]), np.int32), count=np.zeros((B, po["top_k"]), np.uint32),
                        n_drafts=np.zeros(B, np.int32), match_len=np.zeros(B, np.int32)) for _ in inp["corpora"]]
            for b in range(B):
                if served[b]:
                    for si, r in enumerate(res):
                        for name in r:
                            r[name][b] = cache[keys[b]][si][name]
            if len(todo):
                for si, T in enumerate(inp["corpora"]):
                    r = orc.retrieve(T, ctx[todo], cl[todo], po["n_max"], po["n_min"], po["top_k"], d, po["max_occ"])
                    for name in r:
                        res[si][name][todo] = r[name]
                for b in todo:
                    cache[keys[b]] = [{name: r[name][b].copy() for name in r} for r in res]
            root = ctx[np.arange(B), cl - 1]
            tr = orc.build_tree(res, weights, root, kvl, cfg["node_budget"], n_pad)
            if attention and s >= timed_from:
                orc.tree_attn(q, kc, vc, kvl, kt, vt, tr["mask"], tr["n_nodes"])
            am = orc.synth_argmax(tr["tok"], tr["parent"], tr["n_nodes"], inp["plen"][s], inp["rtok"][s], synth.VOCAB)
            ac = orc.accept(tr["tok"], tr["parent"], tr["n_nodes"], am, d + 2)
            kvl, cl, _ = orc.kv_append(ac["path"], ac["acc_len"], ac["bonus"], tr["tok"], kt, vt, kc, vc, kvl, ctx, cl)
            if s >= timed_from:
                times.append(time.perf_counter() - t0)
        return times

    run(np.zeros_like(inp["hits"]), W + K, False)   # recording pass
    times = run(inp["hits"], W, True)
    step_s = statistics.mean(times)
    cores = orc.hardware_threads()
    value = 1.0 / step_s
    sample = (f"every timed step is a full step of all {B} sequences (replay-cache lookup, retrieval on both sources "
              f"for the queries it does not serve, trees, fp64 tree attention of every row, acceptance, append); "
              f"{K} timed steps after {W} warm-up steps and a recording pass")
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": K, "warmup": W,
            "ms_per_step": 1e3 * step_s, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64 attention + u32 retrieval", "data": "synthetic", "impl": "reference",
            "config": {"workload": WORKLOAD if args.scale == 1.0 else WORKLOAD + f" (scaled x{args.scale})",
                       "batch_per_gpu": B, "kv_len0": kv0, "parallelism": "cpu oracle"},
            "step_seconds": {"min": min(times), "max": max(times)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def run_attn(args, rank, ws, local):
    """Tree attention alone: B sequences x 8 KV heads x 32 query heads,
    head dim 128, KV length --kv, seeded random trees of --nodes nodes."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    B, H, Hkv, D, n_pad, L = args.batch, 32, 8, 128, 128, args.kv
    rng = synth.rng_for(5, 500 + rank)
    par = np.full((B, n_pad), -1, np.int32)
    for b in range(B):
        _, pp = synth.random_tree(rng, args.nodes, 10, 4, synth.VOCAB)
        par[b, :args.nodes] = pp
    nn = np.full(B, args.nodes, np.int32)
    kvl = np.full(B, L, np.int32)
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    m = fc.fc_tree_mask(to_dev(par), to_dev(nn), to_dev(kvl))
    g = torch.Generator(device=dev)
    g.manual_seed(7 + rank)
    rnd = lambda *shape: torch.randn(*shape, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    q, kc, vc = rnd(B, n_pad, H, D), rnd(B, Hkv, L, D), rnd(B, Hkv, L, D)
    kt, vt = rnd(B, Hkv, n_pad, D), rnd(B, Hkv, n_pad, D)
    out = torch.empty_like(q)
    args_d = (q, kc, vc, to_dev(kvl), kt, vt, m["mask"], to_dev(nn))
    if args.rope:
        pos = m["pos"]
        kt_rot = fc.fc_rope(kt, pos, 10000.0, layout=1)
        args_d = (q, kc, vc, to_dev(kvl), kt_rot, vt, m["mask"], to_dev(nn))
        attn = lambda: fc.fc_tree_attn_rope(*args_d, pos, 10000.0, out=out)
        rope_k_ms = _gpu_ms(lambda: fc.fc_rope(kt, pos, 10000.0, layout=1, out=kt_rot))
    else:
        attn = lambda: fc.fc_tree_attn(*args_d, out=out)
    for _ in range(args.warmup):
        attn()
    assert fc.fc_get_error() == "FC_OK"
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier(ws)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.wait_first()
    for e0, e1 in evs:
        e0.record()
        attn()
        e1.record()
    torch.cuda.synchronize()
    clock_rec = clocks.stop()
    ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in evs)
    dep = m["depth"].cpu().numpy()
    pairs = sum(H * (args.nodes * L + int((dep[b, :args.nodes] + 1).sum())) for b in range(B))
    flops = 4.0 * D * pairs
    bytes_ = B * (2 * Hkv * L * D * 2 + 2 * Hkv * args.nodes * D * 2 + 2 * args.nodes * H * D * 2)
    peaks = load_peaks()
    return {"metric": "tree-attn TFLOP/s", "value": flops / (ms * 1e-3) / 1e12, "unit": "TFLOP/s",
            "n_gpus": ws, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "config": {"workload": f"tree attention B={B} H=32 Hkv=8 D=128 KV={L} nodes={args.nodes}"
                                   + (", RoPE by node position" if args.rope else "")},
            "frac_tensor_sustained": flops / (ms * 1e-3) / 1e12 / peaks["tc_sustained"],
            "frac_hbm": bytes_ / (ms * 1e-3) / 1e9 / peaks["hbm"], "flops": flops, "bytes": bytes_,
            "rope": ({"queries": "rotated inside the attention kernel", "tree_key_rotation_ms": rope_k_ms}
                     if args.rope else None),
            "clocks": clock_rec}


def run_argmax(args, rank, ws, local):
    """fc_argmax_accept alone: B sequences of seeded random trees (node counts
    uniform in [40, 128], mean ~84 like the step loop's), bf16 N(0,1) logits over
    the 32256-token vocabulary whose argmax follows the first branch for a
    seeded 0-8 prefix.  HBM-bound: every valid row is read once."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    B, n_pad, V = args.batch, 128, synth.VOCAB
    rng = synth.rng_for(6, 600 + rank)
    tok = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(40, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        t, pp = synth.random_tree(rng, int(nn[b]), 10, 4, V)
        tok[b, :nn[b]], par[b, :nn[b]] = t, pp
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32) if a.dtype == np.uint32
                                        else np.ascontiguousarray(a)).to(dev)
    plen, rtok = synth.argmax_draws(rng, B, n_pad, V)
    pred = fc.fc_synth_argmax(to_dev(tok), to_dev(par), to_dev(nn), to_dev(plen), to_dev(rtok), V)
    g = torch.Generator(device=dev)
    g.manual_seed(11 + rank)
    logits = torch.randn((B, n_pad, V), generator=g, device=dev, dtype=torch.float32)
    logits.scatter_(2, pred.long().unsqueeze(2), 8.0)  # the planted predictions win
    logits = logits.to(torch.bfloat16)
    args_d = (logits, to_dev(tok), to_dev(par), to_dev(nn), 12)
    out = fc.fc_argmax_accept(*args_d)
    assert torch.equal(out["argmax"], pred), "planted predictions were not the argmax"
    for _ in range(args.warmup):
        fc.fc_argmax_accept(*args_d, out=out)
    assert fc.fc_get_error() == "FC_OK"
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier(ws)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.wait_first()
    for e0, e1 in evs:
        e0.record()
        fc.fc_argmax_accept(*args_d, out=out)
        e1.record()
    torch.cuda.synchronize()
    clock_rec = clocks.stop()
    ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in evs)
    rows = int(nn.sum())
    bytes_ = rows * V * 2 + B * n_pad * 4 + B * n_pad * 8  # logits rows read, predictions written, tree read
    peaks = load_peaks()
    gbs = bytes_ / (ms * 1e-3) / 1e9
    return {"metric": "argmax+accept GB/s", "value": gbs, "unit": "GB/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "config": {"workload": f"greedy verification from logits B={B} n_pad={n_pad} vocab={V} "
                                   f"rows={rows} (logits {B * n_pad * V * 2 / 1e6:.0f} MB)"},
            "frac_hbm": gbs / peaks["hbm"], "bytes": bytes_,
            "mean_acc_len": float(out["acc_len"].float().mean().item()), "clocks": clock_rec}


def _gpu_ms(fn, reps=20, warm=3, spin_cycles=4_000_000):
    """Mean device time of fn() over `reps` back-to-back calls, with the host
    enqueueing ahead of the device (the stream first spins ~2 ms), so that a
    kernel of a few microseconds is not timed together with the host's own
    per-call overhead."""
    import torch
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(spin_cycles)
    e0.record()
    for _ in range(reps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def _cuda_ms(fn, reps=10, warm=3):
    """Mean CUDA-event time of fn() on the current stream, after warm-up."""
    import torch
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    for e0, e1 in ev:
        e0.record()
        fn()
        e1.record()
    torch.cuda.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in ev)


def _attn_work(fc, tree, kvl, H, Hkv, D):
    """Unmasked (q, k) pair FLOPs and algorithmic bytes of one tree-attention call."""
    nn = tree["n_nodes"].cpu().numpy().astype(np.int64)
    dep = tree["depth"].cpu().numpy().astype(np.int64)
    B = len(nn)
    pairs = sum(H * (nn[b] * kvl[b] + int((dep[b, :nn[b]] + 1).sum())) for b in range(B))
    by = sum(2 * Hkv * kvl[b] * D * 2 + 2 * Hkv * nn[b] * D * 2 + 2 * nn[b] * H * D * 2 for b in range(B))
    return 4.0 * D * pairs, float(by)


def run_configs(args, rank, ws, local):
    """Every stage of the five configurations on this GPU (CUDA events, mean of
    10 after 3 warm-up calls): a report of where each configuration stands
    against its roofline; the benchmark line is the step loop (--mode step)."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    peaks = load_peaks()
    tc, bw = peaks["tc_sustained"] * 1e12, peaks["hbm"] * 1e9
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32) if a.dtype == np.uint32
                                        else np.ascontiguousarray(a)).to(dev)
    out = {"metric": "per-configuration stage times", "unit": "ms", "configs": {}}

    def attn_entry(tree, kvl, H, Hkv, D, L_cap, seed):
        B, n_pad = tree["tok"].shape
        g = torch.Generator(device=dev)
        g.manual_seed(seed)
        rnd = lambda *sh: torch.randn(*sh, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
        q, kc, vc = rnd(B, n_pad, H, D), rnd(B, Hkv, L_cap, D), rnd(B, Hkv, L_cap, D)
        kt, vt = rnd(B, Hkv, n_pad, D), rnd(B, Hkv, n_pad, D)
        o = torch.empty_like(q)
        kv_d = to_dev(np.asarray(kvl, np.int32))
        ms = _gpu_ms(lambda: fc.fc_tree_attn(q, kc, vc, kv_d, kt, vt, tree["mask"], tree["n_nodes"], out=o))
        F, By = _attn_work(fc, tree, kvl, H, Hkv, D)
        t_roof = max(F / tc, By / bw)
        return {"ms": ms, "tflops": F / (ms * 1e-3) / 1e12, "gbs": By / (ms * 1e-3) / 1e9,
                "bound": "tensor" if F / tc >= By / bw else "hbm", "frac_of_roofline": t_roof / (ms * 1e-3)}

    def accept_entry(tree, V, seed, plen_max=8):
        B, n_pad = tree["tok"].shape
        rng = synth.rng_for(7, seed)
        plen, rtok = synth.argmax_draws(rng, B, n_pad, V, plen_max)
        am = fc.fc_synth_argmax(tree["tok"], tree["parent"], tree["n_nodes"], to_dev(plen), to_dev(rtok), V)
        acc = fc.fc_accept(tree["tok"], tree["parent"], tree["n_nodes"], am, 12)
        ms = _gpu_ms(lambda: fc.fc_accept(tree["tok"], tree["parent"], tree["n_nodes"], am, 12, out=acc))
        nn = tree["n_nodes"].cpu().numpy()
        by = float(sum(12 * int(n) + 4 * (12 + 2) for n in nn))
        return {"ms": ms, "gbs": by / (ms * 1e-3) / 1e9, "frac_hbm": by / (ms * 1e-3) / bw,
                "mean_acc_len": float(acc["acc_len"].float().mean().item())}

    def retrieval_entry(sources, ctx, cl, cfg, budget, n_pad, kv0):
        p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
        ctx_d, cl_d = to_dev(ctx), to_dev(cl)
        res = fc.fc_retrieve(sources, ctx_d, cl_d, p)
        ms_r = _gpu_ms(lambda: fc.fc_retrieve(sources, ctx_d, cl_d, p, out=res))
        B = ctx.shape[0]
        root = to_dev(ctx[np.arange(B), cl - 1].astype(np.uint32))
        kvl = to_dev(np.full(B, kv0, np.int32))
        tree = fc.fc_build_tree(res, [1] * len(sources), root, kvl, budget, n_pad)
        ms_t = _gpu_ms(lambda: fc.fc_build_tree(res, [1] * len(sources), root, kvl, budget, n_pad, out=tree))
        ml = res["match_len"].cpu().numpy()
        return tree, {"retrieve_ms": ms_r, "queries_per_s": B / (ms_r * 1e-3),
                      "us_per_query_source": ms_r * 1e3 / (B * len(sources)),
                      "matched_share": float((ml > 0).mean()), "build_tree_ms": ms_t,
                      "mean_tree_nodes": float(tree["n_nodes"].float().mean().item())}

    def build_entry(T):
        t0 = time.perf_counter()
        ds = fc.fc_datastore_build(to_dev(T), synth.VOCAB)
        torch.cuda.synchronize()
        sec = time.perf_counter() - t0
        return ds, {"tokens": int(len(T)), "seconds": sec, "tokens_per_s": len(T) / sec}

    # c1: single source 1M, B=32, attention H = Hkv = 32, KV 512
    cfg = synth.WORKLOADS[1]
    rng = synth.rng_for(1)
    T, _ = synth.build_corpus(rng, cfg["corpus"][0], device="cuda")
    ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], [T], [1.0], 1.1)
    ds, e_build = build_entry(T)
    tree, e_ret = retrieval_entry([ds], ctx, cl, cfg, cfg["node_budget"], cfg["n_pad"], cfg["kv_len"])
    kvl = [cfg["kv_len"]] * cfg["batch"]
    out["configs"]["c1"] = dict(datastore_build=e_build, retrieval_and_tree=e_ret,
                                tree_attn=attn_entry(tree, kvl, cfg["H"], cfg["Hkv"], cfg["D"], cfg["kv_len"], 1),
                                accept=accept_entry(tree, synth.VOCAB, 1))
    del ds, T
    # c2: two sources 5M + 100M, B=256, 64-node trees
    cfg = synth.WORKLOADS[2]
    rng = synth.rng_for(2)
    corpora = [synth.build_corpus(rng, spec, device="cuda")[0] for spec in cfg["corpus"]]
    ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], corpora + [None], cfg["probs"],
                                     1.1)
    built = [build_entry(T) for T in corpora]
    tree, e_ret = retrieval_entry([b[0] for b in built], ctx, cl, cfg, cfg["node_budget"], cfg["n_pad"], 4096)
    out["configs"]["c2"] = dict(datastore_build=[b[1] for b in built], retrieval_and_tree=e_ret)
    del built, corpora
    # c3: attention at the 7B shape, B=16, H = Hkv = 32, KV 4096, 64-node random trees; acceptance
    cfg = synth.WORKLOADS[3]
    rng = synth.rng_for(3)
    B, n_pad, nnod = cfg["batch"], cfg["n_pad"], cfg["n_nodes"]
    tok = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    for b in range(B):
        t, pp = synth.random_tree(rng, nnod, cfg["depth_max"], cfg["branch_max"], synth.VOCAB)
        tok[b, :nnod], par[b, :nnod] = t, pp
    nn = np.full(B, nnod, np.int32)
    kvl = [cfg["kv_len"]] * B
    m = fc.fc_tree_mask(to_dev(par), to_dev(nn), to_dev(np.asarray(kvl, np.int32)))
    tree3 = dict(tok=to_dev(tok), parent=to_dev(par), n_nodes=to_dev(nn), mask=m["mask"], depth=m["depth"])
    out["configs"]["c3"] = dict(tree_attn=attn_entry(tree3, kvl, cfg["H"], cfg["Hkv"], cfg["D"], cfg["kv_len"], 3),
                                accept=accept_entry(tree3, synth.VOCAB, 3))
    # c4: 1B tokens, B=1024, n 24 -> 2, top-64 x 12, 128-node trees
    if not args.skip_1b:
        cfg = synth.WORKLOADS[4]
        rng = synth.rng_for(4)
        T, planted = synth.build_corpus(rng, cfg["corpus"][0], device="cuda")
        ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], [T], [1.0], 1.1,
                                         planted=[planted], planted_share=cfg["planted_share"])
        ds, e_build = build_entry(T)
        tree, e_ret = retrieval_entry([ds], ctx, cl, cfg, cfg["node_budget"], cfg["n_pad"], 0)
        out["configs"]["c4"] = dict(datastore_build=e_build, retrieval_and_tree=e_ret)
        del ds, T
    out["configs"]["c5"] = "the step loop: python bench.py (the benchmark line)"
    return out


def run_retrieve(args, rank, ws, local):
    """Two-source retrieval alone on the step loop's datastores (5M + 100M) for
    --batch contexts of the step loop's query mix: a batch sweep shows where the
    dependent-probe chain stops hiding behind parallelism."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    cfg = synth.WORKLOADS[2]
    rng = synth.rng_for(2)
    corpora = [synth.build_corpus(rng, spec, device="cuda")[0] for spec in cfg["corpus"]]
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32) if a.dtype == np.uint32
                                        else np.ascontiguousarray(a)).to(dev)
    sources = [fc.fc_datastore_build(to_dev(T), synth.VOCAB) for T in corpora]
    ctx, cl, _ = synth.make_contexts(rng, args.batch, cfg["ctx_len"], cfg["n_copy"], corpora + [None], cfg["probs"],
                                     1.1)
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    ctx_d, cl_d = to_dev(ctx), to_dev(cl)
    res = fc.fc_retrieve(sources, ctx_d, cl_d, p)
    ms = _gpu_ms(lambda: fc.fc_retrieve(sources, ctx_d, cl_d, p, out=res), reps=args.steps, warm=args.warmup)
    out = {"metric": "retrievals/s", "value": 2 * args.batch / (ms * 1e-3), "unit": "query-sources/s",
           "n_gpus": ws, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
           "config": {"workload": f"two-source retrieval (5M + 100M tokens), {args.batch} contexts of 128, "
                                  f"n 16->2, top-64 x 10"},
           "us_per_query_source": ms * 1e3 / (2 * args.batch)}
    # the same search without the suffix keys (probes read the suffix array,
    # then the corpus), on the same queries
    plain = [s.without_keys() for s in sources]
    rp = fc.fc_retrieve(plain, ctx_d, cl_d, p)
    assert all(torch.equal(res[k], rp[k]) for k in res) and fc.fc_get_error() == "FC_OK"
    ms_p = _gpu_ms(lambda: fc.fc_retrieve(plain, ctx_d, cl_d, p, out=rp), reps=args.steps, warm=args.warmup)
    out["without_keys"] = {"ms_per_step": ms_p, "us_per_query_source": ms_p * 1e3 / (2 * args.batch),
                           "query_sources_per_s": 2 * args.batch / (ms_p * 1e-3)}
    if args.rev:
        # the reversed-corpus variant on the same queries: n* by one narrowing
        # search in the reversed suffix arrays, then the forward search for n*
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        revs = [fc.fc_datastore_build_reversed(s.tokens, synth.VOCAB) for s in sources]
        torch.cuda.synchronize()
        build_s = time.perf_counter() - t0
        rr = fc.fc_retrieve_rev(sources, revs, ctx_d, cl_d, p)
        same = all(torch.equal(res[k], rr[k]) for k in res)
        assert same and fc.fc_get_error() == "FC_OK"
        ms_r = _gpu_ms(lambda: fc.fc_retrieve_rev(sources, revs, ctx_d, cl_d, p, out=rr), reps=args.steps,
                       warm=args.warmup)
        out["reversed"] = {"ms_per_step": ms_r, "query_sources_per_s": 2 * args.batch / (ms_r * 1e-3),
                           "us_per_query_source": ms_r * 1e3 / (2 * args.batch), "same_outputs": same,
                           "reversed_build_seconds": build_s}
    if args.all_occ:
        # the all-occurrence trie: every distinct continuation of the first 4096
        # occurrences per source, and the weighted trie over all of them
        pa = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
        ra = fc.fc_retrieve_all(sources, ctx_d, cl_d, pa)
        root = to_dev(ctx[np.arange(args.batch), cl - 1])
        kvl = to_dev(np.full(args.batch, 4096, np.int32))
        ws_t = torch.empty(int(fc.LIB.fc_build_tree_all_workspace(2, 4096, cfg["draft_len"], args.batch)),
                           dtype=torch.uint8, device=dev)
        tr = fc.fc_build_tree_all(ra, [1, 1], root, kvl, cfg["node_budget"], cfg["n_pad"], workspace=ws_t)
        assert fc.fc_get_error() == "FC_OK"
        ms_a = _gpu_ms(lambda: fc.fc_retrieve_all(sources, ctx_d, cl_d, pa, out=ra), reps=args.steps,
                       warm=args.warmup)
        ms_t = _gpu_ms(lambda: fc.fc_build_tree_all(ra, [1, 1], root, kvl, cfg["node_budget"], cfg["n_pad"],
                                                    workspace=ws_t, out=tr), reps=args.steps, warm=args.warmup)
        nd = ra["n_drafts"].cpu().numpy()
        out["all_occurrence"] = {"retrieve_all_ms": ms_a, "build_tree_all_ms": ms_t,
                                 "mean_distinct_per_query_source": float(nd.mean()),
                                 "max_distinct_per_query_source": int(nd.max()),
                                 "mean_tree_nodes": float(tr["n_nodes"].float().mean().item()),
                                 "workspace_bytes": int(ws_t.numel())}
    return out


def run_small(args, rank, ws, local):
    """Batch sweep of the step's small kernels on the step loop's own inputs
    (two-source retrieval on the 5M + 100M stores, the step mix of contexts):
    tree build, synthetic predictions, acceptance, KV append and a replay-cache
    lookup that hits.  At the step loop's batch these are latency chains; the
    sweep shows where each one reaches its bandwidth.  Times are means of
    back-to-back calls (`_gpu_ms`); bytes are the algorithmic bytes of each
    call, and the HBM fraction is of the measured copy peak."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    cfg, c5 = synth.WORKLOADS[2], synth.WORKLOADS[5]
    rng = synth.rng_for(2)
    corpora = [synth.build_corpus(rng, spec, device="cuda")[0] for spec in cfg["corpus"]]
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32) if a.dtype == np.uint32
                                        else np.ascontiguousarray(a)).to(dev)
    sources = [fc.fc_datastore_build(to_dev(T), synth.VOCAB) for T in corpora]
    p = fc.params(c5["n_max"], c5["n_min"], c5["top_k"], c5["draft_len"], 4096)
    S, k, d, n_pad, Hkv, D = 2, c5["top_k"], c5["draft_len"], c5["n_pad"], c5["Hkv"], c5["D"]
    path_cap, cap = d + 2, 2 * (d + 2)
    peak = load_peaks()["hbm"]
    batches = [int(x) for x in args.batches.split(",")]
    rows = []
    for B in batches:
        ctx, cl, _ = synth.make_contexts(rng, B, c5["ctx_len"], c5["n_copy"], corpora + [None], c5["probs"], 1.1,
                                         ctx_stride=c5["ctx_len"] + 2 * path_cap)
        ctx_d, cl_d = to_dev(ctx), to_dev(cl)
        res = fc.fc_retrieve(sources, ctx_d, cl_d, p)
        root = to_dev(ctx[np.arange(B), cl - 1])
        kvl = torch.zeros(B, dtype=torch.int32, device=dev)
        tree = fc.fc_build_tree(res, [1, 1], root, kvl, c5["node_budget"], n_pad)
        plen_h, rtok_h = synth.argmax_draws(rng, B, n_pad)
        plen, rtok = to_dev(plen_h), to_dev(rtok_h)
        am = fc.fc_synth_argmax(tree["tok"], tree["parent"], tree["n_nodes"], plen, rtok, synth.VOCAB)
        acc = fc.fc_accept(tree["tok"], tree["parent"], tree["n_nodes"], am, path_cap)
        kt = torch.randn((B, Hkv, n_pad, D), device=dev).to(torch.bfloat16)
        kc = torch.zeros((B, Hkv, cap, D), dtype=torch.bfloat16, device=dev)
        vc = torch.zeros_like(kc)
        kv_out = torch.empty_like(kvl)
        ctx_w = ctx_d.clone()
        cl_out = torch.empty_like(cl_d)
        root_out = torch.empty_like(root)
        rc = fc.RetrievalCache(1 << max(10, int(2 * B - 1).bit_length()), S, p)
        skip = torch.zeros(B, dtype=torch.int32, device=dev)
        fc.fc_rcache_insert(rc, ctx_d, cl_d, skip, res)
        got = fc.retrieve_outputs(S, B, p, dev)
        assert fc.fc_get_error() == "FC_OK"
        calls = {
            "build_tree": lambda: fc.fc_build_tree(res, [1, 1], root, kvl, c5["node_budget"], n_pad, out=tree),
            "synth_argmax": lambda: fc.fc_synth_argmax(tree["tok"], tree["parent"], tree["n_nodes"], plen, rtok,
                                                       synth.VOCAB, out=am),
            "accept": lambda: fc.fc_accept(tree["tok"], tree["parent"], tree["n_nodes"], am, path_cap, out=acc),
            "kv_append": lambda: fc.fc_kv_append(acc, tree["tok"], kt, kt, kc, vc, kvl, kv_out, ctx_w, cl_d, cl_out,
                                                 root_out),
            "rcache_lookup_hit": lambda: fc.fc_rcache_lookup(rc, ctx_d, cl_d, None, skip, got),
        }
        a_len = acc["acc_len"].double()
        nn = tree["n_nodes"].double()
        alg = {  # algorithmic bytes of one call over the batch
            "build_tree": B * (S * k * (d + 2) * 4 + S * 4 + 8) + B * (n_pad * (16 + n_pad // 8) + 4),
            "synth_argmax": B * (n_pad * 16 + 8),
            "accept": float((nn * 12).sum().item()) + B * (4 + 4 * (path_cap + 2)),
            "kv_append": float(((a_len + 1) * Hkv * D * 2 * 2 * 2).sum().item()) + B * 4 * (4 + path_cap + 2),
            "rcache_lookup_hit": B * (2 * S * (k * d + 2 * k + 2) * 4 + 4 * c5["n_max"] + 8),
        }
        rec = {"batch": B, "mean_tree_nodes": float(nn.mean().item()),
               "mean_acc_len": float(a_len.mean().item())}
        for nm, fn in calls.items():
            ms = _gpu_ms(fn, reps=args.steps, warm=args.warmup)
            rec[nm] = {"us": ms * 1e3, "us_per_sequence": ms * 1e3 / B, "alg_bytes": alg[nm],
                       "gbs": alg[nm] / (ms * 1e-3) / 1e9, "hbm_frac": alg[nm] / (ms * 1e-3) / 1e9 / peak}
        assert fc.fc_get_error() == "FC_OK" and int(skip.sum().item()) == B
        rows.append(rec)
        del kt, kc, vc
        torch.cuda.empty_cache()
    return {"metric": "small-kernel batch sweep", "value": None, "unit": "us", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "config": {"workload": "the step's small kernels on two-source retrieval "
                                                          "(5M + 100M), trees <= 128 nodes, GQA 8 KV heads"},
            "hbm_peak_gbs": peak, "sweep": rows}


def run_algorithm1(args, rank, ws, local):
    """The step loop of the default workload with Algorithm 1 in place of the
    replay cache: per sequence a CACHE (l = 50, 20-token output pieces,
    8192 words), a missing table per sub-batch (one for the batch with
    --split 1).  --fill untimed steps fill the CACHE first, so the timed
    steps search active stores.  With --split N > 1 the native step executor
    runs N sub-batches on streams of their own, as in the default mode; the
    stage events then time each sub-batch's retrieval stage (CACHE search,
    datastore fallback, missing-table insert), tree, attention and tail
    (predictions, acceptance, append, CACHE update).  With --split 1 they
    also time the CACHE search and the CACHE update alone."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    K, W, F = args.steps, args.warmup, (100 if args.fill is None else args.fill)
    total = F + W + K + 1
    inp = make_inputs(args.scale, args.batch, rank, total)
    cfg, B = inp["cfg"], inp["B"]
    H, Hkv, D, n_pad, d = cfg["H"], cfg["Hkv"], cfg["D"], cfg["n_pad"], cfg["draft_len"]
    kv0 = inp["kv0"]
    cap = kv0 + total * (d + 1) + 8
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
    sources = [fc.fc_datastore_build(to_dev(T), synth.VOCAB) for T in inp["corpora"]]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], d, 4096)
    kc = torch.empty((B, Hkv, cap, D), dtype=torch.bfloat16, device=dev)
    vc = torch.empty_like(kc)
    g = torch.Generator(device=dev)
    g.manual_seed(inp["seed"])
    kc[:, :, :kv0].normal_(generator=g)
    vc[:, :, :kv0].normal_(generator=g)
    seq = dict(capacity=8192, min_size=50, chunk=20, ctx_keep=cfg["n_max"], missing_capacity=1 << 16, weight=1)
    P = min(16, K + W)
    q_pool = torch.randn((P, B, n_pad, H, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    kt_pool = torch.randn((P, B, Hkv, n_pad, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    vt_pool = torch.randn((P, B, Hkv, n_pad, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
    plen_d, rtok_d = to_dev(inp["plen"]), to_dev(inp["rtok"])
    zeros = torch.zeros(B, dtype=torch.int32, device=dev)
    nsub = max(1, min(args.split, B))

    def make():
        largs = (sources, inp["ctx"], inp["cl"], p, cfg["node_budget"], n_pad, [1, 1], H, Hkv, D, cap, kv0,
                 synth.VOCAB)
        lkw = dict(device=dev, k_cache=kc, v_cache=vc, seq_cache=seq)
        return PipelinedStepLoop(nsub, *largs, **lkw) if nsub > 1 else StepLoop(*largs, **lkw)

    loops_of = lambda lp: lp.loops if nsub > 1 else [lp]

    # untimed pass over the whole trajectory: what each step's retrieval did
    loop = make()
    codes, accs = [], []
    for s in range(F + W + K):
        j = s % P
        loop.step(q_pool[j], kt_pool[j], vt_pool[j], zeros, plen_d[s], rtok_d[s], attention=False)
        if nsub > 1:
            loop.join()
        codes.append(loop.skip.clone())
        accs.append(loop.acc["acc_len"].clone())
    codes = torch.stack(codes).cpu().numpy()[F + W:]
    accs = torch.stack(accs).cpu().numpy()[F + W:]
    kc[:, :, kv0:].zero_()
    vc[:, :, kv0:].zero_()

    loop = make()
    mk = lambda: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    names = ("retrieve", "tree", "attn", "tail") + (() if nsub > 1 else ("cache_search", "cache_update"))
    ev = [[{nm: mk() for nm in names} for _ in range(nsub)] for _ in range(K)]
    for per_step in ev:  # torch creates an event at its first record: do that before the timed region
        for e in per_step:
            for a, b in e.values():
                a.record()
                b.record()

    def do_step(s, i=None):
        j = s % P
        evs = None if i is None else (ev[i] if nsub > 1 else ev[i][0])
        loop.step(q_pool[j], kt_pool[j], vt_pool[j], zeros, plen_d[s], rtok_d[s], events=evs)

    for s in range(F + W):
        do_step(s)
    if nsub > 1:
        loop.join()
    assert step_status(fc, loop) == "FC_OK"
    barrier(ws)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.wait_first()
    stream = torch.cuda.current_stream()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with no_gc():
        start.record(stream)
        for i in range(K):
            do_step(F + W + i, i)
        if nsub > 1:
            loop.join()
        end.record(stream)
        torch.cuda.synchronize()
    clock_rec = clocks.stop()
    barrier(ws)
    status = step_status(fc, loop)
    assert status == "FC_OK", status
    t_max = max_over_ranks(start.elapsed_time(end), ws)
    # each stage's mean time per sub-batch launch (sub-batches overlap: they do not add up)
    stage = {nm: statistics.mean(a.elapsed_time(b) for per_step in ev for e in per_step for a, b in [e[nm]])
             for nm in names}
    subs = loops_of(loop)
    meta = torch.cat([lp.seq_cache.meta for lp in subs]).cpu().numpy()
    m_stored = sum(int(lp.missing.table[0].item()) for lp in subs)
    # the same contexts, retrieved from the datastore alone, and the CACHE
    # search alone on the final stores of one sub-batch (both repeatable:
    # they write only their outputs)
    res_all = fc.fc_retrieve(sources, loop.ctx, loop.ctx_len_now, p)
    ds_ms = _gpu_ms(lambda: fc.fc_retrieve(sources, loop.ctx, loop.ctx_len_now, p, out=res_all), reps=20, warm=3)
    lp0 = subs[0]
    st = torch.empty(lp0.B, dtype=torch.int32, device=dev)
    res_c = fc.retrieve_outputs(len(sources) + 1, lp0.B, p, dev)
    cs_ms = _gpu_ms(lambda: fc.fc_cache_search(lp0.seq_cache, lp0.missing, lp0.ctx, lp0.ctx_len_now, p,
                                               len(sources), res_c, st), reps=20, warm=3)
    n_q = codes.size
    return {"metric": METRIC, "value": weak_value(K, ws, t_max), "unit": UNIT, "n_gpus": ws, "steps": K,
            "warmup": W, "ms_per_step": t_max / K, "higher_is_better": True, "scaling": "weak",
            "dtype": "bf16 attention (fp32 accumulate) + u32 retrieval", "data": "synthetic",
            "config": {"workload": WORKLOAD.replace("50% replay-cache hits", "Algorithm 1: per-sequence CACHE "
                                                    "(l=50, 20-token pieces, 8192 words) + missing table"),
                       "fill_steps": F, "batch_per_gpu": B, "kv_len0": kv0,
                       "l2": "inputs larger than L2 (KV cache 2.2 GB per GPU)",
                       "streams": (f"{nsub} sub-batches of {B // nsub}-{-(-B // nsub)} sequences issued by the "
                                   "native step executor, each with its own missing table" if nsub > 1
                                   else "one stream, one missing table")},
            # per sub-batch step: CACHE search, retrieval, missing insert, tree, attention,
            # predictions, accept, append, CACHE update
            "gpu_launches": 9 * K * nsub,
            "sub_batches": nsub,
            "stages_ms_per_step": stage,
            "cache": {"served_frac": float((codes == 1).sum() / n_q), "skipped_frac": float((codes == 2).sum() / n_q),
                      "datastore_frac": float((codes == 0).sum() / n_q),
                      "acc_len_served": float(accs[codes == 1].mean()) if (codes == 1).any() else None,
                      "acc_len_datastore": float(accs[codes == 0].mean()) if (codes == 0).any() else None,
                      "mean_sequences": float(meta[:, 1].mean()), "mean_words": float(meta[:, 0].mean()),
                      "missing_keys": m_stored, "cache_search_alone_us": cs_ms * 1e3,
                      "cache_search_alone_batch": lp0.B,
                      "datastore_retrieval_all_queries_us": ds_ms * 1e3},
            "clocks": clock_rec}


def run_cache(args, rank, ws, local):
    """fc_cache_search alone on full stores: --batch sequences whose CACHE
    (8192 words, l = 50) was filled through fc_cache_update along a synthetic
    generation of --fill steps (each step the context suffix plus the accepted
    draft tokens, and every 20-token output piece), as in the step loop.
    Three contexts in four then end with a fresh token, as a context whose
    last token is the model's bonus token usually does; the others end inside
    the generation the store was built from."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    B, F, d, n0 = args.batch, (450 if args.fill is None else args.fill), 10, 128
    rng = synth.rng_for(5, 700 + rank)
    stride = n0 + F * (d + 1) + 1
    G = synth.zipf_tokens(rng, B * stride, 1.1).reshape(B, stride)
    acc = np.stack([np.minimum(synth.argmax_draws(rng, B, 1)[0], d) for _ in range(F)])
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
    ctx_d = to_dev(G)
    cache = fc.SequenceCache(B, capacity=8192, min_size=50, chunk=20, ctx_keep=16, device=dev)
    cur = np.full(B, n0, np.int32)
    cache.init(to_dev(cur))
    for s in range(F):
        new = cur + acc[s] + 1
        fc.fc_cache_update(cache, ctx_d, to_dev(cur), to_dev(new), to_dev(acc[s].astype(np.int32)))
        cur = new
    fresh = rng.random(B) < 0.75
    Gq = G.copy()
    Gq[np.arange(B)[fresh], cur[fresh] - 1] = synth.zipf_tokens(rng, int(fresh.sum()), 1.1)
    q_d, ql_d = to_dev(Gq), to_dev(cur)
    missing = fc.MissingTable(1 << 16, 2, device=dev)
    p = fc.params(16, 2, 64, d, 4096)
    res = fc.retrieve_outputs(3, B, p, dev)
    state = torch.empty(B, dtype=torch.int32, device=dev)
    call = lambda: fc.fc_cache_search(cache, missing, q_d, ql_d, p, 2, res, state)
    call()
    assert fc.fc_get_error() == "FC_OK"
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.wait_first()
    ms = _gpu_ms(call, reps=args.steps, warm=args.warmup)
    clock_rec = clocks.stop()
    meta = cache.meta.cpu().numpy()
    words = float(meta[:, 0].sum())
    peaks = load_peaks()
    achieved = 4 * words / (ms * 1e-3) / 1e9
    return {"metric": "CACHE searches/s", "value": B / (ms * 1e-3), "unit": "query-searches/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "config": {"workload": f"fc_cache_search on {B} full stores (8192 words, l=50) filled along {F} "
                                   "generation steps; n 16->2, top-64 x 10"},
            "us_per_call": ms * 1e3, "served_frac": float((state.cpu().numpy() == 1).mean()),
            "mean_words": words / B, "mean_sequences": float(meta[:, 1].mean()),
            "roofline": {"bound": "latency", "achieved": achieved, "peak": peaks["hbm"], "unit": "GB/s",
                         "frac": achieved / peaks["hbm"], "traffic": None, "kernel": "k_cache_search",
                         "note": "bytes = the store words read once; the kernel is bound by its phase latency"},
            "clocks": clock_rec}


def run_decoder(args, rank, ws, local):
    """The step loop with the target model's forward as the verifier: a
    randomly initialised decoder of DeepSeek-Coder 1.3B's shape (24 layers,
    hidden 2048, 16 heads of 128, MLP 5504, vocab 32256) verifies 64-node
    draft trees for --batch sequences over a 2048-token cache, greedy
    acceptance from its logits; retrieval from the default two-source store
    (replay cache off).  With random weights the acceptance carries no
    meaning; the step's cost does."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    from paper_2502_17139_gb300.decoder import DEEPSEEK_CODER_1_3B, TreeDecoder
    from paper_2502_17139_gb300.step import StepLoop

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    s = DEEPSEEK_CODER_1_3B
    K, W = args.steps, args.warmup
    total = K + W + 1
    inp = make_inputs(args.scale, args.batch, rank, total)
    cfg, B = inp["cfg"], inp["B"]
    n_pad, d, kv0 = 64, cfg["draft_len"], 2048
    cap = kv0 + total * (d + 1) + 8
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
    sources = [fc.fc_datastore_build(to_dev(T), synth.VOCAB) for T in inp["corpora"]]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], d, 4096)
    Wt = synth.decoder_weights(s.hidden, s.layers, s.H, s.Hkv, s.D, s.inter, s.vocab, inp["seed"], device=dev)
    caches = []
    for l in range(s.layers):
        kc = torch.zeros((B, s.Hkv, cap, s.D), dtype=torch.bfloat16, device=dev)
        vc = torch.zeros_like(kc)
        kc[:, :, :kv0] = synth.randn_bf16((B, s.Hkv, kv0, s.D), inp["seed"] + 10 + l, dev)
        vc[:, :, :kv0] = synth.randn_bf16((B, s.Hkv, kv0, s.D), inp["seed"] + 500 + l, dev)
        caches.append((kc, vc))
    td = TreeDecoder(s, Wt, B, n_pad, cap, device=dev, caches=caches)
    loop = StepLoop(sources, inp["ctx"], inp["cl"], p, n_pad, n_pad, src_weights(args), s.H, s.Hkv, s.D, cap, kv0,
                    synth.VOCAB, device=dev, k_cache=caches[0][0], v_cache=caches[0][1], decoder=td,
                    cache_capacity=0)
    zeros = torch.zeros(B, dtype=torch.int32, device=dev)
    names = ("retrieve", "tree", "attn", "tail")
    ev = {nm: [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
          for nm in names}
    for _ in range(W):
        loop.step(None, None, None, zeros, zeros, None)
    assert fc.fc_get_error() == "FC_OK"
    barrier(ws)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.wait_first()
    stream = torch.cuda.current_stream()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    accs = []
    start.record(stream)
    for i in range(K):
        loop.step(None, None, None, zeros, zeros, None, events={nm: ev[nm][i] for nm in names})
        accs.append(loop.acc["acc_len"].clone())
    end.record(stream)
    torch.cuda.synchronize()
    clock_rec = clocks.stop()
    barrier(ws)
    assert fc.fc_get_error() == "FC_OK"
    t_max = max_over_ranks(start.elapsed_time(end), ws)
    stage = {nm: statistics.mean(a.elapsed_time(b) for a, b in ev[nm]) for nm in names}
    acc = torch.stack(accs).cpu().numpy()
    # the forward's GEMM work (every row of the padded tree) and its attention
    # share, from one more untimed forward with per-layer events
    T = B * n_pad
    per_layer = s.hidden * (s.H * s.D + 2 * s.Hkv * s.D) + s.H * s.D * s.hidden + s.hidden * 3 * s.inter
    gemm_flops = 2.0 * T * (s.layers * per_layer + s.hidden * s.vocab)
    t = loop.tree
    aev = {"attn": []}
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record()
    td.forward(t["tok"], t["n_nodes"], t["mask"], t["pos"], loop.kv_len_now, events=aev)
    f1.record()
    torch.cuda.synchronize()
    fwd_ms = f0.elapsed_time(f1)
    attn_ms = sum(a.elapsed_time(b) for a, b in aev["attn"])
    # the same forward without per-layer events: host enqueue time, device time
    # eager, and device time replayed from a CUDA graph (no launch gaps)
    torch.cuda.synchronize()
    h0 = time.perf_counter()
    f0.record()
    td.forward(t["tok"], t["n_nodes"], t["mask"], t["pos"], loop.kv_len_now)
    f1.record()
    host_ms = 1e3 * (time.perf_counter() - h0)
    torch.cuda.synchronize()
    eager_ms = f0.elapsed_time(f1)
    g_fwd = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_fwd):
        td.forward(t["tok"], t["n_nodes"], t["mask"], t["pos"], loop.kv_len_now)
    g_fwd.replay()
    torch.cuda.synchronize()
    f0.record()
    for _ in range(3):
        g_fwd.replay()
    f1.record()
    torch.cuda.synchronize()
    graph_ms = f0.elapsed_time(f1) / 3
    peaks = load_peaks()
    gemm_tflops = gemm_flops / ((fwd_ms - attn_ms) * 1e-3) / 1e12
    return {"metric": METRIC, "value": weak_value(K, ws, t_max), "unit": UNIT, "n_gpus": ws, "steps": K, "warmup": W,
            "ms_per_step": t_max / K, "higher_is_better": True, "scaling": "weak",
            "dtype": "bf16 (fp32 accumulate) + u32 retrieval", "data": "synthetic (random-init weights)",
            "config": {"workload": f"step loop verified by a random-init DeepSeek-Coder-1.3B-shaped decoder "
                                   f"(24 x hidden 2048, 16 heads x 128, MLP 5504, vocab 32256), {B} sequences, "
                                   f"64-node trees, cache {kv0}, two-source store 100M + 5M",
                       "batch_per_gpu": B, "n_pad": n_pad, "kv_len0": kv0},
            "stages_ms_per_step": stage,
            "tokens_per_s": float((acc + 1).sum() / (t_max * 1e-3) * ws),
            "mean_accepted": float(acc.mean()),
            "forward": {"ms": fwd_ms, "eager_ms_no_events": eager_ms, "host_enqueue_ms": host_ms,
                        "graph_replay_ms": graph_ms, "attention_ms": attn_ms, "gemm_and_rest_ms": fwd_ms - attn_ms,
                        "gemm_tflops": gemm_tflops, "gemm_frac_of_sustained_bf16": gemm_tflops / peaks["tc_sustained"]},
            "clocks": clock_rec}


def run_gemm(args, rank, ws, local):
    """fc_gemm_bf16 (the library's tcgen05 GEMM) on the decoder's shapes over
    2048 tree rows (32 sequences x 64 nodes, DeepSeek-Coder 1.3B's width),
    timed beside torch.matmul (cuBLAS) on the same operands in the same run.
    Each shape runs back to back on operands that stay resident; the weights
    of the larger shapes exceed L2."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    peaks = load_peaks()
    M = 2048
    shapes = [("q", 2048, 2048), ("kv", 2048, 4096), ("o", 2048, 2048), ("gate_up", 2048, 11008),
              ("down", 5504, 2048), ("lm_head", 2048, 32256)]
    per_layer = {"q", "kv", "o", "gate_up", "down"}
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    rows, ours_t, lib_t, flops_t, lt_t, lt_ok = [], 0.0, 0.0, 0.0, 0.0, True
    for name, K, N in shapes:
        a = torch.randn((M, K), generator=g, device=dev).to(torch.bfloat16)
        b = (torch.randn((K, N), generator=g, device=dev) * K ** -0.5).to(torch.bfloat16)
        c = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
        c_ref = torch.empty_like(c)
        reps, warm = max(args.steps, 5), max(args.warmup, 3)
        t_ours = _cuda_ms(lambda: fc.fc_gemm_bf16(a, b, out=c), reps=reps, warm=warm)
        t_lib = _cuda_ms(lambda: torch.matmul(a, b, out=c_ref), reps=reps, warm=warm)
        t_lt = None
        try:  # the same product through cuBLASLt (torch's other BLAS back end)
            prev = torch.backends.cuda.preferred_blas_library()
            torch.backends.cuda.preferred_blas_library("cublaslt")
            t_lt = _cuda_ms(lambda: torch.matmul(a, b, out=c_ref), reps=reps, warm=warm)
            torch.backends.cuda.preferred_blas_library(prev)
        except (AttributeError, RuntimeError, TypeError):
            pass
        torch.cuda.synchronize()
        assert fc.fc_get_error() == "FC_OK"
        diff = float((c.float() - c_ref.float()).abs().max())
        fl = 2.0 * M * N * K
        w = 24 if name in per_layer else 1  # occurrences in one 24-layer forward
        ours_t += w * t_ours
        lib_t += w * t_lib
        if t_lt is None:
            lt_ok = False
        else:
            lt_t += w * t_lt
        flops_t += w * fl
        rows.append({"gemm": name, "M": M, "N": N, "K": K, "ours_us": 1e3 * t_ours, "cublas_us": 1e3 * t_lib,
                     "cublaslt_us": None if t_lt is None else 1e3 * t_lt,
                     "ours_tflops": fl / t_ours / 1e9, "cublas_tflops": fl / t_lib / 1e9,
                     "cublaslt_tflops": None if t_lt is None else fl / t_lt / 1e9,
                     "ours_frac_of_burst": fl / t_ours / 1e9 / peaks["tc_burst"], "max_abs_diff_vs_cublas": diff})
    # the decoder's two fused epilogues against the unfused pair of calls
    B, n_pad, Hkv, inter = 32, 64, 16, 5504
    h = torch.randn((M, 2048), generator=g, device=dev).to(torch.bfloat16)
    wkv = (torch.randn((2048, 2 * Hkv * 128), generator=g, device=dev) * 2048 ** -0.5).to(torch.bfloat16)
    wgu = (torch.randn((2048, 2 * inter), generator=g, device=dev) * 2048 ** -0.5).to(torch.bfloat16)
    wgu_il = fc.fc_interleave_gate_up(wgu)
    pos = torch.arange(n_pad, device=dev, dtype=torch.int32).repeat(B, 1) + 2048
    k_rot = torch.empty((B, Hkv, n_pad, 128), dtype=torch.bfloat16, device=dev)
    v_h = torch.empty_like(k_rot)
    kv = torch.empty((M, 2 * Hkv * 128), dtype=torch.bfloat16, device=dev)
    gu = torch.empty((M, 2 * inter), dtype=torch.bfloat16, device=dev)
    act = torch.empty((M, inter), dtype=torch.bfloat16, device=dev)

    def unfused_kv():
        fc.fc_gemm_bf16(h, wkv, out=kv)
        fc.fc_rope_heads(kv, 0, 2 * Hkv * 128, k_rot, B, n_pad, Hkv, 128, pos, 10000.0)
        fc.fc_rope_heads(kv, Hkv * 128, 2 * Hkv * 128, v_h, B, n_pad, Hkv, 128, pos, 0.0)

    def unfused_gu():
        fc.fc_gemm_bf16(h, wgu, out=gu)
        fc.fc_silu_mul(gu, act)

    fused = {"kv_heads_us": 1e3 * _cuda_ms(lambda: fc.fc_gemm_kv_heads(h, wkv, B, n_pad, Hkv, pos, 10000.0, k_rot, v_h)),
             "kv_gemm_then_rope_heads_us": 1e3 * _cuda_ms(unfused_kv),
             "silu_mul_us": 1e3 * _cuda_ms(lambda: fc.fc_gemm_silu_mul(h, wgu_il, act)),
             "gu_gemm_then_silu_mul_us": 1e3 * _cuda_ms(unfused_gu)}
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    ach = flops_t / ours_t / 1e9
    return {"metric": "decoder GEMM TFLOP/s", "value": ach, "unit": "TFLOP/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "dtype": "bf16 (fp32 accumulate)",
            "data": "synthetic", "config": {"workload": "decoder GEMMs of a 24-layer DeepSeek-Coder-1.3B-shaped "
                                                        "forward over 2048 tree rows, weighted by occurrences"},
            "cublas_tflops": flops_t / lib_t / 1e9, "ratio_to_cublas": lib_t / ours_t,
            "cublaslt_tflops": flops_t / lt_t / 1e9 if lt_ok else None,
            "ratio_to_cublaslt": lt_t / ours_t if lt_ok else None, "fused_epilogues": fused,
            "roofline": {"bound": "tensor", "achieved": ach, "peak": peaks["tc_burst"], "unit": "TFLOP/s",
                         "frac": ach / peaks["tc_burst"], "peak_source": peaks["source"] + " burst bf16"},
            "shapes": rows}


def run_build(args, rank, ws, local):
    """fc_datastore_build alone: a Zipf(1.1) corpus of --tokens tokens over
    vocab 32256 (the general store's law), built --steps times after
    --warmup builds; CUDA events around each synchronous build."""
    import torch

    import paper_2502_17139_gb300.fastcoder as fc
    import paper_2502_17139_gb300.synth as synth
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    rng = synth.rng_for(2, 77)
    T = synth.zipf_tokens(rng, args.tokens, 1.1, synth.VOCAB, device=dev)
    tok = torch.from_numpy(T.view(np.int32)).to(dev)
    n = tok.numel()
    ws_t = torch.empty(fc.fc_datastore_build_workspace(n, synth.VOCAB), dtype=torch.uint8, device=dev)
    times = []
    for i in range(args.warmup + args.steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        ds = fc.fc_datastore_build(tok, synth.VOCAB, workspace=ws_t)
        e1.record()
        torch.cuda.synchronize()
        if i >= args.warmup:
            times.append(e0.elapsed_time(e1))
        del ds
    assert fc.fc_get_error() == "FC_OK"
    ms = statistics.mean(times)
    return {"metric": "datastore build tokens/s", "value": n / (ms * 1e-3), "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_build": ms, "higher_is_better": True,
            "dtype": "u32", "data": "synthetic",
            "config": {"workload": f"suffix array + bucket table + LCP of {n} Zipf(1.1) tokens, vocab 32256"}}


def main(argv=None):
    args = parse_args(argv)
    rank, ws, local = dist_setup(args.gpus)
    if args.impl == "reference":
        out = run_reference(args, rank, ws)
    elif args.mode == "attn":
        out = run_attn(args, rank, ws, local)
    elif args.mode == "argmax":
        out = run_argmax(args, rank, ws, local)
    elif args.mode == "configs":
        out = run_configs(args, rank, ws, local)
    elif args.mode == "retrieve":
        out = run_retrieve(args, rank, ws, local)
    elif args.mode == "algorithm1":
        out = run_algorithm1(args, rank, ws, local)
    elif args.mode == "cache":
        out = run_cache(args, rank, ws, local)
    elif args.mode == "decoder":
        out = run_decoder(args, rank, ws, local)
    elif args.mode == "gemm":
        out = run_gemm(args, rank, ws, local)
    elif args.mode == "build":
        out = run_build(args, rank, ws, local)
    elif args.mode == "small":
        out = run_small(args, rank, ws, local)
    else:
        out = run_ours(args, rank, ws, local)
    if rank == 0 and out is not None:
        print(json.dumps(out))
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
