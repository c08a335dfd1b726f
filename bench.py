"""Benchmark of one verify step of the VideoSpeculateRAG verifier hot path.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config 72b] [--impl reference]

A step is one pass of the whole hot path over one query batch: shared-prefix
attention, LM-head log-probabilities, CLIP alignment and candidate selection
(the four libfvrag calls).  Inputs are seeded synthetic tensors resident in HBM
before the timed region; L2 is flushed (a 256 MiB write) between timed steps,
outside the per-step CUDA events.

Metric: verified candidate tokens/s = (queries x candidates x tokens) / step time.
Also reported: verify-step microseconds per query, per-kernel times, the roofline
fraction of the dominant kernel (the LM head: tensor-bound at the default 72B-class
shape, HBM-bound at the 7B shape), the
end-to-end number through the public API with host buffers (host->device copies
of the step's inputs and the device->host read of the result inside the timed
region), and the fp64 oracle's time on this host's cores.

Multi-GPU (torchrun): every rank runs an independent replica of the workload
(independent queries, no collective on the data path: weak scaling); the time is
the max over ranks.  --impl reference times the fp64 oracle on the host cores
(rank 0 only).
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2601_01513_gb300 import configs, synth  # noqa: E402

METRIC = "verified candidate tokens/s"
UNIT = "tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# DRAM traffic of one LM-head launch per workload, from an ncu capture of the kernel
# source with this SHA-256 prefix (reported as null once the kernel source changes).
LM_TRAFFIC = {
    "7b": {"sha256_prefix": "fc5d9ea0e4553c80", "bytes_per_launch": 1093830912},
    "72b": {"sha256_prefix": "fc5d9ea0e4553c80", "bytes_per_launch": 2500334080},
}


def peaks():
    p = dict(FALLBACK_PEAKS)
    src = "fallback"
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            m = json.load(f)
        for k in FALLBACK_PEAKS:
            if k in m:
                p[k] = float(m[k])
        src = "measured"
    return p, src


def source_sha(name):
    with open(os.path.join(ROOT, "paper_2601_01513_gb300", "csrc", name), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def algorithmic(cfg):
    """Bytes and flops each kernel must move / perform at minimum (per launch)."""
    Qn, K, L, hq, hkv, D = cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.hq, cfg.hkv, cfg.head_dim
    M, H, V, G = cfg.rows, cfg.hidden, cfg.vocab, cfg.gathers
    plen = synth.prefix_lengths(cfg)
    sumP = int(plen.sum())
    rows = Qn * K * L * hq
    attn_bytes = 2 * sumP * hkv * D * 2 + 2 * rows * D * 2 + 2 * Qn * K * L * hkv * D * 2 + rows * 4
    vis = sum(int(p) * K * L + K * L * (L + 1) // 2 for p in plen) * hq
    attn_flops = 4.0 * D * vis
    lm_bytes = V * H * 2 + M * H * 2 + M * G * 4 + M * G * 4 + M * 4
    lm_flops = 2.0 * M * H * V
    clip_bytes = Qn * (K + cfg.num_frames) * cfg.clip_dim * 2 + Qn * K * 9
    sel_bytes = M * G * 4 + Qn * K * 9 + Qn * 4
    return {"attn": (attn_bytes, attn_flops), "lm": (lm_bytes, lm_flops), "clip": (clip_bytes, 0.0),
            "select": (sel_bytes, 0.0)}


class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs (every 25 ms, so
    that a short run of a few dozen steps still gets several samples)."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
                 "-lms", "25"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def wait_first(self, timeout=5.0):
        """Blocks until nvidia-smi has produced its first sample (it starts slowly); the
        samples then cover the whole timed region that follows."""
        t0 = time.time()
        while self.proc is not None and not self.lines and time.time() - t0 < timeout:
            time.sleep(0.05)
        self.lines.clear()

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def replica_seed(cfg, rank):
    """Seed of rank `rank`'s independent replica (each rank verifies its own queries)."""
    return cfg.seed + 7919 * rank


def max_over_ranks(values, device):
    """Element-wise max of per-rank timings over all ranks (the job time is the slowest rank)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(values, dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_throughput(tokens_per_step, steps, world, max_ms):
    """Whole-job tokens/s: every rank's tokens over the slowest rank's time."""
    return tokens_per_step * steps * world / (max_ms / 1e3)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def run_reference(args, cfg):
    """fp64 oracle on the host cores: each step is a bounded sample of the workload."""
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    from oracle import oracle
    oracle.build()
    x = synth.make_inputs(cfg)
    frac_rows = args.ref_rows
    M = cfg.rows
    rows = np.arange(0, M, max(1, M // frac_rows))[:frac_rows]
    # attention rows of the same candidate tokens, all heads
    tok = rows
    sel = np.zeros((M, cfg.hq), bool)
    sel[tok, :] = True
    sel = sel.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.hq)
    cores = oracle.max_threads()

    def step(rows, sel):
        oracle.verify_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"], x["k_tail"],
                           x["v_tail"], row_sel=sel)
        lp, _ = oracle.score_logprobs(x["hidden"][rows], x["weight"], x["targets"][rows])
        _, mc, _, keep = oracle.clip_align(x["cand_emb"], x["frame_emb"], cfg.threshold)
        full = np.zeros((M, cfg.gathers))
        full[rows] = lp
        oracle.select(full.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.gathers), keep=keep)

    # rows per step: at most --ref-rows, and few enough that the whole run (warm-up and
    # timed steps) stays within about --ref-budget seconds, from a one-step probe
    t0 = time.perf_counter()
    step(rows, sel)
    per_row = (time.perf_counter() - t0) / len(rows)
    n = int(max(1, min(len(rows), args.ref_budget / max(1e-9, per_row * (args.steps + args.warmup)))))
    rows = rows[:n]
    sel = np.zeros((M, cfg.hq), bool)
    sel[rows, :] = True
    sel = sel.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.hq)
    for _ in range(args.warmup):
        step(rows, sel)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step(rows, sel)
    dt = (time.perf_counter() - t0) / args.steps
    value = len(rows) / dt
    sample = ("%d of %d candidate-token rows per step (LM head and all %d heads of attention for "
              "those rows; CLIP and selection in full)" % (len(rows), M, cfg.hq))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_block(cfg),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def config_block(cfg):
    return {"workload": cfg.description, "name": cfg.name, "num_queries": cfg.num_queries,
            "tokens_per_step": cfg.rows, "prefix_len": cfg.prefix_len or list(cfg.prefix_range),
            "hidden": cfg.hidden, "heads": [cfg.hq, cfg.hkv, cfg.head_dim], "vocab": cfg.vocab,
            "clip": [cfg.num_cand, cfg.num_frames, cfg.clip_dim], "selection": "masked mean log-prob",
            "l2": "flushed before every timed step / launch: 256 MiB write, then a 256 MiB read that "
                  "drains the write's dirty lines; both outside the CUDA events",
            "parallelism": "replicas"}


def cpu_baseline(cfg, x, budget_s):
    """The oracle as it stands, timed on this host's cores over a bounded sample."""
    from oracle import oracle
    oracle.build()
    cores = oracle.max_threads()
    M = cfg.rows
    t0 = time.perf_counter()
    done = 0
    nrows = max(1, min(M, 8))
    rows = np.arange(nrows) * max(1, M // nrows)
    # attention for the sampled tokens (all heads) + LM head for the sampled rows, then CLIP + select
    sel = np.zeros((M, cfg.hq), bool)
    sel[rows, :] = True
    sel = sel.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.hq)
    reps = 0
    while True:
        oracle.verify_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"], x["k_tail"],
                           x["v_tail"], row_sel=sel)
        lp, _ = oracle.score_logprobs(x["hidden"][rows], x["weight"], x["targets"][rows])
        _, mc, _, keep = oracle.clip_align(x["cand_emb"], x["frame_emb"], cfg.threshold)
        full = np.zeros((M, cfg.gathers))
        full[rows] = lp
        oracle.select(full.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.gathers), keep=keep)
        done += nrows
        reps += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    return {"value": done / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "%d repetitions of %d of %d candidate-token rows (their attention over all %d "
                      "heads and their LM-head log-probs, plus CLIP and selection in full), %.1f s"
                      % (reps, nrows, M, cfg.hq, dt)}


_TIMED_LAUNCHES = [0]   # library kernel launches inside the timed loops of a row bench


def _time_calls(fn, stream, steps, dev, between=None):
    """CUDA-event time of `steps` calls of fn on `stream` (ms per call, and the list);
    `between` (outside the events) runs before each call.  The library's kernel launches
    inside the loop are added to _TIMED_LAUNCHES (from its own launch counter)."""
    import torch
    from paper_2601_01513_gb300 import fvrag
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    n0 = fvrag.launch_count()
    for i in range(steps):
        if between is not None:
            between()
        ev[i][0].record(stream)
        fn()
        ev[i][1].record(stream)
    _TIMED_LAUNCHES[0] += fvrag.launch_count() - n0
    torch.cuda.synchronize(dev)
    ms = np.array([a.elapsed_time(b) for a, b in ev])
    return float(ms.mean()), ms


def _steps_for_clocks(fn, stream, dev, steps, between=None, min_s=0.6, cap=20000):
    """At least `steps` calls, and enough for the timed loop to last `min_s` seconds of wall
    time, so that the clock sampler (one sample per 100 ms) sees the calls running."""
    import torch
    t0 = time.perf_counter()
    for _ in range(5):
        if between is not None:
            between()
        fn()
    torch.cuda.synchronize(dev)
    per = (time.perf_counter() - t0) / 5
    return int(min(cap, max(steps, np.ceil(min_s / max(per, 1e-7)))))


def bench_row(args):
    """One JSON line for the retrieval or keyframe step (1 GPU; other ranks replicate)."""
    import torch
    import torch.distributed as dist

    from paper_2601_01513_gb300 import fvrag
    from paper_2601_01513_gb300.build import build_all
    from oracle import oracle

    ws_, rank, local = dist_env()
    if ws_ > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if ws_ > 1 else 0)
    if rank == 0:
        build_all()
    if ws_ > 1:
        dist.barrier()
    fvrag.lib()
    pk, pk_src = peaks()
    stream = torch.cuda.Stream(device=dev)
    steps = max(3, min(args.steps, 200))

    if args.row == "retrieve":
        cfg = configs.RETRIEVAL_PRESETS[args.row_config or "retrieve-16q-1m"]
        r = synth.retrieval_inputs(cfg, seed=cfg.seed + 7919 * rank)
        Fr, E, Nt = r["frames"].shape[0], cfg.dim, cfg.num_texts
        texts = torch.from_numpy(r["texts"].view(np.int16)).view(torch.float16).to(dev)
        frames = torch.from_numpy(r["frames"].view(np.int16)).view(torch.float16).to(dev)
        offs = torch.from_numpy(r["frame_offsets"]).to(dev)
        inv = torch.empty(Nt, dtype=torch.float32, device=dev)
        d = fvrag.retrieve_desc(cfg.num_queries, frames, texts, cfg.k_frame, cfg.k_query)
        ws = torch.zeros(fvrag.retrieve_workspace_bytes(d), dtype=torch.uint8, device=dev)
        oi = torch.empty((cfg.num_queries, cfg.k_query), dtype=torch.int32, device=dev)
        os_ = torch.empty((cfg.num_queries, cfg.k_query), dtype=torch.float32, device=dev)
        h_frames = torch.from_numpy(r["frames"].view(np.int16)).view(torch.float16).pin_memory()
        h_offs = torch.from_numpy(r["frame_offsets"]).pin_memory()
        h_oi = torch.empty_like(oi, device="cpu").pin_memory()
        h_os = torch.empty_like(os_, device="cpu").pin_memory()

        def call():
            fvrag.retrieve(frames, offs, texts, cfg.k_frame, oi, os_, ws, text_inv_norm=inv,
                           stream=stream)

        def call_host():
            frames.copy_(h_frames, non_blocking=True)
            offs.copy_(h_offs, non_blocking=True)
            call()
            h_oi.copy_(oi, non_blocking=True)
            h_os.copy_(os_, non_blocking=True)

        with torch.cuda.stream(stream):
            fvrag.embed_inv_norms(texts, inv, stream=stream)      # index build, once per corpus
            inv_ms, _ = _time_calls(lambda: fvrag.embed_inv_norms(texts, inv, stream=stream),
                                    stream, 5, dev)
            for _ in range(args.warmup):
                call()
                call_host()
            torch.cuda.synchronize(dev)
            steps = _steps_for_clocks(call, stream, dev, steps)
            with ClockSampler(dev.index or 0) as clk:
                clk.wait_first()
                t_ms, _ = _time_calls(call, stream, steps, dev)
                e_ms, _ = _time_calls(call_host, stream, steps, dev)
        assert fvrag.read_status(ws) == fvrag.OK
        units = Fr
        metric, unit = "keyframes retrieved/s", "keyframes/s"
        flops = 2.0 * Fr * Nt * E
        nbytes = Nt * E * 2 + Nt * 4 + Fr * E * 2
        t_tc = flops / (pk["bf16_tflops_sustained"] * 1e12)
        t_hbm = nbytes / (pk["hbm_gbs"] * 1e9)
        if t_tc >= t_hbm:
            roof = {"bound": "tensor", "achieved": flops / (t_ms * 1e-3) / 1e12,
                    "peak": pk["bf16_tflops_sustained"], "unit": "TFLOP/s"}
        else:
            roof = {"bound": "hbm", "achieved": nbytes / (t_ms * 1e-3) / 1e9, "peak": pk["hbm_gbs"],
                    "unit": "GB/s"}
        roof.update({"frac": roof["achieved"] / roof["peak"], "traffic": None,
                     "kernel": "fvrag retrieve (tcgen05 fp16 GEMM + per-keyframe top-k), timed "
                               "with its two small merge kernels",
                     "peak_source": pk_src + (" (fp16 tensor peak = the measured bf16 peak; same "
                                              "nominal rate)" if t_tc >= t_hbm else ""),
                     "other_roof_frac": (nbytes / (t_ms * 1e-3) / 1e9) / pk["hbm_gbs"] if t_tc >= t_hbm
                     else (flops / (t_ms * 1e-3) / 1e12) / pk["bf16_tflops_sustained"]})
        h2d = Fr * E * 2 + (cfg.num_queries + 1) * 4
        d2h = cfg.num_queries * cfg.k_query * 8
        config = {"workload": cfg.description, "name": cfg.name, "keyframes": Fr, "texts": Nt,
                  "dim": E, "k_frame": cfg.k_frame, "k_query": cfg.k_query,
                  "l2": "inputs larger than L2 (the %.2f GB corpus is streamed every call)"
                        % (Nt * E * 2 / 1e9),
                  "inv_norm_index_build_ms": inv_ms, "parallelism": "replicas"}
        dtype = "f16"
        cpu = None
        if not args.no_cpu_baseline and ws_ == 1:
            oracle.build()
            sample = np.arange(0, Fr, max(1, Fr // 8))[:8]
            t0 = time.perf_counter()
            fi, fs = oracle.frame_topk(r["frames"][sample], r["texts"], cfg.k_frame)
            oracle.aggregate_topk(np.array([0, len(sample)], np.int32), fi, fs, cfg.k_query)
            dt = time.perf_counter() - t0
            cpu = {"value": len(sample) / dt, "unit": unit, "cores": oracle.max_threads(),
                   "kind": "oracle", "sample": "%d of %d keyframes scanned against the whole corpus "
                   "and aggregated, %.1f s" % (len(sample), Fr, dt)}
    elif args.row == "clip-sweep":
        # the CLIP alignment of Eq. 14-15 alone on a large case, to show its bandwidth
        cfg = configs.V7B.with_(name="clip-16x10x4096x768", num_queries=16, num_cand=10,
                                num_frames=4096, clip_dim=768,
                                description="CLIP alignment alone: 16 queries x 10 candidates x 4096 "
                                            "frames x 768 (fp16)")
        cand, frames = synth.clip_embeddings(cfg, seed=cfg.seed + 7919 * rank)
        tc = torch.from_numpy(cand.view(np.int16)).view(torch.float16).to(dev)
        tf = torch.from_numpy(frames.view(np.int16)).view(torch.float16).to(dev)
        Qn, K = cfg.num_queries, cfg.num_cand
        mc = torch.empty((Qn, K), dtype=torch.float32, device=dev)
        am = torch.empty((Qn, K), dtype=torch.int32, device=dev)
        keep = torch.empty((Qn, K), dtype=torch.uint8, device=dev)
        h_c = torch.from_numpy(cand.view(np.int16)).view(torch.float16).pin_memory()
        h_f = torch.from_numpy(frames.view(np.int16)).view(torch.float16).pin_memory()
        h_keep = torch.empty((Qn, K), dtype=torch.uint8).pin_memory()
        flush_w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

        def call():
            fvrag.clip_align(tc, tf, cfg.threshold, mc, am, keep, stream=stream)

        def call_host():
            tc.copy_(h_c, non_blocking=True)
            tf.copy_(h_f, non_blocking=True)
            call()
            h_keep.copy_(keep, non_blocking=True)

        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                call()
                call_host()
            torch.cuda.synchronize(dev)
            steps = _steps_for_clocks(call, stream, dev, steps, between=flush_w.zero_)
            with ClockSampler(dev.index or 0) as clk:
                clk.wait_first()
                t_ms, _ = _time_calls(call, stream, steps, dev, between=flush_w.zero_)
                e_ms, _ = _time_calls(call_host, stream, steps, dev, between=flush_w.zero_)
        units = Qn * K * cfg.num_frames
        metric, unit = "candidate-frame cosines/s", "cosines/s"
        nbytes = Qn * (K + cfg.num_frames) * cfg.clip_dim * 2 + Qn * K * 9
        roof = {"bound": "hbm", "achieved": nbytes / (t_ms * 1e-3) / 1e9, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "traffic": None, "peak_source": pk_src,
                "kernel": "fvrag CLIP alignment (clip_align_kernel)"}
        roof["frac"] = roof["achieved"] / roof["peak"]
        h2d = (tc.numel() + tf.numel()) * 2
        d2h = Qn * K
        config = {"workload": cfg.description, "name": cfg.name,
                  "clip": [Qn, K, cfg.num_frames, cfg.clip_dim],
                  "l2": "flushed before every timed call (256 MiB write, outside the events); "
                        "the %.0f MB of frames also exceed L2" % (tf.numel() * 2 / 1e6),
                  "parallelism": "replicas"}
        dtype = "f16"
        cpu = None
        if not args.no_cpu_baseline and ws_ == 1:
            oracle.build()
            t0 = time.perf_counter()
            reps = 0
            while True:
                oracle.clip_align(cand[:1], frames[:1], cfg.threshold)
                reps += 1
                if time.perf_counter() - t0 > args.cpu_budget:
                    break
            dt = time.perf_counter() - t0
            cpu = {"value": reps * K * cfg.num_frames / dt, "unit": unit, "cores": oracle.max_threads(),
                   "kind": "oracle", "sample": "%d passes over query 0 (%d candidates x %d frames), %.1f s"
                   % (reps, K, cfg.num_frames, dt)}
    elif args.row == "decode":
        cfg = configs.DECODE_PRESETS[args.row_config or "decode-3b-16q"]
        x = synth.decode_inputs(cfg, seed=cfg.seed + 7919 * rank)

        def up(a):
            t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16) if a.dtype == np.uint16 else a)
            return (t.view(torch.bfloat16) if a.dtype == np.uint16 else t).to(dev)

        q, kp, vp = up(x["q"]), up(x["k_prefix"]), up(x["v_prefix"])
        kc, vc = up(x["k_cache"]), up(x["v_cache"])
        offs, n = up(x["prefix_offsets"]), up(x["cache_len"])
        maxp = int(np.max(np.diff(x["prefix_offsets"])))
        d = fvrag.decode_desc(q, kp, kc, maxp)
        ws = torch.zeros(fvrag.decode_workspace_bytes(d), dtype=torch.uint8, device=dev)
        out = torch.empty_like(q)
        h_q = torch.from_numpy(x["q"].view(np.int16)).view(torch.bfloat16).pin_memory()
        h_n = torch.from_numpy(x["cache_len"]).pin_memory()
        h_out = torch.empty(q.shape, dtype=torch.bfloat16).pin_memory()
        flush_w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

        def call():
            fvrag.decode_attn(q, kp, vp, offs, kc, vc, n, out, ws, maxp, stream=stream)

        def call_host():
            q.copy_(h_q, non_blocking=True)
            n.copy_(h_n, non_blocking=True)
            call()
            h_out.copy_(out, non_blocking=True)

        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                call()
                call_host()
            torch.cuda.synchronize(dev)
            steps = _steps_for_clocks(call, stream, dev, steps, between=flush_w.zero_)
            with ClockSampler(dev.index or 0) as clk:
                clk.wait_first()
                t_ms, _ = _time_calls(call, stream, steps, dev, between=flush_w.zero_)
                e_ms, _ = _time_calls(call_host, stream, steps, dev, between=flush_w.zero_)
        assert fvrag.read_status(ws) == fvrag.OK
        Qn, K, hkv, D = cfg.num_queries, cfg.num_drafts, cfg.hkv, cfg.head_dim
        units = Qn * K
        metric, unit = "draft tokens decoded/s (one attention layer)", "tokens/s"
        sumP = int(x["prefix_offsets"][-1])
        sumN = int(x["cache_len"].sum())
        nbytes = (sumP + sumN) * hkv * D * 2 * 2 + 2 * q.numel() * 2
        roof = {"bound": "hbm", "achieved": nbytes / (t_ms * 1e-3) / 1e9, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "traffic": None, "peak_source": pk_src,
                "kernel": "fvrag shared-prefix attention in decode form (Lq = 1), timed with its "
                          "merge kernel"}
        roof["frac"] = roof["achieved"] / roof["peak"]
        h2d = q.numel() * 2 + n.numel() * 4
        d2h = out.numel() * 2
        config = {"workload": cfg.description, "name": cfg.name, "drafts": units,
                  "prefix_tokens": sumP, "cache_tokens": sumN, "heads": [cfg.hq, hkv, D],
                  "l2": "flushed before every timed call (256 MiB write, outside the events)",
                  "parallelism": "replicas"}
        dtype = "bf16"
        cpu = None
        if not args.no_cpu_baseline and ws_ == 1:
            oracle.build()
            a, b = int(x["prefix_offsets"][0]), int(x["prefix_offsets"][1])
            t0 = time.perf_counter()
            reps = 0
            while True:
                oracle.decode_attn(x["q"][:1], x["k_prefix"][a:b], x["v_prefix"][a:b],
                                   np.array([0, b - a], np.int32), x["k_cache"][:1], x["v_cache"][:1],
                                   x["cache_len"][:1])
                reps += 1
                if time.perf_counter() - t0 > args.cpu_budget:
                    break
            dt = time.perf_counter() - t0
            cpu = {"value": reps * K / dt, "unit": unit, "cores": oracle.max_threads(),
                   "kind": "oracle", "sample": "%d passes over query 0 (%d drafts, all heads), %.1f s"
                   % (reps, K, dt)}
    else:
        cfg = configs.KEYFRAME_PRESETS[args.row_config or "keyframe-8x720p"]
        px, voffs = synth.video_frames(cfg, seed=cfg.seed + 7919 * rank)
        T = int(voffs[-1])
        pixels = torch.from_numpy(px).to(dev)
        vo = torch.from_numpy(voffs).to(dev)
        d = fvrag.keyframe_desc(cfg.num_videos, pixels, cfg.theta)
        ws = torch.zeros(fvrag.keyframes_workspace_bytes(d), dtype=torch.uint8, device=dev)
        sim = torch.empty(T, dtype=torch.float32, device=dev)
        key = torch.empty(T, dtype=torch.uint8, device=dev)
        kidx = torch.empty(T, dtype=torch.int32, device=dev)
        koffs = torch.empty(cfg.num_videos + 1, dtype=torch.int32, device=dev)
        h_px = torch.from_numpy(px).pin_memory()
        h_vo = torch.from_numpy(voffs).pin_memory()
        h_kidx = torch.empty(T, dtype=torch.int32).pin_memory()
        h_koffs = torch.empty(cfg.num_videos + 1, dtype=torch.int32).pin_memory()

        def call():
            fvrag.keyframes(pixels, vo, cfg.theta, sim, key, kidx, koffs, ws, stream=stream)

        def call_host():
            pixels.copy_(h_px, non_blocking=True)
            vo.copy_(h_vo, non_blocking=True)
            call()
            h_koffs.copy_(koffs, non_blocking=True)
            h_kidx.copy_(kidx, non_blocking=True)

        steps = max(3, min(steps, 50))
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                call()
            call_host()
            torch.cuda.synchronize(dev)
            steps = _steps_for_clocks(call, stream, dev, steps)
            with ClockSampler(dev.index or 0) as clk:
                clk.wait_first()
                t_ms, _ = _time_calls(call, stream, steps, dev)
                e_ms, _ = _time_calls(call_host, stream, max(3, steps // 5), dev)
        assert fvrag.read_status(ws) == fvrag.OK
        units = T
        metric, unit = "video frames processed/s", "frames/s"
        nbytes = T * cfg.npix * 3 + T * 512 * 4
        roof = {"bound": "hbm", "achieved": nbytes / (t_ms * 1e-3) / 1e9, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "traffic": None, "peak_source": pk_src,
                "kernel": "fvrag keyframe histogram (bulk-copy ring + shared-memory histograms), "
                          "timed with its similarity and compaction kernels"}
        roof["frac"] = roof["achieved"] / roof["peak"]
        h2d = T * cfg.npix * 3 + (cfg.num_videos + 1) * 4
        d2h = T * 4 + (cfg.num_videos + 1) * 4
        config = {"workload": cfg.description, "name": cfg.name, "frames": T,
                  "resolution": [cfg.width, cfg.height], "theta": cfg.theta,
                  "l2": "inputs larger than L2 (%.2f GB of frames per call)" % (T * cfg.npix * 3 / 1e9),
                  "parallelism": "replicas"}
        dtype = "u8"
        cpu = None
        if not args.no_cpu_baseline and ws_ == 1:
            oracle.build()
            n = int(voffs[1])
            t0 = time.perf_counter()
            reps = 0
            while True:
                oracle.keyframes(px[:n], np.array([0, n], np.int32), cfg.theta)
                reps += 1
                if time.perf_counter() - t0 > args.cpu_budget:
                    break
            dt = time.perf_counter() - t0
            cpu = {"value": reps * n / dt, "unit": unit, "cores": oracle.max_threads(), "kind": "oracle",
                   "sample": "%d passes over video 0 (%d frames), %.1f s" % (reps, n, dt)}

    t_ms, e_ms = max_over_ranks([t_ms, e_ms], dev)
    if rank == 0:
        line = {"metric": metric, "value": units * ws_ / (t_ms * 1e-3), "unit": unit, "n_gpus": ws_,
                "steps": steps, "warmup": args.warmup, "ms_per_step": t_ms, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": dtype, "data": "synthetic",
                "config": config,
                "e2e": {"value": units * ws_ / (e_ms * 1e-3), "unit": unit, "h2d_bytes_per_step": int(h2d),
                        "d2h_bytes_per_step": int(d2h), "ms_per_step": e_ms},
                "gpu_launches": _TIMED_LAUNCHES[0],
                "roofline": roof, "clocks": clk.summary()}
        if cpu:
            line["cpu_baseline"] = cpu
        print(json.dumps(line), flush=True)
    if ws_ > 1:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--kernel-reps", type=int, default=200)
    ap.add_argument("--config", default="72b", choices=sorted(configs.PRESETS),
                    help="verify-step workload (default: the 72B-class verifier, the largest "
                         "single-GPU preset)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--ref-rows", type=int, default=8,
                    help="--impl reference: at most this many candidate-token rows per step")
    ap.add_argument("--ref-budget", type=float, default=150.0,
                    help="--impl reference: seconds the whole run should take at most (fewer "
                         "rows per step, down to one, when it would take longer)")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--row", default="verify",
                    choices=["verify", "retrieve", "keyframes", "decode", "clip-sweep"],
                    help="verify: the verify step (default); retrieve / keyframes / decode: the "
                         "retrieval (Eq. 2-3), keyframe (Eq. 1) or drafter decode-attention "
                         "(Eq. 5) step on its own workload; clip-sweep: the CLIP alignment call "
                         "alone at 16 queries x 10 candidates x 4096 frames x 768 (its bandwidth)")
    ap.add_argument("--row-config", default=None,
                    help="workload preset of --row (default: retrieve-16q-1m / keyframe-8x720p / "
                         "decode-3b-16q)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.row != "verify":
        return bench_row(args)
    cfg = configs.PRESETS[args.config]

    if args.impl == "reference":
        return run_reference(args, cfg)

    import torch
    import torch.distributed as dist

    from paper_2601_01513_gb300 import fvrag
    from paper_2601_01513_gb300.build import build_all
    from paper_2601_01513_gb300.pipeline import VerifyStep

    ws_, rank, local = dist_env()
    if ws_ > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if ws_ > 1 else 0)
    if rank == 0:
        build_all()
    if ws_ > 1:
        dist.barrier()
    fvrag.lib()

    # each rank verifies its own queries (independent replica, rank-dependent seed)
    x = synth.make_inputs(cfg, seed=replica_seed(cfg, rank))
    step = VerifyStep(cfg, device=dev)
    step.upload(x)
    # L2 flush between timed iterations: write a 256 MiB buffer (> the 126.5 MiB L2), then read
    # another 256 MiB buffer so the flush's own dirty lines are written back before the
    # timed kernels start (otherwise the first timed kernel pays for the flush's write-back)
    flush_w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_r = torch.ones((256, 1 << 18), dtype=torch.float32, device=dev)
    flush_sink = torch.empty((256,), dtype=torch.float32, device=dev)

    class _Flush:
        @staticmethod
        def zero_():
            flush_w.zero_()
            torch.amax(flush_r, dim=1, out=flush_sink)

    flush = _Flush()
    names = ["attn", "lm", "clip", "select"]
    # per-kernel numbers: each call alone on all SMs; with an SM split, the attention and the
    # LM head are also timed alone within their budgets ("sm_split" in the line)
    calls = {"attn": lambda: step.attention(sm_budget=0), "lm": lambda: step.lm_head(sm_budget=0),
             "clip": step.clip, "select": step.select}
    split_names = []
    if step.sm_split is not None:
        calls["attn_split"], calls["lm_split"] = step.attention, step.lm_head
        split_names = ["attn_split", "lm_split"]
    for _ in range(args.warmup):
        step.run()
    torch.cuda.synchronize(dev)
    assert fvrag.read_status(step.lm_ws) == fvrag.OK and fvrag.read_status(step.attn_ws) == fvrag.OK
    # kernel launches per step and per call, from the library's own launch counter
    launches_step = step.launches_per_step()
    launches_call = {n: step.launches_of(calls[n]) for n in calls}
    torch.cuda.synchronize(dev)
    # one CUDA graph for the whole step, one per call for the per-kernel numbers
    step.capture()
    graphs = {}
    for n in names + split_names:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            calls[n]()
        graphs[n] = g
    stream = torch.cuda.Stream(device=dev)
    host = step.host_inputs(pin=True)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step.replay()
            for n in names + split_names:
                graphs[n].replay()
            step.run_from_host(host)
        torch.cuda.synchronize(dev)
        # kernels of one end-to-end step (its own SM split may add the attention's merge)
        launches_e2e = step.launches_of(lambda: step.run_from_host(host, stream=stream))
        torch.cuda.synchronize(dev)
        if ws_ > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)
        with ClockSampler(dev.index if dev.index is not None else 0) as clk:
            clk.wait_first()
            # timed region: K whole steps, L2 flushed before each (outside the events)
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(args.steps)]
            t_wall = time.perf_counter()
            for i in range(args.steps):
                flush.zero_()
                ev[i][0].record(stream)
                step.replay()
                ev[i][1].record(stream)
            torch.cuda.synchronize(dev)
            t_wall = time.perf_counter() - t_wall
            step_ms = np.array([a.elapsed_time(b) for a, b in ev])
            # per-kernel launch durations (each call replayed alone, L2 flushed before each)
            kreps = max(3, min(args.steps, args.kernel_reps))
            per_k = np.zeros((kreps, len(names) + len(split_names)))
            for j, n in enumerate(names + split_names):
                kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                       for _ in range(kreps)]
                for i in range(kreps):
                    flush.zero_()
                    kev[i][0].record(stream)
                    graphs[n].replay()
                    kev[i][1].record(stream)
                torch.cuda.synchronize(dev)
                per_k[:, j] = [a.elapsed_time(b) for a, b in kev]
            # end to end through the public API with host buffers: copies of the step's inputs
            # from pinned memory, the step, and the read of the result, all inside the events
            ee = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(args.steps)]
            h2d = d2h = 0
            for i in range(args.steps):
                flush.zero_()
                ee[i][0].record(stream)
                _, _, h2d, d2h = step.run_from_host(host)
                ee[i][1].record(stream)
            torch.cuda.synchronize(dev)
            e2e_ms = float(sum(a.elapsed_time(b) for a, b in ee))
        if ws_ > 1:
            dist.barrier()
        total_ms = float(step_ms.sum())
        assert fvrag.read_status(step.lm_ws) == fvrag.OK and fvrag.read_status(step.attn_ws) == fvrag.OK

    total_ms, e2e_ms = max_over_ranks([total_ms, e2e_ms], dev)
    value = job_throughput(cfg.rows, args.steps, ws_, total_ms)
    e2e_value = job_throughput(cfg.rows, args.steps, ws_, e2e_ms)
    pk, pk_src = peaks()
    alg = algorithmic(cfg)
    names = ["attn", "lm", "clip", "select"]
    kern = {}
    for j, n in enumerate(names):
        us = float(np.mean(per_k[:, j])) * 1e3
        b, f = alg[n]
        kern[n] = {"us": us, "us_median": float(np.median(per_k[:, j])) * 1e3, "GB_s": b / (us * 1e-6) / 1e9,
                   "TFLOP_s": f / (us * 1e-6) / 1e12 if f else 0.0, "alg_bytes": b, "alg_flops": f}
        kern[n]["hbm_frac"] = kern[n]["GB_s"] / pk["hbm_gbs"]
        if f:
            kern[n]["tc_frac"] = kern[n]["TFLOP_s"] / pk["bf16_tflops_sustained"]
    lm = kern["lm"]
    traffic = None   # DRAM bytes per launch from an ncu capture of this workload's LM head
    tr = LM_TRAFFIC.get(cfg.name)
    if tr and tr["bytes_per_launch"] and source_sha("lmhead.cu").startswith(tr["sha256_prefix"]):
        traffic = tr["bytes_per_launch"]
    # the binding roof: HBM below the ridge (at most ~278 rows), the tensor cores above it
    # (the sustained bf16 peak: the call is replayed back to back for seconds)
    ridge = pk["bf16_tflops_sustained"] * 1e12 / (pk["hbm_gbs"] * 1e9)
    if lm["alg_flops"] / lm["alg_bytes"] <= ridge:
        roof = {"bound": "hbm", "achieved": lm["GB_s"], "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": lm["GB_s"] / pk["hbm_gbs"]}
    else:
        roof = {"bound": "tensor", "achieved": lm["TFLOP_s"], "peak": pk["bf16_tflops_sustained"],
                "unit": "TFLOP/s", "frac": lm["TFLOP_s"] / pk["bf16_tflops_sustained"]}
    roof.update({"traffic": traffic, "kernel": "fvrag LM head (tcgen05 GEMM + LSE)",
                 "peak_source": pk_src})
    if rank != 0:
        if ws_ > 1:
            dist.destroy_process_group()
        return 0
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws_, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": config_block(cfg),
            "us_per_query": total_ms / args.steps * 1e3 / cfg.num_queries,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                    "d2h_bytes_per_step": int(d2h), "ms_per_step": e2e_ms / args.steps},
            "gpu_launches": (launches_step + launches_e2e) * args.steps
                            + sum(launches_call[n] for n in names + split_names) * per_k.shape[0],
            "timing": {"step": "CUDA graph of the four calls, CUDA events per step, L2 flushed between steps",
                       "kernels": "each call replayed alone %d times (events per launch), L2 flushed before each"
                                  % per_k.shape[0], "host_wall_s": t_wall,
                       "step_us_p10_p50_p90": [float(np.percentile(step_ms, q)) * 1e3 for q in (10, 50, 90)],
                       "sum_of_call_medians_us": float(sum(k["us_median"] for k in kern.values()))},
            "roofline": roof, "kernels": kern, "clocks": clk.summary()}
    if split_names:
        A, B = step.sm_split
        line["sm_split"] = {
            "attn_sms": A, "lm_sms": B, "e2e": list(step.sm_split_e2e or []),
            "note": "attention beside the LM head on two streams; each timed alone in its budget "
                    "(the host-input path gives the attention the second split: it starts once "
                    "its inputs land)",
            "attn_us": float(np.mean(per_k[:, len(names)])) * 1e3,
            "lm_us": float(np.mean(per_k[:, len(names) + 1])) * 1e3}
    if not args.no_cpu_baseline and ws_ == 1:
        line["cpu_baseline"] = cpu_baseline(cfg, x, args.cpu_budget)
    print(json.dumps(line), flush=True)
    if ws_ > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
