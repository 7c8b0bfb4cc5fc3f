"""Benchmark of one SPIRe speculation round's attention on GB300.

A step is one pass of the whole hot path over one batch: the verification
attention of the k+1 block tokens (split plan, split attention and the
log-sum-exp merge of splits, all in one kernel launch) plus the k draft sink +
window attention steps of the round (draft step j sees
t = L - k + j memory entries).  The default workload is the uniform long-
context config: B=64, L=8192, k=4, 32 query / 8 KV heads, D=128, 64-token pages
in a seeded random order, draft 16 sink + 512 window.  Inputs are seeded
synthetic N(0,1) bf16 tensors resident in HBM.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME]
                    [--impl spire|reference]
    python bench.py --profile-call verify|decode|draft|append|tokens|magicdec
                    [--config NAME] [--max-seqs N] [--warmup W] [--calls C]

Prints one JSON line (rank 0).  `--impl reference` times the fp64 CPU oracle
on a bounded sample of the same workload instead.  `--profile-call` makes only
one kind of library call and exits (for small profiler captures); it prints no
benchmark line.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as wl  # noqa: E402

METRIC = "speculation-round attention tokens/s and HBM GB/s vs 8 TB/s at B=64, k=4, 1 GB300"
HBM_NOMINAL_GBS = 8000.0
SPIRE_TAU_K4_L512 = 3.401   # SPIRe average generation length at L=512, k=4 (Table 1)


# ------------------------------------------------------------------ helpers
def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.QUERY,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self, t0, t1):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.t.join(timeout=2)
        rows = []
        for ts, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            rows.append((ts, parts))
        inside = [r for ts, r in rows if t0 - 0.25 <= ts <= t1 + 0.25] or [r for _, r in rows]
        sm = [float(r[1]) for r in inside if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in inside if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i in range(4)
                          if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "samples": len(inside), "reasons": reasons}


def source_sha16():
    """Hash of the device code and launch configuration (the .cuh kernels and
    spire_launch.h, comments and blank lines left out): the code whose change
    invalidates the ncu counters."""
    import hashlib
    import re
    d = os.path.join(ROOT, "paper_2504_06419_gb300", "csrc")
    h = hashlib.sha256()
    for f in sorted(os.listdir(d)):
        if f.endswith(".cuh") or f == "spire_launch.h":
            h.update(f.encode())
            with open(os.path.join(d, f)) as fh:
                src = re.sub(r"/\*.*?\*/", "", fh.read(), flags=re.S)
            lines = (re.sub(r"//.*", "", ln).rstrip() for ln in src.splitlines())
            h.update("\n".join(ln for ln in lines if ln).encode())
    return h.hexdigest()[:16]


def dram_traffic(key):
    """DRAM bytes per launch from the committed ncu counters, or None when the
    kernels changed since they were taken."""
    try:
        with open(os.path.join(ROOT, "profiles", "counters.json")) as f:
            c = json.load(f)
        if c.get("source_sha16") != source_sha16():
            return None
        k = c["kernels"][key]
        return int(k["dram_bytes_read"]) + int(k["dram_bytes_write"])
    except Exception:
        return None


def verify_bytes(L, k, Hq, Hkv, D):
    """Algorithmic bytes of one verification call: every visible K/V byte once,
    q in (bf16), out (fp32), the block-table entries read and ctx_lens."""
    L = np.asarray(L, dtype=np.int64)
    B = L.size
    kv = int(L.sum()) * 4 * Hkv * D
    qo = B * (k + 1) * Hq * D * (2 + 4)
    meta = int(((L + 63) // 64).sum()) * 4 + 4 * B
    return kv + qo + meta


def draft_bytes(t, S, Hq, Hkv, D):
    t = np.asarray(t, dtype=np.int64)
    B = t.size
    return int(np.minimum(t, S).sum()) * 4 * Hkv * D + B * Hq * D * 6 + 4 * B


def append_bytes(B, n_act, n_dl, d_model, Hkv, D):
    """Algorithmic bytes of one feedback-memory append: the projection weights
    once, the activations, the mixing weights, the new entries and positions."""
    F = 2 * Hkv * D
    return n_dl * F * d_model * 2 + n_act * B * d_model * 2 + n_dl * n_act * 4 + \
        n_dl * B * F * 2 + 4 * B


def tokens_bytes(n_acc, k, V):
    """Algorithmic bytes of one token verification: per sequence the target row
    of the draw and the Exp(1) row, the draft row when a draft was rejected,
    the k gathered entries of p and q, the uniforms, tokens and outputs."""
    n_acc = np.asarray(n_acc, dtype=np.int64)
    B = n_acc.size
    rows = B * 2 * V * 4 + int((n_acc < k).sum()) * V * 4
    return rows + B * (k * 4 * 4 + (k + 1) * 4 + 4)


def verify_flops(L, k, Hq, D):
    L = np.asarray(L, dtype=np.int64)
    rows = sum(int((L - k + i).sum()) for i in range(k + 1))
    return 4 * D * Hq * rows


def reduce_max(values, dist=None, device=None):
    """Element-wise MAX of per-rank timings over all ranks (identity on one
    rank).  Ranks are independent replicas; only the timing is exchanged."""
    if dist is None:
        return [float(v) for v in values]
    import torch
    dev = device if device is not None else "cpu"
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.cpu().tolist()]


def cta_balance(times):
    """Per-SM busy time of one attention call from its per-CTA timing record."""
    busy = [(e - b) / 1e3 for b, e in times]
    mean = statistics.mean(busy)
    first = min(b for b, _ in times)
    return {"ctas": len(times), "busy_us_mean": mean, "busy_us_max": max(busy),
            "busy_us_min": min(busy), "max_over_mean": max(busy) / mean if mean > 0 else None,
            "start_spread_us": (max(b for b, _ in times) - first) / 1e3,
            "span_us": (max(e for _, e in times) - first) / 1e3}


class L2Flush:
    """Empties L2 of every input between timed launches: a 256 MB write (twice
    the 129 MB L2), then a read of that buffer, so that L2 holds only the
    buffer's clean lines.  A write alone leaves L2 full of dirty lines whose
    write-back the next timed kernel would pay (about 16 us for a verify call
    on GB300), which no step of a serving loop, where L2 mostly holds lines
    read by the previous kernels, would see."""

    def __init__(self, dev):
        import torch
        self.buf = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
        self.words = self.buf.view(torch.int64)

    def __call__(self, s, write_only=False):
        self.buf.fill_(s & 0xff)
        if not write_only:
            self.words.amax()


def event_ms(call, n, flush, stream, write_only=False):
    """Mean CUDA-event time (ms) of `call` over n launches, each after the L2
    flush outside the events, on `stream`."""
    import torch
    evs = []
    for s in range(n):
        flush(s, write_only)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call()
        b.record(stream)
        evs.append((a, b))
    torch.cuda.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in evs)


def verify_config_entry(spire, name, dev, stream, flush, args, hbm_peak, max_seqs=0, dist=None):
    """Verification attention on another workload, timed as the headline
    verify call: CUDA events around the C-ABI call, the 256 MB L2 flush
    between launches, the same warm-up.  Frees its inputs before returning."""
    import torch
    cfg = wl.CONFIGS[name]
    k, Hq, Hkv, D = cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
    L = wl.sample_ctx_lens(cfg)
    if max_seqs:
        L = L[:max_seqs]
    vi = wl.make_verify(L, k, Hq, Hkv, D, seed=cfg.seed, device=dev, shuffle=cfg.paged_shuffle)
    desc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
    ws = torch.empty(spire.spire_verify_workspace_bytes(desc, k), dtype=torch.uint8, device=dev)
    out = torch.empty(vi.q.shape, dtype=torch.float32, device=dev)
    sptr = stream.cuda_stream

    def call():
        st = spire.spire_verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table,
                                          vi.ctx_lens, k, desc, out, ws, ws.numel(), sptr)
        if st:
            raise spire.SpireError(st, "spire_verify_attention (%s)" % name)

    for _ in range(args.warmup):
        call()
    torch.cuda.synchronize(dev)
    if spire.spire_get_device_error(ws, stream):
        raise RuntimeError("device error word set by the %s verify call" % name)
    n = max(1, min(args.steps, 100))
    sampler = ClockSampler(dev.index if dev.index is not None else 0)
    sampler.start()
    time.sleep(0.3)
    t0 = time.time()
    ms = reduce_max([event_ms(call, n, flush, stream)], dist, dev)[0]   # the slowest rank
    clocks = sampler.stop(t0, time.time())
    flush(7)
    call()
    bal = cta_balance(spire.spire_get_cta_times(ws, ws.numel()))
    vb = verify_bytes(L, k, Hq, Hkv, D)
    gbs = vb / (ms * 1e-3) / 1e9
    B = int(L.size)
    entry = {"workload": workload_config(cfg, L)["workload"], "calls": n, "ms": ms,
             "algorithmic_bytes": vb, "gbs": gbs, "frac": gbs / hbm_peak,
             "frac_of_8TBs": gbs / HBM_NOMINAL_GBS,
             "verify_tokens_per_s": B * (k + 1) / (ms * 1e-3),
             "tflops": verify_flops(L, k, Hq, D) / (ms * 1e-3) / 1e12,
             "rows_per_kv_head": (Hq // Hkv) * (k + 1),
             "load_balance": bal,
             "traffic": dram_traffic("verify:%s" % name), "clocks": clocks}
    del vi, ws, out
    torch.cuda.empty_cache()

    # the round's k draft steps on this workload's bounded cache (step j sees
    # t = L - k + j entries), each call timed like the verify call, and the
    # speculation-round attention rate of one layer: B (k+1) / (t_verify + sum t_draft)
    S = cfg.n_sink + cfg.window
    di = wl.make_draft(wl.draft_ctx_for_step(L, k, 0), Hq, Hkv, D, cfg.n_sink, cfg.window,
                       seed=cfg.seed + 17, device=dev)
    ctxs = [torch.from_numpy(wl.draft_ctx_for_step(L, k, j)).to(dev) for j in range(k)]
    ddesc = spire.draft_desc(di.q, di.kv)
    dws = torch.empty(spire.spire_draft_workspace_bytes(ddesc, cfg.n_sink, cfg.window),
                      dtype=torch.uint8, device=dev)
    dout = torch.empty(di.q.shape, dtype=torch.float32, device=dev)

    def draft_call(j):
        st = spire.spire_draft_sparse_attention(di.q, di.kv, ctxs[j], cfg.n_sink, cfg.window,
                                                ddesc, dout, dws, dws.numel(), sptr)
        if st:
            raise spire.SpireError(st, "spire_draft_sparse_attention (%s)" % name)

    for _ in range(args.warmup):
        for j in range(k):
            draft_call(j)
    torch.cuda.synchronize(dev)
    if spire.spire_get_device_error(dws, stream):
        raise RuntimeError("device error word set by the %s draft call" % name)
    d_ms = sum(reduce_max([event_ms(lambda: draft_call(j), n, flush, stream)], dist, dev)[0]
               for j in range(k))
    db = sum(draft_bytes(wl.draft_ctx_for_step(L, k, j), S, Hq, Hkv, D) for j in range(k))
    entry["draft"] = {"steps": k, "ms_total": d_ms, "algorithmic_bytes": db,
                      "gbs": db / (d_ms * 1e-3) / 1e9,
                      "frac": db / (d_ms * 1e-3) / 1e9 / hbm_peak,
                      "cache_gb": di.kv.numel() * 2 / 1e9}
    entry["round_tokens_per_s"] = B * (k + 1) / ((ms + d_ms) * 1e-3)
    del di, ctxs, dws, dout
    torch.cuda.empty_cache()
    return entry


def job_value(tokens_per_rank, world, step_ms):
    """Whole-job throughput: every rank processes its own batch (weak scaling)."""
    return world * tokens_per_rank / (step_ms * 1e-3)


def perf_model_detail(L, k, Hq, Hkv, D, S, v_ms, d_ms, dec_ms):
    """Attention-only iteration time multiplier of one layer (Section 2) from
    the measured kernels, beside the model's memory-bound prediction from the
    algorithmic bytes (HOI cancels when every pass is memory-bound)."""
    from paper_2504_06419_gb300 import perf_model as pm
    L = np.asarray(L, dtype=np.int64)
    t_draft = d_ms / k
    dt = pm.measured_delta_t(k, t_draft, v_ms, dec_ms)
    db = sum(draft_bytes(wl.draft_ctx_for_step(L, k, j), S, Hq, Hkv, D) for j in range(k)) / k
    # one attention layer has no weights, and its FLOPs are far below bytes x HOI
    # here, so each pass costs its KV bytes (the paper's form: the target pass and
    # the verification read the same KV_target)
    modeled = pm.iteration_time_multiplier(k, 0.0, 0.0, db, 0.0, 0.0,
                                           verify_bytes(L, k, Hq, Hkv, D), 1.0)
    return {"what": "one attention layer: delta_t = (k t_draft + t_verify) / t_decode, t_decode = "
                    "the verify kernel with k = 0 at length L - k",
            "t_decode_ms": dec_ms, "t_verify_ms": v_ms, "t_draft_ms": t_draft,
            "delta_t_measured": dt, "delta_t_memory_bound_model": modeled,
            "tau_context": SPIRE_TAU_K4_L512,
            "throughput_multiplier_context": pm.throughput_multiplier(SPIRE_TAU_K4_L512, dt)}


# ------------------------------------------------------------------ oracle arm
def run_oracle_sample(cfg, n_seq, threads):
    """Time the fp64 oracle on the first n_seq sequences of the workload:
    the verification call plus the k draft steps.  Returns (seconds, tokens)."""
    import oracle
    L = wl.sample_ctx_lens(cfg)[:n_seq]
    vi = wl.make_verify(L, cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                        seed=cfg.seed, device="cpu", shuffle=cfg.paged_shuffle)
    qb, kb, vb = wl.bf16_bits(vi.q), wl.bf16_bits(vi.k_cache), wl.bf16_bits(vi.v_cache)
    bt, cl = vi.block_table.numpy(), vi.ctx_lens.numpy()
    drafts = []
    for j in range(cfg.k):
        di = wl.make_draft(wl.draft_ctx_for_step(L, cfg.k, j), cfg.num_q_heads,
                           cfg.num_kv_heads, cfg.head_dim, cfg.n_sink, cfg.window,
                           seed=cfg.seed + 17 * (j + 1), device="cpu")
        drafts.append((wl.bf16_bits(di.q), wl.bf16_bits(di.kv), di.ctx_lens.numpy()))
    t0 = time.perf_counter()
    oracle.verify(qb, kb, vb, bt, cl, cfg.k, threads=threads)
    for (q, kv, t) in drafts:
        oracle.draft_ring(q, kv, t, cfg.n_sink, cfg.window, threads=threads)
    dt = time.perf_counter() - t0
    return dt, n_seq * (cfg.k + 1)


def oracle_sample_size(cfg, target_s=15.0, threads=None):
    """Sequences of the workload that keep the oracle leg near target_s: the
    oracle's time grows with the context it reads, so the first sequence's
    time per context token is scaled by the cumulative lengths."""
    L = wl.sample_ctx_lens(cfg).astype(np.float64)
    dt, _ = run_oracle_sample(cfg, 1, threads)
    per_token = max(dt, 1e-3) / L[0]
    n = int(np.searchsorted(np.cumsum(L) * per_token, target_s, side="right"))
    return int(max(1, min(cfg.batch, n)))


def workload_config(cfg, L):
    """The `config` object both arms report for a workload."""
    return {"workload": "%s: B=%d, L=%s, k=%d, %d/%d heads, D=%d, 64-token pages "
                        "(shuffled=%s), draft %d sink + %d window"
                        % (cfg.name, len(L), ("%d" % L[0]) if cfg.ctx_dist == "fixed" else
                           "%s[%d,%d] (sum %d)" % (cfg.ctx_dist, cfg.ctx_lo, cfg.ctx_hi,
                                                   int(L.sum())),
                           cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                           cfg.paged_shuffle, cfg.n_sink, cfg.window),
            "global_batch": int(len(L)), "seq_len": int(L.max()), "parallelism": "replicas"}


def reference_arm(args, cfg):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    threads = os.cpu_count() or 1
    n_seq = oracle_sample_size(cfg, target_s=max(1.0, 20.0 / max(1, args.steps + args.warmup)),
                               threads=threads)
    for _ in range(args.warmup):
        run_oracle_sample(cfg, n_seq, threads)
    times = []
    tokens = 0
    for _ in range(args.steps):
        dt, tok = run_oracle_sample(cfg, n_seq, threads)
        times.append(dt)
        tokens = tok
    per_step = statistics.mean(times)
    value = tokens / per_step
    sample = ("first %d of %d sequences per step (verify + %d draft steps), fp64 C oracle"
              % (n_seq, cfg.batch, cfg.k))
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": per_step * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": dict(workload_config(cfg, wl.sample_ctx_lens(cfg)), sample=sample),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ spire arm
def spire_arm(args, cfg):
    import torch

    import paper_2504_06419_gb300 as spire

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)

    k, Hq, Hkv, D = cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
    L = wl.sample_ctx_lens(cfg)
    if args.max_seqs:
        L = L[:args.max_seqs]     # a smaller case of the same workload (profiling captures)
    vi = wl.make_verify(L, k, Hq, Hkv, D, seed=cfg.seed, device=dev, shuffle=cfg.paged_shuffle)
    drafts = [wl.make_draft(wl.draft_ctx_for_step(L, k, j), Hq, Hkv, D, cfg.n_sink, cfg.window,
                            seed=cfg.seed + 17 * (j + 1), device=dev) for j in range(k)]
    S = cfg.n_sink + cfg.window
    vdesc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
    ddesc = spire.draft_desc(drafts[0].q, drafts[0].kv)
    ws_v = torch.empty(spire.spire_verify_workspace_bytes(vdesc, k), dtype=torch.uint8, device=dev)
    ws_d = torch.empty(spire.spire_draft_workspace_bytes(ddesc, cfg.n_sink, cfg.window),
                       dtype=torch.uint8, device=dev)
    out_v = torch.empty(vi.q.shape, dtype=torch.float32, device=dev)
    out_d = [torch.empty(d.q.shape, dtype=torch.float32, device=dev) for d in drafts]
    sptr = stream.cuda_stream

    def call_verify(q=vi.q, ctx=vi.ctx_lens, bt=vi.block_table, out=out_v, s_handle=None):
        st = spire.spire_verify_attention(q, vi.k_cache, vi.v_cache, bt, ctx, k, vdesc, out,
                                          ws_v, ws_v.numel(), s_handle or sptr)
        if st:
            raise spire.SpireError(st, "spire_verify_attention")

    def call_draft(j, q=None, ctx=None, out=None, s_handle=None):
        d = drafts[j]
        st = spire.spire_draft_sparse_attention(q if q is not None else d.q, d.kv,
                                                ctx if ctx is not None else d.ctx_lens,
                                                cfg.n_sink, cfg.window, ddesc,
                                                out if out is not None else out_d[j], ws_d,
                                                ws_d.numel(), s_handle or sptr)
        if st:
            raise spire.SpireError(st, "spire_draft_sparse_attention")

    flush = L2Flush(dev)

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    # ---- device-resident timing: per-step and per-call CUDA events
    for _ in range(args.warmup):
        call_verify()
        for j in range(k):
            call_draft(j)
    torch.cuda.synchronize(dev)
    err = spire.spire_get_device_error(ws_v, stream)
    if err:
        raise RuntimeError("device error word %d after warm-up" % err)

    # ---- per-call detail (eager launches): verify and draft times, roofline
    n_detail = max(1, min(args.steps, 200))
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(k + 2)] for _ in range(n_detail)]
    barrier()
    for s in range(n_detail):
        flush(s & 0xff)          # L2 flush between steps, outside the events
        e = ev[s]
        e[0].record(stream)
        call_verify()
        e[1].record(stream)
        for j in range(k):
            call_draft(j)
            e[2 + j].record(stream)
    barrier()
    eager_ms = statistics.mean(e[0].elapsed_time(e[-1]) for e in ev)
    # the verify call after a write-only flush (L2 left full of dirty lines), for comparison
    v_ms_dirty = event_ms(call_verify, n_detail, flush, stream, write_only=True)
    v_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in ev)
    d_ms = statistics.mean(sum(e[1 + j].elapsed_time(e[2 + j]) for j in range(k)) for e in ev)

    # ---- plain decoding on the same cache (verify with k = 0 at length L - k): t_target
    q0 = vi.q[:, :1].contiguous()
    ctx0 = (vi.ctx_lens - k).contiguous()
    out0 = torch.empty(q0.shape, dtype=torch.float32, device=dev)
    ws0 = torch.empty(spire.spire_verify_workspace_bytes(vdesc, 0), dtype=torch.uint8, device=dev)

    def call_decode():
        st = spire.spire_verify_attention(q0, vi.k_cache, vi.v_cache, vi.block_table, ctx0, 0,
                                          vdesc, out0, ws0, ws0.numel(), sptr)
        if st:
            raise spire.SpireError(st, "spire_verify_attention (k = 0)")

    for _ in range(args.warmup):
        call_decode()
    dec_ev = []
    for s in range(n_detail):
        flush(s & 0xff)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call_decode()
        b.record(stream)
        dec_ev.append((a, b))
    barrier()
    dec_ms = statistics.mean(a.elapsed_time(b) for a, b in dec_ev)

    # ---- the round as one CUDA graph (verify + k draft steps), replayed per step
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream(dev)
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        call_verify(s_handle=cap.cuda_stream)
        for j in range(k):
            call_draft(j, s_handle=cap.cuda_stream)
        torch.cuda.synchronize(dev)
        with torch.cuda.graph(graph, stream=cap):
            call_verify(s_handle=cap.cuda_stream)
            for j in range(k):
                call_draft(j, s_handle=cap.cuda_stream)
    stream.wait_stream(cap)
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize(dev)

    gev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    sampler = ClockSampler(dev.index if dev.index is not None else 0)
    sampler.start()
    time.sleep(0.6)
    barrier()
    t0 = time.time()
    for s in range(args.steps):
        flush(s & 0xff)          # L2 flush between steps, outside the events
        gev[s][0].record(stream)
        graph.replay()
        gev[s][1].record(stream)
    barrier()
    t1 = time.time()
    clocks = sampler.stop(t0, t1)
    ms = statistics.mean(e[0].elapsed_time(e[1]) for e in gev)
    ms, eager_ms, v_ms, d_ms, dec_ms, v_ms_dirty = reduce_max(
        [ms, eager_ms, v_ms, d_ms, dec_ms, v_ms_dirty], dist, dev)
    del graph

    B = int(L.size)
    tokens = B * (k + 1)
    value = job_value(tokens, world, ms)
    vb = verify_bytes(L, k, Hq, Hkv, D)
    db = sum(draft_bytes(wl.draft_ctx_for_step(L, k, j), S, Hq, Hkv, D) for j in range(k))
    hbm_peak, peak_kind = peaks()
    v_gbs = vb / (v_ms * 1e-3) / 1e9
    d_gbs = db / (d_ms * 1e-3) / 1e9

    # ---- end to end through the C ABI with host buffers
    pin = lambda t: t.detach().cpu().pin_memory()
    h_q, h_ctx, h_bt = pin(vi.q), pin(vi.ctx_lens), pin(vi.block_table)
    h_dq = [pin(d.q) for d in drafts]
    h_dctx = [pin(d.ctx_lens) for d in drafts]
    h_out = torch.empty(out_v.shape, dtype=torch.float32).pin_memory()
    h_dout = [torch.empty(o.shape, dtype=torch.float32).pin_memory() for o in out_d]
    d_q, d_ctx, d_bt = torch.empty_like(vi.q), torch.empty_like(vi.ctx_lens), torch.empty_like(vi.block_table)
    d_dq = [torch.empty_like(d.q) for d in drafts]
    d_dctx = [torch.empty_like(d.ctx_lens) for d in drafts]
    h2d = (h_q.numel() * 2 + h_ctx.numel() * 4 + h_bt.numel() * 4 +
           sum(x.numel() * 2 for x in h_dq) + sum(x.numel() * 4 for x in h_dctx))
    d2h = h_out.numel() * 4 + sum(x.numel() * 4 for x in h_dout)

    # Within a step the uploads run on their own stream ahead of the kernels
    # that need them, and every kernel writes its result straight into pinned
    # host memory (zero-copy over the host link, no separate download); the
    # step ends when the last call is done, nothing crosses a step.
    up = torch.cuda.Stream(device=dev)
    ev = lambda: torch.cuda.Event()

    def e2e_step():
        t0, ins = ev(), [ev() for _ in range(k + 1)]
        t0.record(stream)
        up.wait_event(t0)
        with torch.cuda.stream(up):
            d_q.copy_(h_q, non_blocking=True)
            d_ctx.copy_(h_ctx, non_blocking=True)
            d_bt.copy_(h_bt, non_blocking=True)
            ins[0].record(up)
            for j in range(k):
                d_dq[j].copy_(h_dq[j], non_blocking=True)
                d_dctx[j].copy_(h_dctx[j], non_blocking=True)
                ins[j + 1].record(up)
        stream.wait_event(ins[0])
        call_verify(q=d_q, ctx=d_ctx, bt=d_bt, out=h_out)
        for j in range(k):
            stream.wait_event(ins[j + 1])
            call_draft(j, q=d_dq[j], ctx=d_dctx[j], out=h_dout[j])

    for _ in range(max(3, args.warmup)):
        e2e_step()
    torch.cuda.synchronize(dev)
    if not (torch.equal(h_out, out_v.cpu()) and
            all(torch.equal(h, d.cpu()) for h, d in zip(h_dout, out_d))):
        raise RuntimeError("end-to-end results differ from the device-timed ones")
    e2e_steps = max(1, min(args.steps, 200))
    e2e_ms = []
    for s in range(e2e_steps):
        flush(s & 0xff)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        e2e_step()
        b.record(stream)
        b.synchronize()          # the step's result is on the host
        e2e_ms.append(a.elapsed_time(b))
    e2e_val = job_value(tokens, world, reduce_max([statistics.mean(e2e_ms)], dist, dev)[0])

    # ---- load balance: per-SM busy time of one verify and one draft call
    flush(1)
    call_verify()
    bal_v = cta_balance(spire.spire_get_cta_times(ws_v, ws_v.numel()))
    flush(2)
    call_draft(0)
    bal_d = cta_balance(spire.spire_get_cta_times(ws_d, ws_d.numel()))

    # ---- draft-step pipeline: a draft with n_dl = 2 layers (3 activations mixed,
    # d_model = Hq * D); each step attends on every layer's cache, then appends
    # the new feedback-memory entry to every cache (spire_feedback_append)
    n_dl, n_act, d_model = 2, 3, Hq * D
    t0s = wl.draft_ctx_for_step(L, k, 0)
    ai = wl.make_append(t0s, n_act, n_dl, d_model, Hkv, D, cfg.n_sink, cfg.window,
                        seed=cfg.seed + 101, device=dev)
    adesc = spire.make_append_desc(B, n_act, n_dl, d_model, Hkv, D, cfg.n_sink, cfg.window,
                                   10000.0)
    ws_a = torch.empty(spire.spire_feedback_append_workspace_bytes(adesc), dtype=torch.uint8,
                       device=dev)
    out_l = [torch.empty(d.q.shape, dtype=torch.float32, device=dev) for d in drafts]

    def call_append(j, s_handle=None):
        st = spire.spire_feedback_append(ai.x, ai.mix_w, ai.w_kv, drafts[j].ctx_lens, adesc,
                                         ai.kv, ws_a, ws_a.numel(), s_handle or sptr)
        if st:
            raise spire.SpireError(st, "spire_feedback_append")

    def draft_round(s_handle=None):
        for j in range(k):
            for li in range(n_dl):
                st = spire.spire_draft_sparse_attention(
                    drafts[j].q, ai.kv[li], drafts[j].ctx_lens, cfg.n_sink, cfg.window, ddesc,
                    out_l[j], ws_d, ws_d.numel(), s_handle or sptr)
                if st:
                    raise spire.SpireError(st, "spire_draft_sparse_attention")
            call_append(j, s_handle)

    for _ in range(max(3, args.warmup)):
        call_append(0)
    torch.cuda.synchronize(dev)
    if spire.spire_get_device_error(ws_a, stream):
        raise RuntimeError("device error word set by spire_feedback_append")
    a_steps = max(1, min(args.steps, 200))
    a_ev = []
    for s in range(a_steps):
        flush(s & 0xff)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call_append(s % k)
        b.record(stream)
        a_ev.append((a, b))
    torch.cuda.synchronize(dev)
    app_ms = statistics.mean(a.elapsed_time(b) for a, b in a_ev)
    pgraph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(cap):
        draft_round(cap.cuda_stream)
        torch.cuda.synchronize(dev)
        with torch.cuda.graph(pgraph, stream=cap):
            draft_round(cap.cuda_stream)
    stream.wait_stream(cap)
    for _ in range(max(3, args.warmup)):
        pgraph.replay()
    torch.cuda.synchronize(dev)
    p_ev = []
    for s in range(a_steps):
        flush(s & 0xff)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        pgraph.replay()
        b.record(stream)
        p_ev.append((a, b))
    torch.cuda.synchronize(dev)
    pipe_ms = statistics.mean(a.elapsed_time(b) for a, b in p_ev)
    del pgraph
    app_ms, pipe_ms = reduce_max([app_ms, pipe_ms], dist, dev)
    ab = append_bytes(B, n_act, n_dl, d_model, Hkv, D)
    del ai, ws_a

    # ---- token verification of the round (modified rejection sampling), a
    # Llama 3 sized vocabulary as the stand-in (the paper extrapolates to it)
    V_tok = 128256
    ti = wl.make_tokens(B, k, V_tok, seed=cfg.seed + 202, device=dev)
    ws_t = torch.empty(spire.spire_verify_tokens_workspace_bytes(B, k, V_tok), dtype=torch.uint8,
                       device=dev)
    tok_out = torch.empty((B, k + 1), dtype=torch.int32, device=dev)
    tok_acc = torch.empty((B,), dtype=torch.int32, device=dev)

    def call_tokens():
        st = spire.spire_verify_tokens(ti.p, ti.q, ti.x, ti.u, ti.e, B, k, V_tok, tok_out,
                                       tok_acc, ws_t, ws_t.numel(), sptr)
        if st:
            raise spire.SpireError(st, "spire_verify_tokens")

    for _ in range(max(3, args.warmup)):
        call_tokens()
    torch.cuda.synchronize(dev)
    t_ev = []
    for s in range(a_steps):
        flush(s & 0xff)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call_tokens()
        b.record(stream)
        t_ev.append((a, b))
    torch.cuda.synchronize(dev)
    tok_ms = reduce_max([statistics.mean(a.elapsed_time(b) for a, b in t_ev)], dist, dev)[0]
    n_acc_h = tok_acc.cpu().numpy()
    tb = tokens_bytes(n_acc_h, k, V_tok)
    del ti

    # ---- the MagicDec baseline's draft step: sink 1 + window 64 over the target's
    # own paged cache (Section 4), positions inside the reduced cache
    md_sink, md_win = 1, 64
    md_ws = torch.empty(spire.spire_magicdec_workspace_bytes(vdesc, md_sink, md_win),
                        dtype=torch.uint8, device=dev)
    md_out = torch.empty(drafts[0].q.shape, dtype=torch.float32, device=dev)

    def call_magicdec(j):
        st = spire.spire_magicdec_attention(drafts[j].q, vi.k_cache, vi.v_cache, vi.block_table,
                                            drafts[j].ctx_lens, md_sink, md_win, 10000.0, vdesc,
                                            md_out, md_ws, md_ws.numel(), sptr)
        if st:
            raise spire.SpireError(st, "spire_magicdec_attention")

    for _ in range(max(3, args.warmup)):
        call_magicdec(0)
    torch.cuda.synchronize(dev)
    md_ev = []
    for s in range(a_steps):
        flush(s & 0xff)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call_magicdec(s % k)
        b.record(stream)
        md_ev.append((a, b))
    torch.cuda.synchronize(dev)
    md_ms = reduce_max([statistics.mean(a.elapsed_time(b) for a, b in md_ev)], dist, dev)[0]
    md_bytes = statistics.mean(draft_bytes(wl.draft_ctx_for_step(L, k, j), md_sink + md_win, Hq,
                                           Hkv, D) for j in range(k))
    del md_ws

    # ---- draft sweep: B = 512, t log-uniform in [4096, 262144], sink 16, windows 256 /
    # 1024 / 4096 (bounded caches of 0.57 / 2.2 / 8.6 GB); k steps on one cache per
    # window (step j sees t + j entries); draft tokens/s = B k / sum of the step times
    sw_cfg = wl.CONFIGS["draft_sweep"]
    sw_L = wl.sample_ctx_lens(sw_cfg)
    sw_k, sw_B = sw_cfg.k, int(sw_L.size)
    sweep = []
    for w in sw_cfg.windows:
        sw_S = sw_cfg.n_sink + w
        sdi = wl.make_draft(wl.draft_ctx_for_step(sw_L, sw_k, 0), Hq, Hkv, D, sw_cfg.n_sink, w,
                            seed=sw_cfg.seed + w, device=dev)
        sw_ctx = [torch.from_numpy(wl.draft_ctx_for_step(sw_L, sw_k, j)).to(dev)
                  for j in range(sw_k)]
        sw_desc = spire.draft_desc(sdi.q, sdi.kv)
        sw_ws = torch.empty(spire.spire_draft_workspace_bytes(sw_desc, sw_cfg.n_sink, w),
                            dtype=torch.uint8, device=dev)
        sw_out = torch.empty(sdi.q.shape, dtype=torch.float32, device=dev)

        def call_sweep(j):
            st = spire.spire_draft_sparse_attention(sdi.q, sdi.kv, sw_ctx[j], sw_cfg.n_sink, w,
                                                    sw_desc, sw_out, sw_ws, sw_ws.numel(), sptr)
            if st:
                raise spire.SpireError(st, "spire_draft_sparse_attention")

        for _ in range(max(3, args.warmup)):
            for j in range(sw_k):
                call_sweep(j)
        torch.cuda.synchronize(dev)
        if spire.spire_get_device_error(sw_ws, stream):
            raise RuntimeError("device error word set by the draft sweep")
        sw_ev = []
        for s in range(max(1, min(args.steps, 50))):
            for j in range(sw_k):
                flush((s + j) & 0xff)     # each step streams its cache from HBM
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                call_sweep(j)
                b.record(stream)
                sw_ev.append((a, b))
        torch.cuda.synchronize(dev)
        round_ms = reduce_max([statistics.mean(a.elapsed_time(b) for a, b in sw_ev) * sw_k],
                              dist, dev)[0]
        sw_bytes = sum(draft_bytes(wl.draft_ctx_for_step(sw_L, sw_k, j), sw_S, Hq, Hkv, D)
                       for j in range(sw_k))
        sweep.append({"window": w, "n_sink": sw_cfg.n_sink, "cache_gb": sdi.kv.numel() * 2 / 1e9,
                      "ms_per_round": round_ms,
                      "draft_tokens_per_s": world * sw_B * sw_k / (round_ms * 1e-3),
                      "gbs": sw_bytes / (round_ms * 1e-3) / 1e9,
                      "frac": sw_bytes / (round_ms * 1e-3) / 1e9 / hbm_peak})
        del sdi, sw_ctx, sw_ws, sw_out
        torch.cuda.empty_cache()

    # ---- verification on the other two verify workloads, the ragged serving mix
    # (B = 64, k = 4, L log-uniform in [1024, 131072]) and the large batch with
    # deeper speculation (B = 256, k = 8, 64/8 heads), timed as the headline call
    verify_configs = {}
    for name in ("ragged", "big"):
        if name == cfg.name:
            continue
        verify_configs[name] = verify_config_entry(spire, name, dev, stream, flush, args,
                                                   hbm_peak, dist=dist)

    # ---- the floor of a single launch that reads a call's algorithmic bytes:
    # spire_stream_read streams that many bytes with the attention kernels' copy
    # machinery and computes nothing (same flush, same events)
    floor_buf = torch.empty(int(max(vb, db // k, ab, tb, md_bytes)) + 16, dtype=torch.uint8,
                            device=dev)

    def floor_us(nbytes):
        nb = int(nbytes) // 16 * 16

        def call():
            st = spire.spire_stream_read(floor_buf, nb, sptr)
            if st:
                raise spire.SpireError(st, "spire_stream_read")

        for _ in range(max(3, args.warmup)):
            call()
        return reduce_max([event_ms(call, max(1, min(args.steps, 100)), flush, stream)], dist,
                          dev)[0] * 1e3

    floors = {"verify": floor_us(vb), "draft_step": floor_us(db // k), "append": floor_us(ab),
              "tokens": floor_us(tb), "magicdec": floor_us(md_bytes)}
    del floor_buf

    if rank != 0:
        if dist is not None:
            dist.barrier()
            dist.destroy_process_group()
        return 0

    cpu = None
    if not args.no_cpu_baseline and world == 1:
        threads = os.cpu_count() or 1
        n_seq = oracle_sample_size(cfg, target_s=15.0, threads=threads)
        dt, tok = run_oracle_sample(cfg, n_seq, threads)
        cpu = {"value": tok / dt, "unit": "tokens/s", "cores": threads, "kind": "oracle",
               "sample": "first %d of %d sequences, verify + %d draft steps, fp64 C oracle, "
                         "%.1f s" % (n_seq, cfg.batch, k, dt)}
        # the same oracle on one core, on a smaller sample
        n1 = oracle_sample_size(cfg, target_s=5.0, threads=1)
        dt1, tok1 = run_oracle_sample(cfg, n1, 1)
        cpu["single_core"] = {"value": tok1 / dt1, "unit": "tokens/s", "cores": 1,
                              "sample": "first %d sequences, %.1f s" % (n1, dt1)}

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": dict(workload_config(cfg, L),
                       l2="flushed between steps (a 256 MB write, then a read of that buffer: "
                          "L2 holds none of the inputs and no dirty lines); verify KV %.2f GB "
                          "> L2" % (vb / 1e9)),
        "roofline": {"kernel": "spire_verify_attention: attn_tc_kernel, launched with "
                               "programmatic dependent launch behind the one-CTA merge-counter "
                               "reset; CUDA events around the call",
                     "bound": "hbm", "achieved": v_gbs, "peak": hbm_peak, "unit": "GB/s",
                     "frac": v_gbs / hbm_peak, "peak_kind": peak_kind,
                     "frac_of_8TBs": v_gbs / HBM_NOMINAL_GBS,
                     "algorithmic_bytes": vb, "traffic": dram_traffic("verify:%s" % cfg.name)},
        "detail": {"round": "one CUDA graph per step (verify + %d draft calls); "
                             "eager launches: %.4f ms per step" % (k, eager_ms),
                   "verify_ms": v_ms, "draft_ms_total": d_ms, "verify_gbs": v_gbs,
                   "verify_ms_after_write_only_flush": v_ms_dirty,
                   "stream_floor": {
                       "what": "spire_stream_read: one launch that reads the call's algorithmic "
                               "bytes with the same bulk-copy ring and computes nothing, timed "
                               "like the calls (us); floor_over_us = floor / the call's time",
                       "verify_us": floors["verify"],
                       "verify_floor_over_us": floors["verify"] / (v_ms * 1e3),
                       "draft_step_us": floors["draft_step"],
                       "draft_step_floor_over_us": floors["draft_step"] / (d_ms / k * 1e3)},
                   "draft_gbs": d_gbs, "draft_bytes_per_round": db,
                   "verify_tokens_per_s": world * tokens / (v_ms * 1e-3),
                   "draft_tokens_per_s": world * B * k / (d_ms * 1e-3),
                   "verify_tflops": verify_flops(L, k, Hq, D) / (v_ms * 1e-3) / 1e12,
                   "tau_weighted_tokens_per_s_context": world * B * SPIRE_TAU_K4_L512 / (ms * 1e-3),
                   "feedback_append": {
                       "shape": "%d draft layers, %d activations, d_model %d, %d KV heads x %d, "
                                "keys rotated (theta 1e4)" % (n_dl, n_act, d_model, Hkv, D),
                       "us": app_ms * 1e3, "algorithmic_bytes": ab,
                       "gbs": ab / (app_ms * 1e-3) / 1e9,
                       "frac": ab / (app_ms * 1e-3) / 1e9 / hbm_peak, "bound": "hbm",
                       "floor_us": floors["append"],
                       "floor_over_us": floors["append"] / (app_ms * 1e3),
                       "launches": 1},
                   "perf_model": perf_model_detail(L, k, Hq, Hkv, D, S, v_ms, d_ms, dec_ms),
                   "load_balance": {
                       "what": "per-CTA %globaltimer record (spire_get_cta_times) of one verify "
                               "call and one draft call after an L2 flush: busy = first tile "
                               "to last merge, one CTA per SM",
                       "verify": bal_v, "draft_step": bal_d},
                   "magicdec_draft_step": {
                       "what": "spire_magicdec_attention: sink %d + window %d over the target's "
                               "paged cache, keys and query re-turned to cache positions "
                               "(one fused launch for up to 8 query heads per KV head)"
                               % (md_sink, md_win),
                       "us": md_ms * 1e3, "algorithmic_bytes": md_bytes,
                       "gbs": md_bytes / (md_ms * 1e-3) / 1e9,
                       "floor_us": floors["magicdec"],
                       "floor_over_us": floors["magicdec"] / (md_ms * 1e3),
                       "spire_draft_step_us": d_ms / k * 1e3},
                   "verify_tokens": {
                       "shape": "B=%d, k=%d, vocabulary %d (fp32 distributions)" % (B, k, V_tok),
                       "us": tok_ms * 1e3, "algorithmic_bytes": tb,
                       "gbs": tb / (tok_ms * 1e-3) / 1e9,
                       "frac": tb / (tok_ms * 1e-3) / 1e9 / hbm_peak, "bound": "hbm",
                       "floor_us": floors["tokens"],
                       "floor_over_us": floors["tokens"] / (tok_ms * 1e3),
                       "mean_accepted": float(n_acc_h.mean()), "launches": 3},
                   "verify_configs": verify_configs,
                   "draft_sweep": {
                       "what": "B=%d, t log-uniform [4096, 262144], %d draft steps per round on "
                               "one bounded cache per window, each step's cache streamed from "
                               "HBM (L2 flushed before it)" % (sw_B, sw_k),
                       "windows": sweep},
                   "draft_step_pipeline": {
                       "what": "one CUDA graph per round: %d steps x (%d layer attention calls + "
                               "one feedback append)" % (k, n_dl),
                       "ms_per_round": pipe_ms,
                       "draft_tokens_per_s": world * B * k / (pipe_ms * 1e-3)}},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_val, "unit": "tokens/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h)},
        # each call: the merge-counter reset kernel + one attention kernel
        "gpu_launches": 2 * (k + 1) * args.steps,
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def profile_call(args, cfg):
    """One library call, for profiler captures: allocate only that call's inputs
    (the workload, cut to --max-seqs sequences when given), make --warmup calls
    and then --calls more, each after the 256 MB L2 flush, and exit.  Prints a
    one-line summary, never a benchmark line (times taken under a profiler are
    not measurements)."""
    import torch

    import paper_2504_06419_gb300 as spire

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream
    k, Hq, Hkv, D = cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
    L = wl.sample_ctx_lens(cfg)
    if args.max_seqs:
        L = L[:args.max_seqs]
    B = int(L.size)
    what = args.profile_call
    ws = None
    if what in ("verify", "decode", "magicdec"):
        vi = wl.make_verify(L, k, Hq, Hkv, D, seed=cfg.seed, device=dev, shuffle=cfg.paged_shuffle)
        desc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
        if what == "magicdec":
            t = torch.from_numpy(wl.draft_ctx_for_step(L, k, 0)).to(dev)
            q = vi.q[:, 0].contiguous()
            out = torch.empty(q.shape, dtype=torch.float32, device=dev)
            ws = torch.empty(spire.spire_magicdec_workspace_bytes(desc, 1, 64), dtype=torch.uint8,
                             device=dev)

            def call():
                return spire.spire_magicdec_attention(q, vi.k_cache, vi.v_cache, vi.block_table, t,
                                                      1, 64, 10000.0, desc, out, ws, ws.numel(),
                                                      sptr)
        else:
            kk = k if what == "verify" else 0
            q = vi.q if kk == k else vi.q[:, :1].contiguous()
            ctx = vi.ctx_lens if kk == k else (vi.ctx_lens - k).contiguous()
            out = torch.empty(q.shape, dtype=torch.float32, device=dev)
            ws = torch.empty(spire.spire_verify_workspace_bytes(desc, kk), dtype=torch.uint8,
                             device=dev)

            def call():
                return spire.spire_verify_attention(q, vi.k_cache, vi.v_cache, vi.block_table, ctx,
                                                    kk, desc, out, ws, ws.numel(), sptr)
    elif what == "draft":
        window = args.window or cfg.window
        di = wl.make_draft(wl.draft_ctx_for_step(L, k, 0), Hq, Hkv, D, cfg.n_sink, window,
                           seed=cfg.seed + 17, device=dev)
        desc = spire.draft_desc(di.q, di.kv)
        ws = torch.empty(spire.spire_draft_workspace_bytes(desc, cfg.n_sink, window),
                         dtype=torch.uint8, device=dev)
        out = torch.empty(di.q.shape, dtype=torch.float32, device=dev)

        def call():
            return spire.spire_draft_sparse_attention(di.q, di.kv, di.ctx_lens, cfg.n_sink,
                                                      window, desc, out, ws, ws.numel(), sptr)
    elif what == "append":
        n_dl, n_act, d_model = 2, 3, Hq * D
        ai = wl.make_append(wl.draft_ctx_for_step(L, k, 0), n_act, n_dl, d_model, Hkv, D,
                            cfg.n_sink, cfg.window, seed=cfg.seed + 101, device=dev)
        adesc = spire.make_append_desc(B, n_act, n_dl, d_model, Hkv, D, cfg.n_sink, cfg.window,
                                       10000.0)
        ws = torch.empty(spire.spire_feedback_append_workspace_bytes(adesc), dtype=torch.uint8,
                         device=dev)

        def call():
            return spire.spire_feedback_append(ai.x, ai.mix_w, ai.w_kv, ai.pos, adesc, ai.kv, ws,
                                               ws.numel(), sptr)
    elif what == "tokens":
        V_tok = 128256
        ti = wl.make_tokens(B, k, V_tok, seed=cfg.seed + 202, device=dev)
        ws = torch.empty(spire.spire_verify_tokens_workspace_bytes(B, k, V_tok), dtype=torch.uint8,
                         device=dev)
        tok_out = torch.empty((B, k + 1), dtype=torch.int32, device=dev)
        tok_acc = torch.empty((B,), dtype=torch.int32, device=dev)

        def call():
            return spire.spire_verify_tokens(ti.p, ti.q, ti.x, ti.u, ti.e, B, k, V_tok, tok_out,
                                             tok_acc, ws, ws.numel(), sptr)
    else:
        raise ValueError(what)
    flush = L2Flush(dev)
    n = args.warmup + args.calls
    for s in range(n):
        flush(s & 0xff)
        st = call()
        if st:
            raise spire.SpireError(st, what)
    torch.cuda.synchronize(dev)
    err = spire.spire_get_device_error(ws, stream) if what != "tokens" else 0
    print("profile-call %s on %s (%d sequences): %d calls (%d warm-up), device error word %d"
          % (what, cfg.name, B, n, args.warmup, err), flush=True)
    return 1 if err else 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="uniform8k", choices=sorted(wl.CONFIGS))
    ap.add_argument("--impl", default="spire", choices=["spire", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--max-seqs", type=int, default=0,
                    help="use only the first N sequences of the workload (small profiling "
                         "captures; not a benchmark configuration)")
    ap.add_argument("--profile-call", default=None,
                    choices=["verify", "decode", "draft", "append", "tokens", "magicdec"],
                    help="make only this library call (--warmup + --calls times, each after "
                         "the L2 flush) and exit: small profiler captures, never a benchmark")
    ap.add_argument("--calls", type=int, default=2,
                    help="calls after the warm-up in --profile-call mode")
    ap.add_argument("--window", type=int, default=0,
                    help="draft window for --profile-call draft (default: the workload's)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    cfg = wl.CONFIGS[args.config]
    if args.profile_call:
        return profile_call(args, cfg)
    if args.impl == "reference":
        return reference_arm(args, cfg)
    return spire_arm(args, cfg)


if __name__ == "__main__":
    sys.exit(main())
