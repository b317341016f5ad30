#!/usr/bin/env python
"""Benchmark of the prefix-cached paged-attention path on GB300.

One step = one pass of the hot path over one batch: the new tokens' K/V are
scattered into the paged pool (kv_cache_write), then the batch's attention runs
(paged_attn_decode for decode requests, paged_attn_prefill for suffix or chunk
prefills).  The headline workload is the Llama-3-8B-shaped decode batch
(64 requests sharing a 4096-token policy prefix); its metric is HBM GB/s on
algorithmic bytes (every distinct K/V row read once, shared prefix rows once,
plus the step's Q, O and new-token K/V traffic).  Other workloads are reported
under "workloads" (prefill in TFLOP/s on visible query-key pairs).

Timing: per-step CUDA events on the launching stream, L2 flushed (256 MiB
write) before every step outside the events, W warm-up steps, max over ranks.
Per-kernel times come from a second pass of K steps with the library's own
event tracing (pkv_trace_*); the headline pass runs without it, because an
event between two kernels keeps the second from launching early.

e2e: the headline step driven from pinned host memory through
paged_attn_decode_step (one H2D copy of the packed inputs, cache write,
decode, D2H copy of the output), alternate steps on two streams so that one
step's copies overlap the other's kernels, like a serving loop; host wall time
per step.

--impl reference times the fp64 CPU oracle (the only reference this path has)
on the host cores, one decode request per step.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

HEADLINE = "l8b_decode"
WORKLOAD_DESC = {
    "tiny": "tiny: 8q/2kv heads, d64, 4 requests sharing a 256-token prefix, suffix prefill",
    "l8b_decode": "l8b_decode: Llama-3-8B-shaped decode, 32q/8kv heads, d128, 64 requests "
                  "sharing a 4096-token prefix, suffix U[256,1024], generated U[0,128]",
    "l8b_prefill": "l8b_prefill: Llama-3-8B-shaped suffix prefill, 32q/8kv, d128, 32 requests, "
                   "cached 4096-token prefix, suffix U[512,1024]",
    "qwen_mixed": "qwen_mixed: Qwen2.5-7B-shaped, 28q/4kv, d128, 256 decode requests over "
                  "2048/4096/6144-token prefixes + 8 chunked prefills of 512",
    "l70b_decode": "l70b_decode: Llama-3-70B-shaped decode, 64q/8kv, d128, 512 requests sharing "
                   "a 6144-token prefix, suffix log-U[64,2048], generated U[0,128]",
}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


# ---------------------------------------------------------------------------
# algorithmic work (counted from the workload's lengths, not from the kernels)

def kv_row_bytes(w):
    return 2 * w.num_kv_heads * w.head_dim * 2      # K and V of one token, all kv heads


def decode_bytes(w, req):
    """Distinct K/V rows of the decode requests (shared prefix once) + Q + O."""
    rows = 0
    groups = set()
    for r in range(req.start, req.stop):
        g = int(w.group_of_req[r])
        if g >= 0:
            groups.add(g)
        rows += int(w.context_lens[r]) - w.prefix_len_of(r)
    rows += sum(w.prefix_lens[g] for g in groups)
    nq = req.stop - req.start
    return rows * kv_row_bytes(w) + 2 * nq * w.num_q_heads * w.head_dim * 2


def decode_logical_bytes(w, req):
    """Every decode request's K/V rows (a shared prefix counted once per
    request, as a cache without sharing would read it) + Q + O."""
    rows = sum(int(w.context_lens[r]) for r in range(req.start, req.stop))
    nq = req.stop - req.start
    return rows * kv_row_bytes(w) + 2 * nq * w.num_q_heads * w.head_dim * 2


def write_bytes(w, ntok):
    return 2 * ntok * kv_row_bytes(w)                # read new K/V + write into the pool


def prefill_flops(w, req):
    """4 * d * Hq * visible (query, key) pairs; masked pairs are not counted."""
    pairs = 0
    for r in range(req.start, req.stop):
        S, c = int(w.new_lens[r]), int(w.cached_lens[r])
        pairs += S * c + S * (S + 1) // 2
    return 4 * w.head_dim * w.num_q_heads * pairs


# ---------------------------------------------------------------------------
# clocks during the timed region

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.samples = []   # (t, sm, smmax, reasons)
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm, smmax = float(parts[1]), float(parts[2])
            except ValueError:
                continue
            reasons = [n for n, v in zip(names, parts[5:9]) if v.lower().startswith("active")]
            self.samples.append((time.time(), sm, smmax, reasons))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0, t1):
        inside = [s for s in self.samples if t0 <= s[0] <= t1]
        use = inside if inside else self.samples
        if not use:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        reasons = sorted({r for s in use for r in s[3]})
        return {"sm_mhz": statistics.median(s[1] for s in use), "sm_max_mhz": max(s[2] for s in use),
                "reasons": reasons, "samples": len(use),
                "window": "timed region" if inside else "whole run (timed region shorter than the 100 ms sampling)"}


# ---------------------------------------------------------------------------

def dist_setup(n_gpus):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def _reduce_over_ranks(x, world, op):
    """all-reduce one float over the replicas (on the GPU under NCCL, on the
    CPU under gloo)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=op)
    return float(t.item())


def max_over_ranks(x, world):
    if world == 1:
        return x
    import torch.distributed as dist
    return _reduce_over_ranks(x, world, dist.ReduceOp.MAX)


def sum_over_ranks(x, world):
    if world == 1:
        return x
    import torch.distributed as dist
    return _reduce_over_ranks(x, world, dist.ReduceOp.SUM)


def aggregate_replicas(ms_local, step_bytes, e2e_ms_local, world):
    """Whole-job numbers of N independent replicas: the step time is the
    slowest rank's, the bytes are every rank's, so value = sum of bytes / max
    time (weak scaling).  Returns (ms, total_bytes, GB/s, e2e ms, e2e GB/s)."""
    ms = max_over_ranks(ms_local, world)
    total_bytes = sum_over_ranks(step_bytes, world)
    e2e_ms = max_over_ranks(e2e_ms_local, world)
    return (ms, total_bytes, total_bytes / (ms * 1e-3) / 1e9, e2e_ms,
            total_bytes / (e2e_ms * 1e-3) / 1e9)


def ncu_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if the
    kernel source is unchanged since the capture."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p)).get(kernel)
    if not d or d.get("workload") != workload:
        return None
    src = os.path.join(ROOT, d["source"])
    if not os.path.exists(src) or hashlib.sha256(open(src, "rb").read()).hexdigest() != d["source_sha256"]:
        return None
    return d["dram_bytes_per_launch"]


def run_steps(step_fn, flush, steps, stream):
    """Per-step CUDA events around step_fn on `stream`, L2 flush before each
    step (outside the events)."""
    import torch
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(steps)]
    for a, b in evs:
        flush()
        a.record(stream)
        step_fn()
        b.record(stream)
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in evs]


def measure_workload(name, steps, warmup, use_groups=True, e2e_steps=0):
    """Build a workload, time its steps; returns a dict of results."""
    import numpy as np
    import torch

    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300 import pkv
    from paper_2605_11232_gb300.workloads import make_workload

    w = make_workload(name)
    b = B.build_batch(w, poison=False)
    stream = torch.cuda.current_stream()
    dev = b.device
    Rd, Rp = b.dec.stop - b.dec.start, b.pre.stop - b.pre.start
    out_d = torch.empty((Rd, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device=dev)
    rows_p = B.new_token_rows(w, b.pre)
    out_p = torch.empty((rows_p.stop - rows_p.start, w.num_q_heads, w.head_dim),
                        dtype=torch.bfloat16, device=dev)
    groups_ok = use_groups and b.groups is not None
    ws = B.decode_workspace(b, groups_ok) if Rd else None
    flush_buf = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)

    def flush():
        flush_buf.fill_(1)

    # every new token's K/V is stored by the attention kernel that reads it:
    # the prefill subset's by the prefill kernel (paged_attn_prefill_append),
    # the decode subset's by the decode split pass (paged_attn_decode_append)
    fused_bytes = write_bytes(w, w.num_new_tokens - (rows_p.stop - rows_p.start))

    def step():
        if Rp:
            B.run_prefill_append(b, out_p, None)
        if Rd:
            B.run_decode_append(b, out_d, None, ws, groups_ok)

    # check the configuration runs (prefix pass may be unavailable)
    try:
        step()
    except pkv.PkvError as e:
        if groups_ok and e.code == pkv.PKV_ERR_UNSUPPORTED:
            groups_ok = False
            ws = B.decode_workspace(b, False) if Rd else None
            step()
        else:
            raise
    torch.cuda.synchronize()
    # timed pass: no per-kernel events, so consecutive kernels can overlap
    # their launches (programmatic dependent launch) as in production
    for _ in range(warmup):
        flush()
        step()
    torch.cuda.synchronize()
    step_ms = run_steps(step, flush, steps, stream)
    # the same steps back to back with no flush (warm L2), reported beside
    warm_ms = run_steps(step, lambda: None, steps, stream)
    # a mixed step's decode subset alone, untraced and flushed like the step:
    # the rate of the decode bytes over the time its kernels take together
    # (they overlap one another, which per-kernel events would prevent)
    dec_ms = None
    if Rp and Rd:
        dec_ms = run_steps(lambda: B.run_decode_append(b, out_d, None, ws, groups_ok), flush, steps, stream)
    # traced pass (per-kernel CUDA events from the library) for the roofline
    pkv.pkv_trace_enable(b.pool, True)
    for _ in range(min(warmup, 3)):
        flush()
        step()
    torch.cuda.synchronize()
    pkv.pkv_trace_read(b.pool)            # drop the warm-up launches
    run_steps(step, flush, steps, stream)
    trace = pkv.pkv_trace_read(b.pool)
    pkv.pkv_trace_enable(b.pool, False)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    # algorithmic bytes each decode kernel is responsible for
    kb = {}
    if Rd:
        rows_priv = sum(int(w.context_lens[r]) - w.prefix_len_of(r) for r in range(b.dec.start, b.dec.stop))
        used = {int(w.group_of_req[r]) for r in range(b.dec.start, b.dec.stop)} - {-1}
        rows_pre = sum(w.prefix_lens[gi] for gi in used)
        qo = Rd * w.num_q_heads * w.head_dim * 2
        # private K/V rows read, Q, and the query tokens' own K/V read + stored
        kb["decode_split"] = (rows_priv + (0 if groups_ok else rows_pre)) * kv_row_bytes(w) + qo + fused_bytes
        kb["decode_prefix"] = rows_pre * kv_row_bytes(w) + qo if groups_ok else 0
        kb["decode_combine"] = qo
    res = dict(name=name, w=w, step_ms=step_ms, warm_ms=warm_ms, dec_ms=dec_ms, trace=trace, groups=groups_ok,
               kernel_bytes=kb,
               dec_bytes=decode_bytes(w, b.dec) if Rd else 0,
               dec_logical=decode_logical_bytes(w, b.dec) if Rd else 0,
               wr_bytes=write_bytes(w, w.num_new_tokens),
               pre_flops=prefill_flops(w, b.pre) if Rp else 0, Rd=Rd, Rp=Rp)

    if e2e_steps and Rd and not Rp:
        # End to end through the C ABI from host buffers, as a serving loop
        # runs it: one paged_attn_decode_step call per step copies the step's
        # packed inputs (q, new K/V, context lengths) to the device, decodes
        # with the new tokens stored by the decode kernels
        # (PKV_STEP_FUSED_WRITE) and copies the output back to pinned memory.
        # Alternate steps go to two streams, each with its own device input
        # and output buffers; a step's kernels wait for the previous step's
        # (the steps share one workspace), so its copies overlap the other
        # stream's kernels.  A pinned buffer is refilled
        # only after the step that last used it has completed.
        layout, host, _ = B.step_buffers(b, copies=2, fused=True)
        dev = [torch.empty(layout.bytes, dtype=torch.uint8, device=b.device) for _ in range(2)]
        for k in range(2):
            dev[k].copy_(host[k])
        outs = [torch.empty_like(out_d) for _ in range(2)]
        out_h = [torch.empty(out_d.shape, dtype=out_d.dtype).pin_memory() for _ in range(2)]
        streams = [torch.cuda.Stream() for _ in range(2)]
        done = [torch.cuda.Event() for _ in range(2)]
        steps_k = [pkv.DecodeStep(b.pool, host[k], dev[k], layout, w.num_new_tokens,
                                  b.table[b.dec], w.num_q_heads, w.scale,
                                  b.groups if groups_ok else None, ws, outs[k], None, out_h[k],
                                  None, wait_event=done[1 - k], done_event=done[k],
                                  stream=streams[k]) for k in range(2)]
        torch.cuda.synchronize()
        events = [None, None]
        h2d = layout.bytes
        d2h = out_d.numel() * out_d.element_size()

        def e2e_step(i):
            k = i & 1
            if events[k] is not None:
                events[k].synchronize()   # the step that last used buffer k is done
            steps_k[k]()
            ev = torch.cuda.Event()
            ev.record(streams[k])
            events[k] = ev

        for i in range(max(3, warmup)):
            e2e_step(i)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for i in range(e2e_steps):
            e2e_step(i)
        torch.cuda.synchronize()
        t1 = time.perf_counter()
        assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
        assert torch.equal(out_h[0], out_h[1])   # every step computes the same batch
        res.update(e2e_ms=(t1 - t0) * 1e3 / e2e_steps, h2d=h2d, d2h=d2h)
    b.close()
    del b, flush_buf, ws
    torch.cuda.empty_cache()
    return res


def _timed(step, flush, steps, warmup, stream):
    import torch
    for _ in range(warmup):
        flush()
        step()
    torch.cuda.synchronize()
    return run_steps(step, flush, steps, stream)


def measure_verify(steps, warmup, k=8):
    """Speculative verification of tree-shaped drafts (Sec. 5.3) on the
    Llama-3-8B-shaped decode batch: every request carries k draft tokens in a
    seeded tree (chains, stars and random trees in turn) over its cached
    context (64 requests, shared 4096-token prefix).  A step writes the drafts'
    K/V (kv_cache_write) and verifies them with
    paged_attn_verify_tree_grouped (the shared prefix read once per kv head);
    paged_attn_verify_tree, which reads it once per request, is timed beside
    it.  Reported: TFLOP/s on visible (query, key) pairs, and GB/s on distinct
    K/V bytes (shared prefix once) + Q/O + the write."""
    import numpy as np
    import torch

    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300 import pkv
    from paper_2605_11232_gb300.workloads import make_workload

    w0 = make_workload("l8b_decode", values=False)
    R = w0.num_requests
    cached = [int(c) for c in w0.cached_lens]
    w = make_workload("custom", seed=31, custom=dict(
        Hq=w0.num_q_heads, Hkv=w0.num_kv_heads, d=w0.head_dim, prefix_lens=list(w0.prefix_lens),
        group=[int(x) for x in w0.group_of_req], cached=cached, new=[k] * R, decode=[False] * R))
    rng = np.random.default_rng(31)
    parents = []
    for r in range(R):
        if r % 3 == 0:
            parents += [-1] + list(range(k - 1))
        elif r % 3 == 1:
            parents += [-1] * k
        else:
            parents += [int(rng.integers(-1, i)) if i else -1 for i in range(k)]
    cu = np.arange(0, R * k + 1, k, dtype=np.int32)
    masks_np = pkv.pkv_tree_masks(np.asarray(parents, np.int32), cu)
    b = B.build_batch(w, poison=False)
    masks = torch.from_numpy(masks_np).to(b.device)
    T = R * k
    out = torch.empty((T, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device=b.device)
    vg, keep = B.verify_groups(b)
    ws = B.verify_workspace(b, vg)
    flush_buf = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=b.device)
    flush = lambda: flush_buf.fill_(1)
    stream = torch.cuda.current_stream()

    def step_grouped():
        B.run_write(b)
        B.run_verify_grouped(b, out, None, masks, vg, ws, k)

    def step_plain():
        B.run_write(b)
        pkv.paged_attn_verify_tree(b.pool, b.q, out, None, b.cu_pre, b.context_lens, b.table, k, w.scale, masks)

    def attn_us(step):
        # the verification alone (the drafts' K/V are in the cache by now)
        return 1e3 * statistics.mean(_timed(step, flush, steps, warmup, stream))

    ms = _timed(step_grouped, flush, steps, warmup, stream)
    g_us = attn_us(lambda: B.run_verify_grouped(b, out, None, masks, vg, ws, k))
    ms_plain = _timed(step_plain, flush, steps, warmup, stream)
    p_us = attn_us(lambda: pkv.paged_attn_verify_tree(b.pool, b.q, out, None, b.cu_pre, b.context_lens,
                                                      b.table, k, w.scale, masks))
    # per-kernel times (events around each launch: they keep the passes from overlapping)
    pkv.pkv_trace_enable(b.pool, True)
    _timed(step_grouped, flush, 2, 1, stream)
    pkv.pkv_trace_read(b.pool)
    run_steps(step_grouped, flush, steps, stream)
    trace = pkv.pkv_trace_read(b.pool)
    pkv.pkv_trace_enable(b.pool, False)
    g_kernels = {kk: {"launches": n, "avg_us": 1e3 * t / n} for kk, (n, t) in trace.items()}
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    # visible pairs: each draft sees its cached context and its ancestors (itself included)
    pairs = 0
    for r in range(R):
        for i in range(k):
            pairs += cached[r] + bin(int(masks_np[r * k + i])).count("1")
    flops = 4 * w.head_dim * w.num_q_heads * pairs
    kv_rows = sum(w.prefix_lens) + sum(c - w.prefix_len_of(r) for r, c in enumerate(cached)) + T
    nbytes = kv_rows * kv_row_bytes(w) + 2 * T * w.num_q_heads * w.head_dim * 2 + write_bytes(w, T)
    b.close()
    mean = statistics.mean(ms)
    return {"ms_per_step": mean, "drafts_per_request": k, "requests": R,
            "verify_kernel_us": g_us, "verify_tflops": flops / (g_us * 1e-6) / 1e12,
            "step_hbm_gbs": nbytes / (mean * 1e-3) / 1e9,
            "ungrouped": {"ms_per_step": statistics.mean(ms_plain), "verify_kernel_us": p_us,
                          "verify_tflops": flops / (p_us * 1e-6) / 1e12},
            "kernels": g_kernels,
            "note": "trees: chains, stars and seeded random trees in turn; drafts' K/V written by "
                    "kv_cache_write in the step; verify_kernel_us: the verification call alone"}


def measure_transfer(steps, warmup):
    """KV-block transfer (prefill/decode disaggregation, Sec. 2 / Sec. 7): the
    Llama-3-8B-shaped suffix-prefill batch's blocks (32 requests, shared 4096
    prefix once) gathered from its pool into a staging buffer and scattered
    into another pool's blocks, one GPU.  GB/s on 2 x (read + write) bytes
    of every moved block."""
    import numpy as np
    import torch

    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300 import pkv
    from paper_2605_11232_gb300.workloads import make_workload

    w = make_workload("l8b_prefill")
    b = B.build_batch(w, poison=False)
    B.run_write(b)
    ids = np.unique(np.concatenate([b.table_host[r, :(int(w.context_lens[r]) + 15) // 16]
                                    for r in range(w.num_requests)])).astype(np.int32)
    n = len(ids)
    dk = torch.empty((n,) + tuple(b.k_cache.shape[1:]), dtype=torch.bfloat16, device=b.device)
    dv = torch.empty_like(dk)
    dst = pkv.kv_pool_create(n, w.num_kv_heads, w.head_dim, dk, dv, placement_seed=5)
    dst_ids = torch.from_numpy(pkv.kv_pool_alloc(dst, n)).to(b.device)
    src_ids = torch.from_numpy(ids).to(b.device)
    staging = torch.empty(pkv.pkv_blocks_staging_size(b.pool, n), dtype=torch.uint8, device=b.device)
    flush_buf = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=b.device)

    def step():
        pkv.pkv_blocks_gather(b.pool, src_ids, staging)
        pkv.pkv_blocks_scatter(dst, dst_ids, staging)

    ms = _timed(step, lambda: flush_buf.fill_(1), steps, warmup, torch.cuda.current_stream())
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK and pkv.pkv_check_device_errors(dst) == pkv.PKV_OK
    assert torch.equal(dk[dst_ids.long()].view(torch.int16), b.k_cache[src_ids.long()].view(torch.int16))
    moved = staging.numel()            # bytes of the moved blocks
    mean = statistics.mean(ms)
    pkv.kv_pool_destroy(dst)
    b.close()
    return {"ms_per_step": mean, "blocks": n, "bytes_moved": moved,
            "transfer_hbm_gbs": 4 * moved / (mean * 1e-3) / 1e9,
            "note": "one GPU: source and destination pools on the same device (the cross-GPU copy "
                    "of the staging buffer is not measured)"}


def measure_lora(steps, warmup):
    """Segmented multi-adapter LoRA projection (Sec. 5.6): Llama-3-8B-shaped
    projection (4096 x 4096), rank-16 adapters.  Case C1: the 12-prompt
    4/3/3/2 request over four adapters, batched by pkv_lora_dispatch
    (adapter first, length buckets at 1024 / 2048 tokens); and a larger
    synthetic request (64 prompts, 8 adapters, a quarter base-only).
    TFLOP/s on the base and low-rank products; cuBLAS's base GEMM alone
    (torch.matmul, bf16) on the same rows beside it, for context."""
    import numpy as np
    import torch

    from paper_2605_11232_gb300 import pkv

    def one(lens, ads, n_ad, seed):
        # base-only prompts are dispatched as adapter n_ad (their own group)
        # and run with no adapter (-1)
        order, batches = pkv.pkv_lora_dispatch(np.array([a if a >= 0 else n_ad for a in ads], np.int32),
                                               np.array(lens, np.int32), np.array([1024, 2048], np.int32), 0)
        starts, badapter = [0], []
        for adapter, _bk, b0, b1 in batches:
            starts.append(starts[-1] + sum(lens[order[i]] for i in range(b0, b1)))
            badapter.append(adapter if adapter < n_ad else -1)
        T, d, r = starts[-1], 4096, 16
        g = torch.Generator(device="cuda").manual_seed(seed)
        x = torch.randn((T, d), device="cuda", generator=g).to(torch.bfloat16)
        w = (torch.randn((d, d), device="cuda", generator=g) / d ** 0.5).to(torch.bfloat16)
        a = (torch.randn((n_ad, r, d), device="cuda", generator=g) / d ** 0.5).to(torch.bfloat16)
        b = (torch.randn((n_ad, d, r), device="cuda", generator=g) / r ** 0.5).to(torch.bfloat16)
        scale = np.full(n_ad, 2.0, np.float32)
        y = torch.empty((T, d), dtype=torch.bfloat16, device="cuda")
        flush_buf = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device="cuda")
        step = lambda: pkv.pkv_lora_sgmv(x, w, a, b, scale, starts, badapter, y)
        ms = _timed(step, lambda: flush_buf.fill_(1), steps, warmup, torch.cuda.current_stream())
        t_lora = sum(starts[k + 1] - starts[k] for k in range(len(badapter)) if badapter[k] >= 0)
        flops = 2 * T * d * d + 2 * t_lora * (d * r + r * d)
        base = _timed(lambda: torch.matmul(x, w.t()), lambda: flush_buf.fill_(1), steps, warmup,
                      torch.cuda.current_stream())
        mean, bmean = statistics.mean(ms), statistics.mean(base)
        return {"tokens": T, "segments": len(badapter), "adapters": n_ad, "rank": r,
                "ms_per_call": mean, "tflops": flops / (mean * 1e-3) / 1e12,
                "cublas_base_only_ms": bmean, "cublas_base_only_tflops": 2 * T * d * d / (bmean * 1e-3) / 1e12}

    c1 = one([412, 1830, 2650, 977, 1210, 2205, 388, 1499, 2800, 640, 1750, 2120],
             [0, 0, 0, 0, 1, 1, 1, 2, 2, 2, 3, 3], 4, 11)
    rng = np.random.default_rng(12)
    lens = rng.integers(300, 2900, 64).tolist()
    ads = [int(v) if v < 8 else -1 for v in rng.integers(0, 11, 64)]
    big = one(lens, ads, 8, 12)
    return {"case_c1": c1, "synthetic_64": big}


def summarize(res, peaks):
    hbm, tf_burst, tf_sust, kind = peaks
    ms = statistics.mean(res["step_ms"])
    out = {"ms_per_step": ms, "ms_median": statistics.median(res["step_ms"]),
           "ms_range": [min(res["step_ms"]), max(res["step_ms"])],
           "ms_per_step_warm_l2": statistics.mean(res["warm_ms"]),
           "kernels": {k: {"launches": n, "avg_us": 1e3 * t / n} for k, (n, t) in res["trace"].items()}}
    if res["Rd"]:
        if res["Rp"]:
            # mixed step: the decode bytes over the decode subset's own time
            # (timed alone, untraced, L2 flushed), not over a step that also
            # runs prefill
            dec_us = 1e3 * statistics.mean(res["dec_ms"])
            gbs = res["dec_bytes"] / (dec_us * 1e-6) / 1e9 if dec_us > 0 else float("nan")
            logical = res.get("dec_logical", 0) / (dec_us * 1e-6) / 1e9 if dec_us > 0 else float("nan")
            basis = "decode subset timed alone (its kernels overlapping), L2 flushed"
            out["decode_us_per_step"] = dec_us
            out["decode_kernels_sum_us"] = sum(1e3 * t / n for k, (n, t) in res["trace"].items()
                                               if k.startswith("decode_"))
        else:
            gbs = (res["dec_bytes"] + res["wr_bytes"]) / (ms * 1e-3) / 1e9
            logical = (res.get("dec_logical", 0) + res["wr_bytes"]) / (ms * 1e-3) / 1e9
            basis = "whole step (cache write + decode)"
        out.update(decode_hbm_gbs=gbs, decode_frac_of_measured_hbm=gbs / hbm,
                   decode_frac_of_8tbs=gbs / 8000.0, decode_basis=basis, prefix_pass=res["groups"],
                   decode_logical_gbs=logical,
                   decode_logical_note="logical: every request's K/V rows, a shared prefix counted "
                                       "once per request (what a cache without sharing reads)")
        if not res["Rp"]:
            out["decode_hbm_gbs_warm_l2"] = (res["dec_bytes"] + res["wr_bytes"]) / (
                statistics.mean(res["warm_ms"]) * 1e-3) / 1e9
    if res["Rp"]:
        tp = res["trace"].get("prefill")
        if tp:
            tfs = res["pre_flops"] / (tp[1] / tp[0] * 1e-3) / 1e12
            out.update(prefill_tflops=tfs, prefill_frac_of_measured_bf16=tfs / tf_burst)
    return out


def reference_arm(args, rank, world):
    """The fp64 CPU oracle on the host cores: one step = attention of every
    decode request of the headline batch, bytes counted like the GPU line and
    the cpu_baseline leg (every distinct K/V row once, the shared prefix once
    per step, plus Q and O).  The step's cache write is not run by the oracle
    and its bytes are not counted."""
    import oracle
    from paper_2605_11232_gb300.workloads import make_workload

    if rank != 0:
        return 0
    cores = os.cpu_count() or 1
    w = make_workload(HEADLINE)
    R = w.num_requests
    step_bytes = decode_bytes(w, slice(0, R))
    times = []
    for k in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        for r in range(R):
            oracle.request_attention(w, r, threads=cores)
        dt = time.perf_counter() - t0
        if k >= args.warmup:
            times.append(dt)
    gbs = step_bytes * len(times) / sum(times) / 1e9
    line = {"impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC[HEADLINE], "sample": f"all {R} decode requests per step",
                       "bytes_per_step": step_bytes},
            "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
                             "sample": f"one pass over all {R} l8b_decode requests per step (all q heads, "
                                       "full context), fp64 C oracle, threads = host cores; bytes: distinct "
                                       "K/V rows, shared prefix once per step, plus Q and O"},
            "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


METRIC = "prefix-cached paged-attn: prefill TFLOP/s & decode HBM GB/s, % of GB300 peak"


def cpu_baseline(w_name, budget_s=12.0):
    """The oracle as it stands on this host: passes over the decode requests of
    the headline workload until about budget_s seconds of work, all host cores."""
    import oracle
    from paper_2605_11232_gb300.workloads import make_workload
    cores = os.cpu_count() or 1
    w = make_workload(w_name)
    per_pass_rows = sum(int(w.context_lens[r]) - w.prefix_len_of(r) for r in range(w.num_requests))
    per_pass_rows += sum(w.prefix_lens[g] for g in {int(x) for x in w.group_of_req} if g >= 0)
    per_pass = per_pass_rows * kv_row_bytes(w) + 2 * w.num_requests * w.num_q_heads * w.head_dim * 2
    t0 = time.perf_counter()
    done = 0
    while True:
        for r in range(w.num_requests):
            oracle.request_attention(w, r, threads=cores)
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    # the same oracle on one thread, over the first requests for about a
    # quarter of the budget
    t1 = time.perf_counter()
    n1 = 0
    for r in range(w.num_requests):
        oracle.request_attention(w, r, threads=1)
        n1 += 1
        if time.perf_counter() - t1 > budget_s / 4:
            break
    dt1 = time.perf_counter() - t1
    return {"value": done * per_pass / dt / 1e9, "unit": "GB/s", "cores": cores, "kind": "oracle",
            "sample": f"{done} passes over all {w.num_requests} {w_name} decode requests (all q heads, "
                      f"full context), fp64 C oracle, {cores} threads, {dt:.1f} s; bytes counted like "
                      "the GPU metric (shared prefix once per pass)",
            "one_thread": {"value": per_pass * n1 / w.num_requests / dt1 / 1e9, "unit": "GB/s",
                           "sample": f"{n1} of the {w.num_requests} requests on 1 thread, {dt1:.1f} s; "
                                     "bytes: the pass's, in proportion to the requests done"}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--quick", action="store_true", help="headline workload only")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile", default=None, metavar="WORKLOAD",
                    help="run only WORKLOAD's steps (for ncu captures); prints per-kernel times")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    rank, world, local = dist_setup(args.gpus)
    if args.impl == "reference":
        return reference_arm(args, rank, world)

    import torch
    torch.cuda.set_device(local)
    import __graft_entry__
    if rank == 0:
        __graft_entry__.build()
    barrier(world)
    from paper_2605_11232_gb300 import pkv
    pkv.load()
    peaks = load_peaks()
    if args.profile in ("lora_sgmv", "pd_block_transfer", "spec_verify_tree"):
        fn = {"lora_sgmv": measure_lora, "pd_block_transfer": measure_transfer,
              "spec_verify_tree": measure_verify}[args.profile]
        print(json.dumps({"profile": args.profile, **fn(args.steps, args.warmup)}), flush=True)
        return 0
    if args.profile:
        r = measure_workload(args.profile, args.steps, args.warmup)
        print(json.dumps({"profile": args.profile, **summarize(r, peaks)}), flush=True)
        return 0
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    t_start = time.time()
    head = measure_workload(HEADLINE, args.steps, args.warmup, e2e_steps=max(20, args.steps // 4))
    t_end = time.time()
    extra = {}
    if not args.quick:
        for name in ("l8b_prefill", "qwen_mixed", "l70b_decode"):
            try:
                r = measure_workload(name, max(10, args.steps // 10), 3)
                extra[name] = summarize(r, peaks)
            except Exception as e:   # report, do not hide
                extra[name] = {"error": str(e)}
        for name, fn in (("spec_verify_tree", measure_verify), ("pd_block_transfer", measure_transfer),
                         ("lora_sgmv", measure_lora)):
            try:
                r = fn(max(10, args.steps // 10), 3)
                if "transfer_hbm_gbs" in r:
                    r["frac_of_measured_hbm"] = r["transfer_hbm_gbs"] / peaks[0]
                for sub in ("case_c1", "synthetic_64"):
                    if sub in r:
                        r[sub]["frac_of_measured_bf16"] = r[sub]["tflops"] / peaks[1]
                if "verify_tflops" in r:
                    r["verify_frac_of_measured_bf16"] = r["verify_tflops"] / peaks[1]
                    r["step_frac_of_measured_hbm"] = r["step_hbm_gbs"] / peaks[0]
                extra[name] = r
            except Exception as e:   # report, do not hide
                extra[name] = {"error": str(e)}
    clocks.stop()

    w = head["w"]
    ms_local = statistics.mean(head["step_ms"])
    step_bytes = head["dec_bytes"] + head["wr_bytes"]
    ms, total_bytes, value, e2e_ms, e2e_val = aggregate_replicas(ms_local, step_bytes, head["e2e_ms"], world)
    hbm, tf_burst, tf_sust, pk_kind = peaks
    # roofline of the dominant kernel (largest share of traced time)
    trace = head["trace"]
    dom = max(trace.items(), key=lambda kv: kv[1][1])[0]
    n_dom, t_dom = trace[dom]
    avg_ms = t_dom / n_dom
    alg = head["kernel_bytes"].get(dom)
    achieved = alg / (avg_ms * 1e-3) / 1e9 if alg else None
    traffic = ncu_traffic(dom, HEADLINE)
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC[HEADLINE], "global_batch": int(w.num_requests) * world,
                   "parallelism": f"replicas{world}", "l2": "flushed before every step (256 MiB write), "
                   "per-step CUDA events", "prefix_pass": head["groups"],
                   "bytes_per_step": step_bytes},
        "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm if achieved else None, "peak_kind": pk_kind, "traffic": traffic,
                     "algorithmic_bytes_per_launch": alg, "avg_launch_us": avg_ms * 1e3},
        "e2e": {"value": e2e_val, "unit": "GB/s", "h2d_bytes_per_step": head["h2d"],
                "d2h_bytes_per_step": head["d2h"], "ms_per_step": e2e_ms},
        "gpu_launches": int(sum(n for n, _ in trace.values())),
        "clocks": clocks.summary(t_start, t_end),
        "kernels": {k: {"launches": n, "avg_us": 1e3 * t / n} for k, (n, t) in trace.items()},
        "headline": summarize(head, peaks),
        "workloads": extra,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(HEADLINE)
    elif rank == 0:
        line["cpu_baseline"] = None
    if rank == 0:
        print(json.dumps(line), flush=True)
    barrier(world)
    return 0


if __name__ == "__main__":
    sys.exit(main())
