#!/usr/bin/env python
"""Benchmark of the KV-state graft hot path on GB300 (one JSON line on rank 0).

Workload (default, the 12B-class single graft): L 48, Hq/Hkv 16/8, D 256,
page 64.  One step =
  release the sequence -> own-position graft of an 8,192-token block from an
  HBM store (3 GiB of pages) -> SHA-256 page-digest verification of the
  restored pages -> fresh write of the remaining 24,576 rows -> decode
  attention of one query token over all 32,768 rows of all 48 layers.
value = algorithmic HBM bytes of the step / step time (GB/s); the parts give
each kernel's own figure (graft GB/s, digest GB/s, decode tokens/s).
e2e = the same step through the C ABI with the block in a pinned-host store
(read by the graft kernel over the host link), the query copied from pinned
host memory and the output read back, every step.

--impl reference times the CPU oracle (test infrastructure) on a bounded
sample of the same step.  Under torchrun each rank runs an independent
replica (weak scaling); there is no data-path collective.
"""
from __future__ import annotations

import argparse
import gc
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import kvg_synth as syn  # noqa: E402

METRIC = ("graft GB/s (HBM & host→HBM) + decode-attn tokens/s @32k grafted, % roofline")
ALU_LANES_PER_SM = 64  # 4 SM sub-partitions x 16 ALU-pipe lanes


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p.get("sm_max_mhz", 2070.0)), "measured"
    except Exception:
        return 6800.0, 2070.0, "fallback"


def load_ncu_figures():
    """Per-kernel figures from the committed ncu summary
    (profiles/ncu_traffic.txt: DRAM bytes per launch, and for the hashing
    kernel its ALU-pipe instructions per SHA-256 compression), kept only
    while the kernel's source file is unchanged since the capture."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    out = {}
    if not os.path.exists(path):
        return out
    import hashlib
    for line in open(path):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        parts = dict(kv.split("=", 1) for kv in line.split())
        src = os.path.join(ROOT, "paper_2607_14431_gb300", "csrc", parts["source"])
        if os.path.exists(src) and hashlib.sha256(open(src, "rb").read()).hexdigest()[:16] == parts["sha"]:
            out[parts["kernel"]] = {k: float(v) for k, v in parts.items() if k not in ("kernel", "source", "sha")}
    return out


def load_traffic():
    """Per-launch DRAM bytes from the committed ncu summary, keyed by kernel."""
    return {k: v["bytes_per_launch"] for k, v in load_ncu_figures().items() if "bytes_per_launch" in v}


def sha_alu_ops_per_compression(kernel="graft_verify_ring_kernel"):
    """ALU-pipe instructions per SHA-256 compression of the verified graft's
    kernel, its own instruction mix as ncu counted it (None once the
    kernel's source has changed since that capture)."""
    return load_ncu_figures().get(kernel, {}).get("alu_inst_per_compression")


def aggregate(total_ms: float, steps: int, step_bytes: int, world: int, device) -> tuple:
    """Whole-job figures of a run on `world` replicas: the slowest rank's time
    per step (max over ranks) and the bytes every rank processed over it."""
    if world > 1:
        t = torch.tensor([total_ms], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_step = total_ms / steps
    return ms_step, world * step_bytes / (ms_step * 1e-3) / 1e9


class Clocks:
    """Samples SM clocks and throttle reasons with nvidia-smi during a region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.samples = []
        self.proc = None
        try:
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            sel = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", sel, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            # the sampler must be live before the region it records starts
            t_end = time.perf_counter() + 3.0
            while not self.samples and time.perf_counter() < t_end and self.proc.poll() is None:
                time.sleep(0.005)
            self.n_before = len(self.samples)
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append([x.strip() for x in line.split(",")])

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.t.join(timeout=2)
        # the samples taken during the region (the one that proved the
        # sampler live came before it)
        rows = self.samples[self.n_before:] or self.samples[-1:]
        sm = [float(s[0]) for s in rows if len(s) >= 7 and s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in rows if len(s) >= 7 and s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in rows if len(s) >= 7 for i in range(4)
                          if s[3 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(sm)}


# --------------------------------------------------------------------------
# 12B-class single graft: the default workload
# --------------------------------------------------------------------------

class Step12B:
    """Device state and the per-step call sequence for the 12B workload."""

    def __init__(self, kvg, device, stream, side, n_layers=None, pool_store=False, schedule="overlap",
                 swa=None, kv="bf16"):
        self.kvg = kvg
        self.w = w = syn.B12 if not n_layers else syn.B12.with_layers(n_layers)
        self.dev = device
        self.stream = stream
        self.side = side
        self.ev_graft = torch.cuda.Event()
        self.ev_verify = torch.cuda.Event()
        # completion events of a chunked graft (e2e step), created by one record
        self.chunk_ev = [torch.cuda.Event() for _ in range(16)]
        for e in self.chunk_ev:
            e.record(side)
        self.nb, self.nf = syn.B12_BLOCK, syn.B12_CTX - syn.B12_BLOCK
        P = w.page_size
        # kv "e4m3": the cache (and so the block) holds fp8 E4M3 codes with
        # per-tensor scales; appends quantize the bf16 rows
        self.kv = kv
        fp8 = kv == "e4m3"
        self.dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0,
                                  kv_dtype=kvg.KVG_KV_E4M3 if fp8 else kvg.KVG_KV_BF16,
                                  k_scale=syn.FP8_K_SCALE, v_scale=syn.FP8_V_SCALE)
        elem = 1 if fp8 else 2
        n_pages = syn.B12_CTX // P + self.nb // P
        self.cache = kvg.Cache(self.dims, n_pages + (self.nb // P if pool_store else 0), 2, syn.B12_CTX)
        # pool_store: the block lives in the cache's own pool and grafts by
        # aliasing its pages (no page copy)
        self.store = (kvg.PoolStore(self.cache, 64 << 20) if pool_store
                      else kvg.Store(self.dims, kvg.KVG_RESIDENCY_HBM, 4 << 30))
        self.hstore = kvg.Store(self.dims, kvg.KVG_RESIDENCY_PINNED_HOST, 4 << 30)
        with torch.cuda.stream(stream):
            kb, vb = syn.kv_rows(w, self.nb, w.seed, device)
            pb = torch.arange(self.nb, dtype=torch.int32, device=device)
            kvg.kvg_cache_append(self.cache.h, 1, kb.data_ptr(), vb.data_ptr(), pb.data_ptr(), self.nb, stream)
            self.bid = kvg.kvg_deposit(self.store.h, self.cache.h, 1, 0, self.nb, stream)
            self.hbid = kvg.kvg_deposit(self.hstore.h, self.cache.h, 1, 0, self.nb, stream)
            kvg.kvg_cache_release(self.cache.h, 1, stream)
            self.kf, self.vf = syn.kv_rows(w, self.nf, w.seed + 1, device)
            self.pf = torch.arange(self.nb, syn.B12_CTX, dtype=torch.int32, device=device)
            self.q = syn.queries(w, w.n_layers, 1, w.seed, device)
            self.out = torch.empty_like(self.q)
            # softmax state of the split decode: fp32 [L][1][Hq][D + 4]
            self.state = torch.zeros((w.n_layers, 1, w.n_q_heads, w.head_dim + 4), dtype=torch.float32,
                                     device=device)
        stream.synchronize()
        self.kb, self.vb = kb, vb  # the block's rows, kept for parity tests
        self.scale = 1.0 / math.sqrt(w.head_dim)
        blk_pages = w.n_layers * 2 * (self.nb // P) * w.page_bytes * elem // 2
        self.pool_store = pool_store
        # swa = (W, R): sliding-window layers over the full-size cache, every
        # R-th layer global and the others attending to their last W rows
        self.swa = swa
        self.windows = [0] * w.n_layers
        if swa:
            W, R = swa
            self.windows = [0 if (l + 1) % R == 0 else W for l in range(w.n_layers)]
            kvg.kvg_cache_set_layer_windows(self.cache.h, self.windows)
        rows_read = sum(min(x, syn.B12_CTX) if x else syn.B12_CTX for x in self.windows)
        # HBM algorithmic bytes of each phase: the graft copies the block
        # (read + write); the digest check hashes the block's bytes, which
        # must be read once from HBM only when no copy reads them (the
        # zero-copy graft); the append reads the fresh rows and writes them;
        # the decode reads every valid K/V row once
        self.bytes = {
            "graft": 0 if pool_store else 2 * blk_pages,
            "verify": blk_pages if pool_store else 0,
            "append": (2 + elem) * w.n_layers * 2 * self.nf * w.n_kv_heads * w.head_dim,
            "decode": rows_read * 2 * w.n_kv_heads * w.head_dim * elem + 2 * self.q.numel() * 2,
        }
        # bytes the digest check hashes (not HBM traffic of their own when a
        # copy reads them) and its SHA-256 compressions (65 per 4 KiB leaf)
        self.hashed_bytes = blk_pages
        self.sha_blocks = (blk_pages // 4096) * 65
        self.blk_pages = blk_pages
        # the step's HBM algorithmic bytes, whatever the schedule
        self.step_bytes = sum(self.bytes.values())
        self.schedule = schedule
        # phase -> (stream, first event, last event) of the per-step events
        if schedule == "fused":
            self.bytes["graft_verify"] = self.bytes.pop("graft") + self.bytes.pop("verify")
            self.spans = {"release": ("main", 0, 1), "append": ("main", 1, 2), "graft_join": ("main", 2, 3),
                          "decode": ("main", 3, 4), "graft_verify": ("side", 0, 1)}
        else:
            self.spans = {"release": ("main", 0, 1), "graft": ("main", 1, 2), "append": ("main", 2, 3),
                          "decode": ("main", 3, 4), "verify_join": ("main", 4, 5), "verify": ("side", 0, 1)}
        self.phases = list(self.spans)

    def run_step(self, store=None, bid=None, ev=None):
        """One step.  Schedule "overlap": the graft copies, then the digest
        check (which only reads the grafted pages, written by neither the
        append nor the decode) runs on a side stream, its ALU-bound hashing
        overlapping the HBM-bound append and decode; the main stream waits for
        it before the step ends.  Schedule "fused": see _run_fused.
        ev: optional per-phase timing events (main: 6, side: 2)."""
        if self.schedule == "fused":
            return self._run_fused(store, bid, ev)
        kvg, s, side, c = self.kvg, self.stream, self.side, self.cache.h
        store = store or self.store.h
        bid = self.bid if bid is None else bid
        m = ev["main"] if ev else None
        if m: m[0].record(s)
        kvg.kvg_cache_release(c, 0, s)
        if m: m[1].record(s)
        kvg.kvg_graft(store, bid, c, 0, -1, 0, 0, s)
        if m: m[2].record(s)
        self.ev_graft.record(s)
        side.wait_event(self.ev_graft)
        if ev: ev["side"][0].record(side)
        kvg.kvg_verify(store, bid, c, 0, 0, 0, side)
        if ev: ev["side"][1].record(side)
        self.ev_verify.record(side)
        kvg.kvg_cache_append(c, 0, self.kf.data_ptr(), self.vf.data_ptr(), self.pf.data_ptr(), self.nf, s)
        if m: m[3].record(s)
        kvg.kvg_decode_attention(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads, self.out.data_ptr(),
                                 self.scale, s)
        if m: m[4].record(s)
        s.wait_event(self.ev_verify)
        if m: m[5].record(s)

    def run_step_split(self, store, bid):
        """The fused step with a split decode, for a block that streams in
        from a pinned-host store: the decode over the fresh rows (slots past
        the block) runs on the main stream right after the append, while the
        verified graft is still copying the block over the host link; the
        rows of each chunk of the graft merge in as soon as the chunk has
        landed, and the output is finished once the whole block's digests
        have been checked."""
        kvg, s, side, c = self.kvg, self.stream, self.side, self.cache.h
        kvg.kvg_cache_release(c, 0, s)
        self.ev_graft.record(s)
        side.wait_event(self.ev_graft)
        ends = kvg.kvg_graft_chunked(store, bid, c, 0, [e.cuda_event for e in self.chunk_ev],
                                     flags=kvg.KVG_GRAFT_VERIFY, stream=side)
        self.ev_verify.record(side)
        kvg.kvg_cache_append(c, 0, self.kf.data_ptr(), self.vf.data_ptr(), self.pf.data_ptr(), self.nf, s)
        kvg.kvg_decode_attention_range(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads, self.scale, self.nb,
                                       syn.B12_CTX, 0, self.state.data_ptr(), s)
        lo = 0
        for j, hi in enumerate(ends):
            s.wait_event(self.chunk_ev[j])
            kvg.kvg_decode_attention_range(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads, self.scale, lo, hi,
                                           kvg.KVG_DECODE_MERGE, self.state.data_ptr(), s)
            lo = hi
        s.wait_event(self.ev_verify)
        kvg.kvg_decode_state_finish(self.state.data_ptr(), self.q.numel() // self.w.head_dim, self.w.head_dim,
                                    self.out.data_ptr(), s)

    def _run_fused(self, store=None, bid=None, ev=None):
        """The same step with the digest check folded into the graft: the
        verified graft (one pass: copy + leaf hashes, then page digests) runs
        on a side stream while the main stream appends the fresh rows into
        other pages; the decode waits for both."""
        kvg, s, side, c = self.kvg, self.stream, self.side, self.cache.h
        store = store or self.store.h
        bid = self.bid if bid is None else bid
        m = ev["main"] if ev else None
        if m: m[0].record(s)
        kvg.kvg_cache_release(c, 0, s)
        if m: m[1].record(s)
        self.ev_graft.record(s)
        side.wait_event(self.ev_graft)
        if ev: ev["side"][0].record(side)
        kvg.kvg_graft(store, bid, c, 0, -1, 0, kvg.KVG_GRAFT_VERIFY, side)
        if ev: ev["side"][1].record(side)
        self.ev_verify.record(side)
        kvg.kvg_cache_append(c, 0, self.kf.data_ptr(), self.vf.data_ptr(), self.pf.data_ptr(), self.nf, s)
        if m: m[2].record(s)
        s.wait_event(self.ev_verify)
        if m: m[3].record(s)
        kvg.kvg_decode_attention(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads, self.out.data_ptr(),
                                 self.scale, s)
        if m: m[4].record(s)

def run_kvg(args, rank, world):
    from paper_2607_14431_gb300 import build
    build.build()
    from paper_2607_14431_gb300 import kvg

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    # the main stream (append, decode) at the highest priority: the append's
    # one CTA per SM is placed before the verified graft's queued CTAs, which
    # shortens the window the two share (measured 6.11 -> 6.01 ms per step)
    stream = torch.cuda.Stream(device, priority=torch.cuda.Stream.priority_range()[1])
    side = torch.cuda.Stream(device)
    hbm_peak, sm_max, peak_kind = load_peaks()
    n_sm = torch.cuda.get_device_properties(device).multi_processor_count
    alu_peak = n_sm * ALU_LANES_PER_SM * sm_max * 1e6  # ALU-pipe ops per second at the max SM clock
    swa = tuple(int(x) for x in args.swa.split(":")) if args.swa else None
    st = Step12B(kvg, device, stream, side, args.layers, pool_store=args.store == "pool", schedule=args.schedule,
                 swa=swa, kv=args.kv)
    # the verified graft runs graft_verify_ring_kernel for a full wave of it
    # (five 128-leaf CTAs on every SM) or more on a bf16 cache, else
    # graft_verify_kernel; the append is append_tma_kernel (bf16) or
    # append_e4m3_kernel (fp8)
    gv_kernel = ("graft_verify_ring_kernel" if st.kv == "bf16" and st.sha_blocks // 65 >= n_sm * 5 * 128
                 else "graft_verify_kernel")
    app_kernel = "append_tma_kernel" if st.kv == "bf16" else "append_e4m3_kernel"
    alu_per_c = sha_alu_ops_per_compression(gv_kernel)

    # correctness of the configuration being timed: one verified step
    st.run_step()
    kvg.kvg_sync(st.cache.h, stream, 60.0)
    first_sha = _sha_tensor(st.out)

    for _ in range(args.warmup):
        st.run_step()
    stream.synchronize()

    K = args.steps
    mk = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    evs = [{"main": [mk() for _ in range(6)], "side": [mk(), mk()]} for _ in range(K)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    launches0 = kvg.kvg_launch_count()
    t_start, t_end = mk(), mk()
    torch.cuda.nvtx.range_push("kvg_timed")
    t_start.record(stream)
    for k in range(K):
        st.run_step(ev=evs[k])
    t_end.record(stream)
    torch.cuda.nvtx.range_pop()
    stream.synchronize()
    launches = kvg.kvg_launch_count() - launches0
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    kvg.kvg_sync(st.cache.h, stream, 60.0)  # digest verification of every timed step passed
    step_bytes = st.step_bytes
    ms_step, value = aggregate(total_ms, K, step_bytes, world, device)
    phase_ms = {p: statistics.mean(evs[k][sn][i].elapsed_time(evs[k][sn][j]) for k in range(K))
                for p, (sn, i, j) in st.spans.items()}
    deterministic = _sha_tensor(st.out) == first_sha

    # each graft form alone (CUDA events, median of 40 after 3 untimed): the
    # plain own-position graft (HBM-bound) and the verified one (ALU-bound)
    alone = {}
    if not st.pool_store:
        for name, flags in (("graft_alone", 0), ("graft_verify_alone", kvg.KVG_GRAFT_VERIFY)):
            g0, g1 = mk(), mk()
            gts = []
            clk_g = None
            for k in range(43):
                if k == 3:
                    clk_g = Clocks(local)
                kvg.kvg_cache_release(st.cache.h, 0, stream)
                g0.record(stream)
                kvg.kvg_graft(st.store.h, st.bid, st.cache.h, 0, -1, 0, flags, stream)
                g1.record(stream)
                stream.synchronize()
                if k >= 3:
                    gts.append(g0.elapsed_time(g1))
            ms = statistics.median(gts)
            b = 2 * st.blk_pages
            alone[name] = {"ms": round(ms, 4), "algorithmic_bytes": b, "gbs": round(b / (ms * 1e-3) / 1e9, 1),
                           "hbm_frac": round(b / (ms * 1e-3) / 1e9 / hbm_peak, 3), "clocks": clk_g.stop()}
            if flags and alu_per_c:
                ops = st.sha_blocks * alu_per_c
                alone[name].update({"alu_tops": round(ops / (ms * 1e-3) / 1e12, 3),
                                    "alu_frac": round(ops / (ms * 1e-3) / alu_peak, 3)})
        kvg.kvg_sync(st.cache.h, stream, 60.0)

    # e2e: host-store graft, query from pinned host memory, output read back.
    # With the fused schedule the decode is split: the part over the fresh
    # rows runs while the block still crosses the host link.
    e2e = None
    e2e_vs_device = None
    if not args.no_e2e:
        ref_out = st.out.float().cpu()
        q_host = torch.empty(st.q.shape, dtype=st.q.dtype, pin_memory=True)
        q_host.copy_(st.q.cpu())
        o_host = torch.empty(st.out.shape, dtype=st.out.dtype, pin_memory=True)
        split = st.schedule == "fused"
        ts = []
        for k in range(args.warmup + K):
            t0 = time.perf_counter()
            with torch.cuda.stream(stream):
                st.q.copy_(q_host, non_blocking=True)
            if split:
                st.run_step_split(st.hstore.h, st.hbid)
            else:
                st.run_step(st.hstore.h, st.hbid)
            with torch.cuda.stream(stream):
                o_host.copy_(st.out, non_blocking=True)
            stream.synchronize()
            if k >= args.warmup:
                ts.append(time.perf_counter() - t0)
        kvg.kvg_sync(st.cache.h, stream, 60.0)
        # the split decode's output against the one-call decode of the timed steps
        e2e_vs_device = float((o_host.float() - ref_out).abs().max())
        e2e_ms = statistics.mean(ts) * 1e3
        blk_read = st.blk_pages  # block pages read from host memory by the graft
        e2e = {"value": round(world * step_bytes / (e2e_ms * 1e-3) / 1e9, 2), "unit": "GB/s",
               "ms_per_step": round(e2e_ms, 3),
               "schedule": ("verified host-store graft in chunks; decode split: fresh rows during the graft, "
                            "each chunk's rows as it lands") if split else "verified host-store graft, then the decode",
               "inputs": ("host to device each step: the stored block (pinned-host store) and the query; "
                          "device to host: the output; the fresh rows stay in HBM (the model's own prefill "
                          "writes them on the GPU)"),
               "h2d_bytes_per_step": int(blk_read + st.q.numel() * 2),
               "d2h_bytes_per_step": int(st.out.numel() * 2),
               "host_graft_gbs": None}
        # host->HBM graft alone (the host-store graft kernel)
        e0, e1 = mk(), mk()
        gts = []
        for k in range(5):
            kvg.kvg_cache_release(st.cache.h, 0, stream)
            e0.record(stream)
            kvg.kvg_graft(st.hstore.h, st.hbid, st.cache.h, 0, -1, 0, 0, stream)
            e1.record(stream)
            stream.synchronize()
            gts.append(e0.elapsed_time(e1))
        e2e["host_graft_gbs"] = round(blk_read / (statistics.median(gts) * 1e-3) / 1e9, 2)
        # the host link's ceiling in the same run: pinned cudaMemcpyAsync H2D of 1 GiB
        h2d = measure_h2d(device, 1 << 30, 5)
        e2e["h2d_ceiling_gbs"] = round(h2d, 2)
        e2e["host_graft_link_frac"] = round(e2e["host_graft_gbs"] / h2d, 3)

    # per-launch DRAM bytes from ncu are for the 48-layer launches
    traffic = load_traffic() if st.w.n_layers == syn.B12.n_layers else {}
    parts = {}
    hashing = ("verify", "graft_verify")
    for p in st.phases:
        ms = phase_ms[p]
        if not st.bytes.get(p) and p not in hashing:
            parts[p] = {"ms": round(ms, 4)}
            continue
        b = st.bytes.get(p, 0)
        parts[p] = {"ms": round(ms, 4), "algorithmic_bytes": b}
        if b:
            gbs = b / (ms * 1e-3) / 1e9
            parts[p].update({"gbs": round(gbs, 1), "hbm_frac": round(gbs / hbm_peak, 3)})
        if p in hashing:
            parts[p].update({"hashed_bytes": st.hashed_bytes,
                             "hashed_gbs": round(st.hashed_bytes / (ms * 1e-3) / 1e9, 1),
                             "compressions": st.sha_blocks, "alu_ops_per_compression": alu_per_c})
            if alu_per_c:
                ops = st.sha_blocks * alu_per_c
                parts[p].update({"alu_tops": round(ops / (ms * 1e-3) / 1e12, 3),
                                 "alu_frac": round(ops / (ms * 1e-3) / alu_peak, 3)})
    parts["decode"]["tokens_per_s"] = round(1e3 / phase_ms["decode"], 1)
    kernel_of = {"graft": "graft_kernel", "verify": "sha256_leaves_kernel", "append": app_kernel,
                 "decode": "decode_kernel", "graft_verify": gv_kernel}
    if st.schedule == "fused":
        # The verified graft and the append run side by side on two streams
        # and share one window of HBM (from the release to the decode's
        # start), the longest part of the step; neither kernel alone bounds
        # it (each is slowed by the other's traffic, and the window runs at
        # the rate two plain copies side by side reach).  The roofline unit
        # is that window: both kernels' algorithmic bytes over its duration,
        # each kernel's own figures beside it.
        win = statistics.mean(evs[k]["main"][1].elapsed_time(evs[k]["main"][3]) for k in range(K))
        wb = st.bytes["append"] + st.bytes["graft_verify"]
        # (ncu traffic is kept for the bf16 step's kernels only)
        tr = [traffic.get(app_kernel), traffic.get(gv_kernel)] if st.kv == "bf16" else [None]
        gv = parts["graft_verify"]
        roof = {"bound": "hbm", "kernel": f"{app_kernel} || {gv_kernel}",
                "achieved": round(wb / (win * 1e-3) / 1e9, 1), "peak": hbm_peak, "unit": "GB/s",
                "frac": round(wb / (win * 1e-3) / 1e9 / hbm_peak, 3),
                "traffic": sum(tr) if all(t is not None for t in tr) else None, "peak_kind": peak_kind,
                "window_ms": round(win, 4), "algorithmic_bytes": wb,
                "members": {app_kernel: {k: parts["append"][k] for k in ("ms", "gbs", "hbm_frac")},
                            gv_kernel: {k: gv[k] for k in ("ms", "gbs", "hbm_frac", "alu_tops", "alu_frac") if k in gv}}}
    else:
        # dominant kernel: the longest phase that moves or hashes bytes
        dom = max((p for p in st.phases if st.bytes.get(p) or p in hashing), key=lambda p: phase_ms[p])
        if dom in hashing and alu_per_c:
            ops = st.sha_blocks * alu_per_c
            ach = ops / (phase_ms[dom] * 1e-3) / 1e12
            roof = {"bound": "alu", "kernel": kernel_of[dom], "achieved": round(ach, 3),
                    "peak": round(alu_peak / 1e12, 3), "unit": "Top/s", "frac": round(ach / (alu_peak / 1e12), 3),
                    "traffic": traffic.get(kernel_of[dom]),
                    "peak_kind": f"derived: {n_sm} SMs x {ALU_LANES_PER_SM} ALU-pipe lanes x max SM clock"}
        else:
            ach = st.bytes[dom] / (phase_ms[dom] * 1e-3) / 1e9
            roof = {"bound": "hbm", "kernel": kernel_of[dom], "achieved": round(ach, 1), "peak": hbm_peak,
                    "unit": "GB/s", "frac": round(ach / hbm_peak, 3), "traffic": traffic.get(kernel_of[dom]),
                    "peak_kind": peak_kind}
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(config_12b(st.w.n_layers, world, pool_store=st.pool_store, swa=st.swa, kv=st.kv),
                       schedule="verified graft in one pass, beside the append" if st.schedule == "fused"
                       else "graft, then the digest check beside the append and the decode"),
        "parts": parts, "alone": alone, "roofline": roof, "e2e": e2e, "gpu_launches": int(launches),
        "clocks": clk, "checks": {"deterministic": deterministic, "out_sha256": first_sha,
                                  "digest_verified_steps": K + args.warmup + 1,
                                  "e2e_out_max_abs_vs_device_out": e2e_vs_device},
    }
    return line


# --------------------------------------------------------------------------
# The other workloads (run with --config; the default line is the 12B step)
# --------------------------------------------------------------------------

class Step31B:
    """31B-class relocation: a 16,384-token block deposited at positions
    0..16,383; 8 sequences hold it re-based by delta in {0, 1, 4096, 100000}
    followed by 49,152 fresh rows (65,536-token contexts).  One step =
    relocating graft (delta 4096) of the block into a spare sequence + decode
    of one token for the 8 sequences over all 60 layers.  Every chunk of rows
    (the block's and each sequence's fresh rows) is its own N(0, 1) draw, so
    no two slot ranges hold the same K/V."""

    CHUNK = 2048

    def __init__(self, kvg, device, stream, n_layers=None):
        self.kvg, self.stream = kvg, stream
        self.w = w = syn.B31 if not n_layers else syn.B31.with_layers(n_layers)
        P = w.page_size
        self.nb, self.ctx, self.B = syn.B31_BLOCK, syn.B31_CTX, syn.B31_BATCH
        self.deltas = [syn.B31_DELTAS[i % len(syn.B31_DELTAS)] for i in range(self.B)]
        self.dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0)
        n_pages = self.B * (self.ctx // P) + self.nb // P
        self.cache = kvg.Cache(self.dims, n_pages, self.B + 1, self.ctx)
        blk_bytes = w.n_layers * 2 * (self.nb // P) * w.page_bytes
        self.store = kvg.Store(self.dims, kvg.KVG_RESIDENCY_HBM, blk_bytes + (64 << 20))
        c = self.cache.h
        with torch.cuda.stream(stream):
            # the block: written fresh into the spare sequence, deposited,
            # released; then every sequence's relocated graft and its fresh
            # rows.  Rows are generated one chunk at a time (the cache leaves
            # little room) on this stream, which also frees them.
            for i in range(self.nb // self.CHUNK):
                k, v = self.block_rows(i, device)
                pos = torch.arange(i * self.CHUNK, (i + 1) * self.CHUNK, dtype=torch.int32, device=device)
                kvg.kvg_cache_append(c, self.B, k.data_ptr(), v.data_ptr(), pos.data_ptr(), self.CHUNK, stream)
                del k, v, pos
            self.bid = kvg.kvg_deposit(self.store.h, c, self.B, 0, self.nb, stream)
            kvg.kvg_cache_release(c, self.B, stream)
            for sq in range(self.B):
                kvg.kvg_graft(self.store.h, self.bid, c, sq, -1, self.deltas[sq], 0, stream)
                for i in range(self.n_fresh_chunks):
                    k, v = self.fresh_rows(sq, i, device)
                    p0 = self.deltas[sq] + self.nb + i * self.CHUNK
                    pos = torch.arange(p0, p0 + self.CHUNK, dtype=torch.int32, device=device)
                    kvg.kvg_cache_append(c, sq, k.data_ptr(), v.data_ptr(), pos.data_ptr(), self.CHUNK, stream)
                    del k, v, pos
            self.q = syn.queries(w, w.n_layers, self.B, w.seed, device)
            self.out = torch.empty_like(self.q)
        stream.synchronize()
        kvg.kvg_sync(c, stream, 60.0)
        self.scale = 1.0 / math.sqrt(w.head_dim)
        self.bytes = {"relocate": 2 * blk_bytes,
                      "decode": self.B * w.n_layers * 2 * self.ctx * w.n_kv_heads * w.head_dim * 2
                                + 2 * self.q.numel() * 2}
        self.phases = ["release", "relocate", "decode"]

    @property
    def n_fresh_chunks(self):
        return (self.ctx - self.nb) // self.CHUNK

    def block_rows(self, i, device):
        """K, V of the block's chunk i (rows i*CHUNK ...), bf16 [L][CHUNK][Hkv][D]."""
        return syn.kv_rows(self.w, self.CHUNK, self.w.seed + 17 * i, device)

    def fresh_rows(self, sq, i, device):
        """K, V of sequence sq's fresh chunk i (slots nb + i*CHUNK ...)."""
        return syn.kv_rows(self.w, self.CHUNK, self.w.seed + 100_000 + 64 * sq + i, device)

    def run_step(self, ev=None):
        kvg, s, c = self.kvg, self.stream, self.cache.h
        m = ev["main"] if ev else None
        if m: m[0].record(s)
        kvg.kvg_cache_release(c, self.B, s)
        if m: m[1].record(s)
        kvg.kvg_graft(self.store.h, self.bid, c, self.B, -1, 4096, 0, s)
        if m: m[2].record(s)
        kvg.kvg_decode_attention(c, -1, list(range(self.B)), self.q.data_ptr(), self.w.n_q_heads,
                                 self.out.data_ptr(), self.scale, s)
        if m: m[3].record(s)

class StepTiny:
    """The tiny configuration (2 layers, 4/2 heads, head_dim 64, page 16): a
    256-token block deposited at positions 0..255; one step = own-position
    graft with digest verification into an empty sequence + decode of one
    query token over the 256 rows.  Launch-bound (microseconds), timed for
    completeness (its parity with the oracle is a test)."""

    def __init__(self, kvg, device, stream):
        self.kvg, self.stream = kvg, stream
        self.w = w = syn.TINY
        P = w.page_size
        self.nb = syn.TINY_BLOCK
        self.dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0)
        n_pages = 2 * (self.nb // P) + 2
        self.cache = kvg.Cache(self.dims, n_pages, 2, self.nb)
        self.store = kvg.Store(self.dims, kvg.KVG_RESIDENCY_HBM, 16 << 20)
        c = self.cache.h
        with torch.cuda.stream(stream):
            self.k, self.v = syn.kv_rows(w, self.nb, w.seed, device)
            pos = torch.arange(self.nb, dtype=torch.int32, device=device)
            kvg.kvg_cache_append(c, 1, self.k.data_ptr(), self.v.data_ptr(), pos.data_ptr(), self.nb, stream)
            self.bid = kvg.kvg_deposit(self.store.h, c, 1, 0, self.nb, stream)
            kvg.kvg_cache_release(c, 1, stream)
            self.q = syn.queries(w, w.n_layers, 1, w.seed, device)
            self.out = torch.empty_like(self.q)
        stream.synchronize()
        self.scale = 1.0 / math.sqrt(w.head_dim)
        blk = w.n_layers * 2 * (self.nb // P) * w.page_bytes
        self.bytes = {"graft_verify": 2 * blk, "decode": w.n_layers * 2 * self.nb * w.n_kv_heads * w.head_dim * 2}
        self.phases = ["release", "graft_verify", "decode"]

    def run_step(self, ev=None):
        kvg, s, c = self.kvg, self.stream, self.cache.h
        m = ev["main"] if ev else None
        if m: m[0].record(s)
        kvg.kvg_cache_release(c, 0, s)
        if m: m[1].record(s)
        kvg.kvg_graft(self.store.h, self.bid, c, 0, -1, 0, kvg.KVG_GRAFT_VERIFY, s)
        if m: m[2].record(s)
        kvg.kvg_decode_attention(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads, self.out.data_ptr(),
                                 self.scale, s)
        if m: m[3].record(s)


class StepBatched:
    """Batched library graft on a layer slice of the 12B shape: a 512-block
    HBM store (lengths U{2048..6144}); 32 sequences each graft 4 distinct
    blocks at their own positions (page-aligned, stitched), then 64 decode
    steps append one row per sequence and decode all 32.  consecutive=True:
    blocks 2-4 of each sequence are re-based by the tokens already in it, so
    its position tags run without a gap (the same single batched call, with
    per-graft deltas; their keys are rotated during the copy)."""

    def __init__(self, kvg, device, stream, n_layers=4, consecutive=False, n_store=syn.BATCHED_STORE):
        self.kvg, self.stream = kvg, stream
        self.w = w = syn.BATCHED.with_layers(n_layers or 4)
        P = w.page_size
        self.lens, self.ids = syn.batched_plan(n_store=n_store)
        self.n_store = n_store
        nS = syn.BATCHED_SEQS
        self.steps = syn.BATCHED_STEPS
        self.dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0)
        per_seq_pages = [sum(-(-int(self.lens[b]) // P) for b in self.ids[s]) + -(-self.steps // P) + 1
                         for s in range(nS)]
        self.max_slots = max(per_seq_pages) * P
        n_pages = sum(per_seq_pages) + -(-int(self.lens.max()) // P)
        self.cache = kvg.Cache(self.dims, n_pages, nS + 1, self.max_slots)
        store_bytes = sum(w.n_layers * 2 * -(-int(n) // P) * w.page_bytes + (1 << 20) for n in self.lens)
        self.store = kvg.Store(self.dims, kvg.KVG_RESIDENCY_HBM, store_bytes + (2 << 30))
        c = self.cache.h
        self.bids = []
        with torch.cuda.stream(stream):
            for b, n in enumerate(self.lens):
                n = int(n)
                k, v = syn.kv_rows(w, n, w.seed + b, device)
                pos = torch.arange(n, dtype=torch.int32, device=device)
                kvg.kvg_cache_append(c, nS, k.data_ptr(), v.data_ptr(), pos.data_ptr(), n, stream)
                self.bids.append(kvg.kvg_deposit(self.store.h, c, nS, 0, n, stream))
                kvg.kvg_cache_release(c, nS, stream)
            self.kd, self.vd = syn.kv_rows(w.with_layers(w.n_layers), nS * self.steps, w.seed + 9999, device)
            # kd/vd: [L][steps*nS][Hkv][D] -> per step a [L][nS][Hkv][D] slice
            self.q = syn.queries(w, w.n_layers, nS, w.seed, device)
            self.out = torch.empty_like(self.q)
            ctx0 = torch.tensor([sum(int(self.lens[b]) for b in self.ids[s]) for s in range(nS)], dtype=torch.int32)
            # position tag of step t's row of sequence s: its context length so far
            self.pos = (ctx0[None, :] + torch.arange(self.steps, dtype=torch.int32)[:, None]).to(device)
        stream.synchronize()
        self.scale = 1.0 / math.sqrt(w.head_dim)
        row = w.n_kv_heads * w.head_dim * 2
        graft_b = sum(2 * w.n_layers * 2 * -(-int(self.lens[b]) // P) * w.page_bytes for s in range(nS)
                      for b in self.ids[s])
        ctx0 = [sum(int(self.lens[b]) for b in self.ids[s]) for s in range(nS)]
        dec_b = sum(w.n_layers * 2 * (ctx0[s] + t + 1) * row for s in range(nS) for t in range(self.steps))
        app_b = self.steps * nS * w.n_layers * 2 * row * 2
        self.bytes = {"graft": graft_b, "decode_steps": app_b + dec_b}
        self.phases = ["graft", "decode_steps"]
        self.batch_bids = [self.bids[b] for sq in range(nS) for b in self.ids[sq]]
        self.batch_seqs = [sq for sq in range(nS) for _ in self.ids[sq]]
        self.step_k = [self.kd[:, t * nS:(t + 1) * nS].contiguous() for t in range(self.steps)]
        self.step_v = [self.vd[:, t * nS:(t + 1) * nS].contiguous() for t in range(self.steps)]
        self.set_consecutive(consecutive)

    def set_consecutive(self, consecutive):
        """Own positions (False) or blocks 2-4 of each sequence re-based by the
        tokens already in it (True), from the next step on."""
        nS = syn.BATCHED_SEQS
        self.consecutive = consecutive
        self.batch_deltas = ([int(sum(int(self.lens[b]) for b in self.ids[sq][:i])) for sq in range(nS)
                              for i in range(len(self.ids[sq]))] if consecutive else None)

    def run_step(self, ev=None):
        kvg, s, c = self.kvg, self.stream, self.cache.h
        nS = syn.BATCHED_SEQS
        m = ev["main"] if ev else None
        if m: m[0].record(s)
        for sq in range(nS):
            kvg.kvg_cache_release(c, sq, s)
        # the 128 grafts (4 stitched blocks per sequence) in one batched call
        kvg.kvg_graft_batch(self.store.h, self.batch_bids, c, self.batch_seqs, 0, s, deltas=self.batch_deltas)
        if m: m[1].record(s)
        seqs = list(range(nS))
        for t in range(self.steps):
            kvg.kvg_cache_append_batch(c, seqs, self.step_k[t].data_ptr(), self.step_v[t].data_ptr(),
                                       self.pos[t].data_ptr(), s)
            kvg.kvg_decode_attention(c, -1, seqs, self.q.data_ptr(), self.w.n_q_heads, self.out.data_ptr(),
                                     self.scale, s)
        if m: m[2].record(s)

class StepDeep:
    """Deep-store paging on a 2-layer slice of the 12B shape: 1,394 blocks x
    2,048 tokens in pinned host memory, each with a planted needle (one key
    row aligned with the query, a value row tagged with the block's index).
    One step = graft of one block chosen uniformly over the store's depth,
    read by the kernel straight from host memory, + decode over it."""

    def __init__(self, kvg, device, stream, n_blocks=syn.DEEP_BLOCKS):
        self.kvg, self.stream = kvg, stream
        self.w = w = syn.DEEP
        P = w.page_size
        self.n_blocks = n_blocks
        self.nb = syn.DEEP_BLOCK
        self.dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0)
        self.cache = kvg.Cache(self.dims, syn.DEEP_CTX // P + self.nb // P, 2, syn.DEEP_CTX)
        blk_bytes = w.n_layers * 2 * (self.nb // P) * w.page_bytes
        self.blk_bytes = blk_bytes
        self.store = kvg.Store(self.dims, kvg.KVG_RESIDENCY_PINNED_HOST, n_blocks * (blk_bytes + (1 << 20)) + (2 << 30))
        c = self.cache.h
        # one query per kv head (both query heads of a group equal), unit norm * sqrt(D)
        q = syn.queries(w, w.n_layers, 1, w.seed, device).float()
        q = q.view(w.n_layers, 1, w.n_kv_heads, w.group, w.head_dim)[:, :, :, :1].expand(-1, -1, -1, w.group, -1)
        q = q / q.norm(dim=-1, keepdim=True) * math.sqrt(w.head_dim)
        self.q = q.reshape(w.n_layers, 1, w.n_q_heads, w.head_dim).to(torch.bfloat16).contiguous()
        qhat = self.q.float()[:, 0].view(w.n_layers, w.n_kv_heads, w.group, w.head_dim)[:, :, 0]
        self.needle_pos = [(b * 7919) % self.nb for b in range(n_blocks)]
        self.qhat = qhat
        with torch.cuda.stream(stream):
            for b in range(n_blocks):
                k, v = self.block_rows(b, device)
                pos = torch.arange(self.nb, dtype=torch.int32, device=device)
                kvg.kvg_cache_append(c, 1, k.data_ptr(), v.data_ptr(), pos.data_ptr(), self.nb, stream)
                kvg.kvg_deposit(self.store.h, c, 1, 0, self.nb, stream)
                kvg.kvg_cache_release(c, 1, stream)
            self.out = torch.empty_like(self.q)
        stream.synchronize()
        self.order = syn.deep_plan(n_blocks=n_blocks)
        self.scale = 1.0 / math.sqrt(w.head_dim)
        self.k_iter = 0
        # the next block's host-page translations are resolved (on a side
        # stream, while the current graft runs) before it is grafted
        self.prefetch = True
        self.side = torch.cuda.Stream(device)
        self.ev_start, self.ev_pf = torch.cuda.Event(), torch.cuda.Event()
        self.pf_for = None
        self.bytes = {"host_graft": blk_bytes, "decode": w.n_layers * 2 * self.nb * w.n_kv_heads * w.head_dim * 2}
        self.phases = ["release", "host_graft", "decode"]

    def block_rows(self, b, device):
        """Input rows of block b: N(0,1) K/V with the needle planted at row
        needle_pos[b] (key = 24 * unit query of each kv head, value = tag(b))."""
        w = self.w
        k, v = syn.kv_rows(w, self.nb, w.seed + b, device)
        t = self.needle_pos[b]
        k[:, t] = (self.qhat.to(device) * (24.0 / math.sqrt(w.head_dim))).to(torch.bfloat16)
        v[:, t] = self.tag(b)
        return k, v

    @staticmethod
    def tag(b):
        """The block's needle value: k/64 with |k| <= 127, exact in bf16."""
        return float(((b * 37) % 255) - 127) / 64.0

    def graft(self, b, nxt):
        """Grafts block b on the step's stream; with prefetch, first waits
        for b's prefetch (issued during the previous graft) and issues the
        next block's on the side stream, to run beside this graft."""
        kvg, s = self.kvg, self.stream
        if self.prefetch:
            if self.pf_for == b:
                s.wait_event(self.ev_pf)
            self.ev_start.record(s)
            self.side.wait_event(self.ev_start)
            kvg.kvg_store_prefetch(self.store.h, nxt, self.side)
            self.ev_pf.record(self.side)
            self.pf_for = nxt
        kvg.kvg_graft(self.store.h, b, self.cache.h, 0, -1, 0, 0, s)

    def run_step(self, ev=None):
        kvg, s, c = self.kvg, self.stream, self.cache.h
        b = int(self.order[self.k_iter % len(self.order)])
        nxt = int(self.order[(self.k_iter + 1) % len(self.order)])
        self.k_iter += 1
        m = ev["main"] if ev else None
        if m: m[0].record(s)
        kvg.kvg_cache_release(c, 0, s)
        if m: m[1].record(s)
        self.graft(b, nxt)
        if m: m[2].record(s)
        kvg.kvg_decode_attention(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads, self.out.data_ptr(),
                                 self.scale, s)
        if m: m[3].record(s)
        return b

    def needle_error(self, b):
        """Max |o - tag(b)| over all heads and layers after grafting block b."""
        o = self.out.float()
        return float((o - self.tag(b)).abs().max())


def graft_latencies(kvg, st, stream, blocks, per_hold=100, cycles_per_graft=1_000_000):
    """GPU time (ms) of each graft of the listed blocks of a StepDeep, run back
    to back, and for each whether its launch may have reached the GPU late.
    The grafts go in groups of per_hold: the stream first runs torch's
    cycle-counted sleep kernel (about 0.5 ms per graft of the group at
    2 GHz) while the host enqueues the group's releases, grafts and events,
    so the GPU then runs the group with no launch gap between grafts and no
    idle time before them; a group whose enqueue outlasted half its hold is
    flagged (its times may include launch gaps)."""
    n = len(blocks)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(min(n, per_hold))]
    out, late = [], []
    hold = getattr(torch.cuda, "_sleep", None)  # a private torch helper: without it, no hold
    with torch.cuda.stream(stream):
        for g0 in range(0, n, per_hold):
            grp = blocks[g0:g0 + per_hold]
            if hold is not None:
                hold(cycles_per_graft * len(grp))
            t0 = time.perf_counter()
            for i, b in enumerate(grp):
                nxt = int(blocks[(g0 + i + 1) % n])
                kvg.kvg_cache_release(st.cache.h, 0, stream)
                ev[i][0].record(stream)
                st.graft(int(b), nxt)
                ev[i][1].record(stream)
            slow = hold is None or time.perf_counter() - t0 > 0.5 * cycles_per_graft * len(grp) / 2.0e9
            stream.synchronize()
            for i in range(len(grp)):
                out.append(ev[i][0].elapsed_time(ev[i][1]))
                late.append(slow)
    return np.array(out), np.array(late)


def measure_h2d(device, nbytes=32 << 20, reps=20):
    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    d = torch.empty(nbytes, dtype=torch.uint8, device=device)
    for _ in range(3):
        d.copy_(h, non_blocking=True)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        d.copy_(h, non_blocking=True)
    e1.record()
    torch.cuda.synchronize()
    return nbytes * reps / (e0.elapsed_time(e1) * 1e-3) / 1e9


def measure_other(kvg, device, config, steps, warmup, layers=0, deep_blocks=syn.DEEP_BLOCKS,
                  consecutive=False, st=None, batched_store=syn.BATCHED_STORE):
    """Builds (unless st is given) and times one of the other workloads;
    returns its JSON line (with the set-up time and the clocks of its own
    timed region)."""
    stream = torch.cuda.Stream(device)
    hbm_peak, sm_max, peak_kind = load_peaks()
    mk = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    t_setup = time.perf_counter()
    if st is not None:
        st.stream = stream
    elif config == "tiny":
        st = StepTiny(kvg, device, stream)
    elif config == "31b":
        st = Step31B(kvg, device, stream, layers)
    elif config == "batched":
        st = StepBatched(kvg, device, stream, layers or 4, consecutive=consecutive, n_store=batched_store)
    else:
        st = StepDeep(kvg, device, stream, deep_blocks)
    setup_s = time.perf_counter() - t_setup
    st.run_step()
    kvg.kvg_sync(st.cache.h, stream, 60.0)
    for _ in range(warmup):
        st.run_step()
    stream.synchronize()
    K = steps
    n_ev = len(st.phases) + 1
    evs = [{"main": [mk() for _ in range(n_ev)]} for _ in range(K)]
    clocks = Clocks(device.index or 0)
    launches0 = kvg.kvg_launch_count()
    t0, t1 = mk(), mk()
    blocks = []
    torch.cuda.nvtx.range_push("kvg_timed")
    t0.record(stream)
    for k in range(K):
        r = st.run_step(ev=evs[k])
        blocks.append(r)
    t1.record(stream)
    torch.cuda.nvtx.range_pop()
    stream.synchronize()
    launches = kvg.kvg_launch_count() - launches0
    clk = clocks.stop()
    kvg.kvg_sync(st.cache.h, stream, 60.0)
    ms_step = t0.elapsed_time(t1) / K
    phase_ms = {p: [evs[k]["main"][i].elapsed_time(evs[k]["main"][i + 1]) for k in range(K)]
                for i, p in enumerate(st.phases)}
    step_bytes = sum(st.bytes.values())
    parts = {}
    for p, ts in phase_ms.items():
        ms = statistics.mean(ts)
        parts[p] = {"ms": round(ms, 4)}
        if p in st.bytes:
            gbs = st.bytes[p] / (ms * 1e-3) / 1e9
            parts[p].update({"algorithmic_bytes": st.bytes[p], "gbs": round(gbs, 1),
                             "hbm_frac": round(gbs / hbm_peak, 3)})
    line = {"metric": METRIC, "unit": "GB/s", "n_gpus": 1, "steps": K, "warmup": warmup,
            "ms_per_step": round(ms_step, 4), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic", "parts": parts, "gpu_launches": int(launches), "clocks": clk,
            "setup_s": round(setup_s, 1)}
    if config == "tiny":
        line["value"] = round(step_bytes / (ms_step * 1e-3) / 1e9, 2)
        line["config"] = {"workload": "tiny: L2 Hq4/Hkv2 D64 P16, 256-token block grafted at own positions "
                                      "(digest-verified), decode 1 token over 256 rows; launch-bound"}
        line["parts"]["decode"]["tokens_per_s"] = round(1e3 / statistics.mean(phase_ms["decode"]), 1)
        first = _sha_tensor(st.out)
        st.run_step()
        stream.synchronize()
        line["checks"] = {"deterministic": _sha_tensor(st.out) == first}
    elif config == "31b":
        line["value"] = round(step_bytes / (ms_step * 1e-3) / 1e9, 2)
        line["config"] = {"workload": f"31b-relocation: L{st.w.n_layers} Hq32/Hkv16 D128 P64 theta 1e6, 16384-token "
                                      "block re-based by delta (0,1,4096,100000 across 8 sequences; 4096 timed), "
                                      "decode batch 8 over 65536-token contexts"}
        line["parts"]["decode"]["tokens_per_s"] = round(st.B * 1e3 / statistics.mean(phase_ms["decode"]), 1)
        line["roofline"] = _part_roofline(line["parts"], "decode", "decode_kernel", hbm_peak, peak_kind)
    elif config == "batched":
        line["value"] = round(step_bytes / (ms_step * 1e-3) / 1e9, 2)
        line["config"] = {"workload": f"batched-library: L{st.w.n_layers} slice of 12b, 32 seqs x 4 blocks "
                                      f"U{{2048..6144}} from a {st.n_store}-block HBM store, then 64 decode steps "
                                      "(batch 32)"
                                      + (" [blocks 2-4 re-based to consecutive positions]" if st.consecutive
                                         else "")}
        line["parts"]["decode_steps"]["tokens_per_s"] = round(
            syn.BATCHED_SEQS * st.steps * 1e3 / statistics.mean(phase_ms["decode_steps"]), 1)
        line["roofline"] = _part_roofline(line["parts"], "decode_steps", "decode_kernel", hbm_peak, peak_kind)
    else:
        # The timed loop above keeps the GPU busy (a step's host calls take
        # ~25 us, its GPU work ~0.2 ms).  A graft of a block whose host pages
        # the GPU has not read recently is slower until their address
        # translations are resolved, hence the prefetch of the next block.
        # The per-graft latency distribution is taken in a second pass over
        # the same blocks, enqueued while a short GPU sleep holds the stream.
        g_all, late = graft_latencies(kvg, st, stream, blocks)
        keep = ~late if (~late).sum() >= len(late) // 2 else np.ones(len(late), bool)
        g = g_all[keep]
        depth = np.array(blocks, dtype=np.float64)[keep]
        slope = float(np.polyfit(depth, g, 1)[0]) if len(set(depth.tolist())) > 1 else 0.0
        h2d = measure_h2d(device)
        # the same loop without the prefetch, over another random schedule
        saved = st.order
        st.order, st.k_iter, st.prefetch = syn.deep_plan(seed=st.w.seed + 1, n_blocks=st.n_blocks), 0, False
        evs_np = [{"main": [mk() for _ in range(n_ev)]} for _ in range(K)]
        for k in range(K):
            st.run_step(ev=evs_np[k])
        stream.synchronize()
        st.order, st.k_iter, st.prefetch = saved, 0, True
        g_np = statistics.mean(evs_np[k]["main"][1].elapsed_time(evs_np[k]["main"][2]) for k in range(K))
        # the headline: the timed loop's random grafts (mean GPU time of the
        # graft phase), not the second pass over the same blocks
        gbs = line["parts"]["host_graft"]["gbs"]
        line["value"] = round(gbs, 2)
        line["unit"] = "GB/s host->HBM"
        line["config"] = {"workload": f"deep-store: 2-layer 12b slice, {st.n_blocks} blocks x 2048 tokens "
                                      f"({st.n_blocks * 2048} tokens, {st.n_blocks * st.blk_bytes / 1e9:.1f} GB) in "
                                      "pinned host memory, uniform random grafts"}
        line["roofline"] = {"bound": "host-link", "kernel": "graft_kernel", "achieved": round(gbs, 1),
                            "peak": round(h2d, 1), "unit": "GB/s", "frac": round(gbs / h2d, 3),
                            "peak_kind": "measured in-run: pinned cudaMemcpy H2D, 32 MiB"}
        line["latency_ms"] = {"n": len(g), "mean": round(float(g.mean()), 4), "p50": round(float(np.percentile(g, 50)), 4),
                              "p99": round(float(np.percentile(g, 99)), 4), "max": round(float(g.max()), 4),
                              "slope_ms_per_1000_blocks_depth": round(slope * 1000, 5),
                              "late_launches_left_out": int(len(g_all) - len(g)),
                              "p99_all": round(float(np.percentile(g_all, 99)), 4),
                              "how": "GPU time of each graft (CUDA events), grafts run back to back in groups of "
                                     "100 enqueued while the stream is held; a group whose enqueue outlasted half "
                                     "the hold is left out"}
        # the host graft is bound by the host link, not HBM
        hg = line["parts"]["host_graft"]
        hg.pop("hbm_frac", None)
        hg["link_frac"] = round(hg["gbs"] / h2d, 3)
        hg["note"] = ("timed loop: uniform random grafts over the whole store, each block's host-page "
                      "translations prefetched beside the previous graft (kvg_store_prefetch)")
        line["parts"]["host_graft_no_prefetch"] = {
            "ms": round(g_np, 4), "algorithmic_bytes": st.blk_bytes,
            "gbs": round(st.blk_bytes / (g_np * 1e-3) / 1e9, 1),
            "link_frac": round(st.blk_bytes / (g_np * 1e-3) / 1e9 / h2d, 3),
            "note": "the same loop over another random schedule without the prefetch"}
        line["parts"]["host_graft_gpu"] = {"ms": round(float(g.mean()), 4), "algorithmic_bytes": st.blk_bytes,
                                           "gbs": round(st.blk_bytes / (g.mean() * 1e-3) / 1e9, 1),
                                           "link_frac": round(st.blk_bytes / (g.mean() * 1e-3) / 1e9 / h2d, 3),
                                           "note": "second pass over the timed loop's blocks (latency_ms)"}
        errs = []
        # needle check on 8 sampled blocks
        for b in sorted(set(int(x) for x in blocks))[:8]:
            st.order = np.array([b])
            st.k_iter = 0
            st.run_step()
            stream.synchronize()
            errs.append(st.needle_error(b))
        line["checks"] = {"needle_max_abs_err": max(errs), "needles_checked": len(errs)}
    line["_step"] = st
    return line


def run_other(args):
    from paper_2607_14431_gb300 import build
    build.build()
    from paper_2607_14431_gb300 import kvg
    torch.cuda.set_device(0)
    line = measure_other(kvg, torch.device("cuda", 0), args.config, args.steps, args.warmup, args.layers,
                         args.deep_blocks, args.consecutive, batched_store=args.batched_store)
    line.pop("_step")
    print(json.dumps(line), flush=True)


def _close_step(st):
    for name in ("cache", "store", "hstore"):
        o = getattr(st, name, None)
        if o is not None:
            o.close()
    torch.cuda.synchronize()


def _compact(line, keep_parts):
    """The figures of a workload line that the default line carries."""
    out = {"workload": line["config"]["workload"], "value": line["value"], "unit": line["unit"],
           "ms_per_step": line["ms_per_step"], "steps": line["steps"], "warmup": line["warmup"],
           "setup_s": line["setup_s"], "clocks": line["clocks"],
           "parts": {p: line["parts"][p] for p in keep_parts if p in line["parts"]}}
    for k in ("roofline", "latency_ms", "checks"):
        if k in line:
            out[k] = line[k]
    return out


def run_workloads(args):
    """The other four workloads, each built, timed (with its own clock
    record) and freed in turn, for the default line's `workloads` object.
    The 31B workload runs at its full 60 layers, the batched library at its
    4-layer slice (own positions, then re-based to consecutive positions),
    the deep store with its full 1,394 blocks and 1,000 random grafts."""
    from paper_2607_14431_gb300 import kvg
    device = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    out = {}
    t_all = time.perf_counter()
    plan = [("tiny", dict(steps=500, warmup=5), ("graft_verify", "decode")),
            ("31b", dict(steps=5, warmup=3, layers=args.workload_31b_layers), ("relocate", "decode")),
            ("batched", dict(steps=3, warmup=3), ("graft", "decode_steps")),
            ("deep", dict(steps=syn.DEEP_GRAFTS, warmup=5),
             ("host_graft", "host_graft_no_prefetch", "host_graft_gpu", "decode"))]
    for name, kw, keep in plan:
        try:
            line = measure_other(kvg, device, name, kw["steps"], kw["warmup"], kw.get("layers", 0))
            st = line.pop("_step")
            out[name] = _compact(line, keep)
            if name == "batched":
                # the same store and sequences, blocks 2-4 re-based by the
                # tokens before them (per-graft deltas in the one batched call)
                st.set_consecutive(True)
                line = measure_other(kvg, device, name, kw["steps"], kw["warmup"], st=st)
                line.pop("_step")
                line["setup_s"] = 0.0
                out["batched_consecutive"] = _compact(line, keep)
            _close_step(st)
            del st, line
        except Exception as e:  # reported in the line, never hidden
            out[name] = {"error": f"{type(e).__name__}: {e}"[:300]}
        gc.collect()
        torch.cuda.empty_cache()
    out["total_s"] = round(time.perf_counter() - t_all, 1)
    return out


def _part_roofline(parts, part, kernel, hbm_peak, peak_kind):
    """Roofline object of a workload's longest part (HBM-bound): its
    algorithmic bytes over its CUDA-event time against the measured copy
    peak; no ncu traffic is kept for these workloads."""
    p = parts[part]
    return {"bound": "hbm", "kernel": kernel, "part": part, "achieved": p["gbs"], "peak": round(hbm_peak, 1),
            "unit": "GB/s", "frac": p["hbm_frac"], "traffic": None, "peak_kind": peak_kind}


def _sha_tensor(t):
    import hashlib
    return hashlib.sha256(t.detach().contiguous().view(torch.int16).cpu().numpy().tobytes()).hexdigest()


# --------------------------------------------------------------------------
# CPU oracle on a bounded sample of the same step
# --------------------------------------------------------------------------

def oracle_sample(n_layers_sample: int, chunk: int = 4):
    """One oracle pass of the 12B step over n_layers_sample layers, run in
    chunks of `chunk` layers (inputs are generated per chunk, untimed).
    Returns (seconds, algorithmic bytes of the sample, threads used)."""
    import oracle
    nb, nf = syn.B12_BLOCK, syn.B12_CTX - syn.B12_BLOCK
    total_t, total_b = 0.0, 0
    for c0 in range(0, n_layers_sample, chunk):
        w = syn.B12.with_layers(min(chunk, n_layers_sample - c0))
        k, v = syn.kv_rows(w, syn.B12_CTX, w.seed + c0)
        k, v = syn.as_u16(k), syn.as_u16(v)
        q = syn.as_u16(syn.queries(w, w.n_layers, 1, w.seed + c0))
        d = oracle.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)
        blk = oracle.block_from_kv(d, k[:, :nb], v[:, :nb], syn.positions(0, nb))
        cache = oracle.OracleCache(d, syn.B12_CTX // w.page_size, 1, syn.B12_CTX)
        scale = 1 / math.sqrt(w.head_dim)
        t0 = time.perf_counter()
        cache.graft(0, blk)
        pages = np.stack([cache.pool[l, kv, cache.page_table[0, j]] for l in range(w.n_layers)
                          for kv in range(2) for j in range(blk.n_pages)])
        dig = oracle.page_digests(pages.reshape(-1), w.page_bytes)
        assert np.array_equal(dig.reshape(blk.digests.shape), blk.digests)
        cache.append(0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
        for l in range(w.n_layers):
            cache.decode(0, l, q[l, 0], scale)
        total_t += time.perf_counter() - t0
        blk_pages = w.n_layers * 2 * (nb // w.page_size) * w.page_bytes
        # HBM algorithmic bytes, as the GPU step counts them: block copied,
        # fresh rows read and written, every row decoded (hashing adds none)
        total_b += 2 * blk_pages + 2 * w.n_layers * 2 * nf * w.n_kv_heads * w.head_dim * 2 \
            + w.n_layers * 2 * syn.B12_CTX * w.n_kv_heads * w.head_dim * 2
    return total_t, total_b, oracle.omp_threads()


def oracle_single_thread(n_layers_sample=2):
    """The oracle on one host thread (OMP_NUM_THREADS=1 in a fresh
    interpreter, started by exec, never forked from this CUDA process)."""
    code = ("import json, sys; sys.path.insert(0, %r); import bench; "
            "print(json.dumps(bench.oracle_sample(%d)))" % (os.path.dirname(os.path.abspath(__file__)),
                                                          n_layers_sample))
    env = dict(os.environ, OMP_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    if r.returncode != 0:
        raise RuntimeError("single-thread oracle run failed: " + r.stderr[-2000:])
    dt, b, threads = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": round(b / dt / 1e9, 4), "unit": "GB/s", "threads": threads,
            "sample": f"{n_layers_sample} of 48 layers of one 12b step on one thread: {dt:.2f} s"}


def cpu_baseline(n_layers_sample=48, single_thread_layers=2):
    dt, b, cores = oracle_sample(n_layers_sample)
    out = {"value": round(b / dt / 1e9, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
           "sample": f"{n_layers_sample} of 48 layers of one 12b step (graft, page digests, 24576-row "
                     f"append, fp64 decode of 16 heads over 32768 rows), in 4-layer chunks: {dt:.2f} s"}
    if single_thread_layers > 0:
        out["single_thread"] = oracle_single_thread(single_thread_layers)
    return out


def run_files(args):
    """Block files (the paper's persistent medium): the 12B block (3.2 GB) is
    saved to a file and loaded back, into an HBM store and into a pinned-host
    store, with and without the digest check, each timed over --steps
    transfers.  The file stays in the page cache (as in the paper's restore
    timings); the reads and writes are host-memory copies."""
    import tempfile
    from paper_2607_14431_gb300 import build
    build.build()
    from paper_2607_14431_gb300 import kvg
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    stream, side = torch.cuda.Stream(device), torch.cuda.Stream(device)
    st = Step12B(kvg, device, stream, side)
    digest = bytes(kvg.kvg_store_block_info(st.store.h, st.bid).block_digest)
    tmp = tempfile.mkdtemp(prefix="kvg_files_")
    path = os.path.join(tmp, "block.kvg")
    kvg.kvg_store_save(st.store.h, st.bid, path)
    size = os.path.getsize(path)

    n = max(3, min(args.steps, 8))
    parts = {}
    # one store per residency with room for every load: its first (untimed)
    # load allocates the bounce buffers; each timed load adds a block (and
    # allocates that block's slab, which is part of a store's growth)
    for name, res, flags in (("load_hbm_verified", kvg.KVG_RESIDENCY_HBM, kvg.KVG_GRAFT_VERIFY),
                             ("load_hbm", kvg.KVG_RESIDENCY_HBM, 0),
                             ("load_pinned_host_verified", kvg.KVG_RESIDENCY_PINNED_HOST, kvg.KVG_GRAFT_VERIFY),
                             ("load_pinned_host", kvg.KVG_RESIDENCY_PINNED_HOST, 0)):
        store = kvg.Store(st.dims, res, (n + 1) * (size + (1 << 20)))
        kvg.kvg_store_load(store.h, path, flags)
        ts = []
        for _ in range(n):
            t0 = time.perf_counter()
            bid = kvg.kvg_store_load(store.h, path, flags)
            ts.append(time.perf_counter() - t0)
            assert bytes(kvg.kvg_store_block_info(store.h, bid).block_digest) == digest
        store.close()
        sec = statistics.median(ts)
        parts[name] = {"ms": round(sec * 1e3, 2), "gbs": round(size / sec / 1e9, 2)}
    # saves: each to a new file, removed outside the timed region
    for name, store, bid in (("save_from_hbm", st.store.h, st.bid), ("save_from_pinned_host", st.hstore.h, st.hbid)):
        ts = []
        for k in range(n + 1):
            out = os.path.join(tmp, f"save{k}.kvg")
            t0 = time.perf_counter()
            kvg.kvg_store_save(store, bid, out)
            if k:
                ts.append(time.perf_counter() - t0)
            os.remove(out)
        sec = statistics.median(ts)
        parts[name] = {"ms": round(sec * 1e3, 2), "gbs": round(size / sec / 1e9, 2)}
    # restore latency against block length, the paper's disk-to-GPU restore
    # table's lengths (its figures include an HTTP round trip): block file ->
    # HBM store with every digest checked -> verified graft into an empty
    # sequence of the cache, one block length at a time
    restore = {}
    pb = torch.arange(st.nb, dtype=torch.int32, device=device)
    kvg.kvg_cache_append(st.cache.h, 1, st.kb.data_ptr(), st.vb.data_ptr(), pb.data_ptr(), st.nb, stream)
    for n_tok in (748, 1495, 2990, 5977):
        src_store = kvg.Store(st.dims, kvg.KVG_RESIDENCY_HBM, 4 << 30)
        bid = kvg.kvg_deposit(src_store.h, st.cache.h, 1, 0, n_tok, stream)
        f = os.path.join(tmp, f"block_{n_tok}.kvg")
        kvg.kvg_store_save(src_store.h, bid, f)
        src_store.close()
        nbytes = os.path.getsize(f)
        # room for every load: a block takes its own slab, or a share of a 1 GiB one
        store = kvg.Store(st.dims, kvg.KVG_RESIDENCY_HBM, (n + 1) * max(nbytes + (1 << 20), (1 << 30) + (1 << 20)))
        kvg.kvg_store_load(store.h, f, kvg.KVG_GRAFT_VERIFY)  # untimed: the store's first transfer
        ts = []
        for _ in range(n):
            kvg.kvg_cache_release(st.cache.h, 0, stream)
            stream.synchronize()
            t0 = time.perf_counter()
            b2 = kvg.kvg_store_load(store.h, f, kvg.KVG_GRAFT_VERIFY)
            kvg.kvg_graft(store.h, b2, st.cache.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, stream)
            ts.append(time.perf_counter() - t0)
        store.close()
        os.remove(f)
        restore[str(n_tok)] = {"block_bytes": nbytes, "ms": round(statistics.median(ts) * 1e3, 2)}
    kvg.kvg_cache_release(st.cache.h, 1, stream)
    stream.synchronize()
    parts["restore_from_file_then_graft_verified"] = restore
    os.remove(path)
    os.rmdir(tmp)
    v = parts["load_hbm_verified"]
    line = {"metric": "block file -> HBM store GB/s (digest-verified load of the 12b block, page cache warm)",
            "value": v["gbs"], "unit": "GB/s", "n_gpus": 1, "steps": n, "warmup": args.warmup,
            "ms_per_step": v["ms"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "u8", "data": "synthetic",
            "config": {"workload": f"block files: the 12b block ({size} bytes) saved and loaded back; reads "
                                   f"in 16 MiB chunks by up to 8 threads, HBM stores through pinned bounce "
                                   f"buffers", "cores": len(os.sched_getaffinity(0))},
            "parts": parts}
    print(json.dumps(line), flush=True)


def config_12b(n_layers=48, world=1, pool_store=False, swa=None, kv="bf16"):
    """The 12b workload's config entry, shared by both arms of the bench."""
    return {"workload": f"12b-single-graft: L{n_layers} Hq16/Hkv8 D256 P64, 8192-token block grafted "
                        "at own positions (digest-verified) + 24576 fresh tokens, decode 1 token over 32768"
                        + (" [block in the cache pool: zero-copy graft]" if pool_store else "")
                        + (f" [sliding-window layers: window {swa[0]}, every {swa[1]}th layer global]" if swa else "")
                        + (f" [fp8 E4M3 KV, scales k {syn.FP8_K_SCALE} v {syn.FP8_V_SCALE}]" if kv == "e4m3" else ""),
            "global_batch": world, "seq_len": syn.B12_CTX, "parallelism": f"replicas{world}",
            "l2": ("inputs larger than L2 (3 GiB block, 9.7 GB fresh rows, 12.9 GB cache)" if kv == "bf16" else
                   "inputs larger than L2 (1.6 GB fp8 block, 9.7 GB bf16 fresh rows, 6.4 GB fp8 cache)"),
            "seed": hex(syn.B12.seed)}


def run_reference(args):
    ts, b, cores = [], 0, 1
    for k in range(args.warmup + args.steps):
        dt, b, cores = oracle_sample(1)
        if k >= args.warmup:
            ts.append(dt)
    t = statistics.mean(ts)
    value = b / t / 1e9
    cb = {"value": round(value, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
          "sample": "1 of 48 layers of one 12b step per timed step"}
    return {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t * 1e3, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_12b(world=args.gpus),
            "cpu_baseline": cb, "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                                        "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="kvg", choices=["kvg", "reference"])
    ap.add_argument("--cpu-baseline-layers", type=int, default=48)
    ap.add_argument("--layers", type=int, default=0, help="layer count override (small profiling cases)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--config", default="12b", choices=["12b", "tiny", "31b", "batched", "deep", "files"])
    ap.add_argument("--schedule", default="fused", choices=["overlap", "fused"],
                    help="12b step: digest check on a side stream after the graft (overlap) or folded "
                         "into the graft, which runs beside the append (fused)")
    ap.add_argument("--swa", default="", help="12b step with sliding-window layers, 'W:R' (window W, every "
                                              "R-th layer global), over the full-size cache")
    ap.add_argument("--kv", default="bf16", choices=["bf16", "e4m3"],
                    help="12b step: KV element type of the cache and the block (e4m3: quantized KV blocks)")
    ap.add_argument("--store", default="hbm", choices=["hbm", "pool"],
                    help="12b: block in an HBM store (copying graft) or in the cache pool (zero-copy graft)")
    ap.add_argument("--deep-blocks", type=int, default=syn.DEEP_BLOCKS)
    ap.add_argument("--batched-store", type=int, default=syn.BATCHED_STORE,
                    help="batched: blocks in the store (512; fewer for small profiling cases)")
    ap.add_argument("--consecutive", action="store_true",
                    help="batched: re-base blocks 2-4 of each sequence so its position tags are consecutive")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="12b: leave out the other four workloads (tiny, 31b, batched, deep) from the line")
    ap.add_argument("--workload-31b-layers", type=int, default=0,
                    help="layers of the 31b workload in the default line (0: all 60)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return
    if args.config == "files":
        if rank == 0:
            run_files(args)
        return
    if args.config != "12b":
        if rank == 0:
            run_other(args)
        return
    if world > 1:
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        torch.distributed.init_process_group("nccl")
    line = run_kvg(args, rank, world)
    if rank == 0:
        default_step = not (args.swa or args.kv != "bf16" or args.store != "hbm" or args.layers)
        if world == 1 and default_step and not args.no_workloads:
            gc.collect()
            torch.cuda.empty_cache()
            line["workloads"] = run_workloads(args)
        # the CPU baseline runs at N = 1 only (at N > 1 the other ranks would wait on it)
        if world == 1 and not args.no_cpu_baseline and not args.swa and args.kv == "bf16":
            line["cpu_baseline"] = cpu_baseline(args.cpu_baseline_layers)
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
