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
SHA_OPS_PER_BLOCK = 1400  # fused 32-bit ops per SHA-256 compression (rotate, 3-input logic/add = 1)


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p.get("sm_max_mhz", 2070.0)), "measured"
    except Exception:
        return 6800.0, 2070.0, "fallback"


def load_traffic():
    """Per-launch DRAM bytes from the committed ncu summary, keyed by kernel,
    kept only while the kernel source is unchanged since the capture."""
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
            out[parts["kernel"]] = float(parts["bytes_per_launch"])
    return out


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
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
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
        sm = [float(s[0]) for s in self.samples if len(s) >= 7 and s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in self.samples if len(s) >= 7 and s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in self.samples if len(s) >= 7 for i in range(4)
                          if s[3 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(sm)}


# --------------------------------------------------------------------------
# 12B-class single graft: the default workload
# --------------------------------------------------------------------------

class Step12B:
    """Device state and the per-step call sequence for the 12B workload."""

    def __init__(self, kvg, device, stream):
        self.kvg = kvg
        self.w = w = syn.B12
        self.dev = device
        self.stream = stream
        self.nb, self.nf = syn.B12_BLOCK, syn.B12_CTX - syn.B12_BLOCK
        P = w.page_size
        self.dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0)
        n_pages = syn.B12_CTX // P + self.nb // P
        self.cache = kvg.Cache(self.dims, n_pages, 2, syn.B12_CTX)
        self.store = kvg.Store(self.dims, kvg.KVG_RESIDENCY_HBM, 4 << 30)
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
        stream.synchronize()
        self.kb_cpu_sample = (kb, vb)  # kept on device for the sampled oracle check
        self.scale = 1.0 / math.sqrt(w.head_dim)
        blk_pages = w.n_layers * 2 * (self.nb // P) * w.page_bytes
        self.bytes = {
            "graft": 2 * blk_pages,
            "verify": blk_pages,
            "append": 2 * w.n_layers * 2 * self.nf * w.n_kv_heads * w.head_dim * 2,
            "decode": w.n_layers * 2 * syn.B12_CTX * w.n_kv_heads * w.head_dim * 2
                      + 2 * self.q.numel() * 2,
        }
        self.sha_blocks = (blk_pages // 4096) * 65
        self.phases = ["release", "graft", "verify", "append", "decode"]

    def calls(self, store=None, bid=None):
        kvg, s, c = self.kvg, self.stream, self.cache.h
        store = store or self.store.h
        bid = self.bid if bid is None else bid
        return [
            lambda: kvg.kvg_cache_release(c, 0, s),
            lambda: kvg.kvg_graft(store, bid, c, 0, -1, 0, 0, s),
            lambda: kvg.kvg_verify(store, bid, c, 0, 0, 0, s),
            lambda: kvg.kvg_cache_append(c, 0, self.kf.data_ptr(), self.vf.data_ptr(), self.pf.data_ptr(),
                                         self.nf, s),
            lambda: kvg.kvg_decode_attention(c, -1, [0], self.q.data_ptr(), self.w.n_q_heads,
                                             self.out.data_ptr(), self.scale, s),
        ]

    def sampled_check(self):
        """Oracle attention for two (layer, head) samples of the last step."""
        import oracle
        w = self.w
        kb, vb = self.kb_cpu_sample
        errs = []
        for l, h in [(0, 0), (w.n_layers - 1, w.n_q_heads - 1)]:
            g = h // w.group
            k = torch.cat([kb[l, :, g], self.kf[l, :, g]]).cpu()
            v = torch.cat([vb[l, :, g], self.vf[l, :, g]]).cpu()
            ref = oracle.attention_head(syn.as_u16(self.q[l, 0, h]), syn.as_u16(k), syn.as_u16(v), self.scale)
            got = oracle.bf16_to_f64(syn.as_u16(self.out[l, 0, h]))
            errs.append(float(np.abs(got - ref).max()))
        return max(errs)


def run_kvg(args, rank, world):
    from paper_2607_14431_gb300 import build
    build.build()
    from paper_2607_14431_gb300 import kvg

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    stream = torch.cuda.Stream(device)
    hbm_peak, sm_max, peak_kind = load_peaks()
    st = Step12B(kvg, device, stream)

    # correctness of the configuration being timed: one verified step
    for f in st.calls():
        f()
    kvg.kvg_sync(st.cache.h, stream, 60.0)
    first_sha = _sha_tensor(st.out)

    for _ in range(args.warmup):
        for f in st.calls():
            f()
    stream.synchronize()

    K = args.steps
    n_ph = len(st.phases)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ph + 1)] for _ in range(K)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    launches0 = kvg.kvg_launch_count()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(K):
        calls = st.calls()
        for i, f in enumerate(calls):
            evs[k][i].record(stream)
            f()
        evs[k][n_ph].record(stream)
    t_end.record(stream)
    stream.synchronize()
    launches = kvg.kvg_launch_count() - launches0
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    kvg.kvg_sync(st.cache.h, stream, 60.0)  # digest verification of every timed step passed
    if world > 1:
        t = torch.tensor([total_ms], device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_step = total_ms / K
    phase_ms = {p: statistics.mean(evs[k][i].elapsed_time(evs[k][i + 1]) for k in range(K))
                for i, p in enumerate(st.phases)}
    step_bytes = sum(st.bytes.values())
    value = world * step_bytes / (ms_step * 1e-3) / 1e9
    deterministic = _sha_tensor(st.out) == first_sha
    max_err = st.sampled_check()

    # e2e: host-store graft, query from pinned host memory, output read back
    e2e = None
    if True:
        q_host = torch.empty(st.q.shape, dtype=st.q.dtype, pin_memory=True)
        q_host.copy_(st.q.cpu())
        o_host = torch.empty(st.out.shape, dtype=st.out.dtype, pin_memory=True)
        e2e_calls = st.calls(st.hstore.h, st.hbid)
        ts = []
        for k in range(args.warmup + K):
            t0 = time.perf_counter()
            with torch.cuda.stream(stream):
                st.q.copy_(q_host, non_blocking=True)
            for f in e2e_calls:
                f()
            with torch.cuda.stream(stream):
                o_host.copy_(st.out, non_blocking=True)
            stream.synchronize()
            if k >= args.warmup:
                ts.append(time.perf_counter() - t0)
        kvg.kvg_sync(st.cache.h, stream, 60.0)
        e2e_ms = statistics.mean(ts) * 1e3
        blk_read = st.bytes["verify"]  # block pages read from host memory by the graft
        e2e = {"value": round(world * step_bytes / (e2e_ms * 1e-3) / 1e9, 2), "unit": "GB/s",
               "ms_per_step": round(e2e_ms, 3),
               "h2d_bytes_per_step": int(blk_read + st.q.numel() * 2),
               "d2h_bytes_per_step": int(st.out.numel() * 2),
               "host_graft_gbs": None}
        # host->HBM graft alone (the host-store graft kernel)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        gts = []
        for k in range(5):
            kvg.kvg_cache_release(st.cache.h, 0, stream)
            e0.record(stream)
            kvg.kvg_graft(st.hstore.h, st.hbid, st.cache.h, 0, -1, 0, 0, stream)
            e1.record(stream)
            stream.synchronize()
            gts.append(e0.elapsed_time(e1))
        e2e["host_graft_gbs"] = round(blk_read / (statistics.median(gts) * 1e-3) / 1e9, 2)

    traffic = load_traffic()
    parts = {}
    for p in st.phases:
        ms = phase_ms[p]
        if p == "release":
            parts[p] = {"ms": round(ms, 4)}
            continue
        b = st.bytes[p]
        gbs = b / (ms * 1e-3) / 1e9
        parts[p] = {"ms": round(ms, 4), "algorithmic_bytes": b, "gbs": round(gbs, 1)}
        if p == "verify":
            ops = st.sha_blocks * SHA_OPS_PER_BLOCK
            alu_peak = 152 * 64 * sm_max * 1e6
            parts[p].update({"gops": round(ops / (ms * 1e-3) / 1e9, 1),
                             "alu_frac": round(ops / (ms * 1e-3) / alu_peak, 3)})
        else:
            parts[p]["hbm_frac"] = round(gbs / hbm_peak, 3)
    parts["decode"]["tokens_per_s"] = round(1e3 / phase_ms["decode"], 1)
    kernel_of = {"graft": "graft_kernel", "verify": "sha256_leaves_kernel", "append": "append_kernel",
                 "decode": "decode_split_kernel"}
    dom = max((p for p in st.phases if p != "release"), key=lambda p: phase_ms[p])
    if dom == "verify":
        ops = st.sha_blocks * SHA_OPS_PER_BLOCK
        ach = ops / (phase_ms[dom] * 1e-3) / 1e12
        peak = 152 * 64 * sm_max * 1e6 / 1e12
        roof = {"bound": "alu", "kernel": kernel_of[dom], "achieved": round(ach, 3), "peak": round(peak, 3),
                "unit": "Top/s", "frac": round(ach / peak, 3), "traffic": traffic.get(kernel_of[dom]),
                "peak_kind": "derived: 152 SMs x 64 int32 lanes x max SM clock"}
    else:
        ach = st.bytes[dom] / (phase_ms[dom] * 1e-3) / 1e9
        roof = {"bound": "hbm", "kernel": kernel_of[dom], "achieved": round(ach, 1), "peak": hbm_peak,
                "unit": "GB/s", "frac": round(ach / hbm_peak, 3), "traffic": traffic.get(kernel_of[dom]),
                "peak_kind": peak_kind}
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "12b-single-graft: L48 Hq16/Hkv8 D256 P64, 8192-token block grafted at own "
                               "positions + 24576 fresh tokens, decode 1 token over 32768",
                   "global_batch": world, "seq_len": syn.B12_CTX, "parallelism": f"replicas{world}",
                   "l2": "inputs larger than L2 (3 GiB block, 9.7 GB fresh rows, 12.9 GB cache)"},
        "parts": parts, "roofline": roof, "e2e": e2e, "gpu_launches": int(launches),
        "clocks": clk, "checks": {"sampled_max_abs_err": max_err, "deterministic": deterministic,
                                  "digest_verified_steps": K + args.warmup + 1},
    }
    return line


def _sha_tensor(t):
    import hashlib
    return hashlib.sha256(t.detach().contiguous().view(torch.int16).cpu().numpy().tobytes()).hexdigest()


# --------------------------------------------------------------------------
# CPU oracle on a bounded sample of the same step
# --------------------------------------------------------------------------

def oracle_sample(n_layers_sample: int):
    """One oracle pass of the 12B step restricted to n_layers_sample layers.
    Returns (seconds, algorithmic bytes of the sample, threads used)."""
    import oracle
    w = syn.B12.with_layers(n_layers_sample)
    nb, nf = syn.B12_BLOCK, syn.B12_CTX - syn.B12_BLOCK
    k, v = syn.kv_rows(w, syn.B12_CTX, w.seed)
    k, v = syn.as_u16(k), syn.as_u16(v)
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, w.seed))
    d = oracle.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)
    blk = oracle.block_from_kv(d, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    cache = oracle.OracleCache(d, syn.B12_CTX // w.page_size, 1, syn.B12_CTX)
    scale = 1 / math.sqrt(w.head_dim)
    t0 = time.perf_counter()
    cache.graft(0, blk)
    pages = np.stack([cache.pool[l, kv, cache.page_table[0, j]] for l in range(w.n_layers) for kv in range(2)
                      for j in range(blk.n_pages)])
    dig = oracle.page_digests(pages.reshape(-1), w.page_bytes)
    assert np.array_equal(dig.reshape(blk.digests.shape), blk.digests)
    cache.append(0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    for l in range(w.n_layers):
        cache.decode(0, l, q[l, 0], scale)
    dt = time.perf_counter() - t0
    blk_pages = w.n_layers * 2 * (nb // w.page_size) * w.page_bytes
    b = 2 * blk_pages + blk_pages + 2 * w.n_layers * 2 * nf * w.n_kv_heads * w.head_dim * 2 \
        + w.n_layers * 2 * syn.B12_CTX * w.n_kv_heads * w.head_dim * 2
    return dt, b, oracle.omp_threads()


def cpu_baseline(n_layers_sample=1):
    dt, b, cores = oracle_sample(n_layers_sample)
    return {"value": round(b / dt / 1e9, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
            "sample": f"{n_layers_sample} of 48 layers of one 12b step (graft, page digests, 24576-row "
                      f"append, fp64 decode of 16 heads over 32768 rows): {dt:.2f} s"}


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
    return {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t * 1e3, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": "12b-single-graft (1-layer sample)"},
            "cpu_baseline": cb, "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                                        "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="kvg", choices=["kvg", "reference"])
    ap.add_argument("--cpu-baseline-layers", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return
    if world > 1:
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        torch.distributed.init_process_group("nccl")
    line = run_kvg(args, rank, world)
    if rank == 0:
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(args.cpu_baseline_layers)
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
