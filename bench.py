#!/usr/bin/env python
"""Benchmark of the SideQuest KV-cache hot path on GB300.

Workload (default, "serving-128k"): batched long-horizon serving — 8
requests of 131,072 tokens, each paired with an auxiliary fork (16 decoding
sequences), 32 layers, 32 query / 8 KV heads, head dim 128, page size 64,
bf16.  Synthetic N(0,1) K/V and queries (they stand in for the FRAMES /
BrowseComp agent contexts of the paper's Sec. 4.1, whose lengths pass 100k
tokens, Fig. 2).

One step = one decode token for every sequence: append its K/V row
(all layers) and run decode attention at all 32 layers (each call reads the
shared prefix pages once for main + aux).  Then, timed separately: release
the forks, evict 20-65% of every request in 10-40 spans (Algorithm 1,
clear_kv), re-fork, and decode again.

Prints one JSON line.  `--impl reference` times the CPU oracle on a bounded
sample of the same workload instead (the reference arm).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import shutil
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode-attn tokens/s + achieved HBM GB/s at 128k ctx; span-evict GB/s"
PREFILL_METRIC = "masked-prefill attention tokens/s at 32k ctx (all layers) + achieved bf16 TFLOP/s"
AUX_METRIC = "aux-thread trigger prefill: K/V GB/s read over a 128k shared context (all layers)"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="sq", choices=["sq", "reference"])
    ap.add_argument("--workload", default="serving-128k",
                    choices=["serving-128k", "large-ragged", "agent-32k", "trace", "prefill-32k",
                             "aux-trigger-128k"])
    ap.add_argument("--prefill-ctx", type=int, default=32768, help="prefill-32k: context tokens")
    ap.add_argument("--aux-ctx", type=int, default=131072, help="aux-trigger-128k: context tokens")
    ap.add_argument("--aux-queries", type=int, default=8,
                    help="aux-trigger-128k: trigger-phrase tokens the aux thread prefills")
    ap.add_argument("--turns", type=int, default=50, help="trace: turns per agent")
    ap.add_argument("--requests", type=int, default=8)
    ap.add_argument("--ctx", type=int, default=131072)
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--no-evict", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--ragged", action="store_true",
                    help="trace: evict with sq_evict_spans_ragged")
    ap.add_argument("--no-sub", action="store_true",
                    help="serving-128k at one GPU: skip the other workloads' sub-records")
    return ap.parse_args()


def tensor_peak():
    """Sustained cuBLAS bf16 TFLOP/s (for a kernel timed inside a long step)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["bf16_tflops_sustained"]), "measured (sustained)"
    except Exception:
        return 1700.0, "fallback (sustained)"


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


KERNEL_SOURCES = {
    "sq_decode_splitk_kernel": ["kernels/decode.cu", "kernels/ptx.cuh", "kernels/launch.hpp",
                                "host/plan.hpp"],
    "sq_evict_compact_kernel": ["kernels/kv.cu", "kernels/ptx.cuh", "kernels/launch.hpp",
                                "host/plan.hpp"],
    "sq_prefill_kernel": ["kernels/prefill.cu", "kernels/ptx.cuh", "kernels/tc.cuh",
                          "kernels/launch.hpp", "host/plan.hpp"],
}


def sources_hash(kernel: str) -> str:
    """Hash of a kernel's sources with comments and whitespace removed, so that
    an edit of comments alone does not void a traffic capture."""
    import hashlib
    import re
    m = hashlib.sha256()
    for rel in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2602_22603_gb300", "csrc", rel)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        m.update(" ".join(text.split()).encode())
    return m.hexdigest()[:16]


def recorded_traffic_ratio(kernel: str, workload: str = None):
    """DRAM traffic per algorithmic byte from the ncu capture summarised in
    profiles/, if that capture was taken of the current kernel sources
    (else None).  A kernel captured under several workloads tags each line
    with `workload=`."""
    import re
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir):
        return None, None
    cur = sources_hash(kernel)
    for name in sorted(os.listdir(pdir)):
        if not name.endswith(".md"):
            continue
        with open(os.path.join(pdir, name)) as f:
            for line in f:
                mt = re.search(r"traffic: kernel=(\S+)(?: workload=(\S+))? ratio=([0-9.]+) "
                               r"sources_sha256=([0-9a-f]+)", line)
                if mt and mt.group(1) == kernel and mt.group(2) == workload and mt.group(4) == cur:
                    return float(mt.group(3)), "profiles/" + name
    return None, None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        self.path = None
        exe = shutil.which("nvidia-smi")
        if not exe:
            return
        fd, self.path = tempfile.mkstemp(prefix="sq_clocks_", suffix=".csv")
        os.close(fd)
        self.out = open(self.path, "w")
        self.proc = subprocess.Popen(
            [exe, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
             "-i", str(device_index)], stdout=self.out, stderr=subprocess.DEVNULL)

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


def dist_setup():
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# workload
# ---------------------------------------------------------------------------
def workload_name(args):
    return (f"serving-128k: {args.requests} requests x {args.ctx} tokens + {args.requests} aux forks "
            f"({2 * args.requests} decoding sequences), {args.layers} layers, 32q/8kv heads, d128, "
            f"page 64, bf16")


def read_probe(cache, stream, nbytes=8 << 30, reps=5):
    """Read-only HBM bandwidth of this GPU in this run (sq_probe_read over
    8 GiB, best of 5), reported next to the copy peak."""
    import torch

    import paper_2602_22603_gb300 as sq
    buf = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    st_h = int(stream.cuda_stream)
    sq.sq_probe_read(cache.handle, buf, nbytes, st_h)
    best = 0.0
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        sq.sq_probe_read(cache.handle, buf, nbytes, st_h)
        e1.record(stream)
        torch.cuda.synchronize()
        best = max(best, nbytes / (e0.elapsed_time(e1) / 1e3) / 1e9)
    del buf
    torch.cuda.empty_cache()
    return best


def batched_spec(args):
    """Shapes of the two batched workloads: every request paired with an aux
    fork, all decoding sequences in one call per layer."""
    from synthetic import AGENT_8B, LARGE_70B, random_spans, request_spans, shuffled, sub_seed
    if args.workload == "large-ragged":
        sh = LARGE_70B
        ctxs = [32768, 98304, 196608, 262144]

        def spans(seed, r, n, P):  # 50% of the context in 25 spans
            return shuffled(random_spans(sub_seed(seed, 300 + r), 25, n // 2, P, n,
                                         median=n / 50), r)
        return dict(name=("large-ragged: 4 requests of 32k/96k/192k/262,144 tokens + 4 aux forks "
                          "(8 decoding sequences), 80 layers, 64q/8kv heads, d128, page 64, bf16; "
                          "evict 50% of each in 25 spans"),
                    L=sh.num_layers, Hq=sh.num_q_heads, Hkv=sh.num_kv_heads, D=sh.head_dim,
                    P=sh.page_size, ctxs=ctxs, chunk=2048, spans=spans)
    sh = AGENT_8B
    return dict(name=workload_name(args), L=args.layers, Hq=sh.num_q_heads, Hkv=sh.num_kv_heads,
                D=sh.head_dim, P=sh.page_size, ctxs=[args.ctx] * args.requests, chunk=4096,
                spans=lambda seed, r, n, P: request_spans(seed, r, n, P))


def run_sq(args, world, rank, local):
    import numpy as np
    import torch

    import paper_2602_22603_gb300 as sq
    from synthetic import Bank, bf16_normal, sub_seed

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    spec = batched_spec(args)
    L, Hq, Hkv, D, P = spec["L"], spec["Hq"], spec["Hkv"], spec["D"], spec["P"]
    ctxs = spec["ctxs"]
    R = len(ctxs)
    S = 2 * R
    extra_tokens = 8 + (args.warmup + args.steps) * 3 + 64
    num_pages = sum((c + extra_tokens) // P + 2 for c in ctxs) + R * ((extra_tokens // P) + 2) + 64
    scale = 1.0 / math.sqrt(D)
    seed = args.seed + 1000 * rank
    cache = sq.Cache(L, Hq, Hkv, D, P, num_pages, max_seqs=4 * S + 8)
    stream = torch.cuda.current_stream()

    # K/V source: a seeded N(0,1) bank sliced at seeded offsets
    chunk = spec["chunk"]
    bank = Bank(1 << 28, sub_seed(seed, 1), device="cuda")
    chunk_elems = L * chunk * Hkv * D
    n_chunks = [c // chunk for c in ctxs]
    offs = bank.offsets(sum(n_chunks) * 2, chunk_elems, sub_seed(seed, 2))
    first_off = [2 * sum(n_chunks[:r]) for r in range(R)]
    mains, auxs = [], []

    def build_request(r):
        m = cache.seq_new()
        for c in range(n_chunks[r]):
            i = first_off[r] + 2 * c
            cache.append_kv(m, chunk, bank.view(offs[i], (L, chunk, Hkv, D)),
                            bank.view(offs[i + 1], (L, chunk, Hkv, D)))
        return m

    for r in range(R):
        mains.append(build_request(r))
    tok_elems = L * Hkv * D
    small = bank.offsets(8192, 2 * 8 * tok_elems, sub_seed(seed, 3))
    small_i = [0]

    bank_ptr = bank.data.data_ptr()

    def kv_rows(n):
        """Device addresses of the K and V of n <= 8 new tokens
        ([L, n, Hkv, D] slices of the bank)."""
        o = int(small[small_i[0] % len(small)])
        small_i[0] += 1
        return bank_ptr + 2 * o, bank_ptr + 2 * (o + 8 * tok_elems)

    def fork_all():
        auxs.clear()
        for m in mains:
            a = cache.fork_aux(m)
            k, v = kv_rows(8)                       # trigger phrase (Sec. 3.2)
            cache.append_kv(a, 8, k, v)
            auxs.append(a)

    fork_all()
    seqs = [x for pair in zip(mains, auxs) for x in pair]
    q_all = bf16_normal((L, S, Hq, D), sub_seed(seed, 4), device="cuda")
    out_all = torch.empty(L, S, Hq, D, dtype=torch.bfloat16, device="cuda")
    torch.cuda.synchronize()

    # per-call arguments resolved once: raw pointers, one stream handle
    st_h = int(stream.cuda_stream)
    q_ptr = [q_all[layer].data_ptr() for layer in range(L)]
    o_ptr = [out_all[layer].data_ptr() for layer in range(L)]
    seq_arr = [None]

    def set_seqs():
        import ctypes
        seq_arr[0] = (ctypes.c_int32 * len(seqs))(*seqs)

    set_seqs()

    # new-token K/V of a step: [L][S][Hkv][D] slices of the bank (one batched append)
    step_rows = bank.offsets(512, 2 * S * tok_elems, sub_seed(seed, 6))
    step_i = [0]

    def step(ev=None):
        o = int(step_rows[step_i[0] % len(step_rows)])
        step_i[0] += 1
        sq.sq_append_kv_batch(cache.handle, seq_arr[0], bank_ptr + 2 * o,
                              bank_ptr + 2 * (o + S * tok_elems), st_h)
        if ev is not None:
            ev.record(stream)
        arr = seq_arr[0]
        for layer in range(L):
            sq.sq_decode_attention(cache.handle, arr, layer, q_ptr[layer], o_ptr[layer],
                                   sq.SQ_OUT_BF16, scale, st_h)

    def timed_decode(K, W):
        for _ in range(W):
            step()
        torch.cuda.synchronize()
        barrier(world)
        st0 = cache.stats()
        ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
        ev_m = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
        ev_s[0].record(stream)
        for t in range(K):
            step(ev_m[t])
            ev_s[t + 1].record(stream)
        torch.cuda.synchronize()
        st1 = cache.stats()
        total_ms = ev_s[0].elapsed_time(ev_s[K])
        attn_ms = sum(ev_m[t].elapsed_time(ev_s[t + 1]) for t in range(K))
        calls = st1["decode_calls"] - st0["decode_calls"]
        uniq = st1["decode_unique_bytes"] - st0["decode_unique_bytes"]
        logi = st1["decode_logical_bytes"] - st0["decode_logical_bytes"]
        return {"total_ms": total_ms, "attn_ms": attn_ms, "calls": calls, "unique_bytes": uniq,
                "logical_bytes": logi}

    hbm_peak, peak_kind = peaks()
    probe_gbs = read_probe(cache, stream)
    clocks = ClockSampler(local)
    time.sleep(0.4)
    K, W = args.steps, args.warmup
    before = timed_decode(K, W)
    clock_rec = clocks.stop()
    t_total = max_over_ranks(before["total_ms"], world)
    value = world * S * K / (t_total / 1e3)
    per_call_ms = before["attn_ms"] / before["calls"]
    uniq_per_call = before["unique_bytes"] / before["calls"]
    achieved = uniq_per_call / (per_call_ms / 1e3) / 1e9
    logical_gbs = before["logical_bytes"] / before["calls"] / (per_call_ms / 1e3) / 1e9

    ratio, ratio_src = recorded_traffic_ratio("sq_decode_splitk_kernel")
    res = {
        "metric": METRIC,
        "value": round(value, 3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": round(t_total / K, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V bank, random-init queries; no dataset)",
        "config": {
            "workload": spec["name"],
            "requests_per_gpu": R, "context_tokens": ctxs, "decoding_sequences_per_gpu": S,
            "layers": L, "q_heads": Hq, "kv_heads": Hkv, "head_dim": D, "page_size": P,
            "sm_scale": scale,
            "l2": "inputs larger than L2: %.2f GB of distinct K/V per decode call" % (uniq_per_call / 1e9),
            "parallelism": "replicas: requests partitioned across GPUs, no collective" if world > 1
            else "single GPU",
        },
        "decode": {
            "attn_ms_per_step": round(before["attn_ms"] / K, 4),
            "attn_ms_per_call": round(per_call_ms, 5),
            "tokens_per_s_attention_only": round(S * K / (before["attn_ms"] / 1e3), 3),
            "unique_gb_per_call": round(uniq_per_call / 1e9, 4),
            "logical_gb_per_call": round(before["logical_bytes"] / before["calls"] / 1e9, 4),
            "hbm_gbs_unique": round(achieved, 1),
            "hbm_gbs_logical": round(logical_gbs, 1),
            "frac_of_%s_peak" % peak_kind: round(achieved / hbm_peak, 4),
            "frac_of_nominal_8tbs": round(achieved / 8000.0, 4),
        },
        "roofline": {
            "bound": "hbm",
            "kernel": "sq_decode_splitk_kernel (split-K attention and the merge of its partials)",
            "achieved": round(achieved, 1),
            "peak": hbm_peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": round(achieved / hbm_peak, 4),
            "read_probe_gbs": round(probe_gbs, 1),
            "frac_of_read_probe": round(achieved / probe_gbs, 4),
            "traffic": int(ratio * uniq_per_call) if ratio else None,
            "traffic_source": (ratio_src + ": small-case DRAM bytes per algorithmic byte, scaled "
                               "to this launch's algorithmic bytes") if ratio else None,
            "algorithmic_bytes_per_launch": int(uniq_per_call),
        },
        # per step: the append kernel, then one decode kernel per layer
        "gpu_launches": int(K * (1 + L)),
        "clocks": clock_rec,
    }

    # ---- end to end through the C ABI with host buffers ----------------------
    if not args.no_e2e:
        q_h = q_all.cpu().pin_memory()
        out_h = torch.empty(out_all.shape, dtype=out_all.dtype).pin_memory()
        o_e2e = int(bank.offsets(1, S * 2 * tok_elems, sub_seed(seed, 5))[0])
        kv_h = bank.view(o_e2e, (2, L, S, Hkv, D)).cpu().pin_memory()
        kv_d = torch.empty(2, L, S, Hkv, D, dtype=torch.bfloat16, device="cuda")
        q_d = torch.empty_like(q_all)

        def e2e_step():
            q_d.copy_(q_h, non_blocking=True)
            kv_d.copy_(kv_h, non_blocking=True)
            sq.sq_append_kv_batch(cache.handle, seq_arr[0], kv_d[0], kv_d[1], st_h)
            for layer in range(L):
                cache.decode_attention(seqs, layer, q_d[layer], out_all[layer], sq.SQ_OUT_BF16, scale)
            out_h.copy_(out_all, non_blocking=True)

        for _ in range(W):
            e2e_step()
        torch.cuda.synchronize()
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0 = time.perf_counter()
        e0.record(stream)
        for _ in range(K):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - w0
        e_ms = max_over_ranks(max(e0.elapsed_time(e1), wall * 1e3), world)
        res["e2e"] = {
            "value": round(world * S * K / (e_ms / 1e3), 3), "unit": "tokens/s",
            "h2d_bytes_per_step": int(q_h.numel() * 2 + kv_h.numel() * 2),
            "d2h_bytes_per_step": int(out_h.numel() * 2),
            "note": "pinned host q and new-token K/V copied in, outputs copied out, every step",
        }

    # ---- eviction: release forks, evict per request, re-fork, decode again ---
    if not args.no_evict:
        for a in auxs:
            cache.release(a)
        torch.cuda.synchronize()
        st0 = cache.stats()
        # One eviction per request, enqueued back to back: the host planning
        # of each call overlaps the GPU work of the one before (reads of the
        # input bank keep the GPU busy while the first is planned), and the
        # events between calls give each call's GPU time: copy-on-write
        # copies and the compaction kernel.
        pre_lengths = [cache.seq_info(m)[0] for m in mains]
        span_list = [spec["spans"](seed, r, pre_lengths[r], P) for r in range(len(mains))]
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(mains) + 1)]
        b = []
        for _ in range(4):
            sq.sq_probe_read(cache.handle, bank.data, bank.data.numel() * 2, st_h)
        evs[0].record(stream)
        for r, m in enumerate(mains):
            b.append(cache.stats()["evict_bytes"])
            cache.evict_spans(m, span_list[r])
            evs[r + 1].record(stream)
        torch.cuda.synchronize()
        b.append(cache.stats()["evict_bytes"])
        per_ms = [evs[r].elapsed_time(evs[r + 1]) for r in range(len(mains))]
        ev_ms = sum(per_ms)
        per = [(b[r + 1] - b[r]) / (per_ms[r] / 1e3) / 1e9 for r in range(len(mains))]
        st1 = cache.stats()
        ev_bytes = st1["evict_bytes"] - st0["evict_bytes"]
        assert cache.sync_status() == sq.SQ_OK
        ev_gbs = ev_bytes / (ev_ms / 1e3) / 1e9
        fork_all()
        seqs[:] = [x for pair in zip(mains, auxs) for x in pair]
        set_seqs()
        torch.cuda.synchronize()
        after = timed_decode(K, W)
        pc = after["attn_ms"] / after["calls"]
        up = after["unique_bytes"] / after["calls"]
        ev_ratio, ev_src = recorded_traffic_ratio("sq_evict_compact_kernel")
        res["evict"] = {
            "kernel": "sq_evict_compact_kernel",
            "gbs": round(ev_gbs, 1),
            "traffic_per_call": int(ev_ratio * ev_bytes / len(mains)) if ev_ratio else None,
            "traffic_source": ev_src,
            "frac_of_%s_peak" % peak_kind: round(ev_gbs / hbm_peak, 4),
            "ms_total": round(ev_ms, 4),
            "algorithmic_bytes": int(ev_bytes),
            "evicted_tokens_per_layer": int(st1["evicted_tokens"] - st0["evicted_tokens"]),
            "moved_rows": int(st1["evict_moved_rows"] - st0["evict_moved_rows"]),
            "per_request_gbs": [round(x, 1) for x in per],
            "calls": len(mains),
            "timing": "GPU time per call, calls enqueued back to back (host planning overlapped)",
        }
        res["after_evict"] = {
            "tokens_per_s": round(world * S * K / (max_over_ranks(after["total_ms"], world) / 1e3), 3),
            "attn_ms_per_call": round(pc, 5),
            "unique_gb_per_call": round(up / 1e9, 4),
            "hbm_gbs_unique": round(up / (pc / 1e3) / 1e9, 1),
        }
        st = cache.stats()
        res["peak_live_pages"] = st["peak_live_pages"]

        # ---- ragged-page eviction of the same requests and spans ---------------
        # The requests are rebuilt from the same bank rows to the same length,
        # the same spans are evicted by ragged packing (only the pages the spans
        # touch), and decode runs again over the partial pages.
        lengths = pre_lengths
        for h in mains + auxs:
            cache.release(h)
        torch.cuda.synchronize()
        mains[:] = [build_request(r) for r in range(R)]
        extra_rows = bank.offsets(64, 2 * 64 * tok_elems, sub_seed(seed, 7))
        xi = 0
        for r, m in enumerate(mains):
            k_extra = lengths[r] - ctxs[r]
            while k_extra > 0:
                c = min(k_extra, 64)
                o = int(extra_rows[xi % len(extra_rows)])
                xi += 1
                cache.append_kv(m, c, bank_ptr + 2 * o, bank_ptr + 2 * (o + 64 * tok_elems))
                k_extra -= c
        assert [cache.seq_info(m)[0] for m in mains] == lengths
        torch.cuda.synchronize()
        st0 = cache.stats()
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(mains) + 1)]
        for _ in range(4):
            sq.sq_probe_read(cache.handle, bank.data, bank.data.numel() * 2, st_h)
        evs[0].record(stream)
        for r, m in enumerate(mains):
            cache.evict_spans_ragged(m, span_list[r])
            evs[r + 1].record(stream)
        torch.cuda.synchronize()
        rg_ms = evs[0].elapsed_time(evs[len(mains)])
        st1 = cache.stats()
        assert cache.sync_status() == sq.SQ_OK
        rg_bytes = st1["evict_bytes"] - st0["evict_bytes"]
        partial = sum(sum(1 for f in cache.page_fills(m)[:-1] if f < P) for m in mains)
        fork_all()
        seqs[:] = [x for pair in zip(mains, auxs) for x in pair]
        set_seqs()
        torch.cuda.synchronize()
        after_rg = timed_decode(K, W)
        pc = after_rg["attn_ms"] / after_rg["calls"]
        up = after_rg["unique_bytes"] / after_rg["calls"]
        rg_ratio, rg_src = recorded_traffic_ratio("sq_evict_compact_kernel", "ragged")
        dr_ratio, dr_src = recorded_traffic_ratio("sq_decode_splitk_kernel", "ragged")
        res["evict_ragged"] = {
            "call": "sq_evict_spans_ragged",
            "kernel": "sq_evict_compact_kernel",
            "traffic_per_call": int(rg_ratio * rg_bytes / len(mains)) if rg_ratio else None,
            "traffic_source": rg_src,
            "ms_total": round(rg_ms, 4),
            "ms_total_dense": res["evict"]["ms_total"],
            "moved_rows": int(st1["evict_moved_rows"] - st0["evict_moved_rows"]),
            "moved_rows_dense": res["evict"]["moved_rows"],
            "algorithmic_bytes": int(rg_bytes),
            "gbs": round(rg_bytes / (rg_ms / 1e3) / 1e9, 1),
            "spans": sum(len(x) for x in span_list),
            "partial_pages_left": int(partial),
            "calls": len(mains),
            "timing": "GPU time of the calls enqueued back to back",
        }
        res["after_evict_ragged"] = {
            "tokens_per_s": round(world * S * K / (max_over_ranks(after_rg["total_ms"], world) / 1e3), 3),
            "attn_ms_per_call": round(pc, 5),
            "unique_gb_per_call": round(up / 1e9, 4),
            "hbm_gbs_unique": round(up / (pc / 1e3) / 1e9, 1),
            "frac_of_%s_peak" % peak_kind: round(up / (pc / 1e3) / 1e9 / hbm_peak, 4),
            "unique_gb_per_call_dense": res["after_evict"]["unique_gb_per_call"],
            "traffic_per_call": int(dr_ratio * up) if dr_ratio else None,
            "traffic_source": dr_src,
        }

    # ---- CPU oracle on a bounded sample (rank 0, N = 1) ----------------------
    if not args.no_cpu and rank == 0 and world == 1 and args.workload == "serving-128k":
        res["cpu_baseline"] = cpu_baseline(args, bank, offs, n_chunks[0], chunk, scale)

    cache.close()
    return res


def _timed(stream):
    import torch
    e = torch.cuda.Event(enable_timing=True)
    e.record(stream)
    return e


def run_agent(args, world, rank, local):
    """Single agent, 8B-class GQA: a 32,768-token context and one aux fork;
    256 main and 128 aux decode steps interleaved from one host thread on two
    streams (one sequence per call); then the aux is released and 40% of the
    context is evicted in 12 spans (lognormal lengths, median 1,500).  Keys
    are N(0,1)/sqrt(128) with sm_scale 1."""
    import ctypes

    import torch

    import paper_2602_22603_gb300 as sq
    from synthetic import AGENT_8B, Bank, bf16_normal, random_spans, shuffled, sub_seed
    torch.cuda.set_device(local)
    sh = AGENT_8B
    L, Hq, Hkv, D, P = sh.num_layers, sh.num_q_heads, sh.num_kv_heads, sh.head_dim, sh.page_size
    n0, steps_main, steps_aux = 32768, 256, 128
    seed = args.seed + 1000 * rank
    cache = sq.Cache(L, Hq, Hkv, D, P, (n0 + 1024) // P + 64, max_seqs=8)
    kbank = Bank(1 << 27, sub_seed(seed, 1), device="cuda", scale=1.0 / math.sqrt(D))
    vbank = Bank(1 << 27, sub_seed(seed, 2), device="cuda")
    chunk = 2048
    ce = L * chunk * Hkv * D
    ko, vo = kbank.offsets(n0 // chunk, ce, sub_seed(seed, 3)), vbank.offsets(n0 // chunk, ce, sub_seed(seed, 4))
    main = cache.seq_new()
    for c in range(n0 // chunk):
        cache.append_kv(main, chunk, kbank.view(ko[c], (L, chunk, Hkv, D)),
                        vbank.view(vo[c], (L, chunk, Hkv, D)))
    tok = L * Hkv * D
    ks, vs = kbank.offsets(1024, 8 * tok, sub_seed(seed, 5)), vbank.offsets(1024, 8 * tok, sub_seed(seed, 6))
    kp, vp = kbank.data.data_ptr(), vbank.data.data_ptr()
    cnt = [0]

    def rows(n):
        i = cnt[0] % len(ks)
        cnt[0] += 1
        return kp + 2 * int(ks[i]), vp + 2 * int(vs[i])

    aux = cache.fork_aux(main)
    k, v = rows(8)
    cache.append_kv(aux, 8, k, v)
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    q = {h: bf16_normal((L, 1, Hq, D), sub_seed(seed, 10 + i), device="cuda") for i, h in enumerate((main, aux))}
    out = {h: torch.empty(L, 1, Hq, D, dtype=torch.bfloat16, device="cuda") for h in (main, aux)}
    arr = {h: (ctypes.c_int32 * 1)(h) for h in (main, aux)}
    qp = {h: [q[h][l].data_ptr() for l in range(L)] for h in (main, aux)}
    op = {h: [out[h][l].data_ptr() for l in range(L)] for h in (main, aux)}
    torch.cuda.synchronize()

    def step(h, st):
        sh_ = int(st.cuda_stream)
        k, v = rows(1)
        cache.append_kv(h, 1, k, v, sh_)
        for layer in range(L):
            sq.sq_decode_attention(cache.handle, arr[h], layer, qp[h][layer], op[h][layer],
                                   sq.SQ_OUT_BF16, 1.0, sh_)

    for _ in range(args.warmup):
        step(main, sa)
        step(aux, sb)
    torch.cuda.synchronize()
    st0 = cache.stats()
    clocks = ClockSampler(local)
    time.sleep(0.3)
    w0 = time.perf_counter()
    ea0, eb0 = _timed(sa), _timed(sb)
    done_aux = 0
    for t in range(steps_main):
        step(main, sa)
        if t % 2 == 0 and done_aux < steps_aux:
            step(aux, sb)
            done_aux += 1
    ea1, eb1 = _timed(sa), _timed(sb)
    torch.cuda.synchronize()
    wall = time.perf_counter() - w0
    clock_rec = clocks.stop()
    st1 = cache.stats()
    tokens = steps_main + done_aux
    uniq = st1["decode_unique_bytes"] - st0["decode_unique_bytes"]
    calls = st1["decode_calls"] - st0["decode_calls"]
    # per-call device time: the main thread's steps alone on one stream, the
    # 32 layer calls of each step back to back between two events
    Kc = 32
    evc = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(Kc)]
    sa_h = int(sa.cuda_stream)
    c0 = cache.stats()
    for t in range(Kc):
        k, v = rows(1)
        cache.append_kv(main, 1, k, v, sa_h)
        evc[t][0].record(sa)
        for layer in range(L):
            sq.sq_decode_attention(cache.handle, arr[main], layer, qp[main][layer],
                                   op[main][layer], sq.SQ_OUT_BF16, 1.0, sa_h)
        evc[t][1].record(sa)
    torch.cuda.synchronize()
    c1 = cache.stats()
    call_ms = sum(a.elapsed_time(b) for a, b in evc) / (Kc * L)
    call_bytes = (c1["decode_unique_bytes"] - c0["decode_unique_bytes"]) / (c1["decode_calls"] -
                                                                             c0["decode_calls"])
    call_gbs = call_bytes / (call_ms / 1e3) / 1e9
    # eviction, after releasing the aux (Algorithm 1 order)
    cache.release(aux, int(sb.cuda_stream))
    n = cache.seq_info(main)[0]
    spans = shuffled(random_spans(sub_seed(seed, 20), 12, int(0.4 * n0), P, n, median=1500), 1)
    torch.cuda.synchronize()
    b0 = cache.stats()["evict_bytes"]
    e0 = _timed(sa)
    cache.evict_spans(main, spans, int(sa.cuda_stream))
    e1 = _timed(sa)
    torch.cuda.synchronize()
    ev_ms = e0.elapsed_time(e1)
    ev_bytes = cache.stats()["evict_bytes"] - b0
    assert cache.sync_status() == sq.SQ_OK
    hbm_peak, peak_kind = peaks()
    tr_ratio, tr_src = recorded_traffic_ratio("sq_decode_splitk_kernel", "agent-32k")
    res = {
        "metric": METRIC, "value": round(tokens / wall, 3), "unit": "tokens/s",
        "n_gpus": 1, "steps": steps_main, "warmup": args.warmup,
        "ms_per_step": round(wall * 1e3 / steps_main, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "agent-32k: one 32,768-token context + one aux fork, 32 layers, "
                               "32q/8kv, d128, page 64; 256 main + 128 aux decode steps on two "
                               "streams, one sequence per call; evict 40% in 12 spans",
                   "sm_scale": 1.0, "k_scale": 1.0 / math.sqrt(D)},
        "decode": {
            "calls": calls,
            "gb_per_call": round(uniq / calls / 1e9, 4),
            "hbm_gbs_wall": round(uniq / wall / 1e9, 1),
            "stream_a_ms": round(ea0.elapsed_time(ea1), 3),
            "stream_b_ms": round(eb0.elapsed_time(eb1), 3),
            "main_tokens_per_s": round(steps_main / wall, 3),
            "aux_tokens_per_s": round(done_aux / wall, 3),
        },
        "evict": {"gbs": round(ev_bytes / (ev_ms / 1e3) / 1e9, 1), "ms": round(ev_ms, 4),
                  "algorithmic_bytes": int(ev_bytes),
                  "frac_of_%s_peak" % peak_kind: round(ev_bytes / (ev_ms / 1e3) / 1e9 / hbm_peak, 4)},
        "roofline": {
            "bound": "hbm",
            "kernel": "sq_decode_splitk_kernel, one 32,768-token sequence per call",
            "achieved": round(call_gbs, 1), "peak": hbm_peak, "peak_kind": peak_kind,
            "unit": "GB/s", "frac": round(call_gbs / hbm_peak, 4),
            "algorithmic_bytes_per_launch": int(call_bytes),
            "ms_per_call": round(call_ms, 5),
            "timing": "CUDA events around the 32 layer calls of a main-thread step, "
                      "calls back to back on one stream, 32 steps",
            "traffic": int(tr_ratio * call_bytes) if tr_ratio else None,
            "traffic_source": (tr_src + ": DRAM bytes per algorithmic byte of captured calls of "
                               "this workload, times this call's algorithmic bytes")
                              if tr_ratio else None,
        },
        "clocks": clock_rec,
    }
    if not args.no_cpu and rank == 0 and world == 1:
        res["cpu_baseline"] = agent_cpu_baseline(kbank, vbank, ko, vo, chunk, n0, L, Hq, Hkv, D,
                                                 q[main])
    cache.close()
    return res


def agent_cpu_baseline(kbank, vbank, ko, vo, chunk, n0, L, Hq, Hkv, D, q):
    """The oracle as it stands (oracle/attention.c decode, fp64, OpenMP) on
    the host cores: one main-thread decode step of the agent workload, the
    query of every layer over the 32,768-token context at all 32 layers;
    tokens/s = 1 / seconds of the step."""
    import numpy as np

    from oracle import attention as oatt
    from synthetic import bf16_bits
    hk, hv = bf16_bits(kbank.data.cpu()), bf16_bits(vbank.data.cpu())
    qb = bf16_bits(q.cpu())
    ce = L * chunk * Hkv * D
    total = 0.0
    for layer in range(L):
        k = np.ascontiguousarray(np.concatenate(
            [hk[int(o):int(o) + ce].reshape(L, chunk, Hkv, D)[layer] for o in ko]))
        v = np.ascontiguousarray(np.concatenate(
            [hv[int(o):int(o) + ce].reshape(L, chunk, Hkv, D)[layer] for o in vo]))
        t0 = time.perf_counter()
        oatt.decode(np.ascontiguousarray(qb[layer, 0]), k, v, 1.0)
        total += time.perf_counter() - t0
    return {"value": round(1.0 / total, 4), "unit": "tokens/s", "cores": oatt.num_threads(),
            "kind": "oracle", "cpu_model": cpu_model(),
            "sample": f"one main-thread decode step: the {n0}-token context, all {Hq} heads, "
                      f"all {L} layers",
            "seconds": round(total, 3)}


def run_trace(args, world, rank, local):
    """End-to-end agent-loop trace (Algorithm 1 shape), seed 7: 4 agents in
    lockstep, `--turns` turns each.  A turn: (1) if the aux thread finished,
    release it and evict whole tool responses older than 2 turns, in random
    order, until >= 60% of their tokens are covered; (2) every 4 turns fork an
    aux thread with an 8-token trigger; (3) 256 main decode steps (the aux
    decodes its 128 steps alongside, in the same calls); (4) append a tool
    response of lognormal length (median 3,000, sigma 1, capped at 20,000)."""
    import ctypes

    import numpy as np
    import torch

    import paper_2602_22603_gb300 as sq
    from synthetic import AGENT_8B, Bank, bf16_normal, sub_seed
    torch.cuda.set_device(local)
    sh = AGENT_8B
    L, Hq, Hkv, D, P = sh.num_layers, sh.num_q_heads, sh.num_kv_heads, sh.head_dim, sh.page_size
    A, T = 4, args.turns
    seed = 7 + 1000 * rank
    rng = np.random.default_rng(seed)
    resp = np.minimum(np.rint(rng.lognormal(math.log(3000), 1.0, size=(T, A))), 20000).astype(int)
    resp = np.maximum(resp, 1)
    scale = 1.0 / math.sqrt(D)
    cache = sq.Cache(L, Hq, Hkv, D, P, 6000, max_seqs=16)   # ~2,600 pages at the peak
    bank = Bank(1 << 28, sub_seed(seed, 1), device="cuda")
    tok = L * Hkv * D
    bp = bank.data.data_ptr()
    big = bank.offsets(4096, 2 * 2048 * tok, sub_seed(seed, 2))
    small = bank.offsets(8192, 16 * tok, sub_seed(seed, 3))
    ctr = {"big": 0, "small": 0}
    st = torch.cuda.current_stream()
    sh_ = int(st.cuda_stream)

    def append(h, n):
        while n > 0:
            c = min(n, 2048)
            if c <= 8:
                o = int(small[ctr["small"] % len(small)]); ctr["small"] += 1
                cache.append_kv(h, c, bp + 2 * o, bp + 2 * (o + 8 * tok), sh_)
            else:
                o = int(big[ctr["big"] % len(big)]); ctr["big"] += 1
                cache.append_kv(h, c, bp + 2 * o, bp + 2 * (o + 2048 * tok), sh_)
            n -= c

    mains = [cache.seq_new() for _ in range(A)]
    for m in mains:
        append(m, 256)                      # the user query Q
    responses = [[] for _ in range(A)]      # (turn, start, end), current positions
    q_all = bf16_normal((L, 2 * A, Hq, D), sub_seed(seed, 4), device="cuda")
    out_all = torch.empty(L, 2 * A, Hq, D, dtype=torch.bfloat16, device="cuda")
    qp = [q_all[l].data_ptr() for l in range(L)]
    op = [out_all[l].data_ptr() for l in range(L)]
    auxs = []
    times = {"attention": 0.0, "eviction": 0.0, "append": 0.0}
    ev_list = []
    decoded = 0
    peak_tokens = 0
    st0 = cache.stats()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    w0 = time.perf_counter()
    for t in range(T):
        # phase 1: the aux thread finished last turn -> release, then evict
        if auxs:
            for a in auxs:
                cache.release(a, sh_)
            auxs = []
            e0 = _timed(st)
            for i, m in enumerate(mains):
                old = [r for r in responses[i] if r[0] < t - 2]
                if not old:
                    continue
                order = rng.permutation(len(old))
                total = sum(e - s for _, s, e in old)
                chosen, cov = [], 0
                for j in order:
                    if cov >= 0.6 * total:
                        break
                    chosen.append(old[int(j)])
                    cov += old[int(j)][2] - old[int(j)][1]
                if args.ragged:
                    cache.evict_spans_ragged(m, [(s, e) for _, s, e in chosen], sh_)
                else:
                    cache.evict_spans(m, [(s, e) for _, s, e in chosen], sh_)
                # shift the positions of the responses that stay
                gone = sorted((s, e) for _, s, e in chosen)
                keep = []
                for r in responses[i]:
                    if r in chosen:
                        continue
                    shift = sum(e - s for s, e in gone if e <= r[1])
                    keep.append((r[0], r[1] - shift, r[2] - shift))
                responses[i] = keep
            e1 = _timed(st)
            ev_list.append((e0, e1))
        # phase 2: fork the aux thread every 4 turns
        if t % 4 == 0:
            for m in mains:
                a = cache.fork_aux(m)
                append(a, 8)
                auxs.append(a)
        # phase 3: main decoding, the aux thread alongside for 128 steps
        for s_ in range(256):
            seqs = mains + (auxs if (auxs and s_ < 128) else [])
            ea = _timed(st)
            arr = (ctypes.c_int32 * len(seqs))(*seqs)
            o = int(small[ctr["small"] % len(small)]); ctr["small"] += 1
            sq.sq_append_kv_batch(cache.handle, arr, bp + 2 * o, bp + 2 * (o + 8 * tok), sh_)
            eb = _timed(st)
            for layer in range(L):
                sq.sq_decode_attention(cache.handle, arr, layer, qp[layer], op[layer],
                                       sq.SQ_OUT_BF16, scale, sh_)
            ec = _timed(st)
            decoded += len(seqs)
            if s_ % 64 == 0:
                torch.cuda.synchronize()
            ev_list.append((ea, eb, ec))
        # phase 4: the tool response
        ea = _timed(st)
        for i, m in enumerate(mains):
            n = cache.seq_info(m)[0]
            append(m, int(resp[t, i]))
            responses[i].append((t, n, n + int(resp[t, i])))
        eb = _timed(st)
        ev_list.append(("append", ea, eb))
        peak_tokens = max(peak_tokens, sum(cache.seq_info(m)[0] for m in mains))
    torch.cuda.synchronize()
    wall = time.perf_counter() - w0
    clock_rec = clocks.stop()
    step_append_ms = 0.0   # batched one-row appends of the decode steps (their launch gap included)
    for e in ev_list:
        if e[0] == "append":
            times["append"] += e[1].elapsed_time(e[2])
        elif len(e) == 2:
            times["eviction"] += e[0].elapsed_time(e[1])
        else:
            step_append_ms += e[0].elapsed_time(e[1])
            times["append"] += e[0].elapsed_time(e[1])
            times["attention"] += e[1].elapsed_time(e[2])
    st1 = cache.stats()
    assert cache.sync_status() == sq.SQ_OK
    busy = sum(times.values())
    tr_ratio, tr_src = recorded_traffic_ratio("sq_decode_splitk_kernel",
                                              "ragged" if args.ragged else None)
    call_bytes = (st1["decode_unique_bytes"] - st0["decode_unique_bytes"]) / max(
        1, st1["decode_calls"] - st0["decode_calls"])
    res = {
        "metric": METRIC, "value": round(decoded / wall, 3), "unit": "tokens/s", "n_gpus": 1,
        "steps": T * 256, "warmup": 0, "ms_per_step": round(wall * 1e3 / (T * 256), 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seed 7)",
        "config": {"workload": f"trace: {A} agents x {T} turns, 32 layers, 32q/8kv, d128, page 64; "
                               "tool responses lognormal(median 3000, sigma 1, cap 20000); aux "
                               "every 4 turns (128 steps); evict >= 60% of responses older than "
                               "2 turns"},
        "trace": {
            "decoded_tokens": decoded, "wall_s": round(wall, 3),
            "time_share": {k: round(v / busy, 4) for k, v in times.items()},
            "gpu_ms": {k: round(v, 2) for k, v in times.items()},
            "decode_unique_gb": round((st1["decode_unique_bytes"] - st0["decode_unique_bytes"]) / 1e9, 2),
            "decode_logical_gb": round((st1["decode_logical_bytes"] - st0["decode_logical_bytes"]) / 1e9, 2),
            "attention_gbs": round((st1["decode_unique_bytes"] - st0["decode_unique_bytes"]) /
                                   (times["attention"] / 1e3) / 1e9, 1),
            "evicted_tokens_per_layer": int(st1["evicted_tokens"] - st0["evicted_tokens"]),
            "evict_gbs": round((st1["evict_bytes"] - st0["evict_bytes"]) /
                               max(times["eviction"] / 1e3, 1e-9) / 1e9, 1),
            "peak_tokens_all_agents": int(peak_tokens),
            "peak_live_pages": int(st1["peak_live_pages"]),
            "final_tokens_per_agent": [cache.seq_info(m)[0] for m in mains],
            # the new token's K/V append and its gap to the first layer's
            # attention, as a share of the decode steps' GPU time
            "step_append_share": round(step_append_ms / (step_append_ms + times["attention"]), 5),
            "step_append_us": round(1e3 * step_append_ms / (T * 256), 3),
            "evict_call": "sq_evict_spans_ragged" if args.ragged else "sq_evict_spans",
        },
        "roofline": {
            "bound": "hbm", "kernel": "sq_decode_splitk_kernel (all decode calls of the trace)",
            "achieved": round((st1["decode_unique_bytes"] - st0["decode_unique_bytes"]) /
                              (times["attention"] / 1e3) / 1e9, 1),
            "peak": peaks()[0], "peak_kind": peaks()[1], "unit": "GB/s",
            "timing": "CUDA events around each step's 32 layer calls",
            "traffic": int(tr_ratio * call_bytes) if tr_ratio else None,
            "traffic_source": (tr_src + ": small-case DRAM bytes per algorithmic byte of the same "
                               "kernel (%s), times the mean call's algorithmic bytes"
                               % ("partial pages after a ragged eviction" if args.ragged
                                  else "dense pages")) if tr_ratio else None,
        },
        "clocks": clock_rec,
    }
    res["roofline"]["frac"] = round(res["roofline"]["achieved"] / res["roofline"]["peak"], 4)
    cache.close()
    return res


def prefill_spans(seed, n, P):
    """Closed cursors of the prefill workload: 12 spans holding 40% of the
    context (lognormal lengths, median 1,500), inside [P, n), shuffled."""
    from synthetic import random_spans, shuffled, sub_seed
    return shuffled(random_spans(sub_seed(seed, 20), 12, int(0.4 * n), P, n, median=1500), 1)


def prefill_tile_flops(n, n_q, spans, G, Hkv, D):
    """FLOPs the tile loop issues (every 128 x 128 tile it computes, masked
    parts included) for one call: 4 x 128 x 128 x D per (query tile, key
    tile) pair; a CTA's two query tiles both run over the key tiles its
    later tile reaches.  Key tiles (pages of 64 tokens): the 64-key boxes
    holding a visible key, two by two."""
    import numpy as np
    vis = np.ones(n, dtype=bool)
    for a, b in spans:
        vis[a:b] = False
    n_box = (n + 63) // 64
    box_has = np.array([vis[b * 64:(b + 1) * 64].any() for b in range(n_box)])
    key0 = (np.nonzero(box_has)[0] * 64)[::2]
    span = 2 * (128 // G)
    n_qt = (n_q + span - 1) // span
    total = 0
    for qt in range(n_qt):
        p_last = n - n_q + min((qt + 1) * span, n_q) - 1
        total += 2 * int(np.searchsorted(key0, p_last, side="right"))
    return total * Hkv * 4 * 128 * 128 * D


def run_prefill(args, world, rank, local):
    """Masked prefill attention (Algorithm 2, BuildMask): one 32,768-token
    agent context (8B-class GQA, 32 layers), 40% of it in 12 closed-cursor
    spans that no query sees; every token is a query (a training-style
    forward).  One step = the attention of all layers."""
    import numpy as np
    import torch

    import paper_2602_22603_gb300 as sq
    from synthetic import AGENT_8B, Bank, sub_seed
    torch.cuda.set_device(local)
    sh = AGENT_8B
    L, Hq, Hkv, D, P = args.layers, sh.num_q_heads, sh.num_kv_heads, sh.head_dim, sh.page_size
    G = Hq // Hkv
    n = args.prefill_ctx
    seed = args.seed + 1000 * rank
    scale = 1.0 / math.sqrt(D)
    cache = sq.Cache(L, Hq, Hkv, D, P, n // P + 64, max_seqs=4)
    bank = Bank(1 << 28, sub_seed(seed, 1), device="cuda")
    chunk = 2048
    sizes = [chunk] * (n // chunk) + ([n % chunk] if n % chunk else [])
    offs = bank.offsets(2 * len(sizes), L * chunk * Hkv * D, sub_seed(seed, 2))
    m = cache.seq_new()
    for i, c in enumerate(sizes):
        cache.append_kv(m, c, bank.view(offs[2 * i], (L, c, Hkv, D)),
                        bank.view(offs[2 * i + 1], (L, c, Hkv, D)))
    spans = prefill_spans(seed, n, P)
    q_offs = bank.offsets(L, n * Hq * D, sub_seed(seed, 4))
    q_ptr = [bank.data.data_ptr() + 2 * int(o) for o in q_offs]
    out = torch.empty(n, Hq, D, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(n, Hq, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    st_h = int(stream.cuda_stream)
    torch.cuda.synchronize()

    def step(evs=None):
        for layer in range(L):
            if evs is not None:
                evs[2 * layer].record(stream)
            sq.sq_prefill_attention(cache.handle, m, layer, n, q_ptr[layer], out, sq.SQ_OUT_BF16,
                                    lse, scale, spans, st_h)
            if evs is not None:
                evs[2 * layer + 1].record(stream)

    K, W = args.steps, args.warmup
    for _ in range(W):
        step()
    torch.cuda.synchronize()
    assert cache.sync_status() == sq.SQ_OK
    barrier(world)
    clocks = ClockSampler(local)
    time.sleep(0.4)
    st0 = cache.stats()
    e_begin, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    call_evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2 * L)] for _ in range(K)]
    e_begin.record(stream)
    for t in range(K):
        step(call_evs[t])
    e_end.record(stream)
    torch.cuda.synchronize()
    clock_rec = clocks.stop()
    st1 = cache.stats()
    assert cache.sync_status() == sq.SQ_OK
    total_ms = max_over_ranks(e_begin.elapsed_time(e_end), world)
    call_ms = [call_evs[t][2 * l].elapsed_time(call_evs[t][2 * l + 1]) for t in range(K) for l in range(L)]
    calls = st1["prefill_calls"] - st0["prefill_calls"]
    pairs = (st1["prefill_pairs"] - st0["prefill_pairs"]) / calls
    flops = 4.0 * D * Hq * pairs                       # per call, visible pairs only
    tile_flops = prefill_tile_flops(n, n, spans, G, Hkv, D)
    mean_call = statistics.mean(call_ms)
    achieved = flops / (mean_call / 1e3) / 1e12
    peak, peak_kind = tensor_peak()
    value = world * n * K / (total_ms / 1e3)
    ratio, ratio_src = recorded_traffic_ratio("sq_prefill_kernel", "prefill-32k")
    kv_bytes = n * Hkv * D * 2 * 2                    # K and V of one layer
    res = {
        "metric": PREFILL_METRIC,
        "value": round(value, 2),
        "unit": "tokens/s",
        "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": round(total_ms / K, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V and queries from a bank; no dataset)",
        "config": {
            "workload": (f"prefill-32k: one {n}-token agent context, every token a query, "
                         f"{L} layers, 32q/8kv, d128, page 64, bf16; 12 closed-cursor spans "
                         f"({sum(b - a for a, b in spans)} tokens, 40%) masked for every query"),
            "layers": L, "q_heads": Hq, "kv_heads": Hkv, "head_dim": D, "page_size": P,
            "context_tokens": n, "queries": n, "sm_scale": scale,
            "masked_tokens": int(sum(b - a for a, b in spans)), "spans": len(spans),
            "l2": "each call reads %.2f GB of distinct K/V + %.2f GB of queries (inputs larger than L2)"
                  % (kv_bytes / 1e9, n * Hq * D * 2 / 1e9),
            "parallelism": "replicas" if world > 1 else "single GPU",
        },
        "prefill": {
            "ms_per_call": round(mean_call, 4),
            "ms_per_call_min": round(min(call_ms), 4),
            "visible_pairs_per_head": int(pairs),
            "algorithmic_tflop_per_call": round(flops / 1e12, 4),
            "tile_tflop_per_call": round(tile_flops / 1e12, 4),
            "tile_tflops": round(tile_flops / (mean_call / 1e3) / 1e12, 1),
            "useful_fraction_of_tiles": round(flops / tile_flops, 4),
        },
        "roofline": {
            "bound": "tensor",
            "kernel": "sq_prefill_kernel",
            "achieved": round(achieved, 1),
            "peak": peak,
            "peak_kind": peak_kind,
            "unit": "TFLOP/s",
            "frac": round(achieved / peak, 4),
            "traffic": int(ratio * kv_bytes) if ratio else None,
            "traffic_source": (ratio_src + ": DRAM bytes per byte of the layer's K/V, from the "
                               "capture") if ratio else None,
            "algorithmic_flops_per_launch": int(flops),
        },
        "gpu_launches": int(K * L),
        "clocks": clock_rec,
    }
    if not args.no_e2e:
        # through the C ABI with host buffers: each layer's queries copied in
        # from pinned memory, its outputs and log-sum-exp copied back
        q_h = bank.view(int(q_offs[0]), (n, Hq, D)).cpu().pin_memory()
        q_d = torch.empty(n, Hq, D, dtype=torch.bfloat16, device="cuda")
        out_h = torch.empty(n, Hq, D, dtype=torch.bfloat16).pin_memory()
        lse_h = torch.empty(n, Hq, dtype=torch.float32).pin_memory()
        Ke = min(K, 5)

        def e2e_step():
            for layer in range(L):
                q_d.copy_(q_h, non_blocking=True)
                cache.prefill_attention(m, layer, n, q_d, out, sq.SQ_OUT_BF16, lse, scale, spans)
                out_h.copy_(out, non_blocking=True)
                lse_h.copy_(lse, non_blocking=True)

        e2e_step()
        torch.cuda.synchronize()
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0 = time.perf_counter()
        e0.record(stream)
        for _ in range(Ke):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - w0
        e_ms = max_over_ranks(max(e0.elapsed_time(e1), wall * 1e3), world)
        res["e2e"] = {
            "value": round(world * n * Ke / (e_ms / 1e3), 2), "unit": "tokens/s",
            "h2d_bytes_per_step": int(L * q_h.numel() * 2),
            "d2h_bytes_per_step": int(L * (out_h.numel() * 2 + lse_h.numel() * 4)),
            "steps": Ke,
            "note": "per layer: pinned host queries in, outputs and log-sum-exp out",
        }
    if not args.no_cpu and rank == 0 and world == 1:
        res["cpu_baseline"] = prefill_cpu_baseline(bank, offs, sizes, q_offs, spans, L, Hq, Hkv, D,
                                                   n, scale)
    cache.close()
    return res


def prefill_cpu_baseline(bank, offs, sizes, q_offs, spans, L, Hq, Hkv, D, n, scale):
    """The oracle as it stands (oracle/attention.c prefill, fp64, OpenMP) on
    the host cores: the last 1,024 queries of the context at 2 layers, every
    head (about 10-15 s on 16 cores); tokens/s = queries / (seconds per layer
    x layers)."""
    import numpy as np

    from oracle import attention as oatt
    from synthetic import bf16_bits
    host = bf16_bits(bank.data.cpu())
    n_sample = 1024
    layers = (0, L - 1) if L > 1 else (0,)
    total = 0.0
    for layer in layers:
        ks, vs = [], []
        for i, c in enumerate(sizes):
            for which, dst in ((0, ks), (1, vs)):
                o = int(offs[2 * i + which])
                a = host[o:o + L * c * Hkv * D].reshape(L, c, Hkv, D)
                dst.append(a[layer])
        k = np.ascontiguousarray(np.concatenate(ks))
        v = np.ascontiguousarray(np.concatenate(vs))
        qo = int(q_offs[layer])
        q = host[qo:qo + n * Hq * D].reshape(n, Hq, D)[n - n_sample:]
        t0 = time.perf_counter()
        oatt.prefill(np.ascontiguousarray(q), k, v, scale, spans)
        total += time.perf_counter() - t0
    per_layer = total / len(layers)
    return {"value": round(n_sample / (per_layer * L), 4), "unit": "tokens/s",
            "cores": oatt.num_threads(), "kind": "oracle", "cpu_model": cpu_model(),
            "sample": f"the last {n_sample} queries of the {n}-token context, all {Hq} heads, at "
                      f"{len(layers)} of {L} layers; tokens/s = queries / (seconds per layer x {L})",
            "seconds": round(total, 3)}


def run_aux_trigger(args, world, rank, local):
    """The auxiliary thread's spawn (Algorithm 1, Phase 2): fork the main
    thread's 131,072-token context (8B-class GQA, 32 layers), append the
    trigger phrase (8 tokens by default) and run its masked prefill over the
    whole shared context at every layer, then release the fork.  One step =
    one such spawn; the prefill reads every K/V row of the context once per
    layer, so it is bound by HBM."""
    import torch

    import paper_2602_22603_gb300 as sq
    from synthetic import AGENT_8B, Bank, sub_seed
    torch.cuda.set_device(local)
    sh = AGENT_8B
    L, Hq, Hkv, D, P = args.layers, sh.num_q_heads, sh.num_kv_heads, sh.head_dim, sh.page_size
    n0, n_q = args.aux_ctx, args.aux_queries
    n = n0 + n_q
    seed = args.seed + 1000 * rank
    scale = 1.0 / math.sqrt(D)
    cache = sq.Cache(L, Hq, Hkv, D, P, n // P + 64, max_seqs=4)
    bank = Bank(1 << 28, sub_seed(seed, 1), device="cuda")
    chunk = 4096
    sizes = [chunk] * (n0 // chunk) + ([n0 % chunk] if n0 % chunk else [])
    offs = bank.offsets(2 * len(sizes) + 2, L * chunk * Hkv * D, sub_seed(seed, 2))
    m = cache.seq_new()
    for i, c in enumerate(sizes):
        cache.append_kv(m, c, bank.view(offs[2 * i], (L, c, Hkv, D)),
                        bank.view(offs[2 * i + 1], (L, c, Hkv, D)))
    trig_k = bank.view(offs[-2], (L, n_q, Hkv, D))
    trig_v = bank.view(offs[-1], (L, n_q, Hkv, D))
    q_offs = bank.offsets(L, n_q * Hq * D, sub_seed(seed, 4))
    q_ptr = [bank.data.data_ptr() + 2 * int(o) for o in q_offs]
    out = torch.empty(n_q, Hq, D, dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.current_stream()
    st_h = int(stream.cuda_stream)
    torch.cuda.synchronize()

    def step(evs=None):
        a = cache.fork_aux(m)
        cache.append_kv(a, n_q, trig_k, trig_v)
        for layer in range(L):
            if evs is not None:
                evs[2 * layer].record(stream)
            sq.sq_prefill_attention(cache.handle, a, layer, n_q, q_ptr[layer], out,
                                    sq.SQ_OUT_BF16, None, scale, [], st_h)
            if evs is not None:
                evs[2 * layer + 1].record(stream)
        cache.release(a)

    K, W = args.steps, args.warmup
    for _ in range(W):
        step()
    torch.cuda.synchronize()
    assert cache.sync_status() == sq.SQ_OK
    barrier(world)
    clocks = ClockSampler(local)
    time.sleep(0.4)
    e_begin, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    call_evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2 * L)] for _ in range(K)]
    e_begin.record(stream)
    for t in range(K):
        step(call_evs[t])
    e_end.record(stream)
    torch.cuda.synchronize()
    clock_rec = clocks.stop()
    assert cache.sync_status() == sq.SQ_OK
    total_ms = max_over_ranks(e_begin.elapsed_time(e_end), world)
    call_ms = [call_evs[t][2 * l].elapsed_time(call_evs[t][2 * l + 1]) for t in range(K) for l in range(L)]
    mean_call = statistics.mean(call_ms)
    kv_bytes = n * Hkv * D * 2 * 2                    # K and V of one layer, every row read once
    value = world * kv_bytes * L * K / (total_ms / 1e3) / 1e9
    achieved = kv_bytes / (mean_call / 1e3) / 1e9
    hbm_peak, peak_kind = peaks()
    ratio, ratio_src = recorded_traffic_ratio("sq_prefill_kernel", "aux-trigger-128k")
    res = {
        "metric": AUX_METRIC,
        "value": round(value, 1),
        "unit": "GB/s",
        "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": round(total_ms / K, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V and queries from a bank; no dataset)",
        "config": {
            "workload": (f"aux-trigger-128k: fork of a {n0}-token context, {n_q}-token trigger "
                         f"phrase appended and prefilled over all {n} keys at {L} layers, fork "
                         f"released; 32q/8kv, d128, page 64, bf16"),
            "layers": L, "q_heads": Hq, "kv_heads": Hkv, "head_dim": D, "page_size": P,
            "context_tokens": n0, "trigger_tokens": n_q, "sm_scale": scale,
            "l2": "each call reads %.2f GB of distinct K/V (inputs larger than L2)" % (kv_bytes / 1e9),
            "parallelism": "replicas" if world > 1 else "single GPU",
        },
        "aux_prefill": {
            "us_per_call": round(mean_call * 1e3, 2),
            "us_per_call_min": round(min(call_ms) * 1e3, 2),
            "kv_gb_per_call": round(kv_bytes / 1e9, 4),
            "step": "fork + append of the trigger tokens + one prefill call per layer + release",
        },
        "roofline": {
            "bound": "hbm",
            "kernel": "sq_prefill_kernel (+ sq_prefill_combine_kernel, timed together per call)",
            "achieved": round(achieved, 1),
            "peak": hbm_peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": round(achieved / hbm_peak, 4),
            "traffic": int(ratio * kv_bytes) if ratio else None,
            "traffic_source": (ratio_src + ": DRAM bytes per byte of the layer's K/V, from the "
                               "capture") if ratio else None,
            "algorithmic_bytes_per_launch": int(kv_bytes),
        },
        # per step: the append kernel, then per layer the prefill and the split merge
        "gpu_launches": int(K * (1 + 2 * L)),
        "clocks": clock_rec,
    }
    if not args.no_e2e:
        # through the C ABI with host buffers: the trigger tokens' K/V and each
        # layer's queries copied in from pinned memory, each layer's output back
        tk_h, tv_h = trig_k.cpu().pin_memory(), trig_v.cpu().pin_memory()
        tk_d, tv_d = torch.empty_like(trig_k), torch.empty_like(trig_v)
        q_h = [bank.view(int(o), (n_q, Hq, D)).cpu().pin_memory() for o in q_offs]
        q_d = torch.empty(n_q, Hq, D, dtype=torch.bfloat16, device="cuda")
        out_h = torch.empty(L, n_q, Hq, D, dtype=torch.bfloat16).pin_memory()
        Ke = min(K, 5)

        def e2e_step():
            a = cache.fork_aux(m)
            tk_d.copy_(tk_h, non_blocking=True)
            tv_d.copy_(tv_h, non_blocking=True)
            cache.append_kv(a, n_q, tk_d, tv_d)
            for layer in range(L):
                q_d.copy_(q_h[layer], non_blocking=True)
                cache.prefill_attention(a, layer, n_q, q_d, out, sq.SQ_OUT_BF16, None, scale, [])
                out_h[layer].copy_(out, non_blocking=True)
            cache.release(a)

        e2e_step()
        torch.cuda.synchronize()
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0 = time.perf_counter()
        e0.record(stream)
        for _ in range(Ke):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - w0
        e_ms = max_over_ranks(max(e0.elapsed_time(e1), wall * 1e3), world)
        res["e2e"] = {
            "value": round(world * kv_bytes * L * Ke / (e_ms / 1e3) / 1e9, 1), "unit": "GB/s",
            "h2d_bytes_per_step": int(2 * tk_h.numel() * 2 + L * n_q * Hq * D * 2),
            "d2h_bytes_per_step": int(out_h.numel() * 2),
            "steps": Ke,
            "note": "per step: pinned trigger K/V and per-layer queries in, per-layer outputs out",
        }
    if not args.no_cpu and rank == 0 and world == 1:
        res["cpu_baseline"] = aux_trigger_cpu_baseline(bank, offs, sizes, q_offs, L, Hq, Hkv, D,
                                                       n0, n_q, scale)
    cache.close()
    return res


def aux_trigger_cpu_baseline(bank, offs, sizes, q_offs, L, Hq, Hkv, D, n0, n_q, scale):
    """The oracle as it stands (oracle/attention.c prefill, fp64, OpenMP) on
    the host cores: the trigger tokens' prefill over the whole context at
    every layer, every head (one step, about 10-15 s on 16 cores); GB/s = K/V
    bytes of a layer / seconds per layer."""
    import numpy as np

    from oracle import attention as oatt
    from synthetic import bf16_bits
    host = bf16_bits(bank.data.cpu())
    layers = range(L)
    total = 0.0
    n = n0 + n_q
    for layer in layers:
        ks, vs = [], []
        for i, c in enumerate(sizes):
            for which, dst in ((0, ks), (1, vs)):
                o = int(offs[2 * i + which])
                dst.append(host[o:o + L * c * Hkv * D].reshape(L, c, Hkv, D)[layer])
        for which, dst in ((0, ks), (1, vs)):
            o = int(offs[len(offs) - 2 + which])
            dst.append(host[o:o + L * n_q * Hkv * D].reshape(L, n_q, Hkv, D)[layer])
        k = np.ascontiguousarray(np.concatenate(ks))
        v = np.ascontiguousarray(np.concatenate(vs))
        qo = int(q_offs[layer])
        q = host[qo:qo + n_q * Hq * D].reshape(n_q, Hq, D)
        t0 = time.perf_counter()
        oatt.prefill(np.ascontiguousarray(q), k, v, scale, [])
        total += time.perf_counter() - t0
    per_layer = total / len(layers)
    kv_bytes = n * Hkv * D * 2 * 2
    return {"value": round(kv_bytes / per_layer / 1e9, 4), "unit": "GB/s",
            "cores": oatt.num_threads(), "kind": "oracle", "cpu_model": cpu_model(),
            "sample": f"the {n_q} trigger queries over all {n} keys, all {Hq} heads, at "
                      f"{len(layers)} of {L} layers; GB/s = K/V bytes of a layer / seconds per layer",
            "seconds": round(total, 3)}


def cpu_model() -> str:
    import platform
    try:
        fields = {}
        with open("/proc/cpuinfo") as f:
            for line in f:
                if ":" in line:
                    k, v = line.split(":", 1)
                    fields.setdefault(k.strip().lower(), v.strip())
        if "model name" in fields:
            return fields["model name"]
        if "cpu part" in fields:
            return f"{platform.machine()} (CPU implementer {fields.get('cpu implementer', '?')}, part {fields['cpu part']})"
    except OSError:
        pass
    return platform.machine()


def _oracle_rows(host_bank, offs, n_chunks, chunk, L, Hkv, D, layer, which):
    """K (which = 0) or V (1) bits [n, Hkv, D] of one main sequence at one
    layer, rebuilt from its bank chunks."""
    import numpy as np
    parts = []
    for c in range(n_chunks):
        o = int(offs[c * 2 + which])
        a = host_bank[o:o + L * chunk * Hkv * D].reshape(L, chunk, Hkv, D)
        parts.append(a[layer])
    return np.ascontiguousarray(np.concatenate(parts))


def cpu_baseline(args, bank, offs, n_chunks, chunk, scale):
    """The oracle as it stands (oracle/attention.c, fp64, OpenMP) on the host
    cores: one decode call of the whole batch (the 8 main sequences and their
    forks, every head) at 2 of the layers, over the full context; scaled to
    tokens/s = sequences / (time per layer x layers)."""
    import numpy as np

    from oracle import attention as oatt
    from synthetic import bf16_bits, bf16_normal
    L, Hq, Hkv, D = args.layers, 32, 8, 128
    R = args.requests
    host_bank = bf16_bits(bank.data.cpu())
    layers = (0, L - 1) if L > 1 else (0,)
    oatt_threads = oatt.num_threads()
    total = 0.0
    n_tok = 0
    for layer in layers:
        ks, vs = [], []
        for r in range(R):
            sub = offs[r * n_chunks * 2:(r + 1) * n_chunks * 2]
            k = _oracle_rows(host_bank, sub, n_chunks, chunk, L, Hkv, D, layer, 0)
            v = _oracle_rows(host_bank, sub, n_chunks, chunk, L, Hkv, D, layer, 1)
            ks += [k, k]   # main and its fork read the same prefix rows
            vs += [v, v]
        n_tok = ks[0].shape[0]
        q = bf16_bits(bf16_normal((2 * R, Hq, D), 99 + layer))
        t0 = time.perf_counter()
        oatt.decode_batch(q, ks, vs, scale)
        total += time.perf_counter() - t0
    per_layer = total / len(layers)
    # the same oracle on one thread, over the first sequence only
    oatt.set_threads(1)
    t0 = time.perf_counter()
    oatt.decode_batch(q[:1], ks[:1], vs[:1], scale)
    t1 = time.perf_counter() - t0
    oatt.set_threads(oatt_threads)
    single = round(1 / (t1 * L), 5)
    return {"value": round(2 * R / (per_layer * L), 4), "unit": "tokens/s",
            "cores": oatt_threads, "kind": "oracle", "cpu_model": cpu_model(),
            "single_thread_value": single,
            "sample": f"one decode call of all {2 * R} sequences ({n_tok} tokens each, {Hq} heads) "
                      f"at {len(layers)} of {L} layers; tokens/s = sequences / "
                      f"(seconds per layer x {L} layers)",
            "seconds": round(total, 3)}


def run_reference(args, world, rank):
    """Reference arm: the CPU oracle as it stands, on this machine's host cores,
    for the same metric; each step is one decode call of the whole batch at
    one layer (a bounded sample of the workload)."""
    import numpy as np

    from oracle import attention as oatt
    from synthetic import Bank, bf16_bits, bf16_normal, sub_seed
    if rank != 0:
        return None
    L, Hq, Hkv, D = args.layers, 32, 8, 128
    R, n = args.requests, args.ctx
    scale = 1.0 / math.sqrt(D)
    row = Hkv * D
    # room for a sequence's rows at any of many offsets (at least two
    # sequences' worth, so the draw below never has an empty range)
    bank = bf16_bits(Bank(max(1 << 27, 2 * n * row), sub_seed(args.seed, 11)).data)
    rng = np.random.default_rng(sub_seed(args.seed, 12))

    def rows():
        o = int(rng.integers(0, (bank.size - n * row) // 8)) * 8
        return bank[o:o + n * row].reshape(n, Hkv, D)

    ks, vs = [], []
    for _ in range(R):
        k, v = rows(), rows()
        ks += [k, k]
        vs += [v, v]
    q = bf16_bits(bf16_normal((2 * R, Hq, D), sub_seed(args.seed, 13)))
    for _ in range(args.warmup):
        oatt.decode_batch(q[:1], [ks[0][:4096]], [vs[0][:4096]], scale)
    ts = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oatt.decode_batch(q, ks, vs, scale)
        ts.append(time.perf_counter() - t0)
    t = sum(ts)
    value = 2 * R * args.steps / (t * L)
    sample = (f"per step: one decode call of all {2 * R} sequences (main + fork) x 1 of {L} layers "
              f"at {n} tokens, all {Hq} heads, fp64 C oracle with OpenMP; "
              f"tokens/s = sequences / (seconds per layer x {L} layers)")
    return {
        "metric": METRIC, "value": round(value, 4), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "impl": "reference",
        "config": {"workload": workload_name(args)},
        "cpu_baseline": {"value": round(value, 4), "unit": "tokens/s", "cores": oatt.num_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


# The other workloads, measured in the same process after the headline one
# (its cache closed first), so that one default run records every workload:
# (workload, overrides of the command-line arguments).
SUB_WORKLOADS = [
    ("large-ragged", {"steps": 5, "warmup": 3, "no_cpu": True, "no_e2e": True}),
    ("agent-32k", {}),
    ("trace", {"turns": 16, "ragged": True}),
    ("prefill-32k", {"steps": 3, "warmup": 3, "no_cpu": True, "no_e2e": True}),
    ("aux-trigger-128k", {"steps": 10, "warmup": 3, "no_cpu": True, "no_e2e": True}),
]
SUB_DROP = ("metric", "data", "n_gpus", "higher_is_better", "scaling", "vs_baseline", "dtype",
            "gpu_launches", "e2e")


def run_sub_records(args, rank, local):
    import gc

    import torch
    runners = {"large-ragged": run_sq, "agent-32k": run_agent, "trace": run_trace,
               "prefill-32k": run_prefill, "aux-trigger-128k": run_aux_trigger}
    out = {}
    for name, over in SUB_WORKLOADS:
        a = argparse.Namespace(**vars(args))
        a.workload = name
        for k, v in over.items():
            setattr(a, k, v)
        gc.collect()
        torch.cuda.empty_cache()
        try:
            r = runners[name](a, 1, rank, local)
        except Exception as e:  # a failed sub-record is reported, not fatal
            out[name] = {"error": f"{type(e).__name__}: {e}"}
            continue
        rec = {k: v for k, v in r.items() if k not in SUB_DROP}
        rec["note"] = ("measured in the same process after the headline workload, whose cache "
                       "was closed first; steps and warm-up as listed")
        out[name] = rec
    return out


def main():
    args = parse_args()
    if args.impl == "reference":
        world = int(os.environ.get("WORLD_SIZE", "1"))
        rank = int(os.environ.get("RANK", "0"))
        res = run_reference(args, world, rank)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    world, rank, local = dist_setup()
    if args.workload == "agent-32k":
        res = run_agent(args, world, rank, local)
    elif args.workload == "trace":
        res = run_trace(args, world, rank, local)
    elif args.workload == "prefill-32k":
        res = run_prefill(args, world, rank, local)
    elif args.workload == "aux-trigger-128k":
        res = run_aux_trigger(args, world, rank, local)
    else:
        res = run_sq(args, world, rank, local)
        if args.workload == "serving-128k" and world == 1 and not args.no_sub:
            res["sub_records"] = run_sub_records(args, rank, local)
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
