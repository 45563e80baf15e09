"""Benchmark of one extend step on GB300: KV append + extend attention over a paged KV pool.

A step is the whole hot path for one batch of returning agents: on-device
schedule, KV append of every uncached suffix token into its pool slot, and
extend attention of every suffix row over its agent's cached prefix and
suffix.  Default workload: the coding-agent long-context batch, the largest
that fits one GPU (16 agents, 64 query / 8 KV heads, d128, page size 16,
cached prefixes U[128k,256k], suffixes U[1024,4096], pages scattered over a
pool of 90 % of free HBM), synthetic N(0,1) bf16 data.  The other long-context
batches (Llama-3-8B shape, the LRU / RR-Evict skew pair, the shared-prefix
batch) are timed in the same run as `configs` legs.

Prints one JSON line.  `value` is the algorithmic attention TFLOP/s of the
whole step (append included) with inputs resident in HBM; `e2e` is the same
metric through the public API with host (pinned) inputs and output, copies
inside the timed region.  The roofline object is for the dominant kernel
(extend attention, tensor-core bound).  `--impl reference` times the fp64 CPU
oracle on the host cores instead, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
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
sys.path.insert(0, ROOT)

METRIC = "extend-attn TFLOP/s & uncached suffix tokens/s on 1 GB300; % of roofline"
NOMINAL_BF16_TFLOPS = 2250.0
NOMINAL_HBM_GBS = 8000.0


def attn_flops(wl) -> float:
    """Algorithmic flops: 4 * D * Hq * sum_b (S_b * P_b + S_b (S_b + 1) / 2) (masked work not counted)."""
    P = wl.prefix_lens.astype(np.float64)
    S = wl.suffix_lens.astype(np.float64)
    return float(4.0 * wl.D * wl.Hq * np.sum(S * P + S * (S + 1) / 2))


def attn_bytes(wl) -> float:
    """Algorithmic bytes: each agent's K and V once per KV head, q in, out out, lens and page table."""
    kv = float(np.sum((wl.prefix_lens.astype(np.float64) + wl.suffix_lens) * wl.Hkv * wl.D * 2 * 2))
    qo = 2.0 * wl.T * wl.Hq * wl.D * 2
    meta = wl.page_table.size * 4 + 2 * wl.B * 4
    return kv + qo + meta


def append_bytes(wl) -> float:
    return 4.0 * wl.T * wl.Hkv * wl.D * 2


# the sources a kernel's DRAM traffic depends on: its own code and the schedule's unit order
ATTN_SOURCES = ("extend_attn.cu", "ptx.cuh", "rope.cuh", "rr_internal.h", "sched.cu")
DECODE_SOURCES = ("decode_attn.cu", "ptx.cuh", "rope.cuh", "rr_internal.h", "sched.cu")


def kernel_source_hash(files=ATTN_SOURCES) -> str:
    """Hash of a kernel's code: comments, blank lines and indentation are left out, so an edit to the
    comments keeps a recorded ncu figure valid and any code change invalidates it."""
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2609_32278_gb300", "csrc", f), encoding="utf-8") as fh:
            for line in fh:
                code = line.split("//", 1)[0].strip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return dict(hbm=p["hbm_gbs"], bf16=p["bf16_tflops"], bf16_sus=p["bf16_tflops_sustained"], src="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


# The measured bf16 peaks come as a burst (best of ten 8192^3 GEMMs) and as a sustained figure (the same GEMM
# back to back for 4 s under the power cap).  A tensor-bound kernel is held to the one that matches how long its
# timed loop runs back to back: the burst under a second, the sustained beyond.
SUSTAINED_AFTER_MS = 1000.0


def tensor_peak(peaks, timed_ms):
    """(peak TFLOP/s, description) for a tensor-bound kernel whose timed loop ran `timed_ms` back to back."""
    if timed_ms >= SUSTAINED_AFTER_MS:
        return peaks["bf16_sus"], (f"{peaks['src']} bf16 dense sustained (the timed loop runs {timed_ms / 1e3:.1f} s "
                                   f"back to back, the regime the sustained GEMM figure was taken in)")
    return peaks["bf16"], f"{peaks['src']} bf16 dense burst (the timed loop runs {timed_ms:.0f} ms)"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if args.impl == "ours" else "gloo"
        if backend == "nccl":
            import torch
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world, device=None):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sample_agents(wl, seed: int, max_agents: int = 2):
    """At most `max_agents` seeded agents with suffix rows."""
    rng = np.random.default_rng(seed)
    live = [b for b in range(wl.B) if wl.suffix_lens[b] > 0]
    return sorted(int(b) for b in rng.choice(live, size=min(max_agents, len(live)), replace=False))


def cpu_oracle_sample(wl, flop_budget: float, seed: int, agents=None, kv_cache=None):
    """Time the fp64 oracle on seeded suffix rows of a few agents (two seeded ones unless `agents` is given;
    regenerating an agent's K/V on the CPU, which is not timed, is what bounds the sample's wall time on long
    contexts, so `kv_cache` keeps them across calls)."""
    import oracle
    import synth
    rng = np.random.default_rng(seed)
    live = agents if agents is not None else sample_agents(wl, seed)
    per_row = lambda b, i: 4.0 * wl.D * wl.Hq * (int(wl.prefix_lens[b]) + i + 1)
    picks, spent = {}, 0.0
    while spent < flop_budget:
        b = int(rng.choice(live))
        i = int(rng.integers(0, int(wl.suffix_lens[b])))
        picks.setdefault(b, set()).add(i)
        spent += per_row(b, i)
    threads = os.cpu_count() or 1
    total_t, total_f, rows = 0.0, 0.0, 0
    for b, rs in picks.items():
        rs = np.array(sorted(rs), dtype=np.int64)
        pos = int(wl.prefix_lens[b]) + rs
        L = int(pos.max()) + 1
        qr = synth.q_rows(wl, b, pos)
        for g in range(wl.Hkv):
            if kv_cache is not None:
                if (b, g) not in kv_cache:  # every position the agent can attend to
                    kv_cache[(b, g)] = synth.agent_kv(wl, b, int(wl.prefix_lens[b]) + int(wl.suffix_lens[b]), g)
                K, V = (x[:L] for x in kv_cache[(b, g)])
            else:
                K, V = synth.agent_kv(wl, b, L, g)
            t0 = time.perf_counter()
            oracle.attention_rows(qr[:, g * wl.G:(g + 1) * wl.G], pos, K, V, 1.0 / math.sqrt(wl.D), threads)
            total_t += time.perf_counter() - t0
        total_f += sum(per_row(b, int(i)) for i in rs)
        rows += len(rs)
    return total_f, total_t, rows, threads


def run_reference(args, world, rank):
    import synth
    if rank != 0:
        return 0
    wl = workload(synth, args.config, seed=0)
    budget = args.ref_flops
    agents, cache = sample_agents(wl, seed=99), {}  # the same two agents every step; their K/V generated once
    for _ in range(args.warmup):
        cpu_oracle_sample(wl, budget, seed=1000, agents=agents, kv_cache=cache)
    fl, tm, rows, threads = 0.0, 0.0, 0, 1
    for k in range(args.steps):
        f, t, r, threads = cpu_oracle_sample(wl, budget, seed=k, agents=agents, kv_cache=cache)
        fl += f
        tm += t
        rows += r
    value = fl / tm / 1e12
    tok_per_s = rows / tm
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": tm / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_dict(wl, world),
        "inputs": {"sha256": wl.manifest()["sha256"][:16], "num_pages": wl.num_pages,
                   "note": "no pool: the oracle regenerates K/V by logical position"},
        "uncached_suffix_tokens_per_s": tok_per_s,
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
                         "sample": f"{rows} seeded suffix rows (all heads) of agents {agents} over {args.steps} steps, "
                                   f"~{budget:.1e} flop each; fp64 oracle, K/V generation not timed"},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def load_traffic(src_hash, record="extend_attn_traffic.json"):
    """The committed ncu DRAM-traffic records ({workload: record}) if they were taken on this kernel source,
    else None; and the raw file (or None)."""
    path = os.path.join(ROOT, "profiles", record)
    try:
        with open(path) as f:
            rec = json.load(f)
    except Exception:
        return None, None
    if rec.get("kernel_source_hash") != src_hash:
        return None, rec
    return rec.get("records", {}), rec


def traffic_for(workload, src_hash, record="extend_attn_traffic.json"):
    """DRAM bytes per launch recorded for this whole workload on this kernel source, else None."""
    recs, _ = load_traffic(src_hash, record)
    if not recs or workload not in recs:
        return None
    return recs[workload].get("dram_bytes_per_launch")


def config_dict(wl, world):
    """The workload as both arms name it (fields that do not depend on the pool size, which for the
    coding-agent batch follows free HBM)."""
    return {"workload": wl.name, "B": wl.B, "Hq": wl.Hq, "Hkv": wl.Hkv, "D": wl.D, "page_size": wl.ps,
            "uncached_tokens": wl.T, "kv_tokens": int((wl.prefix_lens.astype(np.int64) + wl.suffix_lens).sum()),
            "l2": f"inputs larger than L2 (KV working set {attn_bytes(wl) / 1e9:.1f} GB > 129 MB)",
            "parallelism": f"replicas x{world}"}


def per_agent_latency(rr, wl, g, dev, st, reps=5):
    """Each agent's extend step (append + attention) run alone, as a returning request would be.

    The kernel-level analogue of per-request time to first token: RR-Evict trades a few whole-history
    recomputes (LRU) for many partial ones, which shows up as a lower maximum here (Sec. 3.3, Sec. 4).
    """
    import torch
    cu = wl.cu
    times = []
    for b in range(wl.B):
        if wl.suffix_lens[b] == 0:
            continue
        r0, r1 = int(cu[b]), int(cu[b + 1])
        args_b = (g["page_table"][b:b + 1], g["prefix_lens"][b:b + 1], g["suffix_lens"][b:b + 1])
        out = g["out"][r0:r1]
        ts = []
        for k in range(reps + 1):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            rr.kv_append(g["k_new"][r0:r1], g["v_new"][r0:r1], g["k_pool"], g["v_pool"], *args_b)
            rr.extend_attention(g["q"][r0:r1], g["k_pool"], g["v_pool"], *args_b, out=out)
            e1.record(st)
            torch.cuda.synchronize(dev)
            if k:
                ts.append(e0.elapsed_time(e1))
        times.append(statistics.median(ts))
    if rr.device_error():
        raise RuntimeError("device error in the per-agent leg")
    t = np.array(times)
    return {"agents": len(times), "max_ms": float(t.max()), "p99_ms": float(np.percentile(t, 99)),
            "p50_ms": float(np.percentile(t, 50)), "mean_ms": float(t.mean()), "sum_ms": float(t.sum())}


# The long-context batches timed beside the main workload (each as its own leg, same step, fewer steps).
LEG_CONFIGS = (("c2_llama3_8b", 10), ("c3_lru", 5), ("c3_rr", 5), ("c5_shared", 10), ("c3g_lru", 3), ("c3g_rr", 3))


def config_leg(rr, synth, name, steps, warmup, dev, st, peaks, rank, local):
    """One long-context batch: append + attention steps, device-timed, with the attention's roofline and the
    clocks seen while they ran."""
    import torch
    wl = workload(synth, name, seed=rank)
    g = synth.gpu_tensors(wl, dev)
    g["out"] = torch.empty_like(g["q"])

    def append():
        rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                     g["suffix_lens"])

    def attend():
        rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"],
                            out=g["out"])

    for _ in range(warmup):
        append()
        attend()
    torch.cuda.synchronize(dev)
    if rr.device_error():
        raise RuntimeError(f"device error in the {name} warm-up")
    ev = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(3)) for _ in range(steps)]
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    for e0, e1, e2 in ev:
        e0.record(st)
        append()
        e1.record(st)
        attend()
        e2.record(st)
    torch.cuda.synchronize(dev)
    clk = clocks.stop()
    if rr.device_error():
        raise RuntimeError(f"device error in the {name} timed region")
    F = attn_flops(wl)
    step_ms = statistics.mean(e0.elapsed_time(e2) for e0, e1, e2 in ev)
    attn_ms = statistics.mean(e1.elapsed_time(e2) for e0, e1, e2 in ev)
    app_ms = statistics.mean(e0.elapsed_time(e1) for e0, e1, e2 in ev)
    achieved = F / (attn_ms * 1e-3) / 1e12
    leg_peak, leg_kind = tensor_peak(peaks, steps * step_ms)
    res = {"config": config_dict(wl, 1), "inputs_sha256": wl.manifest()["sha256"][:16], "steps": steps,
           "warmup": warmup, "ms_per_step": step_ms, "value": F / (step_ms * 1e-3) / 1e12, "unit": "TFLOP/s",
           "uncached_suffix_tokens_per_s": wl.T / (step_ms * 1e-3), "attention_ms": attn_ms,
           "attention_ms_median": statistics.median(e1.elapsed_time(e2) for e0, e1, e2 in ev),
           "kv_append_ms": app_ms, "kv_append_gbs": append_bytes(wl) / (app_ms * 1e-3) / 1e9,
           "roofline": {"bound": "tensor", "achieved": achieved, "peak": leg_peak, "unit": "TFLOP/s",
                        "frac": achieved / leg_peak, "peak_kind": leg_kind, "frac_of_burst": achieved / peaks["bf16"],
                        "frac_of_sustained": achieved / peaks["bf16_sus"],
                        "frac_of_nominal": achieved / NOMINAL_BF16_TFLOPS,
                        "traffic": traffic_for(wl.name, kernel_source_hash()),
                        "algorithmic_flops": F, "algorithmic_bytes": attn_bytes(wl)},
           "clocks": clk}
    if wl.shared_len > 0 and wl.shared_len % 128 == 0:
        # the same attention as a cascade over the shared prefix (rr_extend_attention_shared), checked against
        # the plain call's output within the parity bar and timed the same way
        out_c = torch.empty_like(g["out"])

        def cascade():
            rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                                g["suffix_lens"], out=out_c, shared_len=wl.shared_len)

        for _ in range(warmup):
            cascade()
        cev = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(2)) for _ in range(steps)]
        for e0, e1 in cev:
            e0.record(st)
            cascade()
            e1.record(st)
        torch.cuda.synchronize(dev)
        if rr.device_error():
            raise RuntimeError(f"device error in the {name} cascade region")
        if float((out_c.float() - g["out"].float()).abs().max()) > 2e-2:
            raise RuntimeError(f"{name}: the shared-prefix cascade differs from the plain call")
        c_ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in cev)
        res["cascade"] = {"shared_len": int(wl.shared_len), "attention_ms": c_ms,
                          "attention_tflops": F / (c_ms * 1e-3) / 1e12, "vs_plain": attn_ms / c_ms}
        del out_c
    del g
    torch.cuda.empty_cache()
    return res


def decode_bytes(wl) -> float:
    """Algorithmic bytes of one decode call: each agent's K and V once per KV head, q in, out out, the page
    table entries and lengths read."""
    kv_tok = float((wl.prefix_lens.astype(np.int64) + 1).sum())
    pages = float(sum(-(-(int(p) + 1) // wl.ps) for p in wl.prefix_lens))
    return kv_tok * wl.Hkv * wl.D * 2 * 2 + 2.0 * wl.B * wl.Hq * wl.D * 2 + pages * 4 + wl.B * 4


def decode_leg(args, rr, synth, dev, st, peaks, rank):
    """Decode attention on a decode batch (one new token per agent), device-timed per call."""
    import torch
    free = torch.cuda.mem_get_info(dev)[0]
    wl = synth.decode_config(args.decode_config, seed=rank,
                             free_hbm_bytes=free if args.decode_config == "c4_decode" else None)
    if args.decode_agents:
        n = args.decode_agents
        wl = synth.custom(f"{args.decode_config}[:{n}]", n, wl.Hq, wl.Hkv, wl.D, wl.prefix_lens[:n],
                          wl.suffix_lens[:n], ps=wl.ps, shared_len=wl.shared_len, seed=wl.seed)
    g = synth.gpu_tensors(wl, dev)
    rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                 g["suffix_lens"])
    kv_lens = (g["prefix_lens"] + 1).to(torch.int32)
    out = torch.empty_like(g["q"])
    for _ in range(max(3, args.warmup)):
        rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, out=out)
    torch.cuda.synchronize(dev)
    if rr.device_error():
        raise RuntimeError("device error in the decode warm-up")
    n = max(args.steps, 10)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for e0, e1 in ev:
        e0.record(st)
        rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, out=out)
        e1.record(st)
    torch.cuda.synchronize(dev)
    if rr.device_error():
        raise RuntimeError("device error in the decode timed region")
    ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in ev)
    nbytes = decode_bytes(wl)
    gbs = nbytes / (ms * 1e-3) / 1e9
    dec_hash = kernel_source_hash(DECODE_SOURCES)
    traffic = traffic_for(wl.name, dec_hash, "decode_attn_traffic.json")
    res = {"workload": wl.name, "inputs_sha256": wl.manifest()["sha256"][:16], "B": wl.B, "Hq": wl.Hq,
           "Hkv": wl.Hkv, "D": wl.D,
           "kv_tokens": int((wl.prefix_lens.astype(np.int64) + 1).sum()), "calls": n, "ms_per_call": ms,
           "tokens_per_s": wl.B / (ms * 1e-3),
           "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm"], "unit": "GB/s",
                        "frac": gbs / peaks["hbm"], "traffic": traffic, "algorithmic_bytes": nbytes,
                        "kernel": f"decode_attn_kernel<{wl.D},{3 if wl.D == 128 else 6},{wl.G}>",
                        "peak_kind": f"{peaks['src']} HBM copy bandwidth", "kernel_source_hash": dec_hash},
           "l2": f"K/V working set {nbytes / 1e9:.1f} GB > 129 MB"}
    # a batch over a common prefix: the same calls through rr_decode_attention_shared (the shared pages read
    # once per group of 16 / G agents), checked against the plain call's output within the parity bar
    if wl.shared_len > 0 and wl.shared_len % 128 == 0 and wl.B * wl.Hkv <= 1024:
        out_s = torch.empty_like(out)
        for _ in range(max(3, args.warmup)):
            rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, out=out_s,
                                shared_len=wl.shared_len)
        torch.cuda.synchronize(dev)
        for e0, e1 in ev:
            e0.record(st)
            rr.decode_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], kv_lens, out=out_s,
                                shared_len=wl.shared_len)
            e1.record(st)
        torch.cuda.synchronize(dev)
        if rr.device_error():
            raise RuntimeError("device error in the shared-prefix decode region")
        diff = (out_s.float() - out.float()).abs()
        if float(diff.max()) > 2e-2:
            raise RuntimeError("shared-prefix decode differs from the plain decode")
        ms_s = statistics.mean(e0.elapsed_time(e1) for e0, e1 in ev)
        res["shared_prefix"] = {"shared_len": int(wl.shared_len), "ms_per_call": ms_s,
                                "tokens_per_s": wl.B / (ms_s * 1e-3), "vs_plain": ms / ms_s,
                                "algorithmic_gbs_of_plain_bytes": nbytes / (ms_s * 1e-3) / 1e9}
        del out_s
    del g, out, kv_lens
    torch.cuda.empty_cache()
    return res


# Replay leg: the policy's effect on per-request extend cost (Sec. 4's P99 metrics).  Every extend batch a
# policy's replay produces is run through rr_kv_append + rr_extend_attention on this GPU and timed with CUDA
# events; a request's attention time to first token is its batch's time (one layer).
REPLAY_MODELS = {  # attention geometry of the two served models of Sec. 4
    "conversational": {"model": "Qwen3-Coder-30B-A3B attention (32 q / 4 kv heads, d128)", "Hq": 32, "Hkv": 4},
    "coding": {"model": "Qwen3-8B attention (32 q / 8 kv heads, d128)", "Hq": 32, "Hkv": 8},
}
# kind, agents, admitted concurrency, capacity as a fraction of the admitted agents' summed final contexts:
# points inside the regime of Eq. 1 on these traces (active demand fits, live idle demand does not) --
# at 0.6 and above nothing is evicted from live agents, far below it every policy thrashes
REPLAY_SETTINGS = [
    ("conversational", 222, 40, 0.4), ("conversational", 222, 80, 0.4), ("coding", 64, 16, 0.5),
    ("coding", 64, 16, 0.4),
]
REPLAY_POLICIES = [  # label, policy, completion signals
    ("lru", "lru", False), ("lru+cs", "lru", True), ("rr-evict+cs", "rr", True), ("rr-tiered", "tiered", False),
]
REPLAY_WINDOW_S = 0.05  # requests arriving within one 50 ms scheduling tick share an extend batch


def measure_batches(rr, synth, dev, st, batches, Hq, Hkv, D=128, ps=16):
    """CUDA-event time (seconds) of append + extend attention for each (prefix_lens, suffix_lens) batch.

    One pool holds the largest batch: agent i of a batch takes the next distinct pages of a seeded
    placement, every one of them filled with the generator's values; q / k_new / v_new are the first T rows
    of one generated buffer.  Each batch runs once untimed, then once timed."""
    import torch
    need = max(sum(-(-(int(p) + int(s)) // ps) for p, s in zip(P, S)) for P, S in batches)
    t_max = max(sum(int(s) for s in S) for P, S in batches)
    pool = synth.custom("replay_pool", 1, Hq, Hkv, D, [need * ps], [0], ps=ps, seed=13)
    rows = synth.custom("replay_rows", 1, Hq, Hkv, D, [0], [t_max], ps=ps, seed=14)
    gp = synth.gpu_tensors(pool, dev)
    gr = synth.gpu_tensors(rows, dev)
    pages = pool.page_table[0]
    out = torch.empty_like(gr["q"])
    times = []
    for P, S in batches:
        B = len(P)
        pb = [-(-(int(p) + int(s)) // ps) for p, s in zip(P, S)]
        pt = np.full((B, max(pb)), -1, dtype=np.int32)
        off = 0
        for i, n in enumerate(pb):
            pt[i, :n] = pages[off:off + n]
            off += n
        T = int(sum(S))
        a = (torch.from_numpy(pt).to(dev), torch.tensor(np.asarray(P, dtype=np.int32), device=dev),
             torch.tensor(np.asarray(S, dtype=np.int32), device=dev))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for k in range(2):
            if k:
                e0.record(st)
            rr.kv_append(gr["k_new"][:T], gr["v_new"][:T], gp["k_pool"], gp["v_pool"], *a)
            rr.extend_attention(gr["q"][:T], gp["k_pool"], gp["v_pool"], *a, out=out[:T])
        e1.record(st)
        e1.synchronize()
        times.append(e0.elapsed_time(e1) * 1e-3)
    if rr.device_error():
        raise RuntimeError("device error in the replay batches")
    del gp, gr, out
    torch.cuda.empty_cache()
    return times


def replay_leg(rr, synth, dev, st):
    from paper_2609_32278_gb300 import policy as pol
    res = {"note": ("synthetic agent traces (policy.synthetic_traces) replayed under each policy; each extend "
                    f"batch (requests within {REPLAY_WINDOW_S * 1e3:.0f} ms) run through rr_kv_append + "
                    "rr_extend_attention on this GPU and timed with CUDA events (one layer); a request's "
                    "attention time is its batch's"), "models": {k: m["model"] for k, m in REPLAY_MODELS.items()},
           "runs": []}
    for kind, n, conc, frac in REPLAY_SETTINGS:
        m = REPLAY_MODELS[kind]
        traces = pol.synthetic_traces(n, kind, seed=0)
        finals = sorted(sum(t.new_tokens) + sum(t.output_tokens) for t in traces)
        cap = int(frac * sum(finals[-conc:]))
        run = {"workload": kind, "agents": n, "concurrency": conc, "capacity_tokens": cap,
               "capacity_note": f"{frac} x the summed final contexts of the {conc} largest agents", "policies": {}}
        for label, policy, cs in REPLAY_POLICIES:
            reqs = pol.replay(traces, cap, policy, shared_prompt=2048, chunk=1024, completion_signals=cs,
                              concurrency=conc)
            batches = pol.extend_batches(reqs, REPLAY_WINDOW_S)
            bt = measure_batches(rr, synth, dev, st, [(P, S) for _, P, S in batches], m["Hq"], m["Hkv"])
            per_req = [0.0] * len(reqs)
            for (idx, _, _), t in zip(batches, bt):
                for i in idx:
                    per_req[i] = t
            summ = pol.summarize(reqs, per_req)
            sizes = [len(idx) for idx, _, _ in batches]
            summ.update({"batches": len(batches), "batch_size_max": max(sizes), "batch_size_mean": float(np.mean(sizes)),
                         "batch_ms_p50": 1e3 * pol.percentile(bt, 50), "batch_ms_p99": 1e3 * pol.percentile(bt, 99),
                         "batch_ms_max": 1e3 * max(bt), "gpu_s_total": float(sum(bt))})
            run["policies"][label] = summ
        res["runs"].append(run)
    return res


# The LRU / RR-Evict skew pair drawn from the eviction-policy generator rather than from length samplers:
# 64 coding agents (Qwen3-8B attention: 32 q / 8 kv heads, d128) all admitted, a cache of half their summed
# final contexts, and the batch in which every agent returns with its next request after the median request
# time (policy.snapshot_lengths); the 2048-token system prompt stays shared.
POLICY_PAIR = {"c3g_lru": ("lru", False), "c3g_rr": ("rr", True)}


def policy_workload(synth, name, seed=0):
    from paper_2609_32278_gb300 import policy as pol
    policy, cs = POLICY_PAIR[name]
    traces = pol.synthetic_traces(64, "coding", seed=seed)
    cap = int(0.5 * sum(sum(t.new_tokens) + sum(t.output_tokens) for t in traces))
    reqs = pol.replay(traces, cap, policy, shared_prompt=2048, chunk=1024, completion_signals=cs, concurrency=64)
    P, S = pol.snapshot_lengths(reqs, 0.5)
    return synth.custom(name, len(P), 32, 8, 128, P, S, shared_len=2048, seed=seed)


def workload(synth, name, seed=0, free_hbm_bytes=None):
    if name in POLICY_PAIR:
        return policy_workload(synth, name, seed)
    return synth.config(name, seed=seed, free_hbm_bytes=free_hbm_bytes)


def slice_workload(synth, wl, agents=0, stride=1):
    """A small profiling case: every `stride`-th agent of `wl` (a systematic sample keeps the batch's mix of
    agent kinds), the first `agents` of those if nonzero, in a pool of twice the pages they need."""
    idx = np.arange(0, wl.B, max(1, stride))
    if agents:
        idx = idx[:agents]
    name = wl.name + (f"[::{stride}]" if stride > 1 else "") + (f"[:{agents}]" if agents else "")
    return synth.custom(name, len(idx), wl.Hq, wl.Hkv, wl.D, wl.prefix_lens[idx], wl.suffix_lens[idx], ps=wl.ps,
                        shared_len=wl.shared_len, seed=wl.seed)


def run_ours(args, world, rank, local):
    import torch
    import synth
    import paper_2609_32278_gb300 as rr

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    free = torch.cuda.mem_get_info(dev)[0]
    wl = workload(synth, args.config, seed=rank, free_hbm_bytes=free if args.config == "c4_coding" else None)
    if args.agents or args.agent_stride > 1:
        wl = slice_workload(synth, wl, args.agents, args.agent_stride)
    g = synth.gpu_tensors(wl, dev)
    st = torch.cuda.current_stream(dev)
    F = attn_flops(wl)
    peaks = load_peaks()

    def step():
        rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                     g["suffix_lens"])
        return rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                                   g["suffix_lens"], out=g["out"])

    g["out"] = torch.empty_like(g["q"])
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    code = rr.device_error()
    if code:
        raise RuntimeError(f"device error {code} during warm-up")

    # ---- device-timed steps (inputs resident in HBM; working set > L2)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize(dev)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(st)
    for k in range(args.steps):
        e0, e1, e2 = ev[k]
        e0.record(st)
        rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                     g["suffix_lens"])
        e1.record(st)
        rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"], g["suffix_lens"],
                            out=g["out"])
        e2.record(st)
    t_end.record(st)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop()
    code = rr.device_error()
    if code:
        raise RuntimeError(f"device error {code} in the timed region")
    total_ms = t_start.elapsed_time(t_end)
    total_ms = max_over_ranks(total_ms, world, dev)
    ms_step = total_ms / args.steps
    attn_ms = statistics.mean(ev[k][1].elapsed_time(ev[k][2]) for k in range(args.steps))
    app_ms = statistics.mean(ev[k][0].elapsed_time(ev[k][1]) for k in range(args.steps))
    value = world * F / (ms_step * 1e-3) / 1e12
    tok_s = world * wl.T / (ms_step * 1e-3)

    # ---- the same step as one launch (rr_extend_step: the kernel appends, crosses a grid barrier, attends)
    fused = None
    if not args.no_fused:
        fev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for _ in range(args.warmup):
            rr.extend_step(g["q"], g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"],
                           g["prefix_lens"], g["suffix_lens"], out=g["out"])
        torch.cuda.synchronize(dev)
        for e0, e1 in fev:
            e0.record(st)
            rr.extend_step(g["q"], g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"],
                           g["prefix_lens"], g["suffix_lens"], out=g["out"])
            e1.record(st)
        torch.cuda.synchronize(dev)
        if rr.device_error():
            raise RuntimeError("device error in the fused-step region")
        f_ms = max_over_ranks(statistics.mean(e0.elapsed_time(e1) for e0, e1 in fev), world, dev)
        fused = {"ms_per_step": f_ms, "value": world * F / (f_ms * 1e-3) / 1e12, "unit": "TFLOP/s",
                 "uncached_suffix_tokens_per_s": world * wl.T / (f_ms * 1e-3),
                 "vs_two_calls": ms_step / f_ms}

    e2e = None
    if not args.no_e2e:
        # ---- end to end through the public API: every step copies its inputs from pinned host memory to
        # the device and its output back.  As a serving loop would, the copies run on their own streams
        # and overlap the neighbouring steps' kernels (double-buffered: step k's inputs land while step
        # k-1 computes, step k-1's output leaves while step k computes); each step's copies are inside
        # the timed region.
        keys = ("q", "k_new", "v_new", "page_table", "prefix_lens", "suffix_lens")
        host = {k: g[k].cpu().pin_memory() for k in keys}
        out_h = [torch.empty(g["q"].shape, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
        dev_in = [{k: torch.empty_like(g[k]) for k in keys} for _ in range(2)]
        dev_out = [torch.empty_like(g["q"]) for _ in range(2)]
        h2d = sum(v.numel() * v.element_size() for v in host.values())
        d2h = out_h[0].numel() * out_h[0].element_size()
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        ev_in = [torch.cuda.Event() for _ in range(2)]
        ev_done = [torch.cuda.Event() for _ in range(2)]
        ev_out = [torch.cuda.Event() for _ in range(2)]

        def e2e_steps(n):
            for k in range(n):
                i = k & 1
                with torch.cuda.stream(s_in):
                    if k >= 2:
                        s_in.wait_event(ev_done[i])      # step k-2 has finished reading dev_in[i]
                    for key, v in host.items():
                        dev_in[i][key].copy_(v, non_blocking=True)
                    ev_in[i].record(s_in)
                st.wait_event(ev_in[i])
                if k >= 2:
                    st.wait_event(ev_out[i])             # step k-2's output has left dev_out[i]
                d = dev_in[i]
                rr.kv_append(d["k_new"], d["v_new"], g["k_pool"], g["v_pool"], d["page_table"], d["prefix_lens"],
                             d["suffix_lens"], stream=st)
                rr.extend_attention(d["q"], g["k_pool"], g["v_pool"], d["page_table"], d["prefix_lens"],
                                    d["suffix_lens"], out=dev_out[i], stream=st)
                ev_done[i].record(st)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(ev_done[i])
                    out_h[i].copy_(dev_out[i], non_blocking=True)
                    ev_out[i].record(s_out)
            st.wait_stream(s_out)

        e2e_steps(args.warmup)
        torch.cuda.synchronize(dev)
        barrier(world)
        s0 = torch.cuda.Event(enable_timing=True)
        s1 = torch.cuda.Event(enable_timing=True)
        s0.record(st)
        s_in.wait_stream(st)
        e2e_steps(args.steps)
        s1.record(st)
        torch.cuda.synchronize(dev)
        e2e_ms = max_over_ranks(s0.elapsed_time(s1) / args.steps, world, dev)
        if rr.device_error():
            raise RuntimeError("device error in the end-to-end region")
        # the last step's output must have reached the host intact
        if not torch.equal(out_h[(args.steps - 1) & 1], g["out"].cpu()):
            raise RuntimeError("end-to-end output differs from the device-timed output")
        e2e = {"value": world * F / (e2e_ms * 1e-3) / 1e12, "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
               "overlap": "double-buffered: copies on two side streams overlap the neighbouring steps' kernels"}
        del dev_in, dev_out, out_h, host

    # ---- the same step with rotary position embedding (q and k_new un-rotated; K rotated by the append as
    # it writes the pool, q by the attention kernel as its tiles land), Llama-3's base 500000
    rope = None
    if not args.no_rope:
        table = rr.rope_table(int((wl.prefix_lens + wl.suffix_lens).max()) + 1, wl.D, 500000.0, device=dev)
        out_r = torch.empty_like(g["q"])

        def rope_step():
            rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                         g["suffix_lens"], rope=table)
            rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                                g["suffix_lens"], out=out_r, rope=table)

        for _ in range(args.warmup):
            rope_step()
        torch.cuda.synchronize(dev)
        rev = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(3)) for _ in range(args.steps)]
        for e0, e1, e2 in rev:
            e0.record(st)
            rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                         g["suffix_lens"], rope=table)
            e1.record(st)
            rr.extend_attention(g["q"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                                g["suffix_lens"], out=out_r, rope=table)
            e2.record(st)
        torch.cuda.synchronize(dev)
        if rr.device_error():
            raise RuntimeError("device error in the rotary-step region")
        r_ms = max_over_ranks(statistics.mean(e0.elapsed_time(e2) for e0, e1, e2 in rev), world, dev)
        r_app = statistics.mean(e0.elapsed_time(e1) for e0, e1, e2 in rev)
        r_att = statistics.mean(e1.elapsed_time(e2) for e0, e1, e2 in rev)
        rope = {"ms_per_step": r_ms, "value": world * F / (r_ms * 1e-3) / 1e12, "unit": "TFLOP/s",
                "attention_ms": r_att, "attention_tflops": F / (r_att * 1e-3) / 1e12, "kv_append_ms": r_app,
                "kv_append_gbs": append_bytes(wl) / (r_app * 1e-3) / 1e9, "vs_plain_step": ms_step / r_ms,
                "base": 500000.0}
        if not args.no_fused:  # the same rotated step as one launch (rr_extend_step_rope)
            def rope_one():
                rr.extend_step(g["q"], g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"],
                               g["prefix_lens"], g["suffix_lens"], out=out_r, rope=table)

            for _ in range(args.warmup):
                rope_one()
            torch.cuda.synchronize(dev)
            oev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
            for e0, e1 in oev:
                e0.record(st)
                rope_one()
                e1.record(st)
            torch.cuda.synchronize(dev)
            if rr.device_error():
                raise RuntimeError("device error in the one-launch rotary-step region")
            o_ms = max_over_ranks(statistics.mean(e0.elapsed_time(e1) for e0, e1 in oev), world, dev)
            rope.update({"one_launch_ms": o_ms, "one_launch_value": world * F / (o_ms * 1e-3) / 1e12,
                         "one_launch_vs_two_calls": r_ms / o_ms})
        # restore the un-rotated suffix keys for the legs that follow
        rr.kv_append(g["k_new"], g["v_new"], g["k_pool"], g["v_pool"], g["page_table"], g["prefix_lens"],
                     g["suffix_lens"])
        del table, out_r

    per_agent = None
    if args.per_agent:
        per_agent = per_agent_latency(rr, wl, g, dev, st)
    g.clear()
    torch.cuda.empty_cache()
    replay = None
    if args.replay and rank == 0:
        replay = replay_leg(rr, synth, dev, st)
    legs = None
    if not args.no_legs:
        legs = [config_leg(rr, synth, name, min(args.steps, n), args.warmup, dev, st, peaks, rank, local)
                for name, n in LEG_CONFIGS if name != args.config]
    decode = None
    if not args.no_decode:
        decode = decode_leg(args, rr, synth, dev, st, peaks, rank)

    achieved = F / (attn_ms * 1e-3) / 1e12
    src_hash = kernel_source_hash()
    traffic = traffic_for(wl.name, src_hash)  # recorded for this whole batch (scaled from a slice), or None
    peak, peak_kind = tensor_peak(peaks, args.steps * ms_step)
    roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
            "frac": achieved / peak, "traffic": traffic, "peak_kind": peak_kind,
            "frac_of_burst": achieved / peaks["bf16"], "frac_of_sustained": achieved / peaks["bf16_sus"],
            "frac_of_nominal": achieved / NOMINAL_BF16_TFLOPS,
            "kernel": "extend_attn_kernel<128,2,3>" if wl.D == 128 else "extend_attn_kernel<64,4,4>",
            "algorithmic_bytes": attn_bytes(wl), "algorithmic_flops": F,
            "bytes_bound_frac": attn_bytes(wl) / (attn_ms * 1e-3) / 1e9 / peaks["hbm"],
            "kernel_source_hash": src_hash}

    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config_dict(wl, world),
        "inputs": {"sha256": wl.manifest()["sha256"][:16], "num_pages": wl.num_pages,
                   "pool_gb": 2.0 * wl.num_pages * wl.ps * wl.Hkv * wl.D * 2 / 1e9},
        "uncached_suffix_tokens_per_s": tok_s,
        "attention_ms": attn_ms, "kv_append_ms": app_ms,
        "attention_ms_median": statistics.median(ev[k][1].elapsed_time(ev[k][2]) for k in range(args.steps)),
        "attention_ms_min": min(ev[k][1].elapsed_time(ev[k][2]) for k in range(args.steps)),
        "kv_append_gbs": append_bytes(wl) / (app_ms * 1e-3) / 1e9,
        "roofline": roof,
        "e2e": e2e,
        # per step: the append (one kernel up to 2047 agents, else schedule + append), schedule + attention
        "gpu_launches": (3 if wl.B <= 2047 else 4) * args.steps,
        "clocks": clk,
    }
    if per_agent is not None:
        line["per_agent_extend"] = per_agent
    if fused is not None:
        line["fused_step"] = fused
    if rope is not None:
        line["rope_step"] = rope
    if legs is not None:
        line["configs"] = legs
    if decode is not None:
        line["decode"] = decode
    if replay is not None:
        line["replay"] = replay
    if rank == 0 and not args.no_cpu_baseline:
        f, t, rows, threads = cpu_oracle_sample(wl, args.baseline_flops, seed=7)
        line["cpu_baseline"] = {"value": f / t / 1e12, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
                                "sample": f"{rows} seeded suffix rows (all {wl.Hq} heads) of 2 seeded agents of {args.config}, "
                                          f"{f:.2e} flop; fp64 oracle; K/V generation not timed"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--config", default="c4_coding")
    ap.add_argument("--no-legs", action="store_true", help="skip the other long-context batches' legs")
    ap.add_argument("--ref-flops", type=float, default=5e9, help="oracle flops per reference-arm step")
    ap.add_argument("--baseline-flops", type=float, default=3e11, help="oracle flops of the cpu_baseline sample (~10 s on 16 cores)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--agents", type=int, default=0, help="only the first N agents (small profiling case)")
    ap.add_argument("--agent-stride", type=int, default=1,
                    help="only every K-th agent (small profiling case with the batch's mix of agent kinds)")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    ap.add_argument("--per-agent", action="store_true", help="also time each agent's extend step alone")
    ap.add_argument("--decode-config", default="c2_decode", help="decode batch of the decode leg")
    ap.add_argument("--no-decode", action="store_true", help="skip the decode-attention leg")
    ap.add_argument("--no-fused", action="store_true", help="skip the fused extend-step leg")
    ap.add_argument("--no-rope", action="store_true", help="skip the rotary-embedding step leg")
    ap.add_argument("--decode-agents", type=int, default=0, help="only the first N agents of the decode batch")
    ap.add_argument("--replay", action="store_true",
                    help="also replay synthetic agent traces under each eviction policy, timing every extend batch")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    world, rank, local = dist_setup(args)
    try:
        if args.impl == "reference":
            return run_reference(args, world, rank)
        return run_ours(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
