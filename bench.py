"""Benchmark of the SimSD verification step on GB300.

One step = the whole verification hot path over one batch: temporal-mask
metadata, the masked attention of every layer, greedy acceptance and the KV
commit, all through the C ABI (libsimsd.so), captured in a CUDA graph.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c4|c3|c2|c1]
    python bench.py --impl reference ...     # the fp64 CPU oracle on the host cores

Prints one JSON line.  ``value`` = verified tokens/s = sum_b (a_b + 1) per
step (accepted drafts plus the target's token) / device time per step,
summed over all ranks.  With N > 1 every rank runs an independent replica on
its own GPU (the step has no exchange between sequences): weak scaling.
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
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "verified draft tokens/sec per GB300; attention HBM GB/s vs 8 TB/s"
UNIT = "tokens/s"
# the largest configuration that fits one GPU: SDAR-8B head shapes, 64
# sequences, 36 layers (48.3 GB of KV cache), the KV-bound shape
DEFAULT_WORKLOAD = "c4"
DEFAULT_STEPS = {"c1": 2000, "c2": 2000, "c3": 400, "c4": 60}
UNROLL = {"c1": 50, "c2": 50, "c3": 20, "c4": 1}


def _dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


# the sources each stored traffic figure depends on: a kernel's own file and
# the headers it includes
TRAFFIC_SOURCES = {
    "attention": ("attention_tc.cu", "ptx.cuh", "common.cuh"),
    "accept": ("accept.cu", "ptx.cuh", "common.cuh"),
    "attention_tc256": ("attention_tc256.cu", "ptx.cuh", "common.cuh"),
}


def _kernel_sha(kernel):
    h = hashlib.sha256()
    for fn in TRAFFIC_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2606_02544_gb300", "csrc", fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


TRAFFIC_SOURCE = ("stored: profiles/traffic.json (ncu dram__bytes_read.sum + dram__bytes_write.sum per launch), "
                  "used only while the kernel's sources hash to the value recorded there")


def _traffic(workload, kernel):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the kernel's current sources; else None."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            d = json.load(f)
        entry = d.get(kernel, {})
        if entry.get("sha") != _kernel_sha(kernel):
            return None
        return entry.get(workload)
    except Exception:
        return None


def workload_config(wl, layers):
    """The workload description both arms print in ``config``."""
    return {"workload": wl.name, "Bt": wl.Bt, "Hq": wl.Hq, "Hkv": wl.Hkv, "head_dim": wl.d, "gamma": wl.gamma,
            "prefix": list(wl.prefix), "layers": layers, "vocab": wl.vocab, "page_size": wl.page_size,
            "p_agree": wl.p_agree, "seed": wl.seed, "draft_tokens_per_step": wl.Bt * wl.gamma}


def combine_over_ranks(total_ms, local_tokens, world):
    """Whole-job figures of N independent replicas (one per GPU, no data
    exchange): the slowest rank's timed milliseconds and every rank's
    verified tokens.  Needs an initialised process group when world > 1."""
    if world <= 1:
        return float(total_ms), float(local_tokens)
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(total_ms), float(local_tokens)], dtype=torch.float64)
    tmax = t.clone()
    dist.all_reduce(tmax, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(tmax[0]), float(t[1])


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled while the timed loop runs."""

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join(tempfile.gettempdir(), f"simsd_clocks_{os.getpid()}.csv")

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(self.gpu)], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [p.strip() for p in line.split(",")]
                    if len(parts) < 9:
                        continue
                    try:
                        sm.append(float(parts[1]))
                        mx = float(parts[2])
                    except ValueError:
                        continue
                    for nm, v in zip(names, parts[5:9]):
                        if v.lower() == "active":
                            reasons.add(nm)
            os.remove(self.path)
        except Exception:
            pass
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "samples": len(sm),
                "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------
def run_gpu(args):
    import torch

    from paper_2606_02544_gb300 import build, inputs, simsd
    from paper_2606_02544_gb300.measure import L2_BYTES, algorithmic_bytes, flush_l2
    from paper_2606_02544_gb300.step import VerifyStep

    rank, world, local = _dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    build.build()
    simsd.load_library()
    wl = inputs.WORKLOADS[args.workload]
    si = inputs.make_step_inputs(wl, device="cuda", layers=args.layers)
    st = VerifyStep(si, restore_prefix=True)
    torch.cuda.synchronize()

    attn_bytes, attn_flops, acc_bytes = algorithmic_bytes(si)
    step_bytes = attn_bytes * st.L + acc_bytes
    need_flush = step_bytes < 4 * L2_BYTES
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device="cuda") if need_flush else None
    M = UNROLL.get(args.workload, 1)
    M = max(1, min(M, args.steps))

    # one graph = M steps, each preceded by an L2 flush and bracketed by two
    # event-record nodes; nothing is recorded inside a step (an event node
    # between two kernels stops the next one from being scheduled early)
    ev = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] for _ in range(M)]
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        st.run()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for m in range(M):
            if flush is not None:
                flush_l2(flush)
            e = ev[m]
            # the prefix lengths are reset before the step starts (benchmark
            # plumbing that makes every step verify the same block)
            st.restore()
            e[0].record()
            st.run(restore=False)
            e[1].record()
    # accept-only timing graph piece: events around simsd_accept are taken
    # from the step's own graph nodes via a second capture of one step
    acc_ev = (torch.cuda.Event(enable_timing=True, external=True),
              torch.cuda.Event(enable_timing=True, external=True))
    g_acc = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_acc, stream=stream):
        if flush is not None:
            flush_l2(flush)
        acc_ev[0].record()
        simsd.simsd_accept(si.logits, si.draft, st.accepted_len, st.out_tokens, st.row_argmax, err_word=st.err)
        acc_ev[1].record()

    # attention-only graph: the layers' attention launches between two
    # events (after an L2 flush when the step is flushed too)
    attn_ev = (torch.cuda.Event(enable_timing=True, external=True),
               torch.cuda.Event(enable_timing=True, external=True))
    g_attn = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_attn, stream=stream):
        if flush is not None:
            flush_l2(flush)
        attn_ev[0].record()
        st.run_attention()
        attn_ev[1].record()

    reps = max(1, math.ceil(args.steps / M))
    warm_reps = max(1, math.ceil(args.warmup / M))
    for _ in range(warm_reps):
        graph.replay()
    torch.cuda.synchronize()

    step_ms, attn_ms, toks = [], [], []
    tokens_per_step = st.verified_tokens()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t_wall0 = time.perf_counter()
        for _ in range(reps):
            graph.replay()
            torch.cuda.synchronize()
            for m in range(M):
                step_ms.append(ev[m][0].elapsed_time(ev[m][1]))
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall0
    if world > 1:
        torch.distributed.barrier()
    clocks = clk.summary()
    K = len(step_ms)
    word = simsd.simsd_check_error(st.err)
    if word != 0:
        raise RuntimeError(f"device error word {word}")
    acc_times = []
    for _ in range(20):
        g_acc.replay()
        torch.cuda.synchronize()
        acc_times.append(acc_ev[0].elapsed_time(acc_ev[1]))
    for _ in range(max(3, min(20, int(2000 / max(1.0, 0.25 * st.L))))):
        g_attn.replay()
        torch.cuda.synchronize()
        attn_ms.append(attn_ev[0].elapsed_time(attn_ev[1]))

    total_ms = sum(step_ms)
    local_tokens = tokens_per_step * K
    total_ms_max, all_tokens = combine_over_ranks(total_ms, local_tokens, world)
    value = all_tokens / (total_ms_max / 1e3)

    # ---- end to end through the public API with host buffers
    e2e = run_e2e(args, si, st, stream) if rank == 0 else None

    hbm_peak, tf_peak, peak_kind = _peaks()
    attn_launch_ms = statistics.median(attn_ms) / st.L
    acc_launch_ms = statistics.median(acc_times)
    attn_gbs = attn_bytes / (attn_launch_ms * 1e-3) / 1e9
    acc_gbs = acc_bytes / (acc_launch_ms * 1e-3) / 1e9
    attn_roof = {"kernel": "simsd_verify_attention (attention_tc_kernel + combine_kernel when split)", "bound": "hbm",
                 "achieved": round(attn_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                 "frac": round(attn_gbs / hbm_peak, 4), "frac_of_8TBs": round(attn_gbs / 8000.0, 4),
                 "peak_source": peak_kind, "algorithmic_bytes_per_launch": int(attn_bytes),
                 "launch_us": round(attn_launch_ms * 1e3, 3),
                 "tensor_tflops": round(attn_flops / (attn_launch_ms * 1e-3) / 1e12, 2),
                 "tensor_frac": round(attn_flops / (attn_launch_ms * 1e-3) / 1e12 / tf_peak, 4),
                 "traffic": _traffic(args.workload, "attention"), "traffic_source": TRAFFIC_SOURCE}
    acc_roof = {"kernel": "simsd_accept (accept_kernel)", "bound": "hbm", "achieved": round(acc_gbs, 1),
                "peak": hbm_peak, "unit": "GB/s", "frac": round(acc_gbs / hbm_peak, 4), "peak_source": peak_kind,
                "algorithmic_bytes_per_launch": int(acc_bytes), "launch_us": round(acc_launch_ms * 1e3, 3),
                # rows up to the first rejection only: what a kernel that stopped
                # at the first mismatch would have to read
                "early_stop_bytes": int(tokens_per_step) * int(wl.vocab) * 4,
                "traffic": _traffic(args.workload, "accept"), "traffic_source": TRAFFIC_SOURCE}
    dominant, other = (attn_roof, acc_roof) if attn_launch_ms * st.L >= acc_launch_ms else (acc_roof, attn_roof)

    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            cpu = run_cpu_baseline(args, si, max_seconds=args.cpu_seconds)
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": warm_reps * M, "ms_per_step": round(total_ms_max / K, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32",
            "data": "synthetic (seeded; SDAR-shaped Q/K/V, logits and drafts; no weights)",
            "config": {**workload_config(wl, st.L),
                       "verified_tokens_per_step": tokens_per_step,
                       "l2": "flushed before every step (258 MB write + read)" if need_flush else
                       "inputs larger than L2 (no flush)",
                       "timing": f"CUDA graph of {M} steps; per-step CUDA events (the reset of the prefix "
                                 f"lengths between steps is outside them; no event inside a step); attention "
                                 f"and acceptance launch times from graphs of their own; max over ranks",
                       "parallelism": f"replicas x{world}"},
            "draft_tokens_per_s": round(wl.Bt * wl.gamma * K * world / (total_ms_max / 1e3), 1),
            "roofline": dominant, "roofline_other": other, "clocks": clocks, "e2e": e2e,
            "gpu_launches": st.launches_per_step() * K, "cpu_baseline": cpu,
            "wall_s_timed_region": round(t_wall, 3),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def run_e2e(args, si, st, stream):
    """Verified tokens/s through the public API with pinned host inputs:
    every step copies Q, K_new, V_new, logits, drafts and the step map host ->
    device, runs the step and reads accepted lengths + tokens back.  Two input
    sets alternate so that the copy of step k+1 (on a copy stream) overlaps
    step k (on the compute stream); the host reads step k's results while
    step k+1 runs."""
    import dataclasses

    import torch

    from paper_2606_02544_gb300.step import VerifyStep

    keys = ("q", "k_new", "v_new", "logits", "draft", "step_map")
    host_in = {k: getattr(si, k).cpu().pin_memory() for k in keys}
    # the second set has its own inputs and outputs and shares the caches;
    # steps still run one after the other on the compute stream
    si_b = dataclasses.replace(si, **{k: getattr(si, k).clone() for k in keys})
    sets = [st, VerifyStep(si_b, restore_prefix=True, rope_theta=st.rope_theta)]
    graphs = []
    for s_ in sets:
        with torch.cuda.stream(stream):
            s_.run()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            s_.run()
        graphs.append(g)
    h_a = [torch.empty_like(st.accepted_len, device="cpu").pin_memory() for _ in sets]
    h_t = [torch.empty_like(st.out_tokens, device="cpu").pin_memory() for _ in sets]
    bi = sum(t.numel() * t.element_size() for t in host_in.values())
    bo = h_a[0].numel() * 4 + h_t[0].numel() * 4
    steps = max(3, min(args.steps, 200 if si.w.layers == 1 else 10))
    copy_stream = torch.cuda.Stream()
    copied = [torch.cuda.Event() for _ in sets]
    done = [torch.cuda.Event() for _ in sets]
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)

    def issue(k):
        x = k % 2
        s_ = sets[x]
        with torch.cuda.stream(copy_stream):
            if k >= 2:
                copy_stream.wait_event(done[x])          # step k-2 is done with this set
            for name, t in host_in.items():
                getattr(s_.si, name).copy_(t, non_blocking=True)
            copied[x].record(copy_stream)
        with torch.cuda.stream(stream):
            stream.wait_event(copied[x])
            graphs[x].replay()
            h_a[x].copy_(s_.accepted_len, non_blocking=True)
            h_t[x].copy_(s_.out_tokens, non_blocking=True)
            done[x].record(stream)

    tokens = 0
    warm = 2
    torch.cuda.synchronize()
    for k in range(warm + steps):
        if k == warm:
            done[(k - 1) % 2].synchronize()
            e0.record(stream)
            tokens = 0
        issue(k)
        if k >= warm + 1:
            x = (k - 1) % 2
            done[x].synchronize()                         # step k-1's results on the host
            tokens += int(h_a[x].sum()) + si.w.Bt
    x = (warm + steps - 1) % 2
    done[x].synchronize()
    tokens += int(h_a[x].sum()) + si.w.Bt
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    return {"value": round(tokens / (ms / 1e3), 1), "unit": UNIT, "h2d_bytes_per_step": int(bi),
            "d2h_bytes_per_step": int(bo), "steps": steps, "ms_per_step": round(ms / steps, 4),
            "overlap": "inputs of step k+1 copied (copy stream) while step k runs"}


# ----------------------------------------------------------------------------
def _oracle_sample_step(orc, inputs, si, seqs, layers):
    """The oracle's whole step (mask, attention of the given layers, accept,
    commit) on the listed sequences; returns verified tokens."""
    import numpy as np
    import torch

    w = si.w
    idx = torch.as_tensor(seqs)
    P = w.page_size
    n = si.prefix_len.cpu()[idx]
    bt = si.block_table.cpu()[idx]
    need = [(int(n[r]) + w.gamma + P - 1) // P for r in range(len(seqs))]
    pages = torch.cat([bt[r, :need[r]] for r in range(len(seqs))]).long()
    uniq, inv = torch.unique(pages, return_inverse=True)
    nbt = torch.full_like(bt, -1)
    pos = 0
    for r in range(len(seqs)):
        nbt[r, :need[r]] = inv[pos:pos + need[r]].to(torch.int32)
        pos += need[r]
    sm = si.step_map.cpu()[idx].numpy()
    dev_idx = idx.to(si.q.device)
    for l in layers:
        orc.verify_attention(inputs.host_bits(si.q[l][dev_idx]), inputs.host_bits(si.k_new[l][dev_idx]),
                             inputs.host_bits(si.v_new[l][dev_idx]),
                             inputs.host_bits(si.k_cache[l][uniq.to(si.q.device)]),
                             inputs.host_bits(si.v_cache[l][uniq.to(si.q.device)]), nbt.numpy(), n.numpy(), sm,
                             w.gamma)
    a, _, _, _ = orc.accept(si.logits[dev_idx].cpu().numpy(), si.draft[dev_idx].cpu().numpy(), w.gamma)
    L = len(layers)
    kn = inputs.host_bits(si.k_new[: L][:, dev_idx]) if L else None
    if L:
        orc.kv_commit(kn, inputs.host_bits(si.v_new[: L][:, dev_idx]), sm, a,
                      inputs.host_bits(si.k_cache[: L][:, uniq.to(si.q.device)]),
                      inputs.host_bits(si.v_cache[: L][:, uniq.to(si.q.device)]), nbt.numpy(), n.numpy(), w.gamma)
    return int(np.sum(a)) + len(seqs)


def run_cpu_baseline(args, si, max_seconds=12.0):
    """The oracle as it stands, on this host's cores, on a bounded sample of
    the workload: whole sequences (all layers), repeated until about
    max_seconds of CPU work.  Host-side marshalling is excluded: only the
    oracle calls are timed."""
    from oracle import simsd_oracle as orc
    from paper_2606_02544_gb300 import inputs

    orc.build()
    w = si.w
    layers = list(range(si.q.shape[0]))
    order = list(range(w.Bt))
    done_tokens, t_used, seqs_done = 0, 0.0, 0
    i = 0
    while t_used < max_seconds and seqs_done < 100000:
        b = order[i % w.Bt]
        i += 1
        t0 = time.perf_counter()
        done_tokens += _oracle_sample_step(orc, inputs, si, [b], layers)
        t_used += time.perf_counter() - t0
        seqs_done += 1
    return {"value": round(done_tokens / t_used, 2), "unit": UNIT, "cores": orc.max_threads(), "kind": "oracle",
            "sample": f"{seqs_done} whole sequences x {len(layers)} layers of {w.name} (mask, attention, accept, "
                      f"commit), one sequence per oracle call, {t_used:.1f} s; the value is extrapolated to the "
                      f"workload as verified tokens of the sample / oracle seconds of the sample",
            "extrapolated": True}


def run_reference(args):
    """--impl reference: the fp64 oracle on the host cores (rank 0 only)."""
    rank, world, local = _dist_env()
    if rank != 0:
        return
    import torch

    from oracle import simsd_oracle as orc
    from paper_2606_02544_gb300 import inputs

    orc.build()
    wl = inputs.WORKLOADS[args.workload]
    device = "cuda" if torch.cuda.is_available() else "cpu"
    si = inputs.make_step_inputs(wl, device=device, layers=min(wl.layers, 2) if wl.layers > 2 else None)
    L = si.q.shape[0]
    layer_scale = wl.layers / L
    # each reference "step": one sequence through the whole oracle step,
    # cycling over the batch; throughput scaled to all layers of the workload
    per_step_budget = max(0.5, min(10.0, 120.0 / max(1, args.steps + args.warmup)))
    times, toks = [], []
    b = 0
    for k in range(args.warmup + args.steps):
        t_sum, tok = 0.0, 0
        while True:
            t0 = time.perf_counter()
            tok += _oracle_sample_step(orc, inputs, si, [b % wl.Bt], list(range(L)))
            t_sum += (time.perf_counter() - t0) * layer_scale
            b += 1
            if t_sum >= per_step_budget or b % wl.Bt == 0:
                break
        if k >= args.warmup:
            times.append(t_sum)
            toks.append(tok)
    value = sum(toks) / sum(times)
    cpu = {"value": round(value, 2), "unit": UNIT, "cores": orc.max_threads(), "kind": "oracle",
           "sample": f"{sum(toks)} verified tokens from whole sequences of {wl.name}; "
                     f"{L} of {wl.layers} layers timed, time scaled x{layer_scale:g}"}
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * sum(times) / len(times), 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic (seeded)",
            "config": {**workload_config(wl, wl.layers),
                       "timing": "the oracle on the host cores, wall clock per step of whole sequences"},
            "cpu_baseline": cpu,
            "e2e": {"value": round(value, 2), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=["c1", "c2", "c3", "c4"])
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="oracle time of the cpu_baseline sample (whole sequences until this much is spent)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=None,
                    help="run only this many layers of the workload (a smaller case of the same per-layer "
                         "kernels, for profiler captures)")
    args = ap.parse_args()
    if args.steps is None:
        args.steps = DEFAULT_STEPS[args.workload] if args.impl == "ours" else 10
    args.warmup = max(3, args.warmup)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
