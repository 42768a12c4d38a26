"""The SDAR-8B head-shape sweep: verified tokens/s and the attention's share
of the HBM copy peak at every point of batch x prefix x draft length x draft
agreement (32 query / 8 KV heads, d 128, bf16, one layer, V 151936).

    python -m paper_2606_02544_gb300.sweep [--out table.md] [--steps 10]
        [--batch 1,8,32,128] [--prefix 512,2048,8192,32768]
        [--gamma 4,8,16,32] [--agree 0.3,0.6,0.9] [--sampled]

One JSON line per point on stdout.  Each point captures its step (mask,
attention, acceptance, commit; the prefix lengths reset before every step)
in a CUDA graph and times every step with CUDA events; the attention
launches are timed in a graph of their own.  When a step's bytes are below
4x the L2 size, L2 is flushed before every step.

--sampled times the stochastic acceptance alone over batch x gamma instead.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics

import torch

from . import build, inputs, simsd
from .measure import L2_BYTES, algorithmic_bytes, flush_l2
from .step import VerifyStep

_HERE = os.path.dirname(os.path.abspath(__file__))


def _hbm_peak():
    try:
        with open(os.path.join(_HERE, "..", "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _tensor_peak():
    try:
        with open(os.path.join(_HERE, "..", "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"])
    except Exception:
        return 1900.0


def run_point(w: inputs.Workload, steps: int, peak: float) -> dict:
    si = inputs.make_step_inputs(w, device="cuda")
    st = VerifyStep(si, restore_prefix=True)
    attn_bytes, attn_flops, acc_bytes = algorithmic_bytes(si)
    need_flush = attn_bytes + acc_bytes < 4 * L2_BYTES
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device="cuda") if need_flush else None
    ev = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] for _ in range(steps)]
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        st.run()
    torch.cuda.synchronize()
    # the steps (no event inside a step) and, apart, the attention launches
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for e in ev:
            if flush is not None:
                flush_l2(flush)
            st.restore()
            e[0].record()
            st.run(restore=False)
            e[1].record()
    ea = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] for _ in range(steps)]
    ga = torch.cuda.CUDAGraph()
    with torch.cuda.graph(ga, stream=stream):
        for e in ea:
            if flush is not None:
                flush_l2(flush)
            e[0].record()
            st.run_attention()
            e[1].record()
    for _ in range(2):
        g.replay()
        ga.replay()
    torch.cuda.synchronize()
    step_ms, attn_ms = [], []
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        step_ms += [e[0].elapsed_time(e[1]) for e in ev]
        ga.replay()
        torch.cuda.synchronize()
        attn_ms += [e[0].elapsed_time(e[1]) for e in ea]
    assert simsd.simsd_check_error(st.err) == 0
    tokens = st.verified_tokens()
    t_step = statistics.median(step_ms)
    t_attn = statistics.median(attn_ms)
    gbs = attn_bytes / (t_attn * 1e-3) / 1e9
    row = {"Bt": w.Bt, "prefix": w.prefix[0], "gamma": w.gamma, "p_agree": w.p_agree,
           "verified_tokens_per_step": tokens, "tokens_per_s": round(tokens / (t_step * 1e-3), 1),
           "step_us": round(t_step * 1e3, 2), "attention_us": round(t_attn * 1e3, 2),
           "attention_gbs": round(gbs, 1), "attention_frac": round(gbs / peak, 4),
           "attention_tflops": round(attn_flops / (t_attn * 1e-3) / 1e12, 1),
           "attention_tensor_frac": round(attn_flops / (t_attn * 1e-3) / 1e12 / _tensor_peak(), 4),
           "l2": "flushed" if need_flush else "larger than L2"}
    del g, st, si, flush
    torch.cuda.empty_cache()
    return row


def run_sampled_point(Bt: int, gamma: int, vocab: int, steps: int, peak: float) -> dict:
    """Times simsd_accept_sampled_ws alone (Sec. 3.2, Eq. (2); few long
    sequences split their log-sum-exp pass over many CTAs): one CUDA graph of
    `steps` calls, L2 flushed before each when the logits fit in 4x L2, every
    call timed by events inside the graph."""
    si = inputs.make_sampled_inputs(Bt, gamma, vocab, seed=Bt * 100 + gamma, device="cuda")
    ws = simsd.simsd_accept_sampled_workspace_bytes(Bt, gamma, vocab)
    work = torch.empty(ws, dtype=torch.uint8, device="cuda") if ws else None
    a = torch.empty(Bt, dtype=torch.int32, device="cuda")
    ot = torch.empty(Bt, gamma + 1, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    nbytes = Bt * (2 * gamma + 1) * vocab * 4          # every row read once
    need_flush = nbytes < 4 * L2_BYTES
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device="cuda") if need_flush else None
    ev = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] for _ in range(steps)]

    def call():
        simsd.simsd_accept_sampled_ws(si.target_logits, si.draft_logits, si.draft, si.u_accept, si.u_sample, a, ot,
                                      work, temperature=si.temperature, err_word=err)

    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        call()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for e in ev:
            if flush is not None:
                flush_l2(flush)
            e[0].record()
            call()
            e[1].record()
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    ts = []
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        ts += [e[0].elapsed_time(e[1]) for e in ev]
    assert simsd.simsd_check_error(err) == 0
    t = statistics.median(ts)
    gbs = nbytes / (t * 1e-3) / 1e9
    row = {"kernel": "accept_sampled" + ("+parts" if ws else ""), "Bt": Bt, "gamma": gamma, "vocab": vocab,
           "us": round(t * 1e3, 2),
           "algorithmic_bytes": nbytes, "gbs": round(gbs, 1), "frac": round(gbs / peak, 4),
           "l2": "flushed" if need_flush else "larger than L2"}
    del g, si, flush
    torch.cuda.empty_cache()
    return row


def points(bts, ns, gs, ps, args):
    """Workloads of batch x prefix x gamma x agreement: the preset sweep
    point where one exists (its seed), else one of the same shape, with the
    heads, page size, layer count and seed of the command line."""
    hq, hkv = (int(v) for v in args.heads.split("/"))
    preset = {(w.Bt, w.prefix[0], w.gamma, w.p_agree): w for w in inputs.sweep_points()}
    out = []
    for Bt in sorted(bts):
        for n in sorted(ns):
            for gm in sorted(gs):
                for pa in sorted(ps):
                    w = preset.get((Bt, n, gm, pa))
                    if w is None:
                        w = inputs.Workload(f"c5_b{Bt}_n{n}_g{gm}_p{pa}", "bf16", Bt, 32, 8, 128, gm, (n, n), 1,
                                            151936, pa, inputs._SD, 2.0, 9000 + Bt + n + gm)
                    w = dataclasses.replace(w, Hq=hq, Hkv=hkv, page_size=args.page_size, layers=args.layers,
                                            seed=w.seed if args.seed is None else args.seed)
                    out.append(w)
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--out", default=None, help="also write a markdown table here")
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--batch", default="1,8,32,128")
    ap.add_argument("--prefix", default="512,2048,8192,32768")
    ap.add_argument("--gamma", default="4,8,16,32")
    ap.add_argument("--agree", default="0.3,0.6,0.9")
    ap.add_argument("--heads", default="32/8", help="query/KV heads, e.g. 64/8")
    ap.add_argument("--page-size", type=int, default=64)
    ap.add_argument("--layers", type=int, default=1, help="stacked layers per step (independent K/V per layer)")
    ap.add_argument("--seed", type=int, default=None, help="seed of every point (default: the preset's)")
    ap.add_argument("--sampled", action="store_true",
                    help="time the stochastic acceptance alone over --batch x --gamma (V 151936)")
    args = ap.parse_args(argv)
    sel = lambda s, cast: {cast(x) for x in s.split(",")}
    bts, ns, gs, ps = sel(args.batch, int), sel(args.prefix, int), sel(args.gamma, int), sel(args.agree, float)
    build.build()
    simsd.load_library()
    peak, kind = _hbm_peak()
    rows = []
    if args.sampled:
        for Bt in sorted(bts):
            for gm in sorted(gs):
                row = run_sampled_point(Bt, gm, 151936, args.steps, peak)
                row["peak_gbs"], row["peak_source"] = peak, kind
                print(json.dumps(row), flush=True)
                rows.append(row)
        if args.out:
            with open(args.out, "w") as f:
                f.write(f"| Bt | gamma | path | us | GB/s (rows read once) | of {peak:.0f} GB/s |\n"
                        "|---|---|---|---|---|---|\n")
                for r in rows:
                    path = "parts + spans" if r["kernel"].endswith("+parts") else "cluster"
                    f.write(f"| {r['Bt']} | {r['gamma']} | {path} | {r['us']:.1f} | {r['gbs']:.0f} | "
                            f"{100 * r['frac']:.1f}% |\n")
        return
    for w in points(bts, ns, gs, ps, args):
            row = run_point(w, args.steps, peak)
            row["peak_gbs"], row["peak_source"] = peak, kind
            print(json.dumps(row), flush=True)
            rows.append(row)
    if args.out:
        with open(args.out, "w") as f:
            f.write(f"Heads {args.heads}, page size {args.page_size}, {args.layers} layer(s) per step.\n\n")
            f.write("| Bt | prefix | gamma | p | tokens/s | step us | attention us | attention GB/s | "
                    f"of {peak:.0f} GB/s | TFLOP/s | of {_tensor_peak():.0f} |\n"
                    "|---|---|---|---|---|---|---|---|---|---|---|\n")
            for r in rows:
                f.write(f"| {r['Bt']} | {r['prefix']} | {r['gamma']} | {r['p_agree']} | {r['tokens_per_s']:.0f} | "
                        f"{r['step_us']:.1f} | {r['attention_us']:.1f} | {r['attention_gbs']:.0f} | "
                        f"{100 * r['attention_frac']:.1f}% | {r['attention_tflops']:.0f} | "
                        f"{100 * r['attention_tensor_frac']:.1f}% |\n")


if __name__ == "__main__":
    main()
