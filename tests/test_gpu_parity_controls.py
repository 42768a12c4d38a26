"""Negative controls of the attention parity bar.

A parity test is only evidence if it can fail.  Each control below takes a
kernel output that passes, plants one plausible mistake on the CPU side (in
the oracle's input, or in a CPU recomputation of one row), and checks that
the comparison of tests/_gpu.py then fails:

* an all-zero output (what a kernel that writes nothing would leave), at
  the SDAR-1.7B, SDAR-4B and SDAR-8B sizes;
* one dropped key tile: the oracle run with the last 64 prefix keys of a
  sequence cut off;
* one Eq. (1) bit flipped: one row's attention recomputed with one new-slot
  column added to or removed from its visible set.

The stated tolerance alone (2e-2 + 2e-2 |r|) accepts an all-zero output at
these sizes; the derived bound rejects it.
"""
import math

import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs
from tests._gpu import attention_check, gpu_attention, oracle_attention

pytestmark = pytest.mark.gpu


def _case(name, seqs=None, layers=None):
    wl = inputs.WORKLOADS[name]
    si = inputs.make_step_inputs(wl, device="cuda", layers=layers, poison_unused_rows=True)
    out, word, _ = gpu_attention(si)
    assert word == 0
    ref = oracle_attention(si, seqs=seqs)
    got = out if seqs is None else out[torch.as_tensor(seqs, device="cuda")]
    st = attention_check(got, ref)
    assert st["ok"], st
    return si, got, ref


@pytest.mark.parametrize("name,seqs,layers", [("c2", None, None), ("c3", [0, 17], None), ("c4", [3, 40], 1)])
def test_zero_output_fails(name, seqs, layers):
    _, got, ref = _case(name, seqs, layers)
    st = attention_check(torch.zeros_like(got), ref)
    assert st["tolerance_ok"], "the stated tolerance alone accepts zeros at this size"
    assert not st["bound_ok"] and st["out_of_bound"] > 0.5 * st["elements"], st


@pytest.mark.parametrize("name,layers", [("c2", None), ("c3", None), ("c4", 1)])
def test_dropped_last_tile_fails(name, layers):
    si = inputs.make_step_inputs(inputs.WORKLOADS[name], device="cuda", layers=layers, poison_unused_rows=True)
    out, word, _ = gpu_attention(si)
    # the sequence with the shortest prefix: one 64-key tile of 8000 keys
    # moves the output by less than the bf16 rounding bound
    n = si.prefix_len.cpu().numpy()
    b = int(np.argmin(n))
    ok = oracle_attention(si, seqs=[b])
    assert word == 0 and attention_check(out[b:b + 1], ok)["ok"]
    cut = int(n[b]) - 64
    bad = oracle_attention(si, seqs=[b], prefix_override=[cut])
    st = attention_check(out[b:b + 1], bad)
    assert not st["bound_ok"], st


def _row_attention(si, b, s, visible):
    """fp64 attention of slot s of sequence b for every query head, over the
    whole prefix and the new slots marked in ``visible`` (CPU, direct
    softmax)."""
    w = si.w
    P, g, d = w.page_size, w.g, w.d
    n = int(si.prefix_len[b])
    pages = si.block_table[b, :(n + P - 1) // P].long()
    kc = si.k_cache[0][pages].double().cpu().permute(1, 0, 2, 3).reshape(w.Hkv, -1, d)[:, :n]
    vc = si.v_cache[0][pages].double().cpu().permute(1, 0, 2, 3).reshape(w.Hkv, -1, d)[:, :n]
    cols = torch.as_tensor(np.flatnonzero(visible))
    kn = si.k_new[0][b].double().cpu().permute(1, 0, 2)[:, cols]
    vn = si.v_new[0][b].double().cpu().permute(1, 0, 2)[:, cols]
    K = torch.cat([kc, kn], dim=1)
    V = torch.cat([vc, vn], dim=1)
    q = si.q[0][b, s].double().cpu()
    out = torch.empty(w.Hq, d, dtype=torch.float64)
    for h in range(w.Hq):
        sc = K[h // g] @ q[h] / math.sqrt(d)
        p = torch.softmax(sc, dim=0)
        out[h] = p @ V[h // g]
    return out.numpy()


@pytest.mark.parametrize("name,prefix", [("c2", None), ("small", [40, 130])])
def test_flipped_mask_bit_fails(name, prefix):
    wl = inputs.WORKLOADS["c2"]
    si = inputs.make_step_inputs(wl if name == "c2" else
                                 inputs.Workload("f", "bf16", 2, 16, 8, 128, 4, (0, 200), 1, 64, 0.5,
                                                 1 / math.sqrt(128), 1.0, 9),
                                 device="cuda", prefix_override=prefix, random_step_map=True)
    out, word, _ = gpu_attention(si)
    n = si.prefix_len.cpu().numpy()
    b = int(np.argmin(n))
    ref = oracle_attention(si, seqs=[b])
    got = out[b:b + 1]
    assert word == 0 and attention_check(got, ref)["ok"]
    dense = orc.build_mask(si.step_map.cpu().numpy(), n, wl.gamma)["dense"][b].astype(bool)
    S = wl.S
    # the recomputation reproduces the oracle with the true mask
    for s in range(S):
        np.testing.assert_allclose(_row_attention(si, b, s, dense[s]), ref.out[0, s], rtol=0, atol=1e-12)
    # a row's own pair (never visible), a later data slot, an earlier mask slot
    g = wl.gamma
    for s, t in ((0, g), (1, 2), (g + 2, g + 1), (g + 1, 0)):
        vis = dense[s].copy()
        vis[t] = not vis[t]
        bad_out = ref.out.copy()
        bad_out[0, s] = _row_attention(si, b, s, vis)
        bad = type(ref)(bad_out, ref.err, ref.absv, ref.delta, ref.tiles, ref.dtype)
        st = attention_check(got, bad)
        assert not st["bound_ok"], (s, t, st)
