"""Attention parity at the full sizes of the SDAR-shaped workloads, in the
launch configuration the benchmark times (both bars of tests/_gpu.py).

* SDAR-1.7B layer (8 sequences) and SDAR-4B layer (32 sequences of 4096
  cached tokens): every sequence against the oracle;
* SDAR-8B step over 36 layers through ``VerifyStep`` (mask, every layer's
  attention, acceptance, commit): eight sequences of every layer, drawn by
  seed, against the oracle; acceptance bit-exact on all 64 sequences; the
  prefix lengths advanced by the accepted lengths;
* the target's own block decoding (every block position decoded earlier or
  still [MASK]) at the SDAR-1.7B and SDAR-4B sizes.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd
from paper_2606_02544_gb300.step import VerifyStep
from tests._gpu import assert_attention_close, gpu_attention, oracle_attention

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["c2", "c3"])
def test_full_size_layer_every_sequence(name):
    wl = inputs.WORKLOADS[name]
    si = inputs.make_step_inputs(wl, device="cuda", poison_unused_rows=True)
    out, word, _ = gpu_attention(si)
    ref = oracle_attention(si)
    assert word == ref.err == 0
    assert_attention_close(out, ref)


def test_c4_whole_step_every_layer():
    wl = inputs.WORKLOADS["c4"]
    si = inputs.make_step_inputs(wl, device="cuda")
    ra, rot, _, aerr = orc.accept(si.logits.cpu().numpy(), si.draft.cpu().numpy(), wl.gamma)
    n0 = si.prefix_len.cpu().numpy()
    st = VerifyStep(si, restore_prefix=True)
    st.run()
    assert simsd.simsd_check_error(st.err) == 0 and aerr == 0
    np.testing.assert_array_equal(st.accepted_len.cpu().numpy(), ra)
    np.testing.assert_array_equal(st.out_tokens.cpu().numpy(), rot)
    np.testing.assert_array_equal(st.n.cpu().numpy(), n0 + ra)
    rng = np.random.default_rng(36)
    for layer in range(wl.layers):
        seqs = sorted(rng.choice(wl.Bt, 8, replace=False).tolist())
        ref = oracle_attention(si, layer=layer, seqs=seqs)
        assert ref.err == 0
        assert_attention_close(st.out[layer][torch.as_tensor(seqs, device="cuda")], ref)


@pytest.mark.parametrize("name", ["c2", "c3"])
def test_full_size_target_block_decoding(name):
    w = dataclasses.replace(inputs.WORKLOADS[name], layers=1)
    si = inputs.make_step_inputs(w, device="cuda", with_logits=False)
    si.step_map = inputs.block_step_maps(w.Bt, w.gamma, seed=5, n_draft=0).cuda()
    out, word, _ = gpu_attention(si)
    ref = oracle_attention(si)
    assert word == ref.err == 0
    assert_attention_close(out, ref)
