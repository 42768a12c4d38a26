"""Full-size points of the SDAR-8B sweep (32/8 heads, d 128, bf16, V 151936)
run through the step runner the sweep times: attention checked against the
oracle on sampled sequences (both bars of tests/_gpu.py), acceptance on
every sequence (bit-exact).  The points cover every batch size, the longest
prefix and the 256-row units of 32 drafts (two row blocks per KV head)."""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd
from paper_2606_02544_gb300.step import VerifyStep
from tests._gpu import assert_attention_close, oracle_attention

pytestmark = pytest.mark.gpu


def _point(Bt, n, gamma, p):
    for w in inputs.sweep_points():
        if (w.Bt, w.prefix[0], w.gamma, w.p_agree) == (Bt, n, gamma, p):
            return w
    raise KeyError((Bt, n, gamma, p))


@pytest.mark.parametrize("Bt,n,gamma,p,seqs", [(128, 512, 32, 0.6, [0, 63, 127]),
                                               (1, 32768, 4, 0.3, [0]),
                                               (32, 8192, 16, 0.9, [0, 31]),
                                               (8, 2048, 8, 0.6, [3]),
                                               (32, 8192, 32, 0.3, [5, 20]),
                                               (8, 32768, 32, 0.9, [2]),
                                               (1, 8192, 32, 0.6, [0]),
                                               (128, 32768, 32, 0.6, [77]),
                                               (128, 8192, 16, 0.3, [0, 100])])
def test_sweep_point(Bt, n, gamma, p, seqs):
    w = _point(Bt, n, gamma, p)
    si = inputs.make_step_inputs(w, device="cuda")
    ref = oracle_attention(si, seqs=seqs)
    ra, rot, _, aerr = orc.accept(si.logits.cpu().numpy(), si.draft.cpu().numpy(), gamma)
    st = VerifyStep(si, restore_prefix=True)
    st.run()
    assert simsd.simsd_check_error(st.err) == 0 and ref.err == 0 and aerr == 0
    assert_attention_close(st.out[0][torch.as_tensor(seqs, device="cuda")], ref)
    np.testing.assert_array_equal(st.accepted_len.cpu().numpy(), ra)
    np.testing.assert_array_equal(st.out_tokens.cpu().numpy(), rot)


def test_sampled_sweep_point_runs_and_reports():
    from paper_2606_02544_gb300 import sweep
    row = sweep.run_sampled_point(4, 4, 151936, steps=3, peak=6800.0)
    assert row["us"] > 0 and row["algorithmic_bytes"] == 4 * 9 * 151936 * 4
    assert 0 < row["frac"] < 2
