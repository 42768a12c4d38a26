"""GPU parity of simsd_accept_sampled_ws: stochastic acceptance with a caller
workspace, where the log-sum-exp pass of a small batch is split over many
CTAs (per-part (max, sum) pairs, merged by a second launch over spans of
row a whose last CTA per sequence draws the token).  The
comparison with the oracle is the one of tests/test_gpu_accept_sampled.py:
identical results wherever the oracle's own numbers put every decision
outside the fp32 band, a valid choice inside it."""
import numpy as np
import pytest
import torch

from paper_2606_02544_gb300 import inputs, simsd
from tests import test_gpu_accept_sampled as base

pytestmark = pytest.mark.gpu


def _gpu_ws(si):
    Bt, rows, V = si.target_logits.shape
    ws = simsd.simsd_accept_sampled_workspace_bytes(Bt, rows - 1, V)
    work = torch.full((ws,), 0xAB, dtype=torch.uint8, device="cuda") if ws else None
    a = torch.full((Bt,), -9, dtype=torch.int32, device="cuda")
    ot = torch.full((Bt, rows), -9, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_accept_sampled_ws(si.target_logits, si.draft_logits, si.draft, si.u_accept, si.u_sample, a, ot,
                                  work, temperature=si.temperature, err_word=err)
    torch.cuda.synchronize()
    return a.cpu().numpy(), ot.cpu().numpy(), simsd.simsd_check_error(err)


@pytest.mark.parametrize("Bt,gamma,V,T,eta", [
    (1, 8, 151936, 1.0, 0.5), (1, 32, 151936, 1.0, 0.3), (3, 16, 151936, 0.7, 0.5), (8, 16, 151936, 1.0, 0.4),
    (9, 12, 151936, 1.3, 0.5), (2, 16, 151935, 1.0, 0.5), (8, 4, 151936, 1.0, 0.5), (8, 8, 151936, 0.8, 0.6),
    (1, 2, 262144, 1.0, 0.5), (5, 1, 400000, 1.0, 0.5),
    # 3 rows over 192 parts: each row's pairs span ~64 parts, more than a
    # warp's lanes take in one round
    (1, 1, 1048576, 1.0, 0.5),
])
def test_split_matches_oracle(monkeypatch, Bt, gamma, V, T, eta):
    # at most SMs / 16 sequences with at least 3 MiB of logits each: split
    # (the last CTA of each sequence draws the token)
    assert simsd.simsd_accept_sampled_workspace_bytes(Bt, gamma, V) > 0
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=Bt * 31 + gamma, eta=eta, temperature=T, device="cuda")
    monkeypatch.setattr(base, "_gpu", _gpu_ws)
    base._compare(si)


@pytest.mark.parametrize("Bt,gamma,V", [(10, 4, 151936), (16, 8, 151936), (1, 4, 1024), (4, 1, 100000)])
def test_no_split_is_the_cluster_kernel(monkeypatch, Bt, gamma, V):
    # under 3 MiB a sequence, or more sequences than SMs / 16: no workspace,
    # the same bits as simsd_accept_sampled
    assert simsd.simsd_accept_sampled_workspace_bytes(Bt, gamma, V) == 0
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=Bt + gamma, device="cuda")
    got = _gpu_ws(si)
    ref = base._gpu(si)
    for x, y in zip(got[:2], ref[:2]):
        assert (x == y).all()
    assert got[2] == ref[2]


def test_split_equal_models_accept_everything(monkeypatch):
    # p_theta = p_phi: alpha = 1 for every draft (to rounding)
    si = inputs.make_sampled_inputs(2, 16, 151936, seed=4, device="cuda")
    si.draft_logits = si.target_logits[:, :16].contiguous()
    si.u_accept = si.u_accept * 0.999
    monkeypatch.setattr(base, "_gpu", _gpu_ws)
    a, _ = base._compare(si)
    assert (a == 16).all()


def test_workspace_checks():
    si = inputs.make_sampled_inputs(1, 16, 151936, seed=2, device="cuda")
    ws = simsd.simsd_accept_sampled_workspace_bytes(1, 16, 151936)
    assert ws > 0 and ws % 8 == 0
    a = torch.zeros(1, dtype=torch.int32, device="cuda")
    ot = torch.zeros(1, 17, dtype=torch.int32, device="cuda")
    small = torch.zeros(ws - 8, dtype=torch.uint8, device="cuda")
    with pytest.raises(simsd.SimsdError) as exc:
        simsd.simsd_accept_sampled_ws(si.target_logits, si.draft_logits, si.draft, si.u_accept, si.u_sample, a, ot,
                                      small)
    assert exc.value.status == simsd.SIMSD_ERR_INVALID_ARG


def test_split_bad_draft_with_empty_residual(monkeypatch):
    # equal models: a draft id outside the vocabulary is the only way to
    # reject, the residual is empty and the last CTA draws from p_theta
    Bt, gamma, V = 4, 4, 200000
    assert simsd.simsd_accept_sampled_workspace_bytes(Bt, gamma, V) > 0
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=12, device="cuda")
    si.draft_logits = si.target_logits[:, :gamma].contiguous()
    si.u_accept = si.u_accept * 0.999
    si.draft[0, 0] = V
    si.draft[1, 2] = -1
    monkeypatch.setattr(base, "_gpu", _gpu_ws)
    a, _ = base._compare(si, expect_err=simsd.EW_DRAFT)
    assert list(a[:2]) == [0, 2] and (a[2:] == gamma).all()


def test_split_edge_logits(monkeypatch):
    # masked vocabulary, one dominant token, u at both ends of [0, 1), on
    # the split path
    Bt, gamma, V = 6, 3, 262144
    assert simsd.simsd_accept_sampled_workspace_bytes(Bt, gamma, V) > 0
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=13, device="cuda")
    si.target_logits[0, :, 60000:] = -float("inf")
    si.draft_logits[0, :, 120000:] = -float("inf")
    si.draft[0] = torch.randint(0, 60000, (gamma,), dtype=torch.int32)
    si.target_logits[1, :, 7] = 80.0
    si.target_logits[4, :, V - 3] = 80.0                   # dominant token in the last span
    si.u_accept[2] = 0.0
    si.u_sample[2] = 0.0
    si.u_sample[3] = float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    si.u_accept[3] = 0.9999999
    monkeypatch.setattr(base, "_gpu", _gpu_ws)
    base._compare(si)
