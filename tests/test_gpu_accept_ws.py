"""GPU parity of simsd_accept_ws: greedy acceptance with a caller workspace,
where a small batch's logits are split over more CTAs than one cluster per
sequence holds (per-part argmax keys, then a merge launch).  Outputs must be
bit-exact against the oracle and identical to simsd_accept's."""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import simsd
from tests.test_gpu_mask_accept import _accept_case

pytestmark = pytest.mark.gpu


def _run_ws(logits, draft, expect_split=None):
    Bt, rows, V = logits.shape
    gamma = rows - 1
    ws = simsd.simsd_accept_workspace_bytes(Bt, gamma, V)
    if expect_split is not None:
        assert (ws > 0) == expect_split, ws
    work = torch.full((max(ws, 8),), 0xAB, dtype=torch.uint8, device="cuda") if ws else None
    outs = []
    for use_ws in (True, False):
        a = torch.full((Bt,), -9, dtype=torch.int32, device="cuda")
        ot = torch.full((Bt, rows), -9, dtype=torch.int32, device="cuda")
        am = torch.full((Bt, rows), -9, dtype=torch.int32, device="cuda")
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        if use_ws:
            simsd.simsd_accept_ws(logits, draft, a, ot, work, am, err)
        else:
            simsd.simsd_accept(logits, draft, a, ot, am, err)
        outs.append((a.cpu().numpy(), ot.cpu().numpy(), am.cpu().numpy(), simsd.simsd_check_error(err)))
    ra, rot, ram, rerr = orc.accept(logits.cpu().numpy(), draft.cpu().numpy(), gamma)
    for a, ot, am, word in outs:
        np.testing.assert_array_equal(am, ram)
        np.testing.assert_array_equal(a, ra)
        np.testing.assert_array_equal(ot, rot)
        assert word == rerr
    return ra


@pytest.mark.parametrize("Bt,gamma,V", [(1, 16, 151936), (1, 32, 151936), (2, 16, 151936), (5, 16, 151936),
                                        (9, 12, 151936), (2, 16, 151935), (3, 32, 50001), (8, 8, 151936),
                                        (4, 8, 151936)])
def test_split_bit_exact(Bt, gamma, V):
    # few sequences with at least 4 MiB of logits each: the logits of each
    # split over many CTAs; an odd vocabulary streams scalars
    logits, draft = _accept_case(Bt, gamma, V, seed=Bt * 100 + gamma + V % 7)
    _run_ws(logits, draft, expect_split=True)


@pytest.mark.parametrize("Bt,gamma,V", [(64, 16, 151936), (10, 16, 151936), (8, 4, 151936), (1, 4, 151936),
                                        (2, 4, 1024), (1, 1, 64)])
def test_no_split_keeps_the_cluster_kernel(Bt, gamma, V):
    # more sequences than SMs / 16, or under 4 MiB of logits a sequence: no
    # workspace, the cluster kernel, same results
    logits, draft = _accept_case(Bt, gamma, V, seed=7 + Bt)
    _run_ws(logits, draft, expect_split=False)


def test_split_edge_values():
    Bt, gamma, V = 8, 12, 151936
    logits, draft = _accept_case(Bt, gamma, V, seed=5, p=1.0)
    logits[0, 0] = 0.5                                     # all equal: index 0
    logits[1, 1, 7] = float("nan")
    logits[1, 1, V - 1] = float("nan")                     # first NaN wins
    logits[2, :, 100] = 50.0
    logits[2, :, 140000] = 50.0                            # exact tie across parts: lower index
    logits[3, 0] = -float("inf")
    logits[3, 0, 123456] = float("inf")
    logits[4, 2] = -1.0
    logits[4, 2, 70000] = -0.0
    logits[4, 2, 90000] = 0.0                              # -0.0 == +0.0: the lower index
    logits[5, 0, 0] = float("nan")
    draft[6, 2] = V                                        # out of range: flagged, rejected
    draft[7, 0] = -1
    am = torch.argmax(logits, -1)
    draft[:6] = am[:6, :gamma].to(torch.int32)
    _run_ws(logits, draft, expect_split=True)


def test_workspace_checks():
    logits, draft = _accept_case(1, 16, 151936, seed=3)
    ws = simsd.simsd_accept_workspace_bytes(1, 16, 151936)
    assert ws > 0 and ws % 8 == 0
    a = torch.zeros(1, dtype=torch.int32, device="cuda")
    ot = torch.zeros(1, 17, dtype=torch.int32, device="cuda")
    small = torch.zeros(ws - 8, dtype=torch.uint8, device="cuda")
    with pytest.raises(simsd.SimsdError) as exc:
        simsd.simsd_accept_ws(logits, draft, a, ot, small)
    assert exc.value.status == simsd.SIMSD_ERR_INVALID_ARG
    with pytest.raises(simsd.SimsdError):
        simsd.simsd_accept_ws(logits, draft, a, ot, None)
    # reusing one workspace call after call gives the same results
    work = torch.empty(ws, dtype=torch.uint8, device="cuda")
    ref = None
    for _ in range(3):
        simsd.simsd_accept_ws(logits, draft, a, ot, work)
        got = (a.clone(), ot.clone())
        ref = ref or got
        assert torch.equal(got[0], ref[0]) and torch.equal(got[1], ref[1])
