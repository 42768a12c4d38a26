"""Failure detection on the GPU: a bounded on-device wait that runs out.

Every wait in the library's kernels gives up after a time limit, sets
SIMSD_EW_TIMEOUT in the caller's error word and lets the kernel finish in
order (in-flight copies and MMAs drained, tensor memory freed), so that the
context stays usable.  A test hook (simsd_debug_expire_next_wait) arms one
launch so that one of its barriers expects an arrival that never comes and
its waits give up after 200 us; nothing traps, faults or spins without a
limit.  The next, normal launch on the same stream must then give the same
bits as before the planted expiry and match the oracle.
"""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd
from tests._gpu import assert_attention_close, gpu_attention, gpu_mask, oracle_attention

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("Bt,Hq,gamma,prefix", [(40, 16, 4, (100, 300)), (20, 32, 32, (100, 300)),
                                               (20, 32, 32, (3000, 4000)), (2, 32, 32, (1500, 2000))])
def test_attention_wait_runs_out_and_the_context_stays_usable(Bt, Hq, gamma, prefix):
    # 40 sequences x 8 KV heads of 16 rows: 320 unsplit units in two waves
    # of the one-row-block kernel; 20 x 8 units of 256 rows: the persistent
    # two-row-block kernel on whole short units, or in stream-K runs of long
    # ones, then their merge (each block's PV issuer waits for P that the
    # planted count never completes); 2 x 8 units of 256 rows: the same
    # kernel with key-tile ranges, then the combine kernel
    w = inputs.Workload("we", "bf16", Bt, Hq, 8, 128, gamma, prefix, 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 31)
    si = inputs.make_step_inputs(w, device="cuda", random_step_map=True, with_logits=False)
    tau, sect, _, _, merr = gpu_mask(si, mask_bits=False)
    assert simsd.simsd_check_error(merr) == 0
    before, word, ws = gpu_attention(si, mask=(tau, sect))
    # a workspace for the ranges and the stream-K partials of the 256-row units
    assert word == 0 and (ws > 0) == (gamma == 32 and (Bt == 2 or prefix[0] >= 3000))
    simsd.simsd_debug_expire_next_wait(simsd.DEBUG_WAIT_ATTENTION, 200)
    out = torch.full_like(si.q[0], float("nan"))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    work = torch.zeros(ws, dtype=torch.uint8, device="cuda") if ws else None
    simsd.simsd_verify_attention(si.q[0], si.k_new[0], si.v_new[0], si.k_cache[0], si.v_cache[0], si.block_table,
                                 si.prefix_len, tau, sect, out, workspace=work, err_word=err)
    word = simsd.simsd_check_error(err)
    assert word == simsd.EW_TIMEOUT
    after, word, _ = gpu_attention(si, mask=(tau, sect))
    assert word == 0 and torch.equal(after, before)
    assert_attention_close(after, oracle_attention(si))


def test_accept_wait_runs_out_and_the_context_stays_usable():
    # 700 sequences: too many for one resident cluster each, so every
    # sequence runs as a single CTA (the only form the hook arms)
    Bt, gamma, V = 700, 4, 1024
    g = torch.Generator(device="cuda").manual_seed(5)
    logits = torch.randn(Bt, gamma + 1, V, generator=g, device="cuda")
    am = logits[:, :gamma].argmax(-1).to(torch.int32)
    draft = torch.where(torch.rand(Bt, gamma, generator=g, device="cuda") < 0.7, am,
                        torch.randint(0, V, (Bt, gamma), generator=g, device="cuda", dtype=torch.int32))
    a = torch.full((Bt,), -9, dtype=torch.int32, device="cuda")
    ot = torch.full((Bt, gamma + 1), -9, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_debug_expire_next_wait(simsd.DEBUG_WAIT_ACCEPT, 200)
    simsd.simsd_accept(logits, draft, a, ot, err_word=err)
    assert simsd.simsd_check_error(err) == simsd.EW_TIMEOUT
    err.zero_()
    simsd.simsd_accept(logits, draft, a, ot, err_word=err)
    assert simsd.simsd_check_error(err) == 0
    ra, rot, _, rerr = orc.accept(logits.cpu().numpy(), draft.cpu().numpy(), gamma)
    assert rerr == 0
    np.testing.assert_array_equal(a.cpu().numpy(), ra)
    np.testing.assert_array_equal(ot.cpu().numpy(), rot)


def test_hook_arguments_and_small_batches():
    with pytest.raises(simsd.SimsdError):
        simsd.simsd_debug_expire_next_wait(7, 200)
    with pytest.raises(simsd.SimsdError):
        simsd.simsd_debug_expire_next_wait(simsd.DEBUG_WAIT_ACCEPT, 1)
    # a small batch runs in clusters: the hook refuses to arm it, launches
    # nothing, and the arm is consumed
    logits = torch.randn(2, 5, 1024, device="cuda")
    draft = torch.zeros(2, 4, dtype=torch.int32, device="cuda")
    a = torch.full((2,), -9, dtype=torch.int32, device="cuda")
    ot = torch.full((2, 5), -9, dtype=torch.int32, device="cuda")
    simsd.simsd_debug_expire_next_wait(simsd.DEBUG_WAIT_ACCEPT, 200)
    with pytest.raises(simsd.SimsdError) as exc:
        simsd.simsd_accept(logits, draft, a, ot)
    assert exc.value.status == simsd.SIMSD_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert (a == -9).all()
    simsd.simsd_accept(logits, draft, a, ot)
    ra, _, _, _ = orc.accept(logits.cpu().numpy(), draft.cpu().numpy(), 4)
    np.testing.assert_array_equal(a.cpu().numpy(), ra)
