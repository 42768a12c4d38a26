"""simsd_verify_attention_noalloc against simsd_verify_attention.

The allocation-free entry point serves callers that cannot call cudaMalloc
(engines that hand all device memory to their own pool at start-up and must
not stall on the allocator, or code running where allocation is not
allowed).  Both entry points run the same kernels on the same plan and
differ only in where the split partials live (the library's static array
instead of caller memory), so their outputs must be bit-identical, on
consecutive calls that share the static array.  The one exception: where
simsd_verify_attention gives every CTA an equal share of all key tiles
(stream-K, whose partials would not fit the array), the no-alloc entry
point keeps the plan it had without that option; both are checked against
the oracle there.  This file is collected
last, so that a run that stops at the first failure has run every other
test first.
"""
import numpy as np
import pytest
import torch

from paper_2606_02544_gb300 import inputs, simsd
from tests._gpu import gpu_mask

pytestmark = pytest.mark.gpu

NOALLOC_SCRATCH_BYTES = 12 << 20


def _regular(si, tau, sect):
    w = si.w
    dt = simsd.SIMSD_BF16 if si.q.dtype == torch.bfloat16 else simsd.SIMSD_F32
    ws = simsd.simsd_verify_workspace_bytes(dt, w.Bt, w.gamma, w.Hq, w.Hkv, w.d, si.block_table.shape[1],
                                            w.page_size)
    work = torch.zeros(ws, dtype=torch.uint8, device="cuda") if ws else None
    out = torch.full_like(si.q[0], float("nan"))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_verify_attention(si.q[0], si.k_new[0], si.v_new[0], si.k_cache[0], si.v_cache[0], si.block_table,
                                 si.prefix_len, tau, sect, out, workspace=work, err_word=err)
    assert simsd.simsd_check_error(err) == 0
    return out, ws


def _noalloc(si, tau, sect):
    out = torch.full_like(si.q[0], float("nan"))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_verify_attention_noalloc(si.q[0], si.k_new[0], si.v_new[0], si.k_cache[0], si.v_cache[0],
                                         si.block_table, si.prefix_len, tau, sect, out, err_word=err)
    assert simsd.simsd_check_error(err) == 0
    return out


def test_noalloc_matches_regular_entry_point_on_consecutive_calls():
    # Small batches with long prefixes make the kernel split each sequence's
    # prefix more than eight ways, so the split partials go through the
    # static scratch (up to eight splits merge in shared memory).  The
    # second call has other sizes and values and reads what it wrote over
    # the first call's partials; both must equal the regular entry point.
    cases = [
        inputs.Workload("na1", "bf16", 1, 16, 8, 128, 4, (1200, 3000), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 21),
        inputs.Workload("na2", "bf16", 2, 32, 8, 128, 8, (300, 3000), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 22),
    ]
    for w in cases:
        si = inputs.make_step_inputs(w, device="cuda", random_step_map=True, with_logits=False)
        tau, sect, _, _, merr = gpu_mask(si, mask_bits=False)
        assert simsd.simsd_check_error(merr) == 0
        want, ws = _regular(si, tau, sect)
        assert 0 < ws <= NOALLOC_SCRATCH_BYTES, "the case must use the static scratch"
        got = _noalloc(si, tau, sect)
        assert torch.equal(got, want)


def test_noalloc_fp32_and_unsplit_shapes():
    for w in (inputs.WORKLOADS["c1"],
              inputs.Workload("na3", "bf16", 200, 8, 8, 128, 4, (64, 256), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 23)):
        si = inputs.make_step_inputs(w, device="cuda", with_logits=False)
        tau, sect, _, _, _ = gpu_mask(si, mask_bits=False)
        want, _ = _regular(si, tau, sect)
        got = _noalloc(si, tau, sect)
        assert torch.equal(got, want)


def test_noalloc_keeps_whole_units_where_streamk_runs():
    # 20 sequences of 32 drafts: simsd_verify_attention walks stream-K runs
    # (40 MB of partials); the no-alloc entry point keeps the units whole,
    # no scratch: another order of summation, both within the bars
    from tests._gpu import assert_attention_close, oracle_attention
    w = inputs.Workload("na5", "bf16", 20, 32, 8, 128, 32, (3000, 4000), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 25)
    si = inputs.make_step_inputs(w, device="cuda", random_step_map=True, with_logits=False)
    tau, sect, _, _, _ = gpu_mask(si, mask_bits=False)
    want, ws = _regular(si, tau, sect)
    assert ws > NOALLOC_SCRATCH_BYTES
    got = _noalloc(si, tau, sect)
    ref = oracle_attention(si, seqs=[0, 9, 19])
    for out in (want, got):
        assert_attention_close(out[torch.as_tensor([0, 9, 19], device=out.device)], ref)


def test_noalloc_rejects_sizes_beyond_the_static_scratch():
    # one sequence of 32 drafts with a 32k-token prefix: 16 units split ~19
    # ways need ~20 MB of partials, more than the static array holds
    w = inputs.Workload("na4", "bf16", 1, 32, 8, 128, 32, (32768, 32768), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 24)
    si = inputs.make_step_inputs(w, device="cuda", with_logits=False)
    ws = simsd.simsd_verify_workspace_bytes(simsd.SIMSD_BF16, 1, 32, 32, 8, 128, si.block_table.shape[1], 64)
    assert ws > NOALLOC_SCRATCH_BYTES
    tau, sect, _, _, _ = gpu_mask(si, mask_bits=False)
    out = torch.full_like(si.q[0], float("nan"))
    with pytest.raises(simsd.SimsdError) as exc:
        simsd.simsd_verify_attention_noalloc(si.q[0], si.k_new[0], si.v_new[0], si.k_cache[0], si.v_cache[0],
                                             si.block_table, si.prefix_len, tau, sect, out)
    assert exc.value.status == simsd.SIMSD_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert torch.isnan(out.float()).all(), "nothing may be launched for a rejected call"
