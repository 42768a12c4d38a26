"""simsd_verify_attention_noalloc against simsd_verify_attention.

The allocation-free entry point serves callers that cannot call cudaMalloc
(code inside a CUDA-graph capture, or engines that give all device memory
to their own pool and must not stall on the allocator).  It must produce the
same attention as the regular entry point, whose scratch the caller
allocates, on consecutive calls that share the library's static scratch.
"""
import numpy as np
import pytest
import torch

from paper_2606_02544_gb300 import inputs, simsd
from tests._gpu import BF16_ATOL, BF16_RTOL, F32_ATOL, gpu_mask

pytestmark = pytest.mark.gpu


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


def _close(got, want, dtype):
    g = got.float().cpu().numpy()
    r = want.float().cpu().numpy()
    assert np.isfinite(g).all()
    if dtype == "f32":
        assert np.abs(g - r).max() <= F32_ATOL
    else:
        assert (np.abs(g - r) <= BF16_ATOL + BF16_RTOL * np.abs(r)).all()


def test_noalloc_matches_regular_entry_point_on_consecutive_calls():
    # Small batches with long prefixes make the kernel split each sequence's
    # prefix more than eight ways, so the split partials go through the
    # static scratch (up to eight splits merge in shared memory); the second
    # call uses other sizes and values, so stale contents would show.
    cases = [
        inputs.Workload("na1", "bf16", 1, 16, 8, 128, 4, (1200, 3000), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 21),
        inputs.Workload("na2", "bf16", 2, 32, 8, 128, 8, (300, 3000), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 22),
    ]
    for w in cases:
        si = inputs.make_step_inputs(w, device="cuda", random_step_map=True, with_logits=False)
        tau, sect, _, _, merr = gpu_mask(si, mask_bits=False)
        assert simsd.simsd_check_error(merr) == 0
        want, ws = _regular(si, tau, sect)
        assert ws > 0, "the case must use scratch"
        got = _noalloc(si, tau, sect)
        _close(got, want, w.dtype)


def test_noalloc_fp32_and_unsplit_shapes():
    for w in (inputs.WORKLOADS["c1"],
              inputs.Workload("na3", "bf16", 200, 8, 8, 128, 4, (64, 256), 1, 64, 0.5, 1 / np.sqrt(128), 1.0, 23)):
        si = inputs.make_step_inputs(w, device="cuda", with_logits=False)
        tau, sect, _, _, _ = gpu_mask(si, mask_bits=False)
        want, _ = _regular(si, tau, sect)
        got = _noalloc(si, tau, sect)
        _close(got, want, w.dtype)
