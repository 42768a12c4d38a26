"""GPU parity of the fused rotary-embedding prologue (Sec. 3.1 "Position
Encoding Alignment") against the fp64 oracle: attention with un-rotated q
and k_new at the RoPE-copy positions of simsd_build_mask, at the physical
positions of the Table 4 ablation, the commit of rotated keys, and a whole
step.  Tolerances as for the plain paths (bf16: 2e-2 + 2e-2*|ref|; fp32:
1e-5); committed bf16 keys within one bf16 unit in the last place (the
kernel rotates in fp32 and rounds once, the oracle rounds the fp64 value).
"""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd
from paper_2606_02544_gb300.step import VerifyStep
from tests._gpu import assert_attention_close, gpu_attention, gpu_mask, oracle_attention

pytestmark = pytest.mark.gpu


def _w(dtype="bf16", Bt=3, Hq=16, Hkv=8, d=128, gamma=4, P=64, seed=0):
    std = 1.0 if dtype == "f32" else 1 / np.sqrt(128)
    return inputs.Workload("r", dtype, Bt, Hq, Hkv, d, gamma, (0, 300), 1, 64, 0.5, std, 1.0, seed, P)


def _rope_check(si, theta, mode=1):
    tau, sect, rope, _, merr = gpu_mask(si, mask_bits=False)
    assert simsd.simsd_check_error(merr) == 0
    if mode == 2:
        n = si.prefix_len.long()[:, None]
        rope = (n + torch.arange(si.w.S, device=n.device)[None]).to(torch.int32).contiguous()
    out, word, _ = gpu_attention(si, mask=(tau, sect), rope_pos=rope, rope_theta=theta)
    ref = oracle_attention(si, rope_theta=theta, rope_mode=mode)
    assert word == ref.err == 0
    return assert_attention_close(out, ref)


@pytest.mark.parametrize("gamma,Hq,Hkv", [(4, 16, 8), (8, 32, 8), (16, 32, 8), (32, 32, 8)])
def test_bf16_rope_copy(gamma, Hq, Hkv):
    w = _w(Bt=3, Hq=Hq, Hkv=Hkv, gamma=gamma, seed=gamma)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=[0, 65, 1000], random_step_map=True,
                                 poison_unused_rows=True)
    _rope_check(si, 1e6)


@pytest.mark.parametrize("P", [16, 64, 128])
def test_bf16_rope_split_and_pages(P):
    # two sequences: the prefix is split across CTAs, the new tile is in the first split
    w = _w(Bt=2, Hq=16, Hkv=8, gamma=4, P=P, seed=P)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=[3000, 129], random_step_map=True)
    _rope_check(si, 1e4)


def test_bf16_rope_large_positions():
    # positions near 2^15 exercise the angle reduction
    w = _w(Bt=2, Hq=8, Hkv=8, gamma=8, seed=3)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=[32700, 16000])
    _rope_check(si, 1e6)


def test_bf16_physical_positions_ablation():
    w = _w(Bt=3, gamma=8, Hq=32, Hkv=8, seed=4)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=[5, 70, 400], random_step_map=True)
    _rope_check(si, 1e6, mode=2)


@pytest.mark.parametrize("d", [64, 128])
def test_fp32_rope_copy(d):
    w = _w("f32", Bt=4, Hq=4, Hkv=2, d=d, gamma=3, P=16, seed=d)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=[0, 17, 64, 1030], random_step_map=True,
                                 poison_unused_rows=True)
    _rope_check(si, 1e4)
    _rope_check(si, 1e4, mode=2)


def test_noalloc_with_rope():
    w = _w(Bt=2, Hq=16, Hkv=8, gamma=4, seed=9)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=[700, 90], random_step_map=True)
    tau, sect, rope, _, _ = gpu_mask(si, mask_bits=False)
    out = torch.full_like(si.q[0], float("nan"))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_verify_attention_noalloc(si.q[0], si.k_new[0], si.v_new[0], si.k_cache[0], si.v_cache[0],
                                         si.block_table, si.prefix_len, tau, sect, out, err_word=err,
                                         rope_pos=rope, rope_theta=1e6)
    assert simsd.simsd_check_error(err) == 0
    assert_attention_close(out, oracle_attention(si, rope_theta=1e6))


def _values(bits, dtype):
    """Stored bits (uint16 bf16 patterns or float32) as float64 values."""
    if dtype == "bf16":
        return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return bits.astype(np.float64)


def _assert_keys_close(got_bits, want_bits, dtype):
    g = _values(got_bits, dtype)
    r = _values(want_bits, dtype)
    if dtype == "bf16":
        # one unit in the last place of an 8-bit significand
        tol = np.ldexp(1.0, np.frexp(np.abs(r))[1] - 8)
        assert (np.abs(g - r) <= tol + 1e-30).all()
    else:
        np.testing.assert_allclose(g, r, rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("dtype,P", [("bf16", 64), ("bf16", 16), ("f32", 8)])
def test_commit_rotates_keys(dtype, P):
    gamma = 8
    n = [0, 63, 64, 5, 2000, 127]
    w = inputs.Workload("c", dtype, len(n), 8, 4, 128 if dtype == "bf16" else 64, gamma, (0, 0), 2, 16, 0.5, 1.0,
                        1.0, 7, P)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=n, random_step_map=True, with_logits=False)
    a = torch.as_tensor(np.random.default_rng(1).integers(0, gamma + 1, len(n)).astype(np.int32), device="cuda")
    tau, sect, rope, _, err = gpu_mask(si, mask_bits=False)
    kc0, vc0 = si.k_cache.clone(), si.v_cache.clone()
    nn = si.prefix_len.clone()
    simsd.simsd_kv_commit(si.k_new, si.v_new, tau, sect, a, si.k_cache, si.v_cache, si.block_table, nn, err,
                          rope_pos=rope, rope_theta=1e6)
    word = simsd.simsd_check_error(err)
    rk, rv, rn, rerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), a.cpu().numpy(), inputs.host_bits(kc0),
                                     inputs.host_bits(vc0), si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), gamma, rope_theta=1e6)
    assert word == rerr == 0
    np.testing.assert_array_equal(nn.cpu().numpy(), rn)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)
    _assert_keys_close(inputs.host_bits(si.k_cache), rk, dtype)


@pytest.mark.parametrize("name,theta", [("c1", 1e4), ("c2", 1e6)])
def test_whole_step_with_rope(name, theta):
    wl = inputs.WORKLOADS[name]
    si = inputs.make_step_inputs(wl, device="cuda")
    ref = oracle_attention(si, rope_theta=theta)
    ra, rot, _, aerr = orc.accept(si.logits.cpu().numpy(), si.draft.cpu().numpy(), wl.gamma)
    kc0, vc0 = inputs.host_bits(si.k_cache), inputs.host_bits(si.v_cache)
    st = VerifyStep(si, restore_prefix=True, rope_theta=theta)
    st.capture()
    for _ in range(2):
        st.replay()
    word = simsd.simsd_check_error(st.err)
    assert word == ref.err == aerr == 0
    assert_attention_close(st.out[0], ref)
    np.testing.assert_array_equal(st.accepted_len.cpu().numpy(), ra)
    np.testing.assert_array_equal(st.out_tokens.cpu().numpy(), rot)
    rk, rv, rn, _ = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                  si.step_map.cpu().numpy(), ra, kc0, vc0, si.block_table.cpu().numpy(),
                                  si.prefix_len.cpu().numpy(), wl.gamma, rope_theta=theta)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)
    _assert_keys_close(inputs.host_bits(si.k_cache), rk, wl.dtype)
