"""GPU parity of simsd_kv_commit (bit-exact cache and prefix lengths) and of
the whole verification step, eager and captured in a CUDA graph."""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd
from paper_2606_02544_gb300.step import VerifyStep
from tests._gpu import assert_attention_close, gpu_mask, oracle_attention

pytestmark = pytest.mark.gpu


def _commit_case(dtype, L, gamma, P, n, seed):
    w = inputs.Workload("c", dtype, len(n), 8, 4, 128 if dtype == "bf16" else 64, gamma, (0, 0), L, 16, 0.5,
                        1.0, 1.0, seed, P)
    return inputs.make_step_inputs(w, device="cuda", prefix_override=n, random_step_map=True, with_logits=False)


@pytest.mark.parametrize("dtype,L,gamma,P", [("bf16", 3, 8, 64), ("bf16", 2, 32, 16), ("f32", 2, 4, 8),
                                             ("bf16", 1, 1, 64)])
def test_commit_bit_exact(dtype, L, gamma, P):
    n = [0, 63, 64, 5, 200, 127]
    si = _commit_case(dtype, L, gamma, P, n, seed=gamma + P)
    rng = np.random.default_rng(gamma)
    a = torch.as_tensor(rng.integers(0, gamma + 1, len(n)).astype(np.int32), device="cuda")
    tau, sect, _, _, err = gpu_mask(si, mask_bits=False)
    kc0, vc0 = si.k_cache.clone(), si.v_cache.clone()
    nn = si.prefix_len.clone()
    simsd.simsd_kv_commit(si.k_new, si.v_new, tau, sect, a, si.k_cache, si.v_cache, si.block_table, nn, err)
    word = simsd.simsd_check_error(err)
    rk, rv, rn, rerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), a.cpu().numpy(), inputs.host_bits(kc0),
                                     inputs.host_bits(vc0), si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), gamma)
    assert word == rerr == 0
    np.testing.assert_array_equal(nn.cpu().numpy(), rn)
    np.testing.assert_array_equal(inputs.host_bits(si.k_cache), rk)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)


@pytest.mark.parametrize("dtype,Hkv,d,gamma,P", [("bf16", 8, 128, 16, 8), ("f32", 8, 128, 8, 16),
                                                 ("bf16", 2, 64, 32, 1)])
def test_commit_rows_beyond_the_first_32_pages(dtype, Hkv, d, gamma, P):
    # destination rows past a sequence's first 32 pages (their page ids come
    # from a window that starts at the first destination page), rows that
    # straddle a page boundary, one-row pages (32 accepted rows on 32
    # pages), and rows of 8 heads x 128 fp32 (256 chunks of 16 bytes)
    n = [32 * P - 1, 32 * P, 41 * P - 2, 500, 7, 33 * P + 1]
    w = inputs.Workload("c", dtype, len(n), 2 * Hkv, Hkv, d, gamma, (0, 0), 2, 16, 0.5, 1.0, 1.0, gamma + P, P)
    si = inputs.make_step_inputs(w, device="cuda", prefix_override=n, random_step_map=True, with_logits=False)
    rng = np.random.default_rng(P)
    a = rng.integers(1, gamma + 1, len(n)).astype(np.int32)
    a[2] = gamma
    a = torch.as_tensor(a, device="cuda")
    tau, sect, _, _, err = gpu_mask(si, mask_bits=False)
    kc0, vc0 = si.k_cache.clone(), si.v_cache.clone()
    nn = si.prefix_len.clone()
    simsd.simsd_kv_commit(si.k_new, si.v_new, tau, sect, a, si.k_cache, si.v_cache, si.block_table, nn, err)
    word = simsd.simsd_check_error(err)
    rk, rv, rn, rerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), a.cpu().numpy(), inputs.host_bits(kc0),
                                     inputs.host_bits(vc0), si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), gamma)
    assert word == rerr == 0
    np.testing.assert_array_equal(nn.cpu().numpy(), rn)
    np.testing.assert_array_equal(inputs.host_bits(si.k_cache), rk)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)


def test_commit_bad_page_past_the_first_32():
    P = 8
    si = _commit_case("bf16", 2, 8, P, [300, 40 * P + 5, 9], seed=3)
    bt = si.block_table.clone()
    bt[1, (40 * P + 5) // P + 1] = -3               # a destination page id below zero
    si.block_table = bt
    a = torch.tensor([4, 8, 2], dtype=torch.int32, device="cuda")
    tau, sect, _, _, err = gpu_mask(si, mask_bits=False)
    kc0, vc0 = si.k_cache.clone(), si.v_cache.clone()
    nn = si.prefix_len.clone()
    simsd.simsd_kv_commit(si.k_new, si.v_new, tau, sect, a, si.k_cache, si.v_cache, si.block_table, nn, err)
    word = simsd.simsd_check_error(err)
    rk, rv, rn, rerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), a.cpu().numpy(), inputs.host_bits(kc0),
                                     inputs.host_bits(vc0), si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), 8)
    assert word == rerr == simsd.EW_PAGE
    np.testing.assert_array_equal(nn.cpu().numpy(), rn)
    np.testing.assert_array_equal(inputs.host_bits(si.k_cache), rk)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)


@pytest.mark.parametrize("gamma", [4, 16])
def test_commit_with_undrafted_and_decoded_positions(gamma):
    # only drafted data slots are ever committed: a decoded slot (tau 0) and
    # an undrafted one (no data slot) never match an accepted step
    n = [0, 63, 64, 5, 200, 127, 31, 9]
    si = _commit_case("bf16", 2, gamma, 16, n, seed=gamma)
    si.step_map = inputs.block_step_maps(len(n), gamma, seed=gamma + 3).cuda()
    drafted = (si.step_map > 0).sum(1).cpu().numpy()
    rng = np.random.default_rng(gamma)
    a = torch.as_tensor(np.array([rng.integers(0, k + 1) for k in drafted], np.int32), device="cuda")
    tau, sect, _, _, err = gpu_mask(si, mask_bits=False)
    kc0, vc0 = si.k_cache.clone(), si.v_cache.clone()
    nn = si.prefix_len.clone()
    simsd.simsd_kv_commit(si.k_new, si.v_new, tau, sect, a, si.k_cache, si.v_cache, si.block_table, nn, err)
    word = simsd.simsd_check_error(err)
    rk, rv, rn, rerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), a.cpu().numpy(), inputs.host_bits(kc0),
                                     inputs.host_bits(vc0), si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), gamma)
    assert word == rerr == 0
    np.testing.assert_array_equal(nn.cpu().numpy(), rn)
    np.testing.assert_array_equal(inputs.host_bits(si.k_cache), rk)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)


def test_commit_error_paths():
    si = _commit_case("bf16", 2, 4, 16, [0, 14, 30, 7], seed=1)
    sm = si.step_map.clone()
    sm[3] = 0                                   # no source slot for sequence 3
    si.step_map = sm
    bt = si.block_table.clone()
    bt[2, 30 // 16] = si.num_pages              # destination page outside the pool
    si.block_table = bt
    a = torch.tensor([2, 9, 3, 1], dtype=torch.int32, device="cuda")  # sequence 1: a > gamma
    tau, sect, _, _, err = gpu_mask(si, mask_bits=False)
    kc0, vc0 = si.k_cache.clone(), si.v_cache.clone()
    nn = si.prefix_len.clone()
    simsd.simsd_kv_commit(si.k_new, si.v_new, tau, sect, a, si.k_cache, si.v_cache, si.block_table, nn, err)
    word = simsd.simsd_check_error(err)
    rk, rv, rn, rerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), a.cpu().numpy(), inputs.host_bits(kc0),
                                     inputs.host_bits(vc0), si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), 4)
    assert word == rerr and word & simsd.EW_PAGE and word & simsd.EW_ACCEPT_LEN and word & simsd.EW_STEP_MAP
    np.testing.assert_array_equal(nn.cpu().numpy(), rn)
    np.testing.assert_array_equal(inputs.host_bits(si.k_cache), rk)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)


@pytest.mark.parametrize("name", ["c1", "c2"])
@pytest.mark.parametrize("graph", [False, True])
def test_whole_step(name, graph):
    wl = inputs.WORKLOADS[name]
    si = inputs.make_step_inputs(wl, device="cuda")
    ref = oracle_attention(si)
    ra, rot, ram, aerr = orc.accept(si.logits.cpu().numpy(), si.draft.cpu().numpy(), wl.gamma)
    kc0, vc0 = inputs.host_bits(si.k_cache), inputs.host_bits(si.v_cache)
    st = VerifyStep(si, restore_prefix=True)
    if graph:
        st.capture()
        for _ in range(3):
            st.replay()
    else:
        st.run()
        st.run()
    word = simsd.simsd_check_error(st.err)
    assert word == 0 and ref.err == 0 and aerr == 0
    assert_attention_close(st.out[0], ref)
    np.testing.assert_array_equal(st.accepted_len.cpu().numpy(), ra)
    np.testing.assert_array_equal(st.out_tokens.cpu().numpy(), rot)
    np.testing.assert_array_equal(st.n.cpu().numpy(), si.prefix_len.cpu().numpy() + ra)
    rk, rv, rn, cerr = orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new),
                                     si.step_map.cpu().numpy(), ra, kc0, vc0, si.block_table.cpu().numpy(),
                                     si.prefix_len.cpu().numpy(), wl.gamma)
    np.testing.assert_array_equal(inputs.host_bits(si.k_cache), rk)
    np.testing.assert_array_equal(inputs.host_bits(si.v_cache), rv)


@pytest.mark.parametrize("with_table", [True, False])
def test_commit_without_layers_only_advances_prefix(with_table):
    # L = 0: there is no row to place, so the call only advances the prefix
    # lengths; the caller may then pass no K/V, no cache and no block table
    import ctypes
    lib = simsd.load_library()
    Bt, gamma = 4, 8
    dev = "cuda"
    n = torch.tensor([0, 5, 64, 100], dtype=torch.int32, device=dev)
    a = torch.tensor([0, 3, 8, 1], dtype=torch.int32, device=dev)
    sm = torch.arange(1, gamma + 1, dtype=torch.int32, device=dev).repeat(Bt, 1)
    tau = torch.empty(Bt, 2 * gamma, dtype=torch.int32, device=dev)
    sect = torch.empty(Bt, 2 * gamma, dtype=torch.uint8, device=dev)
    rope = torch.empty_like(tau)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    simsd.simsd_build_mask(sm, n, gamma, tau, sect, rope, err_word=err)
    bt = torch.zeros(Bt, 3, dtype=torch.int32, device=dev) if with_table else None
    n0 = n.clone()
    P = ctypes.c_void_p
    rc = lib.simsd_kv_commit(simsd.SIMSD_BF16, None, None, 0, P(tau.data_ptr()), P(sect.data_ptr()), None,
                             ctypes.c_float(0.0), P(a.data_ptr()), None, None, 0,
                             P(bt.data_ptr()) if bt is not None else None, 3, 64, P(n.data_ptr()), Bt, gamma, 8,
                             128, P(err.data_ptr()), P(torch.cuda.current_stream().cuda_stream))
    assert rc == simsd.SIMSD_OK
    assert simsd.simsd_check_error(err) == 0
    assert torch.equal(n, n0 + a)
