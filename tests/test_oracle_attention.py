"""Pins of the oracle's verification attention (SimSD Sec. 3.2, Sec. 3.3).

The oracle's masked attention is checked against: torch's
scaled_dot_product_attention in fp64 with the mask taken from the prose
statement; closed forms (constant values, zero keys); invariances (page
placement, shifting all keys); and the single-layer equivalence with
ordinary step-by-step decoding that the paper's precision analysis (Sec. 4.3)
states: each position's direct attention visibility matches its denoising
step, so one attention layer reproduces sequential decoding exactly.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs
from tests._pins import dense_prefix, library_attention, widen


def _tiny(dtype="f32", Bt=3, Hq=4, Hkv=2, d=16, gamma=4, prefix=(0, 130), P=16, seed=0):
    return inputs.Workload("tiny", dtype, Bt, Hq, Hkv, d, gamma, prefix, 1, 64, 0.5, 1.0, 1.0, seed, P)


def _run_oracle(si, layer=0, threads=0):
    return orc.verify_attention(
        inputs.host_bits(si.q[layer]), inputs.host_bits(si.k_new[layer]), inputs.host_bits(si.v_new[layer]),
        inputs.host_bits(si.k_cache[layer]), inputs.host_bits(si.v_cache[layer]), si.block_table.numpy(),
        si.prefix_len.numpy(), si.step_map.numpy(), si.w.gamma, threads=threads)


def _run_library(si, layer=0):
    return library_attention(
        inputs.host_bits(si.q[layer]), inputs.host_bits(si.k_new[layer]), inputs.host_bits(si.v_new[layer]),
        inputs.host_bits(si.k_cache[layer]), inputs.host_bits(si.v_cache[layer]), si.block_table.numpy(),
        si.prefix_len.numpy(), si.step_map.numpy(), si.w.gamma)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("gamma,P", [(1, 16), (2, 64), (4, 16), (5, 8)])
def test_matches_library_sdpa(dtype, gamma, P):
    w = _tiny(dtype, gamma=gamma, P=P, seed=gamma)
    for n in ([0, 1, 63], [64, 65, 130], [17, 0, 128]):
        si = inputs.make_step_inputs(w, prefix_override=n, random_step_map=True, with_logits=False)
        out, err = _run_oracle(si)
        assert err == 0
        ref = _run_library(si)
        np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_poisoned_unused_rows_are_never_read():
    # Rows of the page pool that hold no prefix row are NaN; the result must
    # be finite and equal to the library result.
    w = _tiny("bf16", gamma=4, P=16)
    si = inputs.make_step_inputs(w, prefix_override=[5, 33, 70], poison_unused_rows=True, with_logits=False)
    out, err = _run_oracle(si)
    assert err == 0 and np.isfinite(out).all()
    np.testing.assert_allclose(out, _run_library(si), rtol=1e-12, atol=1e-12)


def test_constant_values_give_that_constant():
    # softmax weights sum to one: if every visible V row equals c, O = c.
    w = _tiny("f32", gamma=3, P=16)
    si = inputs.make_step_inputs(w, prefix_override=[0, 20, 47], random_step_map=True, with_logits=False)
    c = torch.linspace(-2, 3, w.d)
    si.v_cache[:] = c
    si.v_new[:] = c
    out, _ = _run_oracle(si)
    np.testing.assert_allclose(out, np.broadcast_to(c.double().numpy(), out.shape), rtol=0, atol=1e-13)


def test_zero_keys_average_exactly_n_plus_gamma_values():
    # With K = 0 every visible key scores 0, so O is the mean of the visible
    # V rows; each row sees the n prefix rows and exactly gamma new slots.
    w = _tiny("f32", gamma=4, P=16)
    si = inputs.make_step_inputs(w, prefix_override=[0, 9, 64], random_step_map=True, with_logits=False)
    si.k_cache.zero_()
    si.k_new.zero_()
    out, _ = _run_oracle(si)
    vn = si.v_new[0].double().numpy()
    vc = si.v_cache[0].double().numpy()
    bt = si.block_table.numpy()
    mu_all = si.step_map.numpy()
    for b in range(w.Bt):
        n = int(si.prefix_len[b])
        mu = mu_all[b]
        for kvh in range(w.Hkv):
            pref_sum = dense_prefix(vc, bt, b, n, kvh).sum(0)
            for s in range(w.S):
                k, is_mask = s % w.gamma, s >= w.gamma
                t = mu[k]
                # new slots seen: data slots with smaller label (and itself for a
                # data row), mask slots with larger label (and itself for a mask row)
                seen = [j for j in range(w.gamma) if (mu[j] < t or (not is_mask and mu[j] == t))]
                seen_m = [j for j in range(w.gamma) if (mu[j] > t or (is_mask and mu[j] == t))]
                assert len(seen) + len(seen_m) == w.gamma
                tot = pref_sum + vn[b, seen, kvh].sum(0) + vn[b, [w.gamma + j for j in seen_m], kvh].sum(0)
                want = tot / (n + w.gamma)
                for h in range(kvh * w.g, (kvh + 1) * w.g):
                    np.testing.assert_allclose(out[b, s, h], want, rtol=1e-12, atol=1e-13)


def test_shift_of_all_keys_leaves_output_unchanged():
    # Adding one vector c to every key changes all scores of a row by the
    # same amount q.c, which the softmax cancels.
    w = _tiny("f32", gamma=4, P=16)
    si = inputs.make_step_inputs(w, prefix_override=[3, 40, 64], random_step_map=True, with_logits=False)
    # keys on a 2^-10 grid and an integer shift keep k + c exact in fp32
    si.k_cache = torch.round(si.k_cache * 1024) / 1024
    si.k_new = torch.round(si.k_new * 1024) / 1024
    base, _ = _run_oracle(si)
    c = torch.randint(-3, 4, (w.d,), generator=torch.Generator().manual_seed(4)).float()
    si.k_cache += c
    si.k_new += c
    shifted, _ = _run_oracle(si)
    np.testing.assert_allclose(shifted, base, rtol=1e-11, atol=1e-12)


def test_page_placement_does_not_change_result():
    w = _tiny("bf16", gamma=4, P=8)
    si = inputs.make_step_inputs(w, prefix_override=[30, 8, 57], with_logits=False)
    out1, _ = _run_oracle(si)
    # move every page to a new physical slot
    perm = torch.randperm(si.num_pages, generator=torch.Generator().manual_seed(1))
    inv = torch.argsort(perm)
    kc = si.k_cache[0][inv]   # new page p holds old page perm[p]
    vc = si.v_cache[0][inv]
    bt = si.block_table.clone()
    valid = bt >= 0
    bt[valid] = perm.to(torch.int32)[bt[valid].long()]
    out2, err = orc.verify_attention(
        inputs.host_bits(si.q[0]), inputs.host_bits(si.k_new[0]), inputs.host_bits(si.v_new[0]),
        inputs.host_bits(kc), inputs.host_bits(vc), bt.numpy(), si.prefix_len.numpy(), si.step_map.numpy(),
        w.gamma)
    assert err == 0
    np.testing.assert_array_equal(out1, out2)


def test_thread_count_does_not_change_bits():
    w = _tiny("bf16", gamma=4, P=16)
    si = inputs.make_step_inputs(w, prefix_override=[30, 100, 57], random_step_map=True, with_logits=False)
    a, _ = _run_oracle(si, threads=1)
    b, _ = _run_oracle(si, threads=4)
    np.testing.assert_array_equal(a, b)


def test_padding_rows_zero_and_error_paths():
    w = _tiny("f32", gamma=4, P=16)
    si = inputs.make_step_inputs(w, prefix_override=[10, 20, 30], with_logits=False)
    sm = si.step_map.clone()
    sm[0, 1] = 0                      # padding position in sequence 0
    si.step_map = sm
    out, err = _run_oracle(si)
    assert err == 0
    assert (out[0, [1, 1 + w.gamma]] == 0).all()
    assert np.abs(out[0, [0, 2, 3]]).sum() > 0
    # prefix longer than the block table can hold
    n = si.prefix_len.clone()
    n[1] = si.block_table.shape[1] * w.page_size + 1
    si.prefix_len = n
    out, err = _run_oracle(si)
    assert err & orc.ERR_PREFIX_LEN and (out[1] == 0).all() and np.abs(out[2]).sum() > 0
    # a page id outside the pool
    si.prefix_len = torch.tensor([10, 20, 30], dtype=torch.int32)
    bt = si.block_table.clone()
    bt[2, 0] = si.num_pages
    si.block_table = bt
    out, err = _run_oracle(si)
    assert err & orc.ERR_PAGE and (out[2] == 0).all() and np.abs(out[1]).sum() > 0


# --------------------------------------------------------------------------
# Single-layer equivalence with step-by-step decoding (Sec. 3.2, Sec. 4.3)
# --------------------------------------------------------------------------

@dataclasses.dataclass
class _Toy:
    E: np.ndarray
    emask: np.ndarray
    pos: np.ndarray
    Wq: np.ndarray
    Wk: np.ndarray
    Wv: np.ndarray
    Wo: np.ndarray
    Wr: np.ndarray

    @staticmethod
    def make(seed, Vt=48, dm=16, Hq=2, Hkv=1, d=16, npos=256):
        r = np.random.default_rng(seed)
        return _Toy(r.normal(size=(Vt, dm)), r.normal(size=dm), 0.5 * r.normal(size=(npos, dm)),
                    r.normal(size=(Hq, dm, d)) / 4, r.normal(size=(Hkv, dm, d)) / 4,
                    r.normal(size=(Hkv, dm, d)) / 4, r.normal(size=(Hq * d, Vt)),
                    r.normal(size=(Hq * d, dm)) / 8)

    def qkv(self, h):
        """Per-slot projections of hidden states h [m][dm], rounded to the
        float32 values that both sides then read."""
        q = np.einsum("md,hde->mhe", h, self.Wq).astype(np.float32)
        k = np.einsum("md,hde->mhe", h, self.Wk).astype(np.float32)
        v = np.einsum("md,hde->mhe", h, self.Wv).astype(np.float32)
        return q, k, v


def _bidir(q, K, V):
    """Plain unmasked attention of one query row per head (library sdpa)."""
    Hq, d = q.shape
    g = Hq // K.shape[1]
    out = np.zeros((Hq, d))
    for h in range(Hq):
        o = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[h][None, None].astype(np.float64)),
            torch.from_numpy(K[:, h // g][None].astype(np.float64)),
            torch.from_numpy(V[:, h // g][None].astype(np.float64)), scale=1.0 / np.sqrt(d))
        out[h] = o[0, 0].numpy()
    return out


def _paged(K, V, P, rng):
    """Places prefix rows K, V [n][Hkv][d] into a shuffled page pool whose
    other rows hold unrelated values; returns (k_cache, v_cache, table)."""
    n, Hkv, d = K.shape
    npages = max((n + P - 1) // P, 1)
    num_pages = npages + 2
    order = rng.permutation(num_pages)[:npages]
    kc = rng.normal(size=(num_pages, Hkv, P, d)).astype(np.float32)
    vc = rng.normal(size=(num_pages, Hkv, P, d)).astype(np.float32)
    for j in range(n):
        kc[order[j // P], :, j % P] = K[j]
        vc[order[j // P], :, j % P] = V[j]
    return kc, vc, order.astype(np.int32)[None]


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_single_layer_equals_step_by_step_decode(seed):
    rng = np.random.default_rng(100 + seed)
    toy = _Toy.make(seed)
    gamma = 5
    n = int(rng.integers(0, 40))
    mu = (rng.permutation(gamma) + 1).astype(np.int32)
    prefix_tok = rng.integers(0, toy.E.shape[0], n)
    hp = toy.E[prefix_tok] + toy.pos[:n]
    _, Kp, Vp = toy.qkv(hp)
    slot_of = {int(t): k for k, t in enumerate(mu)}

    # sequential greedy decoding of the block along the step map
    x = [None] * gamma
    seq_logits, seq_mask_out, seq_data_out = [], {}, {}

    def block_hidden(state):
        return np.stack([(toy.E[state[k]] if state[k] is not None else toy.emask) + toy.pos[n + k]
                         for k in range(gamma)])

    for r in range(1, gamma + 1):
        ks = slot_of[r]
        qb, Kb, Vb = toy.qkv(block_hidden(x))
        o = _bidir(qb[ks], np.concatenate([Kp, Kb]), np.concatenate([Vp, Vb]))
        seq_mask_out[r] = o
        lg = (o.reshape(-1) @ toy.Wo).astype(np.float32)
        seq_logits.append(lg)
        x[ks] = int(np.argmax(lg))
        # the data token of step r is read with the state after step r
        qb2, Kb2, Vb2 = toy.qkv(block_hidden(x))
        seq_data_out[r] = _bidir(qb2[ks], np.concatenate([Kp, Kb2]), np.concatenate([Vp, Vb2]))

    # one verification forward with the drafts equal to the decoded tokens
    hD = np.stack([toy.E[x[k]] + toy.pos[n + k] for k in range(gamma)])
    hM = np.stack([toy.emask + toy.pos[n + k] for k in range(gamma)])      # RoPE copy: same position
    q, k, v = toy.qkv(np.concatenate([hD, hM]))
    kc, vc, bt = _paged(Kp, Vp, 8, rng)
    out, err = orc.verify_attention(q[None], k[None], v[None], kc, vc, bt, [n], mu[None], gamma)
    assert err == 0
    for r in range(1, gamma + 1):
        ks = slot_of[r]
        np.testing.assert_allclose(out[0, gamma + ks], seq_mask_out[r], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(out[0, ks], seq_data_out[r], rtol=1e-12, atol=1e-13)

    # acceptance over the verification logits accepts every correct draft
    ver_logits = [(out[0, gamma + slot_of[r]].reshape(-1) @ toy.Wo).astype(np.float32)
                  for r in range(1, gamma + 1)]
    ver_logits.append((out[0, slot_of[gamma]].reshape(-1) @ toy.Wo).astype(np.float32))
    drafts = np.array([x[slot_of[r]] for r in range(1, gamma + 1)], np.int32)
    a, ot, am, err = orc.accept(np.stack(ver_logits)[None], drafts[None], gamma)
    assert err == 0 and a[0] == gamma
    np.testing.assert_array_equal(ot[0, :gamma], drafts)


@pytest.mark.parametrize("seed,n_draft", [(0, 3), (1, 1), (2, 5), (3, 0), (4, 0), (5, 2)])
def test_single_layer_with_undrafted_and_decoded_positions(seed, n_draft):
    """A block of B positions: some decoded earlier in the block (code -2),
    n_draft drafted along a random order, the rest left [MASK] (code -1).
    Each prediction row must equal plain bidirectional attention over the
    block as it stands when that row predicts: positions known before its
    step hold their clean token, every other position its [MASK] input.
    Each data row equals the same after its own step.  n_draft = 0 is the
    target completing the block itself (Sec. 3.2)."""
    rng = np.random.default_rng(500 + seed)
    toy = _Toy.make(40 + seed)
    B = 6
    n = int(rng.integers(0, 30))
    order = rng.permutation(B)
    codes = np.full(B, orc.STEP_UNDRAFTED, np.int32)
    codes[order[:n_draft]] = rng.permutation(n_draft) + 1
    n_dec = int(rng.integers(1, B - n_draft + 1)) if n_draft < B else 0
    codes[order[n_draft:n_draft + n_dec]] = orc.STEP_DECODED
    tok = rng.integers(0, toy.E.shape[0], B)
    big = 10 ** 9
    known = [0 if c == orc.STEP_DECODED else (big if c == orc.STEP_UNDRAFTED else int(c)) for c in codes]
    hp = toy.E[rng.integers(0, toy.E.shape[0], n)] + toy.pos[:n]
    _, Kp, Vp = toy.qkv(hp)

    def block_hidden(t):
        # the block when every position known before step t is decoded
        return np.stack([(toy.E[tok[k]] if known[k] < t else toy.emask) + toy.pos[n + k] for k in range(B)])

    hD = np.stack([toy.E[tok[k]] + toy.pos[n + k] for k in range(B)])
    hM = np.stack([toy.emask + toy.pos[n + k] for k in range(B)])
    q, k, v = toy.qkv(np.concatenate([hD, hM]))
    kc, vc, bt = _paged(Kp, Vp, 8, rng)
    out, err = orc.verify_attention(q[None], k[None], v[None], kc, vc, bt, [n], codes[None], B)
    assert err == 0
    for j in range(B):
        if codes[j] != orc.STEP_DECODED:        # a prediction row, at its step
            qb, Kb, Vb = toy.qkv(block_hidden(known[j]))
            want = _bidir(qb[j], np.concatenate([Kp, Kb]), np.concatenate([Vp, Vb]))
            np.testing.assert_allclose(out[0, B + j], want, rtol=1e-12, atol=1e-13)
        else:
            assert (out[0, B + j] == 0).all()
        if codes[j] != orc.STEP_UNDRAFTED:      # a data row, just after its step
            qb, Kb, Vb = toy.qkv(block_hidden(known[j] + 1))
            want = _bidir(qb[j], np.concatenate([Kp, Kb]), np.concatenate([Vp, Vb]))
            np.testing.assert_allclose(out[0, j], want, rtol=1e-12, atol=1e-13)
        else:
            assert (out[0, j] == 0).all()


def test_two_layers_are_only_approximate():
    # With two layers the data slots' hidden states were formed under their
    # own decoding step, not the current one, so the match is no longer exact
    # (Sec. 4.3: the approximation comes from higher-order interactions).
    rng = np.random.default_rng(7)
    toy1, toy2 = _Toy.make(11), _Toy.make(12)
    gamma = 4
    mu = (rng.permutation(gamma) + 1).astype(np.int32)
    slot_of = {int(t): k for k, t in enumerate(mu)}
    x = [int(t) for t in rng.integers(0, toy1.E.shape[0], gamma)]
    empty_k = np.zeros((1, 1, 8, 16), np.float32)
    bt = np.zeros((1, 1), np.int32)

    def layer2_seq(r):
        state = [x[k] if mu[k] < r else None for k in range(gamma)]
        h0 = np.stack([(toy1.E[state[k]] if state[k] is not None else toy1.emask) + toy1.pos[k]
                       for k in range(gamma)])
        q, K, V = toy1.qkv(h0)
        h1 = np.stack([h0[k] + _bidir(q[k], K, V).reshape(-1) @ toy1.Wr for k in range(gamma)])
        q2, K2, V2 = toy2.qkv(h1)
        return _bidir(q2[slot_of[r]], K2, V2)

    hD = np.stack([toy1.E[x[k]] + toy1.pos[k] for k in range(gamma)])
    hM = np.stack([toy1.emask + toy1.pos[k] for k in range(gamma)])
    h0 = np.concatenate([hD, hM])
    q, k, v = toy1.qkv(h0)
    o1, _ = orc.verify_attention(q[None], k[None], v[None], empty_k, empty_k, bt, [0], mu[None], gamma)
    h1 = h0 + o1[0].reshape(2 * gamma, -1) @ toy1.Wr
    q2, k2, v2 = toy2.qkv(h1)
    o2, _ = orc.verify_attention(q2[None], k2[None], v2[None], empty_k, empty_k, bt, [0], mu[None], gamma)
    gap = max(np.abs(o2[0, gamma + slot_of[r]] - layer2_seq(r)).max() for r in range(1, gamma + 1))
    assert gap > 1e-6
