"""Pins of the oracle's greedy acceptance (SimSD Sec. 3.2, Eq. (2)).

At temperature 0 the draft and target distributions are one-hot, so
alpha_r = min(1, p_theta/p_phi) is 1 when the target's argmax equals the
draft and 0 otherwise; the longest prefix before the first rejection is
accepted and the target supplies the token at the first rejected position.
Pins: numpy's argmax (first occurrence, NaN first) with a cumulative-product
form of the prefix length, the p = 1 and forced-mismatch special cases, and
the expected accepted length sum_k p^k of independent agreements.
"""
import numpy as np
import pytest

from oracle import simsd_oracle as orc


def _numpy_reference(logits, draft):
    am = np.argmax(logits, axis=-1).astype(np.int32)       # first maximum; first NaN wins
    gamma = draft.shape[1]
    agree = draft == am[:, :gamma]
    a = np.cumprod(agree, axis=1).sum(1).astype(np.int32)
    ot = np.full((draft.shape[0], gamma + 1), -1, np.int32)
    for b in range(draft.shape[0]):
        ot[b, : a[b]] = draft[b, : a[b]]
        ot[b, a[b]] = am[b, a[b]]
    return a, ot, am


@pytest.mark.parametrize("gamma,V", [(1, 7), (4, 1024), (8, 333), (32, 64)])
def test_matches_numpy_with_ties_and_nans(gamma, V):
    rng = np.random.default_rng(gamma * 1000 + V)
    Bt = 24
    logits = rng.normal(0, 2, (Bt, gamma + 1, V)).astype(np.float32)
    logits[0, 0] = 1.5                                          # all equal -> index 0
    logits[1, :, 3] = logits[1].max(-1) + 1
    logits[1, :, V - 1] = logits[1, :, 3]                       # tie between 3 and V-1
    logits[2, 0, V // 2] = np.nan                               # NaN beats every number
    logits[2, 1, [1, V - 1]] = np.nan                           # first NaN wins
    logits[3, 0, :] = -np.inf
    logits[4, 0, 2] = -0.0
    logits[4, 0, :2] = -1.0
    logits[4, 0, 3:] = -1.0
    logits[4, 0, V - 1] = 0.0                                   # -0.0 == +0.0: lower index
    am = np.argmax(logits, -1)
    agree = rng.random((Bt, gamma)) < 0.7
    draft = np.where(agree, am[:, :gamma], rng.integers(0, V, (Bt, gamma))).astype(np.int32)
    a, ot, am_o, err = orc.accept(logits, draft, gamma)
    ra, rot, ram = _numpy_reference(logits, draft)
    assert err == 0
    np.testing.assert_array_equal(am_o, ram)
    np.testing.assert_array_equal(a, ra)
    np.testing.assert_array_equal(ot, rot)


def test_all_correct_and_first_wrong():
    rng = np.random.default_rng(0)
    gamma, V = 6, 500
    logits = rng.normal(size=(5, gamma + 1, V)).astype(np.float32)
    am = np.argmax(logits, -1).astype(np.int32)
    a, ot, _, _ = orc.accept(logits, am[:, :gamma], gamma)
    assert (a == gamma).all()
    np.testing.assert_array_equal(ot, am)                   # gamma drafts + the extra row's token
    bad = am[:, :gamma].copy()
    bad[:, 0] = (bad[:, 0] + 1) % V
    a, ot, _, _ = orc.accept(logits, bad, gamma)
    assert (a == 0).all()
    np.testing.assert_array_equal(ot[:, 0], am[:, 0])
    assert (ot[:, 1:] == -1).all()


def test_expected_accepted_length():
    # independent agreement with probability p' per draft: E[a] = sum_k p'^k
    rng = np.random.default_rng(42)
    gamma, V, Bt, p = 4, 64, 6000, 0.7
    logits = rng.normal(size=(Bt, gamma + 1, V)).astype(np.float32)
    am = np.argmax(logits, -1)
    agree = rng.random((Bt, gamma)) < p
    draft = np.where(agree, am[:, :gamma], rng.integers(0, V, (Bt, gamma))).astype(np.int32)
    a, _, _, _ = orc.accept(logits, draft, gamma)
    pe = p + (1 - p) / V
    want = sum(pe ** k for k in range(1, gamma + 1))
    assert abs(a.mean() - want) < 4 * a.std() / np.sqrt(Bt)


def test_out_of_range_draft_is_flagged_and_rejected():
    rng = np.random.default_rng(1)
    gamma, V = 4, 50
    logits = rng.normal(size=(3, gamma + 1, V)).astype(np.float32)
    am = np.argmax(logits, -1).astype(np.int32)
    draft = am[:, :gamma].copy()
    draft[0, 2] = V
    draft[1, 0] = -5
    draft[2, 3] = 1 << 30
    draft[2, 1] = (draft[2, 1] + 1) % V          # rejection happens before the bad id
    a, ot, _, err = orc.accept(logits, draft, gamma)
    assert err & orc.ERR_DRAFT
    np.testing.assert_array_equal(a, [2, 0, 1])
    assert ot[0, 2] == am[0, 2] and ot[1, 0] == am[1, 0]
