"""Pins of the oracle's stochastic acceptance (Sec. 3.2, Eq. (2)).

The expectations come from outside the oracle: the speculative-sampling
theorem (the first emitted token is distributed as p_theta when the draft is
drawn from p_phi), numpy softmax / cumsum / searchsorted, hand-worked
two-token cases, and the low-temperature limit, which must reduce to the
greedy rule.
"""
import numpy as np
import pytest

from oracle import simsd_oracle as orc


def np_softmax(x, t=1.0):
    z = np.asarray(x, np.float64) / t
    z = np.exp(z - z.max(axis=-1, keepdims=True))
    return z / z.sum(axis=-1, keepdims=True)


def test_hand_worked_two_token_case():
    # p_theta = (0.8, 0.2), p_phi = (0.5, 0.5)
    tl = np.log(np.array([[[0.8, 0.2], [0.5, 0.5]]], np.float64)).astype(np.float32)
    dl = np.log(np.array([[[0.5, 0.5]]], np.float64)).astype(np.float32)
    for x, u, want_a, want_tok in ((0, 0.99, 1, None), (1, 0.39, 1, None), (1, 0.41, 0, 0)):
        a, ot, al, _, err = orc.accept_sampled(tl, dl, np.array([[x]], np.int32), np.array([[u]], np.float32),
                                               np.array([0.5], np.float32), 1)
        assert err == 0
        np.testing.assert_allclose(al[0, 0], 1.0 if x == 0 else 0.4, rtol=1e-6)
        assert a[0] == want_a
        if want_tok is not None:
            # residual max(0, p_theta - p_phi) = (0.3, 0): the target token is 0
            assert ot[0, 0] == want_tok and ot[0, 1] == -1


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_first_token_is_distributed_as_the_target(seed):
    """Speculative-sampling theorem: with x ~ p_phi and independent uniform
    u_accept, u_sample, P(first emitted token = v) = p_theta(v)."""
    r = np.random.default_rng(seed)
    V, N = 6, 20000
    tl = r.normal(size=(1, 2, V)).astype(np.float32) * 1.5
    dl = r.normal(size=(1, 1, V)).astype(np.float32) * 1.5
    pt = np_softmax(tl[0, 0])
    pd = np_softmax(dl[0, 0])
    us = ((np.arange(N) + 0.5) / N).astype(np.float32)   # midpoint grid of u_sample
    dist = np.zeros(V)
    for x in range(V):
        # acceptance: the oracle's alpha (accept iff u_accept < alpha)
        _, _, al, _, _ = orc.accept_sampled(tl, dl, np.array([[x]], np.int32), np.zeros((1, 1), np.float32),
                                            np.zeros(1, np.float32), 1)
        alpha = al[0, 0]
        np.testing.assert_allclose(alpha, min(1.0, pt[x] / pd[x]), rtol=1e-6)
        # after a rejection: the drawn token over the u_sample grid
        reps = np.repeat(tl, N, axis=0), np.repeat(dl, N, axis=0)
        a, ot, _, _, _ = orc.accept_sampled(reps[0], reps[1], np.full((N, 1), x, np.int32),
                                            np.ones((N, 1), np.float32), us, 1)
        assert (a == 0).all()
        freq = np.bincount(ot[:, 0], minlength=V) / N
        dist += pd[x] * (alpha * np.eye(V)[x] + (1.0 - alpha) * freq)
    np.testing.assert_allclose(dist, pt, atol=2e-4)


def test_equal_distributions_accept_all_and_draw_from_the_bonus_row():
    r = np.random.default_rng(4)
    Bt, gamma, V = 5, 3, 50
    tl = r.normal(size=(Bt, gamma + 1, V)).astype(np.float32)
    dl = tl[:, :gamma].copy()
    dr = r.integers(0, V, (Bt, gamma)).astype(np.int32)
    ua = r.random((Bt, gamma)).astype(np.float32) * 0.999
    us = r.random(Bt).astype(np.float32)
    a, ot, al, _, err = orc.accept_sampled(tl, dl, dr, ua, us, gamma)
    assert err == 0 and (a == gamma).all()
    np.testing.assert_allclose(al, 1.0)
    for b in range(Bt):
        c = np.cumsum(np_softmax(tl[b, gamma]))
        want = int(np.searchsorted(c, np.float64(us[b]) * c[-1], side="right"))
        assert ot[b, gamma] == want
        np.testing.assert_array_equal(ot[b, :gamma], dr[b])


def test_longest_prefix_walk():
    r = np.random.default_rng(5)
    Bt, gamma, V = 1, 6, 30
    tl = r.normal(size=(Bt, gamma + 1, V)).astype(np.float32)
    dl = r.normal(size=(Bt, gamma, V)).astype(np.float32)
    dr = r.integers(0, V, (Bt, gamma)).astype(np.int32)
    _, _, al, _, _ = orc.accept_sampled(tl, dl, dr, np.zeros((Bt, gamma), np.float32), np.zeros(Bt, np.float32),
                                        gamma)
    for stop in range(gamma + 1):
        # accept rows < stop (u just below alpha), reject row stop (u at alpha)
        ua = np.array([[al[0, r_] * 0.5 if r_ < stop else (1.0 if al[0, r_] >= 1 else al[0, r_] + (1 - al[0, r_]) / 2)
                        for r_ in range(gamma)]], np.float32)
        a, ot, _, _, _ = orc.accept_sampled(tl, dl, dr, ua, np.zeros(Bt, np.float32), gamma)
        want = stop if stop < gamma and al[0, stop] < 1.0 else None
        if want is None:
            continue
        assert a[0] == want
        np.testing.assert_array_equal(ot[0, :want], dr[0, :want])
        assert (ot[0, want + 1:] == -1).all()


def test_low_temperature_reduces_to_the_greedy_rule():
    r = np.random.default_rng(6)
    Bt, gamma, V = 40, 4, 64
    # the draft model's greedy choice: x = argmax of its own logits, which
    # agrees with the target's argmax in about 60% of the rows
    tl = r.normal(size=(Bt, gamma + 1, V)).astype(np.float32)
    dl = r.normal(size=(Bt, gamma, V)).astype(np.float32)
    am = tl[:, :gamma].argmax(axis=2)
    agree = r.random((Bt, gamma)) < 0.6
    bi, ri = np.nonzero(agree)
    dl[bi, ri, am[bi, ri]] = dl[bi, ri].max(axis=1) + 1.0
    dr = dl.argmax(axis=2).astype(np.int32)
    ua = (0.01 + 0.98 * r.random((Bt, gamma))).astype(np.float32)
    us = (0.01 + 0.98 * r.random(Bt)).astype(np.float32)
    a, ot, _, _, err = orc.accept_sampled(tl, dl, dr, ua, us, gamma, temperature=1e-3)
    ga, got, _, gerr = orc.accept(tl, dr, gamma)
    assert err == gerr == 0
    np.testing.assert_array_equal(a, ga)
    np.testing.assert_array_equal(ot, got)


def test_temperature_scales_the_logits():
    r = np.random.default_rng(7)
    Bt, gamma, V = 6, 3, 40
    tl = r.normal(size=(Bt, gamma + 1, V)).astype(np.float32)
    dl = r.normal(size=(Bt, gamma, V)).astype(np.float32)
    dr = r.integers(0, V, (Bt, gamma)).astype(np.int32)
    ua = r.random((Bt, gamma)).astype(np.float32)
    us = r.random(Bt).astype(np.float32)
    one = orc.accept_sampled(tl, dl, dr, ua, us, gamma, temperature=1.0)
    two = orc.accept_sampled(2 * tl, 2 * dl, dr, ua, us, gamma, temperature=2.0)
    np.testing.assert_array_equal(one[0], two[0])
    np.testing.assert_array_equal(one[1], two[1])
    np.testing.assert_allclose(one[2], two[2], rtol=1e-12)


def test_out_of_range_draft_is_rejected_and_flagged():
    r = np.random.default_rng(8)
    tl = r.normal(size=(2, 3, 10)).astype(np.float32)
    dl = tl[:, :2].copy()
    dr = np.array([[3, 4], [10, 1]], np.int32)
    a, ot, al, _, err = orc.accept_sampled(tl, dl, dr, np.zeros((2, 2), np.float32), np.zeros(2, np.float32), 2)
    assert err & 8
    assert a[0] == 2 and a[1] == 0 and al[1, 0] == 0.0
