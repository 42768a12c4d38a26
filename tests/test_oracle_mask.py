"""Pins of the oracle's temporal mask (SimSD Sec. 3.1, Eq. (1)).

Each check compares the oracle with something other than Eq. (1)'s case
table: hand-derived fixtures, the textbook triangular masks that the
identity step map reduces to, the paper's prose statements of the visible
sets (Sec. 3.1 "Masked Token Prediction", Sec. 3.2 "Target Model
Verification"), and structural invariants that follow from the rule.
"""
import itertools
import os

import numpy as np
import pytest

from oracle import simsd_oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    rows, mu = [], None
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            if line.startswith("step_map:"):
                mu = [int(x) for x in line.split(":")[1].split()]
                continue
            rows.append([int(x) for x in line.split()])
    return np.array(mu, np.int32), np.array(rows, np.uint8)


@pytest.mark.parametrize("name", ["mask_B4_identity.txt", "mask_B4_mu2413.txt"])
def test_golden_hand_derived(name):
    mu, want = _read_golden(name)
    r = orc.build_mask(mu[None, :], [7], len(mu))
    assert r["err"] == 0
    np.testing.assert_array_equal(r["dense"][0], want)


@pytest.mark.parametrize("gamma", [1, 2, 3, 4, 8, 16, 32])
def test_identity_reduces_to_triangular_masks(gamma):
    # With mu = identity, tau = block position.  D x D is the inclusive causal
    # (lower-triangular) mask of AR decoding; the verification slot of the r-th
    # draft sees the drafts before it only (Sec. 3.2), i.e. D~ x D is strictly
    # lower-triangular; D x D~ strictly upper and D~ x D~ inclusive upper.
    r = orc.build_mask(None, [0], gamma)
    A = r["dense"][0].astype(bool)
    one = np.ones((gamma, gamma), bool)
    np.testing.assert_array_equal(A[:gamma, :gamma], np.tril(one))
    np.testing.assert_array_equal(A[:gamma, gamma:], np.triu(one, 1))
    np.testing.assert_array_equal(A[gamma:, :gamma], np.tril(one, -1))
    np.testing.assert_array_equal(A[gamma:, gamma:], np.triu(one))


def _prose_mask(mu):
    """Visible sets as the paper's prose states them, by block position.

    Sec. 3.1 "Masked Token Prediction": a prediction slot D~_i sees data
    tokens from earlier steps and mask placeholders of the current and later
    steps.  Sec. 3.1 (after Eq. (1)): a data token D_i sees earlier data
    tokens (and itself) and later mask placeholders.
    """
    B = len(mu)
    A = np.zeros((2 * B, 2 * B), np.uint8)
    for i in range(B):
        data_seen_by_Di = {k for k in range(B) if mu[k] < mu[i]} | {i}
        mask_seen_by_Di = {k for k in range(B) if mu[k] > mu[i]}
        data_seen_by_Dti = {k for k in range(B) if mu[k] < mu[i]}
        mask_seen_by_Dti = {k for k in range(B) if mu[k] >= mu[i]}
        for k in data_seen_by_Di:
            A[i, k] = 1
        for k in mask_seen_by_Di:
            A[i, B + k] = 1
        for k in data_seen_by_Dti:
            A[B + i, k] = 1
        for k in mask_seen_by_Dti:
            A[B + i, B + k] = 1
    return A


@pytest.mark.parametrize("gamma", [1, 2, 3, 4, 5])
def test_every_permutation_matches_prose(gamma):
    perms = np.array(list(itertools.permutations(range(1, gamma + 1))), np.int32)
    r = orc.build_mask(perms, np.zeros(len(perms), np.int32), gamma)
    assert r["err"] == 0
    for b, mu in enumerate(perms):
        np.testing.assert_array_equal(r["dense"][b], _prose_mask(list(mu)), err_msg=str(mu))


@pytest.mark.parametrize("gamma", [6, 8, 16, 32])
def test_random_permutations_match_prose(gamma):
    rng = np.random.default_rng(gamma)
    perms = np.stack([rng.permutation(gamma) + 1 for _ in range(40)]).astype(np.int32)
    r = orc.build_mask(perms, np.zeros(len(perms), np.int32), gamma)
    for b, mu in enumerate(perms):
        np.testing.assert_array_equal(r["dense"][b], _prose_mask(list(mu)))


@pytest.mark.parametrize("gamma", [1, 3, 4, 7, 16])
def test_structure_invariants(gamma):
    # Every row sees exactly gamma of the 2*gamma new slots: for each block
    # position exactly one of (D_k, D~_k); each row sees itself and never the
    # other member of its own pair.
    rng = np.random.default_rng(100 + gamma)
    perms = np.stack([rng.permutation(gamma) + 1 for _ in range(25)]).astype(np.int32)
    r = orc.build_mask(perms, np.zeros(len(perms), np.int32), gamma)
    for A in r["dense"].astype(int):
        assert (A.sum(1) == gamma).all()
        assert ((A[:, :gamma] + A[:, gamma:]) == 1).all()
        for i in range(2 * gamma):
            assert A[i, i] == 1
            pair = i + gamma if i < gamma else i - gamma
            assert A[i, pair] == 0


def test_verification_row_equals_previous_data_row():
    # The verification slot of step r sees exactly the context of the data
    # token of step r-1 (both: steps < r as data, steps >= r as masks); the
    # first verification slot sees only masks and the last data token only
    # data (the fully decoded block).
    gamma = 6
    rng = np.random.default_rng(5)
    for _ in range(20):
        mu = rng.permutation(gamma) + 1
        A = orc.build_mask(mu[None].astype(np.int32), [0], gamma)["dense"][0]
        slot_of = {int(t): k for k, t in enumerate(mu)}
        for r in range(2, gamma + 1):
            np.testing.assert_array_equal(A[gamma + slot_of[r]], A[slot_of[r - 1]])
        np.testing.assert_array_equal(A[gamma + slot_of[1]], np.r_[np.zeros(gamma), np.ones(gamma)])
        np.testing.assert_array_equal(A[slot_of[gamma]], np.r_[np.ones(gamma), np.zeros(gamma)])


def test_permutation_equivariance():
    # Eq. (1) depends only on (section, tau): slot (s, k) under mu behaves as
    # slot (s, mu_k - 1) under the identity map.
    gamma = 7
    rng = np.random.default_rng(9)
    ident = orc.build_mask(None, [0], gamma)["dense"][0]
    for _ in range(30):
        mu = (rng.permutation(gamma) + 1).astype(np.int32)
        A = orc.build_mask(mu[None], [0], gamma)["dense"][0]
        idx = np.r_[mu - 1, gamma + mu - 1]
        np.testing.assert_array_equal(A, ident[np.ix_(idx, idx)])


def test_padding_zeroes_rows_and_columns():
    # Sec. 3.1: padding positions have their rows and columns zeroed; the
    # remaining positions see each other as if the padded ones were absent
    # (Eq. (1) only compares labels).
    gamma = 8
    rng = np.random.default_rng(3)
    for _ in range(30):
        mu = (rng.permutation(gamma) + 1).astype(np.int32)
        pad = rng.random(gamma) < 0.35
        mu_p = np.where(pad, 0, mu).astype(np.int32)
        r = orc.build_mask(mu_p[None], [0], gamma)
        assert r["err"] == 0
        A = r["dense"][0]
        padslots = np.r_[pad, pad]
        assert (A[padslots] == 0).all() and (A[:, padslots] == 0).all()
        assert (r["section"][0][padslots] == orc.SECT_PAD).all()
        keep = ~pad
        if keep.sum() == 0:
            continue
        # relabel the kept positions 1..m in the same order
        kept_mu = mu[keep]
        ranks = np.argsort(np.argsort(kept_mu)) + 1
        m = int(keep.sum())
        B = orc.build_mask(ranks[None].astype(np.int32), [0], m)["dense"][0]
        idx = np.r_[np.nonzero(keep)[0], gamma + np.nonzero(keep)[0]]
        np.testing.assert_array_equal(A[np.ix_(idx, idx)], B)


def test_rope_copy_and_labels():
    # Sec. 3.1 "Position Encoding Alignment": D~_k reuses the RoPE index of
    # D_k, which keeps its absolute index (prefix length + k).
    gamma = 5
    n = np.array([0, 1, 63, 64, 1000], np.int32)
    rng = np.random.default_rng(1)
    mu = np.stack([rng.permutation(gamma) + 1 for _ in range(len(n))]).astype(np.int32)
    r = orc.build_mask(mu, n, gamma)
    for b in range(len(n)):
        want = n[b] + np.arange(gamma)
        np.testing.assert_array_equal(r["rope_pos"][b, :gamma], want)
        np.testing.assert_array_equal(r["rope_pos"][b, gamma:], want)
        np.testing.assert_array_equal(r["tau"][b, :gamma], mu[b])
        np.testing.assert_array_equal(r["tau"][b, gamma:], mu[b])
        assert (r["section"][b, :gamma] == orc.SECT_D).all()
        assert (r["section"][b, gamma:] == orc.SECT_DT).all()


def test_mask_bits_match_dense():
    gamma = 32
    rng = np.random.default_rng(2)
    mu = np.stack([rng.permutation(gamma) + 1 for _ in range(4)]).astype(np.int32)
    r = orc.build_mask(mu, np.zeros(4, np.int32), gamma)
    for b in range(4):
        for i in range(2 * gamma):
            bits = int(r["mask_bits"][b, i])
            got = np.array([(bits >> j) & 1 for j in range(2 * gamma)], np.uint8)
            np.testing.assert_array_equal(got, r["dense"][b, i])


@pytest.mark.parametrize("bad", [[1, 1, 2, 3], [1, 2, 5, 3], [1, -3, 2, 3], [4, 2, 2, 0], [-1, 1, 1, -2]])
def test_invalid_step_map_is_flagged_and_padded(bad):
    r = orc.build_mask(np.array([bad], np.int32), [3], 4)
    assert r["err"] & orc.ERR_STEP_MAP
    assert (r["section"][0] == orc.SECT_PAD).all()
    assert (r["dense"][0] == 0).all()


# ---- blocks with fewer drafts than positions, and the target completing
# the block itself (Sec. 3.2, last sentences of "Target Model Verification")

INF = 10 ** 9


def _prose_mask_block(codes):
    """Visible sets by the step at which each position becomes known.

    A position decoded earlier in the block is known before every step
    (step 0), a drafted position at its draft step, an undrafted one never
    within this step.  Its data slot exists iff it holds a token (decoded or
    drafted), its mask slot iff a prediction is made there (drafted or
    undrafted).  A data token sees the data tokens known no later than it and
    the placeholders of positions still unknown at that time; a prediction
    slot sees the data tokens known strictly earlier and the placeholders of
    positions unresolved at its step (Sec. 3.1).
    """
    B = len(codes)
    known = [0 if c == orc.STEP_DECODED else (INF if c == orc.STEP_UNDRAFTED else c) for c in codes]
    has_d = [c > 0 or c == orc.STEP_DECODED for c in codes]
    has_m = [c > 0 or c == orc.STEP_UNDRAFTED for c in codes]
    A = np.zeros((2 * B, 2 * B), np.uint8)
    for i in range(B):
        for k in range(B):
            if has_d[i] and has_d[k] and known[k] <= known[i]:
                A[i, k] = 1
            if has_d[i] and has_m[k] and known[k] > known[i]:
                A[i, B + k] = 1
            if has_m[i] and has_d[k] and known[k] < known[i]:
                A[B + i, k] = 1
            if has_m[i] and has_m[k] and known[k] >= known[i]:
                A[B + i, B + k] = 1
    return A


def _random_block(rng, B, n_draft, n_decoded):
    codes = np.full(B, orc.STEP_UNDRAFTED, np.int32)
    pos = rng.permutation(B)
    codes[pos[:n_draft]] = rng.permutation(n_draft) + 1
    codes[pos[n_draft:n_draft + n_decoded]] = orc.STEP_DECODED
    return codes


@pytest.mark.parametrize("B", [1, 2, 4, 5, 8, 16, 32])
def test_undrafted_and_decoded_positions_match_prose(B):
    rng = np.random.default_rng(300 + B)
    maps = []
    for _ in range(30):
        n_draft = int(rng.integers(0, B + 1))
        n_dec = int(rng.integers(0, B - n_draft + 1))
        codes = _random_block(rng, B, n_draft, n_dec)
        codes[rng.random(B) < 0.1] = 0       # some padding as well
        maps.append(codes)
    maps = np.stack(maps)
    r = orc.build_mask(maps, np.zeros(len(maps), np.int32), B)
    assert r["err"] == 0
    for b, codes in enumerate(maps):
        np.testing.assert_array_equal(r["dense"][b], _prose_mask_block(list(codes)), err_msg=str(codes))


@pytest.mark.parametrize("B", [1, 3, 4, 8, 32])
def test_target_completing_the_block_is_bidirectional(B):
    # With no drafts (decoded tokens and [MASK] placeholders only) the step
    # is the dLLM's own block decoding: every real slot sees every other.
    rng = np.random.default_rng(400 + B)
    for _ in range(10):
        codes = _random_block(rng, B, 0, int(rng.integers(0, B + 1)))
        r = orc.build_mask(codes[None], [5], B)
        assert r["err"] == 0
        real = np.concatenate([codes == orc.STEP_DECODED, codes == orc.STEP_UNDRAFTED])
        A = r["dense"][0].astype(bool)
        assert real.sum() == B
        assert A[np.ix_(real, real)].all()
        assert not A[~real].any() and not A[:, ~real].any()


def test_drafted_part_is_the_mask_of_the_drafts_alone():
    # Removing the undrafted and decoded positions leaves the plain mask of
    # the drafted permutation: the extra kinds change nothing among drafts.
    rng = np.random.default_rng(9)
    for _ in range(20):
        B = int(rng.integers(2, 17))
        codes = _random_block(rng, B, int(rng.integers(1, B + 1)), 0)
        codes[codes == orc.STEP_UNDRAFTED] = np.where(rng.random((codes == orc.STEP_UNDRAFTED).sum()) < 0.5,
                                                      orc.STEP_UNDRAFTED, orc.STEP_DECODED)
        d = np.nonzero(codes > 0)[0]
        full = orc.build_mask(codes[None], [0], B)["dense"][0]
        alone = orc.build_mask(codes[d][None], [0], len(d))["dense"][0]
        idx = np.concatenate([d, B + d])
        np.testing.assert_array_equal(full[np.ix_(idx, idx)], alone)
