"""Pins of the oracle's rotary position embedding and of the RoPE-copy rule.

Sec. 3.1 "Position Encoding Alignment": D~_k reuses the RoPE index of D_k,
so both sit at n + k; the Table 4 ablation ("without aligned RoPE") puts the
mask slots at their physical positions n + gamma + k instead.  The rotation
itself is RoFormer's (Su et al.) in the rotate-half layout: x_i + j x_{i+d/2}
is multiplied by exp(j * pos * theta^(-2i/d)).  Every expectation below is
computed independently of the oracle: numpy complex arithmetic, the textbook
2x2 rotation matrix, algebraic identities, or step-by-step decoding.
"""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


def np_rope(x, pos, theta):
    """RoPE by complex multiplication (independent of the oracle)."""
    x = np.asarray(x, np.float64)
    d = x.shape[-1]
    half = d // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = theta ** (-2.0 * np.arange(half) / d)
    z = z * np.exp(1j * pos * freq)
    return np.concatenate([z.real, z.imag], axis=-1)


@pytest.mark.parametrize("d", [2, 8, 64, 128])
@pytest.mark.parametrize("pos", [0, 1, 7, 1000, 32767])
@pytest.mark.parametrize("theta", [1e4, 1e6])
def test_rotation_matches_complex_multiplication(d, pos, theta):
    x = np.random.default_rng(d + pos).normal(size=(3, d))
    # the angle pos * theta^(-2i/d) carries about pos * 1e-16 of rounding
    np.testing.assert_allclose(orc.rope_rotate(x, pos, theta), np_rope(x, pos, theta), rtol=0,
                               atol=1e-12 + 4e-16 * pos)


def test_d2_is_the_textbook_rotation_matrix():
    x = np.array([0.3, -1.7])
    for pos in (0.0, 0.5, 2.0, 100.0):
        R = np.array([[np.cos(pos), -np.sin(pos)], [np.sin(pos), np.cos(pos)]])
        np.testing.assert_allclose(orc.rope_rotate(x, pos, 1e4), R @ x, rtol=0, atol=1e-14)


def test_identity_norm_composition_and_relative_position():
    r = np.random.default_rng(3)
    q, k = r.normal(size=128), r.normal(size=128)
    theta = 1e6
    np.testing.assert_array_equal(orc.rope_rotate(q, 0, theta), q)
    for pos in (5, 4096):
        rq = orc.rope_rotate(q, pos, theta)
        # each (i, i + d/2) pair keeps its length
        np.testing.assert_allclose(rq[:64] ** 2 + rq[64:] ** 2, q[:64] ** 2 + q[64:] ** 2, rtol=1e-12)
    np.testing.assert_allclose(orc.rope_rotate(orc.rope_rotate(q, 300, theta), 45, theta),
                               orc.rope_rotate(q, 345, theta), rtol=1e-10, atol=1e-12)
    # the score depends only on the position difference
    for m, n, c in ((10, 3, 1000), (0, 77, 5), (4096, 4100, 123)):
        a = orc.rope_rotate(q, m, theta) @ orc.rope_rotate(k, n, theta)
        b = orc.rope_rotate(q, m + c, theta) @ orc.rope_rotate(k, n + c, theta)
        assert abs(a - b) < 1e-10 * max(1.0, abs(a))


def _inputs(seed, Bt=2, gamma=4, Hq=4, Hkv=2, d=16, P=8):
    r = np.random.default_rng(seed)
    S = 2 * gamma
    n = r.integers(0, 30, Bt).astype(np.int32)
    max_pages = 6
    num_pages = Bt * max_pages
    bt = r.permutation(num_pages).astype(np.int32).reshape(Bt, max_pages)
    q = r.normal(size=(Bt, S, Hq, d)).astype(np.float32)
    kn = r.normal(size=(Bt, S, Hkv, d)).astype(np.float32)
    vn = r.normal(size=(Bt, S, Hkv, d)).astype(np.float32)
    kc = r.normal(size=(num_pages, Hkv, P, d)).astype(np.float32)
    vc = r.normal(size=(num_pages, Hkv, P, d)).astype(np.float32)
    mu = np.stack([r.permutation(gamma) + 1 for _ in range(Bt)]).astype(np.int32)
    return q, kn, vn, kc, vc, bt, n, mu, gamma


@pytest.mark.parametrize("mode", [1, 2])
def test_attention_rotates_q_and_new_keys_at_the_rope_copy_positions(mode):
    q, kn, vn, kc, vc, bt, n, mu, gamma = _inputs(5 + mode)
    theta = 1e4
    S = 2 * gamma
    qr, kr = np.empty_like(q, dtype=np.float64), np.empty_like(kn, dtype=np.float64)
    for b in range(q.shape[0]):
        for t in range(S):
            # Sec. 3.1: D_k and D~_k both at n + k; Table 4 ablation: slot t at n + t
            pos = n[b] + (t % gamma if mode == 1 else t)
            qr[b, t] = np_rope(q[b, t], pos, theta)
            kr[b, t] = np_rope(kn[b, t], pos, theta)
    # fp64 pre-rotated inputs are not representable in float32, so compare the
    # oracle's own rotation against attention over float32-rounded rotations
    # at a tolerance set by that rounding
    want, e1 = orc.verify_attention(qr.astype(np.float32), kr.astype(np.float32), vn, kc, vc, bt, n, mu, gamma)
    got, e2 = orc.verify_attention(q, kn, vn, kc, vc, bt, n, mu, gamma, rope_theta=theta, rope_mode=mode)
    assert e1 == 0 and e2 == 0
    np.testing.assert_allclose(got, want, rtol=1e-5, atol=1e-5)


def test_aligned_and_physical_positions_differ():
    q, kn, vn, kc, vc, bt, n, mu, gamma = _inputs(9)
    a, _ = orc.verify_attention(q, kn, vn, kc, vc, bt, n, mu, gamma, rope_theta=1e4, rope_mode=1)
    p, _ = orc.verify_attention(q, kn, vn, kc, vc, bt, n, mu, gamma, rope_theta=1e4, rope_mode=2)
    # data rows see the same data positions in both modes only where no mask
    # slot is visible; mask rows always differ
    assert np.abs(a[:, gamma:] - p[:, gamma:]).max() > 1e-3


def test_commit_stores_rotated_keys_and_plain_values():
    q, kn, vn, kc, vc, bt, n, mu, gamma = _inputs(11)
    L = 1
    kn5, vn5 = kn[None], vn[None]
    kc5, vc5 = kc[None], vc[None]
    acc = np.array([gamma, 2], np.int32)
    theta = 1e6
    k2, v2, n2, err = orc.kv_commit(kn5, vn5, mu, acc, kc5, vc5, bt, n, gamma, rope_theta=theta)
    assert err == 0
    np.testing.assert_array_equal(n2, n + acc)
    P = kc.shape[2]
    for b in range(2):
        for r in range(acc[b]):
            k = int(np.where(mu[b] == r + 1)[0][0])       # data slot of the r-th draft
            row = n[b] + r
            pg, off = bt[b, row // P], row % P
            np.testing.assert_allclose(k2[0, pg, :, off], np_rope(kn[b, k], n[b] + k, theta).astype(np.float32),
                                       rtol=1e-6, atol=1e-6)
            np.testing.assert_array_equal(v2[0, pg, :, off], vn[b, k])


def _bf16_bits_nearest_even(v):
    """Rounds a float64 to bfloat16 (8 significant bits), ties to even, with
    Python's own frexp and banker's round; returns the 16-bit pattern."""
    import math
    if v == 0.0:
        return np.uint16(np.float32(v).view(np.uint32) >> 16)
    m, e = math.frexp(float(v))
    r = math.ldexp(round(m * 256.0), e - 8)
    return np.uint16(np.float32(r).view(np.uint32) >> 16)


def test_commit_rounds_rotated_bf16_keys_to_nearest_even():
    q, kn, vn, kc, vc, bt, n, mu, gamma = _inputs(13)
    bits = lambda a: (a.view(np.uint32) >> 16).astype(np.uint16)
    widen = lambda b: (b.astype(np.uint32) << 16).view(np.float32)
    kb, vb = bits(kn), bits(vn)
    acc = np.array([gamma, gamma], np.int32)
    theta = 1e4
    k2, v2, _, err = orc.kv_commit(kb[None], vb[None], mu, acc, bits(kc)[None], bits(vc)[None], bt, n, gamma,
                                   rope_theta=theta)
    assert err == 0
    P = kc.shape[2]
    for b in range(2):
        for r in range(gamma):
            k = int(np.where(mu[b] == r + 1)[0][0])
            row = n[b] + r
            pg, off = bt[b, row // P], row % P
            rot = np_rope(widen(kb[b, k]).astype(np.float64), n[b] + k, theta)
            want = np.vectorize(_bf16_bits_nearest_even, otypes=[np.uint16])(rot)
            np.testing.assert_array_equal(k2[0, pg, :, off], want)
            np.testing.assert_array_equal(v2[0, pg, :, off], vb[b, k])


# ------------------------------------------------------------------ decode
def _bidir(q, K, V):
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


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_aligned_rope_reproduces_step_by_step_decode(seed):
    """One layer with rotary positions and no additive ones.  Step r of
    sequential decoding rotates the block's queries and keys at their
    positions n + k; the verification forward with the aligned RoPE copy
    gives the same outputs, physical positions do not."""
    r = np.random.default_rng(200 + seed)
    Vt, dm, Hq, Hkv, d, gamma, theta = 40, 16, 2, 1, 16, 4, 1e4
    E, emask = r.normal(size=(Vt, dm)), r.normal(size=dm)
    Wq, Wk, Wv = (r.normal(size=(H, dm, d)) / 4 for H in (Hq, Hkv, Hkv))
    Wo = r.normal(size=(Hq * d, Vt))
    proj = lambda h, W: np.einsum("md,hde->mhe", h, W).astype(np.float32)
    n = int(r.integers(1, 30))
    mu = (r.permutation(gamma) + 1).astype(np.int32)
    slot_of = {int(t): k for k, t in enumerate(mu)}
    hp = E[r.integers(0, Vt, n)]
    Kp = np.stack([np_rope(proj(hp, Wk)[j], j, theta) for j in range(n)])     # cache holds rotated keys
    Vp = proj(hp, Wv).astype(np.float64)

    x = [None] * gamma
    mask_out, data_out = {}, {}

    def block(state):
        hb = np.stack([E[state[k]] if state[k] is not None else emask for k in range(gamma)])
        qb = np.stack([np_rope(proj(hb, Wq)[k], n + k, theta) for k in range(gamma)])
        kb = np.stack([np_rope(proj(hb, Wk)[k], n + k, theta) for k in range(gamma)])
        return qb, kb, proj(hb, Wv)

    for step in range(1, gamma + 1):
        ks = slot_of[step]
        qb, kb, vb = block(x)
        mask_out[step] = _bidir(qb[ks], np.concatenate([Kp, kb]), np.concatenate([Vp, vb]))
        x[ks] = int(np.argmax(mask_out[step].reshape(-1) @ Wo))
        qb2, kb2, vb2 = block(x)
        data_out[step] = _bidir(qb2[ks], np.concatenate([Kp, kb2]), np.concatenate([Vp, vb2]))

    hv = np.concatenate([np.stack([E[x[k]] for k in range(gamma)]), np.stack([emask] * gamma)])
    q, k, v = proj(hv, Wq), proj(hv, Wk), proj(hv, Wv)
    P = 8
    npages = (n + P - 1) // P
    kc = np.zeros((npages, Hkv, P, d), np.float32)
    vc = np.zeros((npages, Hkv, P, d), np.float32)
    for j in range(n):
        kc[j // P, :, j % P] = Kp[j]
        vc[j // P, :, j % P] = Vp[j]
    bt = np.arange(npages, dtype=np.int32)[None]
    # the rotated cache keys were rounded to float32; the decode used fp64 ones
    out, err = orc.verify_attention(q[None], k[None], v[None], kc, vc, bt, [n], mu[None], gamma, rope_theta=theta,
                                    rope_mode=1)
    assert err == 0
    for step in range(1, gamma + 1):
        ks = slot_of[step]
        np.testing.assert_allclose(out[0, gamma + ks], mask_out[step], rtol=1e-5, atol=1e-6)
        np.testing.assert_allclose(out[0, ks], data_out[step], rtol=1e-5, atol=1e-6)
    phys, _ = orc.verify_attention(q[None], k[None], v[None], kc, vc, bt, [n], mu[None], gamma, rope_theta=theta,
                                   rope_mode=2)
    worst = max(np.abs(phys[0, gamma + slot_of[s]] - mask_out[s]).max() for s in range(1, gamma + 1))
    assert worst > 1e-3
