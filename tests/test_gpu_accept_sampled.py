"""GPU parity of simsd_accept_sampled (Sec. 3.2, Eq. (2)) against the oracle.

The accepted length and the tokens are integers, but each is decided by a
floating-point comparison: u_accept against alpha, and u_sample * total
against a cumulative sum.  The kernel forms the probabilities in fp32, the
oracle in fp64.  Where the oracle's own numbers put the decision farther than
the fp32 error from its boundary the results must be identical; inside that
band the GPU's choice must be one of the valid ones (its alpha on the right
side of u within the band, its token's cumulative interval within the band of
the threshold).  The speculative-sampling theorem gives a size-independent
property: the first emitted token is distributed as p_theta.
"""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd

pytestmark = pytest.mark.gpu

ALPHA_BAND = 2e-5   # |u_accept - alpha|: fp32 softmax ratio error is about 1e-6
DRAW_BAND = 2e-5    # distance of the threshold to a cumulative boundary, relative to the total


def _gpu(si):
    Bt, rows, _ = si.target_logits.shape
    a = torch.full((Bt,), -9, dtype=torch.int32, device="cuda")
    ot = torch.full((Bt, rows), -9, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_accept_sampled(si.target_logits, si.draft_logits, si.draft, si.u_accept, si.u_sample, a, ot,
                               temperature=si.temperature, err_word=err)
    torch.cuda.synchronize()
    return a.cpu().numpy(), ot.cpu().numpy(), simsd.simsd_check_error(err)


def _softmax64(x, t):
    z = np.asarray(x, np.float64) / t
    z = np.exp(z - z.max())
    return z / z.sum()


def _draw_is_valid(tl, dl, a, gamma, u, tok, t):
    """The GPU's token has positive weight and its cumulative interval lies
    within DRAW_BAND of the threshold (fp64 weights of the oracle's rule)."""
    pt = _softmax64(tl[a], t)
    w = pt
    if a < gamma:
        r = np.maximum(0.0, pt - _softmax64(dl[a], t))
        if r.sum() > 0.0:
            w = r
    if not (0 <= tok < w.size) or w[tok] <= 0.0:
        return False
    c = np.cumsum(w)
    tot = c[-1]
    thr = float(u) * tot
    lo = c[tok] - w[tok]
    return lo <= thr + DRAW_BAND * tot and c[tok] >= thr - DRAW_BAND * tot


def _compare(si, expect_err=0):
    """Every sequence whose decisions all lie outside the fp32 band (by the
    oracle's own fp64 numbers) must match the oracle exactly; a sequence
    with a decision inside the band must make a valid choice.  Band hits are
    counted: at V = 151936 most draws are band hits, since one token's
    probability (~7e-6 of the total) is below the band."""
    tl = si.target_logits.cpu().numpy()
    dl = si.draft_logits.cpu().numpy()
    dr = si.draft.cpu().numpy()
    ua = si.u_accept.cpu().numpy()
    us = si.u_sample.cpu().numpy()
    Bt, rows, V = tl.shape
    gamma = rows - 1
    ga, got, gerr = _gpu(si)
    ra, rot, ral, rmg, rerr = orc.accept_sampled(tl, dl, dr, ua, us, gamma, temperature=si.temperature)
    assert gerr == rerr == expect_err
    band_hits = 0
    for b in range(Bt):
        a = int(ga[b])
        assert 0 <= a <= gamma
        # the acceptance decisions that matter: rows up to the first rejection
        last = min(max(a, int(ra[b])), gamma - 1)
        near_alpha = any(abs(float(ua[b, r]) - ral[b, r]) < ALPHA_BAND for r in range(last + 1))
        near_draw = rmg[b] < DRAW_BAND
        if not (near_alpha or near_draw):
            assert a == ra[b], (b, a, ra[b])
            np.testing.assert_array_equal(got[b], rot[b])
            continue
        band_hits += 1
        if a != ra[b]:
            r = min(a, int(ra[b]))
            assert abs(float(ua[b, r]) - ral[b, r]) < ALPHA_BAND, (b, a, ra[b], ua[b, r], ral[b, r])
        np.testing.assert_array_equal(got[b, :a], dr[b, :a])
        assert (got[b, a + 1:] == -1).all()
        if a == ra[b] and got[b, a] != rot[b, a]:
            assert near_draw, (b, a, got[b, a], rot[b, a], rmg[b])
        assert _draw_is_valid(tl[b], dl[b], a, gamma, us[b], int(got[b, a]), si.temperature), (b, a, got[b, a])
    exact = int(sum(int(ga[b]) == int(ra[b]) and np.array_equal(got[b], rot[b]) for b in range(Bt)))
    print(f"accept_sampled Bt={Bt} gamma={gamma} V={V}: {band_hits} sequence(s) with a decision in the fp32 band, "
          f"{exact} of {Bt} equal to the oracle")
    # measured on the GB300: every sequence of every case equal to the oracle
    # (band hits included, 0-79% of the sequences at V 151936); a valid
    # in-band choice may still differ on at most 2% of them
    assert exact >= Bt - max(1, Bt // 50), (exact, Bt, band_hits)
    return ga, got


@pytest.mark.parametrize("Bt,gamma,V,T,eta", [
    (1, 4, 1024, 1.0, 0.5), (8, 4, 151936, 1.0, 0.5), (32, 8, 151936, 1.0, 0.3), (3, 1, 151936, 0.7, 1.0),
    (5, 32, 50000, 1.0, 0.2), (300, 4, 4096, 1.3, 0.5), (16, 16, 151936, 1.0, 0.4), (2, 5, 3, 1.0, 2.0),
])
def test_accept_sampled_matches_oracle(Bt, gamma, V, T, eta):
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=Bt * 1000 + gamma * 10 + V % 7, eta=eta, temperature=T,
                                    device="cuda")
    _compare(si)


@pytest.mark.parametrize("Bt,V", [(6, 1001), (6, 30001), (400, 1001)])
def test_accept_sampled_scalar_paths(Bt, V):
    # a vocabulary that is not a multiple of 4, and base pointers off 16 bytes;
    # small and large batches take the one- and two-CTA-per-SM variants
    si = inputs.make_sampled_inputs(Bt, 4, V, seed=V, device="cuda")
    _compare(si)
    for name in ("target_logits", "draft_logits"):
        t = getattr(si, name)
        flat = torch.empty(t.numel() + 1, device="cuda")
        flat[1:] = t.reshape(-1)
        setattr(si, name, flat[1:].view(t.shape))
    _compare(si)


def test_accept_sampled_equal_models_accept_everything():
    si = inputs.make_sampled_inputs(24, 8, 151936, seed=11, device="cuda")
    si.draft_logits = si.target_logits[:, :8].contiguous()
    si.u_accept = si.u_accept * 0.999
    a, _ = _compare(si)
    assert (a == 8).all()


def test_accept_sampled_bad_draft_with_empty_residual():
    # equal models: a draft id outside the vocabulary is the only way to
    # reject, and the residual is empty, so the token comes from p_theta
    Bt, gamma, V = 6, 4, 20000
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=12, device="cuda")
    si.draft_logits = si.target_logits[:, :gamma].contiguous()
    si.u_accept = si.u_accept * 0.999
    si.draft[0, 0] = V
    si.draft[1, 2] = -1
    si.draft[2, 3] = 2 ** 30
    a, _ = _compare(si, expect_err=simsd.EW_DRAFT)
    assert list(a[:3]) == [0, 2, 3] and (a[3:] == gamma).all()


def test_accept_sampled_edge_logits():
    Bt, gamma, V = 6, 3, 4096
    si = inputs.make_sampled_inputs(Bt, gamma, V, seed=13, device="cuda")
    # masked vocabulary (-inf logits, as top-k / top-p filtering leaves them)
    si.target_logits[0, :, 1000:] = -float("inf")
    si.draft_logits[0, :, 2000:] = -float("inf")
    si.draft[0] = torch.randint(0, 1000, (gamma,), dtype=torch.int32)
    # one dominant token in every target row
    si.target_logits[1, :, 7] = 80.0
    # u at the ends of [0, 1)
    si.u_accept[2] = 0.0
    si.u_sample[2] = 0.0
    si.u_sample[3] = float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    si.u_accept[3] = 0.9999999
    _compare(si)


def test_accept_sampled_empty_batch():
    si = inputs.make_sampled_inputs(1, 4, 64, seed=14, device="cuda")
    a = torch.full((1,), -9, dtype=torch.int32, device="cuda")
    ot = torch.full((1, 5), -9, dtype=torch.int32, device="cuda")
    simsd.simsd_accept_sampled(si.target_logits[:0], si.draft_logits[:0], si.draft[:0], si.u_accept[:0],
                               si.u_sample[:0], a[:0], ot[:0])
    torch.cuda.synchronize()
    assert int(a[0]) == -9 and (ot == -9).all()


def test_first_token_is_distributed_as_the_target():
    """Speculative-sampling theorem: with x ~ p_phi and independent uniform
    draws, P(first emitted token = v) = p_theta(v), at any temperature."""
    N, V, T = 400000, 12, 0.8
    g = torch.Generator().manual_seed(15)
    tl = torch.randn(1, 2, V, generator=g) * 1.5
    dl = torch.randn(1, 1, V, generator=g) * 1.5
    pd = torch.softmax(dl[0, 0].double() / T, 0)
    pt = torch.softmax(tl[0, 0].double() / T, 0).numpy()
    draft = torch.multinomial(pd, N, replacement=True, generator=g).to(torch.int32).view(N, 1)
    si = inputs.SampledInputs(tl.expand(N, 2, V).contiguous().cuda(), dl.expand(N, 1, V).contiguous().cuda(),
                              draft.cuda(), torch.rand(N, 1, generator=g).cuda(), torch.rand(N, generator=g).cuda(), T)
    _, ot, err = _gpu(si)
    assert err == 0
    freq = np.bincount(ot[:, 0], minlength=V) / N
    sigma = np.sqrt(pt * (1 - pt) / N)
    assert (np.abs(freq - pt) < 5 * sigma + 1e-6).all(), (freq, pt)
