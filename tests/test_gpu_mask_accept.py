"""GPU parity of simsd_build_mask and simsd_accept against the oracle
(bit-exact; both are integer results)."""
import numpy as np
import pytest
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd
from tests._gpu import gpu_mask

pytestmark = pytest.mark.gpu


def _meta(Bt, gamma, seed, pad_frac=0.0, invalid=0):
    rng = np.random.default_rng(seed)
    mu = np.stack([rng.permutation(gamma) + 1 for _ in range(Bt)]).astype(np.int32)
    if pad_frac:
        mu[rng.random(mu.shape) < pad_frac] = 0
    for b in range(invalid):
        mu[b, 0] = mu[b, -1] if gamma > 1 else gamma + 1
    n = rng.integers(0, 5000, Bt).astype(np.int32)
    return mu, n


@pytest.mark.parametrize("gamma", [1, 2, 3, 4, 8, 16, 31, 32])
@pytest.mark.parametrize("identity", [False, True])
def test_build_mask_bit_exact(gamma, identity):
    Bt = 37
    mu, n = _meta(Bt, gamma, gamma, pad_frac=0.0 if identity else 0.15, invalid=0 if identity else 2)
    w = inputs.Workload("m", "bf16", Bt, 2, 1, 128, gamma, (0, 0), 1, 8, 0.5, 1.0, 1.0, 0)
    dev = torch.device("cuda")
    sm = None if identity else torch.as_tensor(mu, device=dev)
    si = inputs.StepInputs(w, torch.as_tensor(n, device=dev), None, 0, sm, *([None] * 7), None)
    tau, sect, rope, bits, err = gpu_mask(si)
    word = simsd.simsd_check_error(err)
    r = orc.build_mask(None if identity else mu, n, gamma)
    np.testing.assert_array_equal(tau.cpu().numpy(), r["tau"])
    np.testing.assert_array_equal(sect.cpu().numpy(), r["section"])
    np.testing.assert_array_equal(rope.cpu().numpy(), r["rope_pos"])
    np.testing.assert_array_equal(bits.cpu().numpy().view(np.uint64), r["mask_bits"])
    assert word == r["err"]


@pytest.mark.parametrize("gamma", [1, 2, 3, 4, 8, 16, 32])
@pytest.mark.parametrize("n_draft", [None, 0])
def test_build_mask_undrafted_and_decoded_bit_exact(gamma, n_draft):
    # blocks with fewer drafts than positions (n_draft None: random counts)
    # and the target's own block decoding (n_draft 0)
    Bt = 41
    mu = inputs.block_step_maps(Bt, gamma, seed=7 * gamma, n_draft=n_draft, pad_frac=0.1).numpy()
    mu[0] = [simsd.STEP_DECODED - 1] + [1] * (gamma - 1) if gamma > 1 else [-3]   # invalid: flagged, all padding
    n = np.random.default_rng(gamma).integers(0, 5000, Bt).astype(np.int32)
    w = inputs.Workload("m", "bf16", Bt, 2, 1, 128, gamma, (0, 0), 1, 8, 0.5, 1.0, 1.0, 0)
    dev = torch.device("cuda")
    si = inputs.StepInputs(w, torch.as_tensor(n, device=dev), None, 0, torch.as_tensor(mu, device=dev),
                           *([None] * 7), None)
    tau, sect, rope, bits, err = gpu_mask(si)
    word = simsd.simsd_check_error(err)
    r = orc.build_mask(mu, n, gamma)
    np.testing.assert_array_equal(tau.cpu().numpy(), r["tau"])
    np.testing.assert_array_equal(sect.cpu().numpy(), r["section"])
    np.testing.assert_array_equal(rope.cpu().numpy(), r["rope_pos"])
    np.testing.assert_array_equal(bits.cpu().numpy().view(np.uint64), r["mask_bits"])
    assert word == r["err"] == simsd.EW_STEP_MAP


def _accept_case(Bt, gamma, V, seed, p=0.6, std=2.0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    logits = torch.randn(Bt, gamma + 1, V, generator=g, device="cuda") * std
    am = torch.argmax(logits[:, :gamma], -1)
    cg = torch.Generator().manual_seed(seed)
    agree = (torch.rand(Bt, gamma, generator=cg) < p).cuda()
    rnd = torch.randint(0, V, (Bt, gamma), generator=cg).cuda()
    draft = torch.where(agree, am, rnd).to(torch.int32)
    return logits, draft


def _run_accept(logits, draft):
    Bt, rows, V = logits.shape
    gamma = rows - 1
    a = torch.full((Bt,), -9, dtype=torch.int32, device="cuda")
    ot = torch.full((Bt, rows), -9, dtype=torch.int32, device="cuda")
    am = torch.full((Bt, rows), -9, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    simsd.simsd_accept(logits, draft, a, ot, am, err)
    word = simsd.simsd_check_error(err)
    ra, rot, ram, rerr = orc.accept(logits.cpu().numpy(), draft.cpu().numpy(), gamma)
    np.testing.assert_array_equal(am.cpu().numpy(), ram)
    np.testing.assert_array_equal(a.cpu().numpy(), ra)
    np.testing.assert_array_equal(ot.cpu().numpy(), rot)
    assert word == rerr
    return ra


@pytest.mark.parametrize("Bt,gamma,V", [(1, 4, 1024), (8, 4, 151936), (32, 8, 151936), (64, 16, 151936),
                                        (3, 1, 151936), (5, 32, 50000), (200, 4, 4096), (7, 3, 1001),
                                        (2, 5, 3), (1, 32, 151936), (2, 4, 64), (19, 8, 151936), (4, 16, 65540),
                                        (700, 2, 512)])
def test_accept_bit_exact(Bt, gamma, V):
    # one cluster per sequence, from 16 CTAs (one sequence of 33 rows) down
    # to single CTAs in several waves (700 sequences); a 64-token vocabulary
    # leaves CTAs with a few units or none; odd vocabularies stream scalars
    logits, draft = _accept_case(Bt, gamma, V, seed=Bt * 100 + gamma)
    _run_accept(logits, draft)


def test_accept_edge_values():
    Bt, gamma, V = 8, 4, 20000
    logits, draft = _accept_case(Bt, gamma, V, seed=5, p=1.0)
    logits[0, 0] = 0.5                                     # all equal: index 0
    logits[1, 1, 7] = float("nan")
    logits[1, 1, 19999] = float("nan")                     # first NaN wins
    logits[2, :, 100] = 50.0
    logits[2, :, 17000] = 50.0                             # exact tie: lower index
    logits[3, 0] = -float("inf")
    logits[3, 0, 12345] = float("inf")
    logits[4, 2] = -1.0
    logits[4, 2, 3] = -0.0
    logits[4, 2, 9] = 0.0                                  # -0.0 == +0.0: index 3
    logits[5, 0, 0] = float("nan")                         # NaN at index 0
    draft[6, 2] = V                                        # out of range: flagged, rejected
    draft[7, 0] = -1
    am = torch.argmax(logits, -1)
    draft[:6] = am[:6, :gamma].to(torch.int32)
    _run_accept(logits, draft)


def test_accept_scalar_paths():
    # vocab not a multiple of 4 and a base pointer that is not 16-byte aligned
    logits, draft = _accept_case(6, 4, 30001, seed=9)
    _run_accept(logits, draft)
    big, draft2 = _accept_case(6, 4, 30001, seed=10)
    flat = torch.empty(big.numel() + 1, device="cuda")
    flat[1:] = big.reshape(-1)
    shifted = flat[1:].view(big.shape)
    _run_accept(shifted, draft2)


def test_accept_agreement_statistics_full_vocab():
    # p = 1 accepts every draft; a forced first mismatch accepts none
    logits, draft = _accept_case(16, 8, 151936, seed=3, p=1.0)
    assert (_run_accept(logits, draft) == 8).all()
    am = torch.argmax(logits, -1)
    draft[:, 0] = ((am[:, 0] + 1) % 151936).to(torch.int32)
    assert (_run_accept(logits, draft) == 0).all()
