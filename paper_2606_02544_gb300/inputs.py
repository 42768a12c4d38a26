"""Seeded synthetic inputs for the SimSD verification step.

This module only draws random tensors and lays them out; it contains none of
the method's arithmetic (no mask, no attention, no acceptance, no commit).
Both the CUDA path and the fp64 oracle are fed from it.

The paper measures end-to-end decoding of SDAR models on GSM8K, TriviaQA,
MBPP and MMLU (Sec. 4.1).  Neither the weights nor the datasets are used
here: the verification forward is driven by synthetic tensors with the head
shapes of SDAR-1.7B/4B/8B, the block lengths of the paper (B = gamma = 4, 8,
plus 16 and 32 for the sweep) and draft agreement rates in the range of the
paper's measured token-level acceptance (Table 2: 0.52 to 0.97).

Recipe (one per workload, all values seeded):
  * prefix lengths: fixed, or uniform integers in [lo, hi];
  * paged cache: page size P (64), every sequence owns ceil((n_b + gamma)/P)
    pages (room to commit gamma rows) drawn from one random permutation of the
    page pool; unused block-table entries are -1;
  * Q, K_new, V_new and the cache ~ N(0, std^2) (std 1 for the fp32 case,
    1/sqrt(128) for the bf16 SDAR-shaped cases), one independent draw per
    layer (seed + 1000*l);
  * logits [Bt][gamma+1][V] ~ N(0, sigma^2) in fp32;
  * drafts: with probability p the row's argmax (torch.argmax), otherwise a
    uniform token in [0, V);
  * step map: the identity (left-to-right) unless a random permutation is
    requested; blocks with fewer drafts than positions draw the number of
    drafted, earlier-decoded and still-[MASK] positions uniformly;
  * stochastic acceptance: target logits ~ N(0, sigma^2); the draft model's
    logits are the target's plus N(0, (eta sigma)^2) noise (eta sets how
    often drafts are accepted); each draft is drawn from the draft model's
    softmax(logits / T) by the Gumbel-max rule (argmax of logits / T plus
    Gumbel noise); u_accept and u_sample ~ U[0, 1).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    dtype: str            # "f32" or "bf16": storage and compute type of Q/K/V/O
    Bt: int               # sequences in the batch
    Hq: int               # query heads
    Hkv: int              # KV heads
    d: int                # head dimension
    gamma: int            # draft length = block length
    prefix: tuple         # (lo, hi) inclusive; lo == hi for a fixed prefix
    layers: int           # stacked attention layers (independent K/V per layer)
    vocab: int
    p_agree: float        # probability that a draft equals the row argmax
    qkv_std: float
    logit_std: float
    seed: int
    page_size: int = 64

    @property
    def S(self) -> int:
        return 2 * self.gamma

    @property
    def g(self) -> int:
        return self.Hq // self.Hkv

    def describe(self) -> dict:
        return dataclasses.asdict(self)


_SD = 1.0 / math.sqrt(128.0)

WORKLOADS = {
    # tiny fp32 correctness case
    "c1": Workload("c1_tiny_fp32", "f32", 1, 2, 1, 64, 4, (128, 128), 1, 1024, 0.7, 1.0, 1.0, 0),
    # SDAR-1.7B-shaped verification layer
    "c2": Workload("c2_sdar1.7b_layer", "bf16", 8, 16, 8, 128, 4, (512, 1024), 1, 151936, 0.6, _SD, 2.0, 1),
    # SDAR-4B-shaped verification layer, paged cache P=64
    "c3": Workload("c3_sdar4b_layer_paged64", "bf16", 32, 32, 8, 128, 8, (4096, 4096), 1, 151936, 0.5, _SD, 2.0, 2),
    # SDAR-8B-shaped step over 36 stacked layers
    "c4": Workload("c4_sdar8b_36layers", "bf16", 64, 32, 8, 128, 16, (2048, 8192), 36, 151936, 0.8, _SD, 2.0, 3),
}


def sweep_points():
    """The SDAR-8B head-shape sweep: batch x prefix x gamma x agreement."""
    pts = []
    i = 0
    for Bt in (1, 8, 32, 128):
        for n in (512, 2048, 8192, 32768):
            for gamma in (4, 8, 16, 32):
                for p in (0.3, 0.6, 0.9):
                    pts.append(Workload(f"c5_b{Bt}_n{n}_g{gamma}_p{p}", "bf16", Bt, 32, 8, 128, gamma,
                                        (n, n), 1, 151936, p, _SD, 2.0, 4 + i))
                    i += 1
    return pts


def torch_dtype(w: Workload):
    return torch.float32 if w.dtype == "f32" else torch.bfloat16


@dataclasses.dataclass
class StepInputs:
    """All tensors of one verification step (device or host)."""
    w: Workload
    prefix_len: torch.Tensor      # int32 [Bt]
    block_table: torch.Tensor     # int32 [Bt][max_pages]
    num_pages: int
    step_map: torch.Tensor        # int32 [Bt][gamma]
    q: torch.Tensor               # [L][Bt][S][Hq][d]
    k_new: torch.Tensor           # [L][Bt][S][Hkv][d]
    v_new: torch.Tensor           # [L][Bt][S][Hkv][d]
    k_cache: torch.Tensor         # [L][num_pages][Hkv][P][d]
    v_cache: torch.Tensor         # [L][num_pages][Hkv][P][d]
    logits: torch.Tensor          # fp32 [Bt][gamma+1][V]
    draft: torch.Tensor           # int32 [Bt][gamma]
    row_valid: np.ndarray         # bool [num_pages][P]: row holds a prefix row


def _cpu_gen(seed: int) -> torch.Generator:
    return torch.Generator(device="cpu").manual_seed(int(seed))


def _dev_gen(seed: int, device) -> torch.Generator:
    return torch.Generator(device=device).manual_seed(int(seed))


def make_metadata(w: Workload, seed: Optional[int] = None, prefix_override=None, random_step_map=False,
                  spare_pages: int = 3):
    """Prefix lengths, page table and step map (host tensors, int32)."""
    seed = w.seed if seed is None else seed
    gen = _cpu_gen(seed)
    lo, hi = w.prefix
    if prefix_override is not None:
        n = torch.as_tensor(np.asarray(prefix_override, dtype=np.int32))
    elif lo == hi:
        n = torch.full((w.Bt,), lo, dtype=torch.int32)
    else:
        n = torch.randint(lo, hi + 1, (w.Bt,), generator=gen, dtype=torch.int64).to(torch.int32)
    P = w.page_size
    pages_b = [(int(x) + w.gamma + P - 1) // P for x in n.tolist()]
    num_pages = sum(pages_b) + spare_pages
    max_pages = max(max(pages_b), 1)
    perm = torch.randperm(num_pages, generator=gen).to(torch.int32)
    bt = torch.full((w.Bt, max_pages), -1, dtype=torch.int32)
    pos = 0
    for b, cnt in enumerate(pages_b):
        bt[b, :cnt] = perm[pos:pos + cnt]
        pos += cnt
    if random_step_map:
        sm = torch.stack([torch.randperm(w.gamma, generator=gen) + 1 for _ in range(w.Bt)]).to(torch.int32)
    else:
        sm = torch.arange(1, w.gamma + 1, dtype=torch.int32).repeat(w.Bt, 1)
    # rows of the pool that hold a prefix row
    row_valid = np.zeros((num_pages, P), dtype=bool)
    bt_np = bt.numpy()
    for b in range(w.Bt):
        nb = int(n[b])
        for p in range(pages_b[b]):
            lo_r = p * P
            cnt = min(max(nb - lo_r, 0), P)
            row_valid[bt_np[b, p], :cnt] = True
    return n, bt, num_pages, sm, row_valid


def make_step_inputs(w: Workload, device="cpu", seed: Optional[int] = None, prefix_override=None,
                     random_step_map=False, poison_unused_rows=False, layers: Optional[int] = None,
                     qkv_std: Optional[float] = None, with_logits=True) -> StepInputs:
    """Draws every tensor of one verification step for workload ``w``.

    ``poison_unused_rows`` fills cache rows that hold no prefix row with NaN,
    so that a kernel which reads past a sequence's prefix shows it.
    """
    seed = w.seed if seed is None else seed
    L = w.layers if layers is None else layers
    std = w.qkv_std if qkv_std is None else qkv_std
    n, bt, num_pages, sm, row_valid = make_metadata(w, seed, prefix_override, random_step_map)
    dt = torch_dtype(w)
    S, P = w.S, w.page_size
    poison = None
    if poison_unused_rows:
        poison = torch.as_tensor(~row_valid, device=device).view(num_pages, 1, P, 1)
    q = torch.empty(L, w.Bt, S, w.Hq, w.d, dtype=dt, device=device)
    k_new = torch.empty(L, w.Bt, S, w.Hkv, w.d, dtype=dt, device=device)
    v_new = torch.empty_like(k_new)
    k_cache = torch.empty(L, num_pages, w.Hkv, P, w.d, dtype=dt, device=device)
    v_cache = torch.empty_like(k_cache)
    for l in range(L):
        g = _dev_gen(seed + 1000 * l, device)
        for dst in (q[l], k_new[l], v_new[l], k_cache[l], v_cache[l]):
            dst.copy_(torch.randn(dst.shape, generator=g, device=device).mul_(std))
        if poison is not None:
            k_cache[l].masked_fill_(poison, float("nan"))
            v_cache[l].masked_fill_(poison, float("nan"))
    if with_logits:
        g = _dev_gen(seed + 7, device)
        logits = torch.randn(w.Bt, w.gamma + 1, w.vocab, generator=g, device=device) * w.logit_std
        cg = _cpu_gen(seed + 11)
        agree = torch.rand(w.Bt, w.gamma, generator=cg) < w.p_agree
        rnd = torch.randint(0, w.vocab, (w.Bt, w.gamma), generator=cg, dtype=torch.int64)
        am = torch.argmax(logits[:, : w.gamma, :], dim=-1).cpu()
        draft = torch.where(agree, am, rnd).to(torch.int32)
    else:
        logits = torch.zeros(w.Bt, w.gamma + 1, 1, device=device)
        draft = torch.zeros(w.Bt, w.gamma, dtype=torch.int32)
    dev = torch.device(device)
    return StepInputs(w, n.to(dev), bt.to(dev), num_pages, sm.to(dev), q, k_new, v_new, k_cache, v_cache,
                      logits, draft.to(dev), row_valid)


STEP_UNDRAFTED, STEP_DECODED = -1, -2


def block_step_maps(Bt: int, gamma: int, seed: int, n_draft=None, pad_frac: float = 0.0) -> torch.Tensor:
    """Step maps of blocks with fewer drafts than positions: per sequence a
    random number of drafted positions (labels 1..n in a random order, or
    exactly n_draft), a random number of positions decoded earlier in the
    block (-2), the rest left [MASK] (-1), then padding (0) with probability
    pad_frac.  n_draft = 0 gives the target's own block decoding."""
    g = _cpu_gen(seed)
    out = torch.empty(Bt, gamma, dtype=torch.int32)
    for b in range(Bt):
        nd = int(torch.randint(0, gamma + 1, (1,), generator=g)) if n_draft is None else min(n_draft, gamma)
        ndec = int(torch.randint(0, gamma - nd + 1, (1,), generator=g))
        pos = torch.randperm(gamma, generator=g)
        row = torch.full((gamma,), STEP_UNDRAFTED, dtype=torch.int32)
        row[pos[:nd]] = (torch.randperm(nd, generator=g) + 1).to(torch.int32)
        row[pos[nd:nd + ndec]] = STEP_DECODED
        if pad_frac > 0:
            row[torch.rand(gamma, generator=g) < pad_frac] = 0
        out[b] = row
    return out


@dataclasses.dataclass
class SampledInputs:
    target_logits: torch.Tensor   # fp32 [Bt][gamma+1][V]
    draft_logits: torch.Tensor    # fp32 [Bt][gamma][V]
    draft: torch.Tensor           # int32 [Bt][gamma]
    u_accept: torch.Tensor        # fp32 [Bt][gamma]
    u_sample: torch.Tensor        # fp32 [Bt]
    temperature: float


def make_sampled_inputs(Bt: int, gamma: int, vocab: int, seed: int, logit_std: float = 2.0, eta: float = 0.5,
                        temperature: float = 1.0, device="cpu") -> SampledInputs:
    """Inputs of the stochastic acceptance; drawn on the CPU so that they
    do not depend on the device."""
    g = _cpu_gen(seed)
    tl = torch.randn(Bt, gamma + 1, vocab, generator=g) * logit_std
    dl = tl[:, :gamma] + torch.randn(Bt, gamma, vocab, generator=g) * (eta * logit_std)
    # Gumbel-max: argmax(l / T + G), G = -log(-log U), U ~ U(0, 1)
    uu = torch.rand(Bt, gamma, vocab, generator=g, dtype=torch.float64).clamp_(1e-300, 1.0 - 1e-16)
    draft = torch.argmax(dl.double() / temperature - torch.log(-torch.log(uu)), dim=-1).to(torch.int32)
    del uu
    ua = torch.rand(Bt, gamma, generator=g)
    us = torch.rand(Bt, generator=g)
    dev = torch.device(device)
    return SampledInputs(tl.contiguous().to(dev), dl.contiguous().to(dev), draft.to(dev), ua.to(dev), us.to(dev),
                         float(temperature))


def host_bits(t: torch.Tensor) -> np.ndarray:
    """Host numpy view of a tensor's stored values: float32 as float32,
    bfloat16 as its uint16 bit patterns (exact; no rounding)."""
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float32:
        return t.numpy()
    return t.numpy()
