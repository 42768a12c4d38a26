"""GPU parity of the 256-row attention kernel (two row blocks of one KV head
in one persistent CTA per SM) against the fp64 oracle, both bars of
tests/_gpu.py.

The kernel serves units of 129..256 query rows per KV head (32 drafts with
32/8 heads, 16 drafts with 64/8 heads, 20 drafts with 32/8 heads, where the
second block is partly empty).  With fewer units than SMs each unit's key
tiles are split into ranges whose partials the combine kernel merges; with
more, when whole units would load the CTAs unevenly, every CTA takes an
equal run of the key tiles of all units (stream-K) and the units cut by run
boundaries are merged by a second launch.
Cases: ragged prefixes across tile and page edges, every page size, random
step maps, padding, undrafted and decoded positions, RoPE applied in the
kernel (both position rules), NaN-poisoned unused cache rows, more
sequences than the ranking handles, split units (small batches, ranges with
no tile, the new-slot tile in range 0 only), stream-K runs (units cut once
or across many CTAs, prefix lengths out of range inside a run), and the
error paths.
"""
import numpy as np
import pytest
import torch

from paper_2606_02544_gb300 import inputs, simsd
from tests import _plan
from tests._gpu import assert_attention_close, gpu_attention, gpu_mask, oracle_attention

pytestmark = pytest.mark.gpu


def _w(Bt, gamma=32, Hq=32, Hkv=8, P=64, prefix=(0, 700), seed=0, std=None):
    std = 1 / np.sqrt(128) if std is None else std
    return inputs.Workload("t256", "bf16", Bt, Hq, Hkv, 128, gamma, prefix, 1, 64, 0.5, std, 1.0, seed, P)


def _uses_tc256(si):
    # two row blocks of 128 rows per KV head
    w = si.w
    rows = w.g * w.S
    return 128 < rows <= 256 and 128 % w.g == 0


def _splits(si):
    # key-tile ranges per unit as the planner chooses them (tests/_plan.py):
    # 1 with at least one unit per SM, 0 when the one-row-block kernel takes
    # the shape
    w = si.w
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    return _plan.tc256_splits(w.Bt, w.Hkv, 2, _plan.max_tiles(si.block_table.shape[1], w.page_size), sms)


def _streamk(si):
    # equal runs of all key tiles instead of those ranges (tests/_plan.py)
    w = si.w
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    T = _plan.max_tiles(si.block_table.shape[1], w.page_size)
    return _plan.tc256_streamk(w.Bt, w.Hkv, T, _splits(si), sms)


def _check(si, seqs=None, rope=None):
    assert _uses_tc256(si)
    if rope is None:
        out, word, ws = gpu_attention(si)
        ref = oracle_attention(si, seqs=seqs)
    else:
        theta, mode = rope
        tau, sect, pos, _, merr = gpu_mask(si, mask_bits=False)
        assert simsd.simsd_check_error(merr) == 0
        if mode == 2:
            n = si.prefix_len.long()[:, None]
            pos = (n + torch.arange(si.w.S, device=n.device)[None]).to(torch.int32).contiguous()
        out, word, ws = gpu_attention(si, mask=(tau, sect), rope_pos=pos, rope_theta=theta)
        ref = oracle_attention(si, seqs=seqs, rope_theta=theta, rope_mode=mode)
    # a workspace when the units are split or walked in stream-K runs, none
    # when the kernel takes them whole
    ns = _splits(si)
    assert (ns > 1 and ws > 0) or (ns == 1 and (ws > 0) == _streamk(si)) or ns == 0
    assert word == ref.err
    got = out if seqs is None else out[torch.as_tensor(seqs, device=out.device)]
    assert_attention_close(got, ref)
    return out, word


@pytest.mark.parametrize("P", [8, 16, 32, 64, 128, 256])
def test_page_sizes_and_ragged_prefixes(P):
    rng = np.random.default_rng(P)
    n = rng.integers(0, 700, 20)
    n[:6] = [0, 1, 63, 64, 65, 129]
    si = inputs.make_step_inputs(_w(20, P=P, seed=P), device="cuda", prefix_override=n, random_step_map=True,
                                 poison_unused_rows=True)
    _check(si, seqs=[0, 1, 2, 3, 4, 5, 11, 19])


@pytest.mark.parametrize("gamma,Hq", [(32, 32), (16, 64), (20, 32), (17, 32)])
def test_row_layouts(gamma, Hq):
    # 64/8 heads with 16 drafts: 256 rows of 8 heads x 32 slots; 20 or 17
    # drafts with 32/8 heads: the second block is partly empty
    si = inputs.make_step_inputs(_w(24, gamma=gamma, Hq=Hq, seed=gamma + Hq), device="cuda", random_step_map=True,
                                 poison_unused_rows=True)
    _check(si, seqs=[0, 7, 13, 23])


def test_many_units_per_cta_and_long_prefixes():
    # 64 sequences x 8 KV heads = 512 units: several units per CTA, prefixes
    # from 0 to 4000 ranked longest first
    si = inputs.make_step_inputs(_w(64, prefix=(0, 4000), seed=3), device="cuda", random_step_map=True)
    n = si.prefix_len.cpu().numpy()
    _check(si, seqs=sorted({int(np.argmax(n)), int(np.argmin(n)), 5, 40, 63}))


def test_more_sequences_than_ranked():
    # beyond 256 sequences the walk keeps the batch order (whole units)
    si = inputs.make_step_inputs(_w(300, prefix=(0, 300), seed=4), device="cuda")
    assert not _streamk(si)
    _check(si, seqs=[0, 150, 299])


def test_whole_units_one_per_sm():
    # 19 x 8 = 152 units: one per SM, the whole-unit walk
    si = inputs.make_step_inputs(_w(19, prefix=(200, 1500), seed=13), device="cuda", random_step_map=True,
                                 poison_unused_rows=True)
    assert _splits(si) == 1 and not _streamk(si)
    _check(si, seqs=[0, 9, 18])


@pytest.mark.parametrize("Bt,lens,P", [
    (20, [9000] + [10] * 19, 64),                        # the long units span many CTAs each
    (20, [9000] + [10] * 19, 16),
    (20, [0, 64, 65, 4000, 1] * 4, 64),                  # ragged; runs start inside and between units
    (20, [0, 64, 65, 4000, 1] * 4, 256),
    (24, [3000, 0, 2500, 0, 700, 129] * 4, 64),
    (40, list(range(0, 4000, 100)), 32),
])
def test_streamk_runs(Bt, lens, P):
    si = inputs.make_step_inputs(_w(Bt, prefix=(0, max(lens)), P=P, seed=Bt + len(set(lens)) + P), device="cuda",
                                 prefix_override=np.array(lens), random_step_map=True, poison_unused_rows=True)
    assert _streamk(si)
    _check(si, seqs=sorted({0, 1, 3, Bt // 2, Bt - 1}))


@pytest.mark.parametrize("mode", [1, 2])
def test_streamk_rope(mode):
    si = inputs.make_step_inputs(_w(20, prefix=(2000, 3000), seed=40 + mode), device="cuda", random_step_map=True)
    assert _streamk(si)
    _check(si, seqs=[0, 10, 19], rope=(1e6, mode))


def test_streamk_deterministic():
    si = inputs.make_step_inputs(_w(24, prefix=(1500, 4000), seed=16), device="cuda", random_step_map=True)
    assert _streamk(si)
    a, _, _ = gpu_attention(si)
    b, _, _ = gpu_attention(si)
    assert torch.equal(a, b)


def test_short_units_stay_whole():
    # 20 sequences of at most 700 keys (12 tiles): the pieces and the merge
    # of equal runs would cost more than the uneven whole units
    si = inputs.make_step_inputs(_w(20, prefix=(0, 700), seed=17), device="cuda")
    assert _splits(si) == 1 and not _streamk(si)


def test_streamk_small_batch_long_prefixes():
    # 8 x 8 units of ~510 tiles, fewer than SMs: equal runs of ~216 tiles
    # (units spanning three CTAs) cost less than seven ranges a unit in three
    # waves of items (measured 262 -> 244 us at 32768 keys)
    si = inputs.make_step_inputs(_w(8, prefix=(32000, 32768), seed=15), device="cuda", random_step_map=True)
    assert _splits(si) > 1 and _streamk(si)
    _check(si, seqs=[0, 7])


def test_split_units_keep_ranges():
    # the split tests above run the ranges walk, not stream-K
    for Bt, prefix, P in [(1, (3000, 3000), 64), (8, (1500, 2000), 64), (12, (2000, 6000), 64), (2, (1000, 1100), 8)]:
        si = inputs.make_step_inputs(_w(Bt, prefix=prefix, P=P, seed=1), device="cuda")
        assert _splits(si) > 1 and not _streamk(si)


def test_streamk_largest_batch():
    # 255 sequences, the most stream-K takes: the tile offsets of all of them
    # fill the CTA's 256-entry table; ~16k-key prefixes (17 GB of cache)
    si = inputs.make_step_inputs(_w(255, prefix=(15000, 16000), seed=18), device="cuda", random_step_map=True)
    assert _streamk(si)
    _check(si, seqs=[0, 127, 254])


def test_streamk_bad_prefix_inside_runs():
    # prefix lengths out of range and a bad page inside runs that cut units
    si = inputs.make_step_inputs(_w(22, prefix=(2000, 3000), seed=14), device="cuda", random_step_map=True)
    n = si.prefix_len.clone()
    n[3] = si.block_table.shape[1] * si.w.page_size + 1
    n[10] = -1
    si.prefix_len = n
    bt = si.block_table.clone()
    bt[7, 5] = si.num_pages
    si.block_table = bt
    assert _streamk(si)
    out, word = _check(si, seqs=[2, 3, 4, 7, 10, 11])
    assert word & simsd.EW_PREFIX_LEN and word & simsd.EW_PAGE
    assert (out[[3, 7, 10]].float() == 0).all()


@pytest.mark.parametrize("n_draft", [None, 0])
def test_undrafted_decoded_and_padding(n_draft):
    si = inputs.make_step_inputs(_w(20, prefix=(0, 500), seed=5), device="cuda")
    si.step_map = inputs.block_step_maps(20, 32, seed=6, n_draft=n_draft, pad_frac=0.1).cuda()
    _check(si, seqs=[0, 3, 9, 19])


@pytest.mark.parametrize("mode", [1, 2])
def test_rope_in_kernel(mode):
    si = inputs.make_step_inputs(_w(20, prefix=(0, 600), seed=7 + mode), device="cuda", random_step_map=True)
    _check(si, seqs=[0, 10, 19], rope=(1e6, mode))


def test_unit_scale_scores():
    si = inputs.make_step_inputs(_w(20, prefix=(100, 900), seed=9, std=1.0), device="cuda", random_step_map=True)
    _check(si, seqs=[2, 17])


def test_error_paths():
    si = inputs.make_step_inputs(_w(20, prefix=(10, 300), seed=10), device="cuda")
    sm = si.step_map.clone()
    sm[0, 2] = 0                                    # padding slot in sequence 0
    sm[3, :2] = 1                                   # invalid map: all padding
    si.step_map = sm
    n = si.prefix_len.clone()
    n[1] = si.block_table.shape[1] * si.w.page_size + 3    # beyond the block table
    si.prefix_len = n
    bt = si.block_table.clone()
    bt[2, 1] = si.num_pages + 5                     # page id outside the pool
    si.block_table = bt
    out, word = _check(si, seqs=[0, 1, 2, 3, 4])
    assert word & simsd.EW_PREFIX_LEN and word & simsd.EW_PAGE and word & simsd.EW_STEP_MAP
    assert (out[1:4].float() == 0).all() and (out[0, [2, 34]].float() == 0).all()


@pytest.mark.parametrize("Bt,prefix,P,split", [(1, (0, 0), 64, 0), (1, (3000, 3000), 64, 2),
                                               (3, (1200, 1500), 16, 2), (8, (1500, 2000), 64, 2),
                                               (8, (0, 40), 32, 0), (12, (2000, 6000), 64, 2),
                                               (18, (500, 1500), 128, 1), (2, (1000, 1100), 8, 2)])
def test_split_units(Bt, prefix, P, split):
    # fewer units than SMs: ranges of key tiles per unit, merged by the
    # combine kernel (ranges of short sequences can hold no tile); nearly
    # one unit per SM stays whole (1), short units go to the one-row-block
    # kernel (0)
    si = inputs.make_step_inputs(_w(Bt, prefix=prefix, P=P, seed=Bt + P), device="cuda", random_step_map=True,
                                 poison_unused_rows=True)
    assert min(_splits(si), 2) == split
    _check(si, seqs=sorted({0, Bt // 2, Bt - 1}))


@pytest.mark.parametrize("gamma,Hq", [(16, 64), (20, 32)])
def test_split_units_row_layouts(gamma, Hq):
    si = inputs.make_step_inputs(_w(4, gamma=gamma, Hq=Hq, prefix=(1000, 1200), seed=gamma), device="cuda",
                                 random_step_map=True, poison_unused_rows=True)
    assert _splits(si) > 1
    _check(si, seqs=[0, 3])


@pytest.mark.parametrize("mode", [1, 2])
def test_split_units_rope(mode):
    si = inputs.make_step_inputs(_w(2, prefix=(1000, 1300), seed=20 + mode), device="cuda", random_step_map=True)
    assert _splits(si) > 1
    _check(si, seqs=[0, 1], rope=(1e6, mode))


def test_split_units_error_paths():
    si = inputs.make_step_inputs(_w(6, prefix=(1000, 1700), seed=30), device="cuda")
    sm = si.step_map.clone()
    sm[0, 5] = 0                                    # padding slot in sequence 0
    sm[3, :2] = 1                                   # invalid map: all padding
    si.step_map = sm
    n = si.prefix_len.clone()
    n[1] = si.block_table.shape[1] * si.w.page_size + 3    # beyond the block table
    si.prefix_len = n
    bt = si.block_table.clone()
    bt[2, 1] = -1                                   # page id outside the pool
    si.block_table = bt
    assert _splits(si) > 1
    out, word = _check(si, seqs=[0, 1, 2, 3, 4])
    assert word & simsd.EW_PREFIX_LEN and word & simsd.EW_PAGE and word & simsd.EW_STEP_MAP
    assert (out[1:4].float() == 0).all() and (out[0, [5, 37]].float() == 0).all()


def test_split_units_deterministic():
    si = inputs.make_step_inputs(_w(2, prefix=(900, 4000), seed=12), device="cuda", random_step_map=True)
    a, _, _ = gpu_attention(si)
    b, _, _ = gpu_attention(si)
    assert torch.equal(a, b)


def test_deterministic_and_equal_to_rerun():
    si = inputs.make_step_inputs(_w(24, prefix=(100, 900), seed=11), device="cuda", random_step_map=True)
    a, _, _ = gpu_attention(si)
    b, _, _ = gpu_attention(si)
    assert torch.equal(a, b)
