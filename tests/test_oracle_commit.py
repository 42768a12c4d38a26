"""Pins of the oracle's KV commit (SimSD Sec. 3.2 commit, Sec. 3.3 KV cache).

The accepted drafts' data-slot K/V are appended to the sequence's pages in
draft (tau) order.  Pins: a numpy gather that locates the source slots with
argsort of the step map; a round trip (attention over the committed cache
equals library attention over the old prefix followed by the accepted rows);
and the error paths.
"""
import numpy as np
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs
from tests._pins import dense_prefix, library_attention


def _setup(dtype="bf16", L=2, gamma=5, P=8, n=(0, 7, 8, 21), seed=0):
    w = inputs.Workload("tiny", dtype, len(n), 4, 2, 16, gamma, (0, 0), L, 32, 0.5, 1.0, 1.0, seed, P)
    si = inputs.make_step_inputs(w, prefix_override=list(n), random_step_map=True, with_logits=False)
    return w, si


def _commit(w, si, a):
    return orc.kv_commit(inputs.host_bits(si.k_new), inputs.host_bits(si.v_new), si.step_map.numpy(), a,
                         inputs.host_bits(si.k_cache), inputs.host_bits(si.v_cache), si.block_table.numpy(),
                         si.prefix_len.numpy(), w.gamma)


def test_commit_matches_numpy_gather():
    w, si = _setup()
    a = np.array([5, 0, 3, 1], np.int32)
    kc, vc, n2, err = _commit(w, si, a)
    assert err == 0
    n = si.prefix_len.numpy()
    np.testing.assert_array_equal(n2, n + a)
    kn, vn = inputs.host_bits(si.k_new), inputs.host_bits(si.v_new)
    kc0, vc0 = inputs.host_bits(si.k_cache), inputs.host_bits(si.v_cache)
    bt = si.block_table.numpy()
    order = np.argsort(si.step_map.numpy(), axis=1)        # slot of tau = 1, 2, ...
    touched = np.zeros(kc0.shape[1:4][:1] + kc0.shape[3:4], bool)   # [num_pages][P]
    for b in range(w.Bt):
        for r in range(a[b]):
            row = n[b] + r
            pg, off = bt[b, row // w.page_size], row % w.page_size
            touched[pg, off] = True
            np.testing.assert_array_equal(kc[:, pg, :, off], kn[:, b, order[b, r]])
            np.testing.assert_array_equal(vc[:, pg, :, off], vn[:, b, order[b, r]])
    # nothing else changed
    untouched = ~touched
    np.testing.assert_array_equal(kc.transpose(1, 3, 0, 2, 4)[untouched],
                                  kc0.transpose(1, 3, 0, 2, 4)[untouched])
    np.testing.assert_array_equal(vc.transpose(1, 3, 0, 2, 4)[untouched],
                                  vc0.transpose(1, 3, 0, 2, 4)[untouched])


def test_round_trip_through_attention():
    # After the commit, attention with prefix n+a over the cache equals
    # library attention whose prefix is the old prefix followed by the
    # accepted drafts' K/V in tau order.
    w, si = _setup("f32", L=1, gamma=4, P=8, n=(5, 16, 0))
    a = np.array([4, 2, 3], np.int32)
    kc, vc, n2, err = _commit(w, si, a)
    assert err == 0
    q = inputs.host_bits(si.q[0])
    out, err = orc.verify_attention(q, inputs.host_bits(si.k_new[0]), inputs.host_bits(si.v_new[0]), kc[0], vc[0],
                                    si.block_table.numpy(), n2, si.step_map.numpy(), w.gamma)
    assert err == 0
    # dense reference: old prefix + accepted rows, contiguous pages
    order = np.argsort(si.step_map.numpy(), axis=1)
    kc0, vc0 = inputs.host_bits(si.k_cache[0]), inputs.host_bits(si.v_cache[0])
    kn, vn = inputs.host_bits(si.k_new[0]), inputs.host_bits(si.v_new[0])
    nmax = int(n2.max())
    P = nmax + 1
    Kd = np.zeros((w.Bt, w.Hkv, P, w.d), np.float32)
    Vd = np.zeros((w.Bt, w.Hkv, P, w.d), np.float32)
    bt0 = si.block_table.numpy()
    for b in range(w.Bt):
        n = int(si.prefix_len[b])
        for h in range(w.Hkv):
            rows_k = [dense_prefix(kc0, bt0, b, n, h)] + [kn[b, order[b, r], h][None] for r in range(a[b])]
            rows_v = [dense_prefix(vc0, bt0, b, n, h)] + [vn[b, order[b, r], h][None] for r in range(a[b])]
            Kd[b, h, : n + a[b]] = np.concatenate(rows_k)
            Vd[b, h, : n + a[b]] = np.concatenate(rows_v)
    ref = library_attention(q, kn, vn, Kd, Vd, np.arange(w.Bt, dtype=np.int32)[:, None], n2,
                            si.step_map.numpy(), w.gamma)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_commit_error_paths():
    w, si = _setup(n=(0, 7, 15, 21))
    bt = si.block_table.clone()
    n = si.prefix_len.numpy()
    # destination page of sequence 2's first accepted row is outside the pool
    bt[2, n[2] // w.page_size] = si.num_pages
    si.block_table = bt
    sm = si.step_map.clone()
    sm[3] = 0                                  # all padding: no source slot
    si.step_map = sm
    a = np.array([1, 7, 2, 1], np.int32)       # sequence 1: accepted length > gamma
    kc, vc, n2, err = _commit(w, si, a)
    assert err & orc.ERR_PAGE and err & orc.ERR_ACCEPT_LEN and err & orc.ERR_STEP_MAP
    np.testing.assert_array_equal(n2, [n[0] + 1, n[1], n[2] + 2, n[3] + 1])
    # sequence 2: the first row was skipped, the second (next page) was written
    row = n[2] + 1
    order = np.argsort(si.step_map.numpy()[2])
    pg = int(bt[2, row // w.page_size])
    np.testing.assert_array_equal(kc[:, pg, :, row % w.page_size],
                                  inputs.host_bits(si.k_new)[:, 2, order[1]])
    # exactly two cache rows changed (sequence 0's row and sequence 2's second
    # row), in every layer and KV head
    kc0 = inputs.host_bits(si.k_cache)
    changed = (kc != kc0).any(-1)               # [L][num_pages][Hkv][P]
    assert changed.sum() == 2 * w.layers * w.Hkv
