"""Independent statements used to pin the oracle (test helpers only).

Nothing here is shared with the oracle or the CUDA path: these are second
statements of the same facts, written from the paper's prose or reduced to
library routines.
"""
import numpy as np
import torch


def prose_mask(mu):
    """Visible new slots per row, from the paper's prose (Sec. 3.1 "Masked
    Token Prediction" and the paragraph after Eq. (1)); block positions with
    mu == 0 are padding (no row, no column)."""
    B = len(mu)
    A = np.zeros((2 * B, 2 * B), bool)
    for i in range(B):
        if mu[i] == 0:
            continue
        for k in range(B):
            if mu[k] == 0:
                continue
            A[i, k] = mu[k] < mu[i] or k == i          # earlier data tokens and itself
            A[i, B + k] = mu[k] > mu[i]                # later mask placeholders
            A[B + i, k] = mu[k] < mu[i]                # data tokens from earlier steps
            A[B + i, B + k] = mu[k] >= mu[i]           # current and later placeholders
    return A


def widen(x):
    """float64 copy of stored values (float32, or bf16 bits held in uint16)."""
    x = np.asarray(x)
    if x.dtype == np.uint16:
        return (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return x.astype(np.float64)


def dense_prefix(cache, block_table, b, n, kvh):
    """Rows 0..n-1 of sequence b read through the page table (numpy gather)."""
    P = cache.shape[2]
    idx = np.arange(n)
    pages = block_table[b, idx // P]
    return cache[pages, kvh, idx % P, :]


def library_attention(q, k_new, v_new, k_cache, v_cache, block_table, prefix_len, step_map, gamma,
                      scale=None):
    """Verification attention through torch's scaled_dot_product_attention in
    fp64, with the mask taken from the prose statement.  Padding rows -> 0."""
    q, k_new, v_new = widen(q), widen(k_new), widen(v_new)
    k_cache, v_cache = widen(k_cache), widen(v_cache)
    Bt, S, Hq, d = q.shape
    Hkv = k_new.shape[2]
    g = Hq // Hkv
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    out = np.zeros_like(q)
    for b in range(Bt):
        n = int(prefix_len[b])
        mu = np.arange(1, gamma + 1) if step_map is None else np.asarray(step_map[b])
        A = prose_mask(list(mu))
        for kvh in range(Hkv):
            Kp = dense_prefix(k_cache, block_table, b, n, kvh)
            Vp = dense_prefix(v_cache, block_table, b, n, kvh)
            K = np.concatenate([Kp, k_new[b, :, kvh]], 0)
            V = np.concatenate([Vp, v_new[b, :, kvh]], 0)
            mask = np.concatenate([np.ones((S, n), bool), A], 1)
            for h in range(kvh * g, (kvh + 1) * g):
                rows = mask.any(1)
                if not rows.any():
                    continue
                o = torch.nn.functional.scaled_dot_product_attention(
                    torch.from_numpy(q[b, rows, h][None]), torch.from_numpy(K[None]),
                    torch.from_numpy(V[None]), attn_mask=torch.from_numpy(mask[rows][None]), scale=scale)
                out[b, rows, h] = o[0].numpy()
    return out
