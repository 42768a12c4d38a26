"""The attention and acceptance planners restated in Python (their rules,
written independently of the library's C++), for tests: the CPU suite
checks the library's plan queries against them over many shapes and SM
counts, and the GPU tests use them to know which path a case takes.

Attention (bf16, d 128): g = Hq/Hkv heads share a KV head, 2*gamma slots a
sequence.  Up to 128 query rows per KV head make one row block; more are
split into blocks of 128 // g slots.  Key tiles of 64 keys: T = ceil(n / 64)
+ 1 (the new slots' tile).  Two row blocks go to the 256-row kernel, which
keeps whole units (sequence, KV head) when there is at least one per SM,
else splits each unit's tiles into the number of ranges ns minimising
ceil(units ns / SMs) (ceil(T / ns) + 14) (the one-row-block kernel keeps
units under 16 tiles), and walks equal runs of all tiles (stream-K)
instead when W + (ceil(W / T) + 1) 14 + 10, W = ceil(units T / SMs), is at
least 3% below that cost (at most 255 sequences).  The one-row-block
kernel splits prefixes only when its units cannot fill two CTAs per SM.
"""

ITEM_COST = 14
MERGE_COST = 10
ROWS = 128
D = 128


def _cdiv(a, b):
    return -(-a // b)


def max_tiles(max_pages, page_size):
    return _cdiv(max_pages * page_size, 64) + 1


def tc256_splits(Bt, Hkv, rb, T, sms):
    if rb != 2:
        return 0
    units = Bt * Hkv
    if units >= sms:
        return 1
    if T < 16:
        return 0
    cost = {ns: _cdiv(units * ns, sms) * (_cdiv(T, ns) + ITEM_COST) for ns in range(1, min(64, max(1, T // 2)) + 1)}
    return min(cost, key=lambda ns: (cost[ns], ns))


def tc256_streamk(Bt, Hkv, T, ns, sms):
    units = Bt * Hkv
    if ns < 1 or Bt > 255 or units * T >= 1 << 30:
        return False
    ranges = _cdiv(units * ns, sms) * (_cdiv(T, ns) + ITEM_COST)
    W = _cdiv(units * T, sms)
    runs = W + (_cdiv(W, T) + 1) * ITEM_COST + MERGE_COST
    return runs * 100 < ranges * 97


def plan_attention(Bt, gamma, Hq, Hkv, max_pages, page_size, sms):
    """dict(kernel, nsplit, streamk, rows_blk, fuse, ws_bytes), or None when
    the bf16 kernels do not take the shape."""
    S, g = 2 * gamma, Hq // Hkv
    if g * S <= ROWS:
        rb, s_blk = 1, S
    else:
        if ROWS % g:
            return None
        s_blk = ROWS // g
        rb = _cdiv(S, s_blk)
    rows_blk = g * s_blk
    if rows_blk > ROWS or g > 256 or s_blk > 256:
        return None
    T = max_tiles(max_pages, page_size)
    ns256 = tc256_splits(Bt, Hkv, rb, T, sms)
    if ns256:
        sk = tc256_streamk(Bt, Hkv, T, ns256, sms)
        ns = 1 if sk else ns256
        if sk:
            ws = sms * (4 * ROWS * (D + 2) * 4 + 16)
        elif ns > 1:
            ws = Bt * Hkv * rb * ns * rows_blk * (D + 2) * 4
        else:
            ws = 0
        return dict(kernel=1, nsplit=ns, streamk=int(sk), rows_blk=rows_blk, fuse=0, ws_bytes=ws)
    units = Bt * Hkv * rb
    slots = 2 * sms
    ns = 1
    if units < slots:
        ns = max(1, slots // units)
        ns = min(ns, max(1, T // 2))
        ns = min(ns, 64)
    fuse = 2 <= ns <= 8
    ws = units * ns * rows_blk * (D + 2) * 4 if ns > 1 and not fuse else 0
    return dict(kernel=0, nsplit=ns, streamk=0, rows_blk=rows_blk, fuse=int(fuse), ws_bytes=ws)


def accept_parts(Bt, gamma, vocab, sms):
    """Greedy acceptance: CTAs per sequence of the split pass (0: cluster kernel)."""
    if Bt * 16 > sms:
        return 0
    if (gamma + 1) * vocab * 4 < 4 << 20:
        return 0
    units = (gamma + 1) * _cdiv(vocab, 4)
    parts = min(units // (8 * 512), 2 * sms // Bt)
    return parts if parts > 16 else 0


def accept_ws(Bt, gamma, vocab, sms):
    p = accept_parts(Bt, gamma, vocab, sms)
    return Bt * p * (gamma + 1) * 8 if p else 0


def samp_parts(Bt, gamma, vocab, sms):
    """Stochastic acceptance: CTAs per sequence of the split pass."""
    if Bt * 16 > sms:
        return 0
    rows = 2 * gamma + 1
    if rows * vocab * 4 < 3 << 20:
        return 0
    units = rows * _cdiv(vocab, 4)
    parts = min(units // (8 * 512), 2 * sms // Bt)
    return parts if parts > 16 else 0


def samp_ws(Bt, gamma, vocab, sms):
    p = samp_parts(Bt, gamma, vocab, sms)
    if not p:
        return 0
    n = Bt * p
    return n * (2 * gamma + 1) * 8 + n * 8 + ((Bt * 4 + 7) & ~7)
