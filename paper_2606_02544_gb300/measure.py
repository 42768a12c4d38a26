"""Byte and flop accounting of one verification step, and the L2 flush
used between timed steps (shared by bench.py and the sweep)."""
from __future__ import annotations

L2_BYTES = 129 * 1024 * 1024  # GB300 L2


def algorithmic_bytes(si):
    """Bytes the verification attention must move per layer (each read
    once): the prefix K/V, Q, K_new/V_new and O, plus metadata; its flops
    over the visible keys; and the bytes of the acceptance logits."""
    w = si.w
    eb = 4 if w.dtype == "f32" else 2
    n = si.prefix_len.double().sum().item()
    kv = n * w.Hkv * w.d * 2 * eb
    q_o = 2 * w.Bt * w.S * w.Hq * w.d * eb
    new = 2 * w.Bt * w.S * w.Hkv * w.d * eb
    meta = w.Bt * (4 + 4 * si.block_table.shape[1] + 5 * w.S)
    attn = kv + q_o + new + meta
    flops = 4.0 * w.d * w.Hq * w.S * (n + w.Bt * w.gamma)
    accept = w.Bt * (w.gamma + 1) * w.vocab * 4.0
    return attn, flops, accept


def flush_l2(buf):
    """Evicts the step's data from L2: write a buffer twice the L2 size, then
    read it back so the dirty lines are written out before the next step."""
    buf.fill_(1)
    buf.view(-1, 4096).amax(dim=1)
