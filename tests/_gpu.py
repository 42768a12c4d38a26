"""Helpers of the GPU parity tests: run one call through the C ABI and the
same call through the oracle, on the same seeded inputs.

The oracle only ever sees host copies of the generator's tensors; it builds
its own mask from the step map and never reads anything the CUDA path made.
"""
import numpy as np
import torch

from oracle import simsd_oracle as orc
from paper_2606_02544_gb300 import inputs, simsd

BF16_ATOL = 2e-2
BF16_RTOL = 2e-2
F32_ATOL = 1e-5


def gpu_mask(si, mask_bits=True):
    w = si.w
    dev = si.prefix_len.device
    tau = torch.full((w.Bt, w.S), -7, dtype=torch.int32, device=dev)
    sect = torch.full((w.Bt, w.S), 77, dtype=torch.uint8, device=dev)
    rope = torch.full((w.Bt, w.S), -7, dtype=torch.int32, device=dev)
    bits = torch.zeros((w.Bt, w.S), dtype=torch.int64, device=dev) if mask_bits else None
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    simsd.simsd_build_mask(si.step_map, si.prefix_len, w.gamma, tau, sect, rope, bits, err)
    return tau, sect, rope, bits, err


def gpu_attention(si, layer=0, mask=None, err=None, rope_pos=None, rope_theta=0.0):
    w = si.w
    if mask is None:
        tau, sect, _, _, merr = gpu_mask(si, mask_bits=False)
    else:
        tau, sect = mask[0], mask[1]
        merr = None
    dt = simsd.SIMSD_BF16 if si.q.dtype == torch.bfloat16 else simsd.SIMSD_F32
    ws = simsd.simsd_verify_workspace_bytes(dt, w.Bt, w.gamma, w.Hq, w.Hkv, w.d, si.block_table.shape[1],
                                            w.page_size)
    work = torch.zeros(ws, dtype=torch.uint8, device=si.q.device) if ws else None
    out = torch.full_like(si.q[layer], float("nan"))
    e = torch.zeros(1, dtype=torch.int32, device=si.q.device) if err is None else err
    simsd.simsd_verify_attention(si.q[layer], si.k_new[layer], si.v_new[layer], si.k_cache[layer],
                                 si.v_cache[layer], si.block_table, si.prefix_len, tau, sect, out,
                                 workspace=work, err_word=e, rope_pos=rope_pos, rope_theta=rope_theta)
    word = simsd.simsd_check_error(e)
    if merr is not None:
        word |= simsd.simsd_check_error(merr)
    return out, word, ws


def oracle_attention(si, layer=0, seqs=None, rope_theta=0.0, rope_mode=1):
    """Oracle attention for all sequences, or for the listed ones only (a
    sub-batch with its own compact page pool).  rope_theta > 0: q and k_new
    are rotated by the oracle first (rope_mode 1: RoPE copy, 2: physical
    positions)."""
    rope = dict(rope_theta=rope_theta, rope_mode=rope_mode)
    if seqs is None:
        return orc.verify_attention(
            inputs.host_bits(si.q[layer]), inputs.host_bits(si.k_new[layer]), inputs.host_bits(si.v_new[layer]),
            inputs.host_bits(si.k_cache[layer]), inputs.host_bits(si.v_cache[layer]),
            si.block_table.cpu().numpy(), si.prefix_len.cpu().numpy(), si.step_map.cpu().numpy(), si.w.gamma,
            **rope)
    idx = torch.as_tensor(seqs, device=si.q.device)
    bt = si.block_table[idx].cpu()
    n = si.prefix_len[idx].cpu()
    P = si.w.page_size
    used = []
    for r in range(len(seqs)):
        cnt = (int(n[r]) + P - 1) // P
        used.append(bt[r, :cnt])
    used = torch.cat(used) if used else torch.zeros(0, dtype=torch.int32)
    uniq, inv = torch.unique(used, return_inverse=True)
    new_bt = torch.full_like(bt, -1)
    pos = 0
    for r in range(len(seqs)):
        cnt = (int(n[r]) + P - 1) // P
        new_bt[r, :cnt] = inv[pos:pos + cnt].to(torch.int32)
        pos += cnt
    pages = uniq.to(si.q.device).long()
    kc = si.k_cache[layer][pages] if len(pages) else si.k_cache[layer][:1]
    vc = si.v_cache[layer][pages] if len(pages) else si.v_cache[layer][:1]
    return orc.verify_attention(
        inputs.host_bits(si.q[layer][idx]), inputs.host_bits(si.k_new[layer][idx]),
        inputs.host_bits(si.v_new[layer][idx]), inputs.host_bits(kc), inputs.host_bits(vc), new_bt.numpy(),
        n.numpy(), si.step_map[idx].cpu().numpy(), si.w.gamma, **rope)


def assert_attention_close(got, want, dtype):
    g = got.float().cpu().numpy().astype(np.float64)
    assert np.isfinite(g).all(), "non-finite output"
    if dtype == "f32":
        err = np.abs(g - want).max()
        assert err <= F32_ATOL, f"max abs error {err}"
    else:
        bad = np.abs(g - want) > BF16_ATOL + BF16_RTOL * np.abs(want)
        assert not bad.any(), (f"{bad.sum()} elements out of tolerance; max abs "
                               f"{np.abs(g - want).max():.3g}")
    return float(np.abs(g - want).max())
