"""One verification step of SimSD through the C ABI.

A step (Sec. 3.2, one target verification forward per speculative step):
  1. simsd_build_mask      tau / section / RoPE-copy positions (Eq. (1))
  2. simsd_verify_attention, once per layer (the masked attention; with
     ``rope_theta`` the un-rotated q / k_new are rotated at the RoPE-copy
     positions inside the kernel, Sec. 3.1)
  3. simsd_accept_ws       greedy longest-prefix acceptance (Eq. (2), T=0)
  4. simsd_kv_commit       append the accepted drafts' K/V, advance n_b
All four run on one stream and are captured into one CUDA graph, so the
step needs no host round trip.  PyTorch only allocates the buffers.
"""
from __future__ import annotations

import torch

from . import simsd
from .inputs import StepInputs


class VerifyStep:
    """Device buffers and the call sequence of one verification step.

    ``restore_prefix`` copies the original prefix lengths back before each
    step (4*Bt bytes, an elementwise kernel) so that repeated steps verify the same
    block against the same prefix: the commit writes rows past the original
    prefix, which the restored lengths never read.
    """

    def __init__(self, si: StepInputs, restore_prefix: bool = True, rope_theta: float = 0.0):
        w = si.w
        self.rope_theta = float(rope_theta)
        dev = si.q.device
        self.si = si
        self.w = w
        self.restore_prefix = restore_prefix
        self.L = si.q.shape[0]
        i32 = dict(dtype=torch.int32, device=dev)
        self.n_orig = si.prefix_len.clone()
        self.n = si.prefix_len.clone()
        self.tau = torch.empty(w.Bt, w.S, **i32)
        self.section = torch.empty(w.Bt, w.S, dtype=torch.uint8, device=dev)
        self.rope_pos = torch.empty(w.Bt, w.S, **i32)
        self.out = torch.empty_like(si.q)
        dt = simsd.SIMSD_BF16 if si.q.dtype == torch.bfloat16 else simsd.SIMSD_F32
        ws = simsd.simsd_verify_workspace_bytes(dt, w.Bt, w.gamma, w.Hq, w.Hkv, w.d, si.block_table.shape[1],
                                                w.page_size)
        self.workspace = torch.empty(max(ws, 16), dtype=torch.uint8, device=dev) if ws > 0 else None
        # the acceptance splits a small batch's logits over more CTAs when a
        # workspace is given (0 bytes: the scratch-free cluster kernel)
        aws = simsd.simsd_accept_workspace_bytes(w.Bt, w.gamma, si.logits.shape[-1]) if si.logits is not None else 0
        self.accept_workspace = torch.empty(aws, dtype=torch.uint8, device=dev) if aws > 0 else None
        self.accepted_len = torch.empty(w.Bt, **i32)
        self.out_tokens = torch.empty(w.Bt, w.gamma + 1, **i32)
        self.row_argmax = torch.empty(w.Bt, w.gamma + 1, **i32)
        self.err = torch.zeros(1, **i32)
        self.graph = None
        self.attn_events = None

    # ------------------------------------------------------------------
    def restore(self):
        """Puts the original prefix lengths back (4*Bt bytes).  An
        elementwise kernel, not a memcpy: a memcpy would be queued on a copy
        engine behind the next step's host-to-device input copies and hold
        this step back until they finish."""
        torch.mul(self.n_orig, 1, out=self.n)

    def run(self, attn_events=None, restore=None):
        """Issues the whole step on the current stream (eager or captured).
        ``attn_events`` = (start, end) events recorded around the layers'
        attention calls.  ``restore`` (default: the ``restore_prefix``
        setting) first puts the original prefix lengths back."""
        si, w = self.si, self.w
        if self.restore_prefix if restore is None else restore:
            self.restore()
        simsd.simsd_build_mask(si.step_map, self.n, w.gamma, self.tau, self.section, self.rope_pos,
                               err_word=self.err)
        rope = self.rope_pos if self.rope_theta > 0 else None
        if attn_events is not None:
            attn_events[0].record()
        self.run_attention()
        if attn_events is not None:
            attn_events[1].record()
        simsd.simsd_accept_ws(si.logits, si.draft, self.accepted_len, self.out_tokens, self.accept_workspace,
                              row_argmax=self.row_argmax, err_word=self.err)
        simsd.simsd_kv_commit(si.k_new, si.v_new, self.tau, self.section, self.accepted_len, si.k_cache,
                              si.v_cache, si.block_table, self.n, err_word=self.err, rope_pos=rope,
                              rope_theta=self.rope_theta)

    def run_attention(self):
        """The layers' verification attention alone, on the step's current
        mask metadata (the last step's simsd_build_mask)."""
        si = self.si
        rope = self.rope_pos if self.rope_theta > 0 else None
        for l in range(self.L):
            simsd.simsd_verify_attention(si.q[l], si.k_new[l], si.v_new[l], si.k_cache[l], si.v_cache[l],
                                         si.block_table, self.n, self.tau, self.section, self.out[l],
                                         workspace=self.workspace, err_word=self.err, rope_pos=rope,
                                         rope_theta=self.rope_theta)

    def launches_per_step(self) -> int:
        """Kernels of this library launched by one step."""
        combine = 1 if self.workspace is not None else 0
        accept = 2 if self.accept_workspace is not None else 1
        # mask, attention (+ combine) per layer, accept (parts + merge), commit
        return 1 + self.L * (1 + combine) + accept + 1

    def capture(self, time_attention: bool = True):
        """Captures one step into a CUDA graph (with event-record nodes
        around the attention layers when ``time_attention``)."""
        if time_attention:
            self.attn_events = (torch.cuda.Event(enable_timing=True, external=True),
                                torch.cuda.Event(enable_timing=True, external=True))
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.run()  # warm-up outside capture (lazy library setup)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run(self.attn_events)
        self.graph = g
        return g

    def replay(self):
        self.graph.replay()

    def verified_tokens(self) -> int:
        """Accepted drafts plus the one target token per sequence."""
        return int(self.accepted_len.sum().item()) + self.w.Bt
