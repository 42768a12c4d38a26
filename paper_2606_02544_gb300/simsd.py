"""Python binding of libsimsd.so (argument marshalling only).

Each function has the name of the C entry point it calls (include/simsd.h)
and takes torch CUDA tensors; it reads shapes and data pointers, passes them
with the current CUDA stream, and raises :class:`SimsdError` on a non-zero
status.  Every step of the computation runs in the library's kernels; there
is no fallback: if the library is missing or fails to load, the first call
raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libsimsd.so")

SIMSD_OK, SIMSD_ERR_INVALID_ARG, SIMSD_ERR_UNSUPPORTED, SIMSD_ERR_CUDA, SIMSD_ERR_DEVICE = 0, 1, 2, 3, 4
SIMSD_F32, SIMSD_BF16 = 0, 1
SECT_DATA, SECT_MASK, SECT_PAD = 0, 1, 255
EW_STEP_MAP, EW_PREFIX_LEN, EW_PAGE, EW_DRAFT, EW_TIMEOUT, EW_ACCEPT_LEN = 1, 2, 4, 8, 16, 32
STEP_UNDRAFTED, STEP_DECODED = -1, -2

EXPORTED = ("simsd_build_mask", "simsd_verify_workspace_bytes", "simsd_verify_attention",
            "simsd_verify_attention_noalloc", "simsd_accept", "simsd_accept_workspace_bytes", "simsd_accept_ws",
            "simsd_accept_sampled", "simsd_accept_sampled_workspace_bytes", "simsd_accept_sampled_ws",
            "simsd_kv_commit", "simsd_plan_attention", "simsd_plan_accept",
            "simsd_check_error", "simsd_debug_expire_next_wait",
            "simsd_last_error", "simsd_version")
DEBUG_WAIT_ATTENTION, DEBUG_WAIT_ACCEPT = 1, 2


class SimsdError(RuntimeError):
    def __init__(self, status, where, detail=""):
        super().__init__(f"{where} failed with status {status}: {detail}")
        self.status = status


_lib = None
_lock = threading.Lock()


def load_library(path: str = LIB_PATH):
    """Loads libsimsd.so once; raises if it is missing (build it with
    ``paper_2606_02544_gb300.build.build()``)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise RuntimeError(f"libsimsd.so not found at {path}; run paper_2606_02544_gb300.build.build()")
            lib = ctypes.CDLL(path)
            P, I, F, Z = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
            lib.simsd_build_mask.argtypes = [P, P, I, I, P, P, P, P, P, P]
            lib.simsd_verify_workspace_bytes.argtypes = [I, I, I, I, I, I, I, I]
            lib.simsd_verify_workspace_bytes.restype = Z
            lib.simsd_verify_attention.argtypes = [I, P, P, P, P, P, I, P, I, I, P, P, P, P, F, I, I, I, I, I, F,
                                                   P, P, Z, P, P]
            lib.simsd_verify_attention_noalloc.argtypes = [I, P, P, P, P, P, I, P, I, I, P, P, P, P, F, I, I, I, I,
                                                           I, F, P, P, P]
            lib.simsd_accept.argtypes = [P, P, I, I, I, P, P, P, P, P]
            lib.simsd_accept_workspace_bytes.argtypes = [I, I, I]
            lib.simsd_accept_workspace_bytes.restype = Z
            lib.simsd_accept_ws.argtypes = [P, P, I, I, I, P, P, P, P, Z, P, P]
            lib.simsd_accept_sampled.argtypes = [P, P, P, P, P, F, I, I, I, P, P, P, P]
            lib.simsd_accept_sampled_workspace_bytes.argtypes = [I, I, I]
            lib.simsd_accept_sampled_workspace_bytes.restype = Z
            lib.simsd_accept_sampled_ws.argtypes = [P, P, P, P, P, F, I, I, I, P, P, P, Z, P, P]
            lib.simsd_kv_commit.argtypes = [I, P, P, I, P, P, P, F, P, P, P, I, P, I, I, P, I, I, I, I, P, P]
            lib.simsd_check_error.argtypes = [P, P, P]
            lib.simsd_debug_expire_next_wait.argtypes = [I, ctypes.c_uint]
            lib.simsd_plan_attention.argtypes = [I, I, I, I, I, I, I, I, I, P, P]
            lib.simsd_plan_accept.argtypes = [I, I, I, I, I, P, P]
            lib.simsd_last_error.restype = ctypes.c_char_p
            for name in ("simsd_build_mask", "simsd_verify_attention", "simsd_verify_attention_noalloc",
                         "simsd_accept", "simsd_accept_sampled", "simsd_kv_commit", "simsd_check_error",
                         "simsd_debug_expire_next_wait", "simsd_version", "simsd_plan_attention",
                         "simsd_plan_accept"):
                getattr(lib, name).restype = ctypes.c_int
            _lib = lib
    return _lib


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _check(rc, where):
    if rc != SIMSD_OK:
        detail = load_library().simsd_last_error().decode(errors="replace")
        raise SimsdError(rc, where, detail)


def _dtype_code(t):
    if t.dtype == torch.bfloat16:
        return SIMSD_BF16
    if t.dtype == torch.float32:
        return SIMSD_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def simsd_version() -> int:
    return load_library().simsd_version()


def simsd_plan_attention(dtype, Bt, gamma, Hq, Hkv, d, max_pages, page_size, num_sms):
    """The plan simsd_verify_attention takes on a GPU with num_sms SMs (no
    device needed): dict of kernel, nsplit, streamk, rows_blk, fuse and
    ws_bytes."""
    plan = (ctypes.c_int32 * 5)()
    ws = ctypes.c_size_t(0)
    rc = load_library().simsd_plan_attention(dtype, Bt, gamma, Hq, Hkv, d, max_pages, page_size, num_sms,
                                             ctypes.cast(plan, ctypes.c_void_p), ctypes.cast(ctypes.pointer(ws),
                                                                                            ctypes.c_void_p))
    _check(rc, "simsd_plan_attention")
    return {"kernel": plan[0], "nsplit": plan[1], "streamk": plan[2], "rows_blk": plan[3], "fuse": plan[4],
            "ws_bytes": ws.value}


def simsd_plan_accept(sampled, Bt, gamma, vocab, num_sms):
    """(parts, ws_bytes) of simsd_accept_ws (sampled False) or
    simsd_accept_sampled_ws (True) on a GPU with num_sms SMs."""
    parts = ctypes.c_int32(0)
    ws = ctypes.c_size_t(0)
    rc = load_library().simsd_plan_accept(int(bool(sampled)), Bt, gamma, vocab, num_sms,
                                          ctypes.cast(ctypes.pointer(parts), ctypes.c_void_p),
                                          ctypes.cast(ctypes.pointer(ws), ctypes.c_void_p))
    _check(rc, "simsd_plan_accept")
    return parts.value, ws.value


def simsd_build_mask(step_map, prefix_len, gamma, tau, section, rope_pos, mask_bits=None, err_word=None,
                     stream=None):
    Bt = prefix_len.shape[0]
    rc = load_library().simsd_build_mask(_p(step_map), _p(prefix_len), Bt, gamma, _p(tau), _p(section),
                                         _p(rope_pos), _p(mask_bits), _p(err_word), _stream(stream))
    _check(rc, "simsd_build_mask")


def simsd_verify_workspace_bytes(dtype_code, Bt, gamma, Hq, Hkv, d, max_pages, page_size) -> int:
    return int(load_library().simsd_verify_workspace_bytes(dtype_code, Bt, gamma, Hq, Hkv, d, max_pages, page_size))


def simsd_verify_attention(q, k_new, v_new, k_cache, v_cache, block_table, prefix_len, tau, section, out,
                           workspace=None, err_word=None, softmax_scale=0.0, rope_pos=None, rope_theta=0.0,
                           stream=None):
    """q/out [Bt][2g][Hq][d]; k_new/v_new [Bt][2g][Hkv][d];
    k_cache/v_cache [num_pages][Hkv][P][d]; block_table [Bt][max_pages].
    rope_pos [Bt][2g] (with rope_theta > 0): q and k_new are rotated first."""
    Bt, S, Hq, d = q.shape
    Hkv = k_new.shape[2]
    num_pages, _, P, _ = k_cache.shape
    max_pages = block_table.shape[1]
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = load_library().simsd_verify_attention(
        _dtype_code(q), _p(q), _p(k_new), _p(v_new), _p(k_cache), _p(v_cache), num_pages, _p(block_table),
        max_pages, P, _p(prefix_len), _p(tau), _p(section), _p(rope_pos), float(rope_theta), Bt, S // 2, Hq, Hkv,
        d, float(softmax_scale), _p(out), _p(workspace), ws_bytes, _p(err_word), _stream(stream))
    _check(rc, "simsd_verify_attention")


def simsd_verify_attention_noalloc(q, k_new, v_new, k_cache, v_cache, block_table, prefix_len, tau, section, out,
                                   err_word=None, softmax_scale=0.0, rope_pos=None, rope_theta=0.0, stream=None):
    """simsd_verify_attention without a workspace: the library's static
    device scratch is used instead (for callers that cannot allocate)."""
    Bt, S, Hq, d = q.shape
    Hkv = k_new.shape[2]
    num_pages, _, P, _ = k_cache.shape
    max_pages = block_table.shape[1]
    rc = load_library().simsd_verify_attention_noalloc(
        _dtype_code(q), _p(q), _p(k_new), _p(v_new), _p(k_cache), _p(v_cache), num_pages, _p(block_table),
        max_pages, P, _p(prefix_len), _p(tau), _p(section), _p(rope_pos), float(rope_theta), Bt, S // 2, Hq, Hkv,
        d, float(softmax_scale), _p(out), _p(err_word), _stream(stream))
    _check(rc, "simsd_verify_attention_noalloc")


def simsd_accept(logits, draft, accepted_len, out_tokens, row_argmax=None, err_word=None, stream=None):
    Bt, rows, V = logits.shape
    rc = load_library().simsd_accept(_p(logits), _p(draft), Bt, rows - 1, V, _p(accepted_len), _p(out_tokens),
                                     _p(row_argmax), _p(err_word), _stream(stream))
    _check(rc, "simsd_accept")


def simsd_accept_workspace_bytes(Bt, gamma, vocab) -> int:
    return int(load_library().simsd_accept_workspace_bytes(Bt, gamma, vocab))


def simsd_accept_ws(logits, draft, accepted_len, out_tokens, workspace=None, row_argmax=None, err_word=None,
                    stream=None):
    """simsd_accept with a caller workspace (uint8 device tensor of
    simsd_accept_workspace_bytes() bytes, or None when that is 0)."""
    Bt, rows, V = logits.shape
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    rc = load_library().simsd_accept_ws(_p(logits), _p(draft), Bt, rows - 1, V, _p(accepted_len), _p(out_tokens),
                                        _p(row_argmax), _p(workspace), nbytes, _p(err_word), _stream(stream))
    _check(rc, "simsd_accept_ws")


def simsd_accept_sampled(target_logits, draft_logits, draft, u_accept, u_sample, accepted_len, out_tokens,
                         temperature=1.0, err_word=None, stream=None):
    """target_logits [Bt][g+1][V], draft_logits [Bt][g][V] fp32; draft [Bt][g];
    u_accept [Bt][g], u_sample [Bt] fp32 uniform draws."""
    Bt, rows, V = target_logits.shape
    rc = load_library().simsd_accept_sampled(_p(target_logits), _p(draft_logits), _p(draft), _p(u_accept),
                                             _p(u_sample), float(temperature), Bt, rows - 1, V, _p(accepted_len),
                                             _p(out_tokens), _p(err_word), _stream(stream))
    _check(rc, "simsd_accept_sampled")


def simsd_kv_commit(k_new, v_new, tau, section, accepted_len, k_cache, v_cache, block_table, prefix_len,
                    err_word=None, rope_pos=None, rope_theta=0.0, stream=None):
    """k_new/v_new [L][Bt][2g][Hkv][d]; k_cache/v_cache [L][num_pages][Hkv][P][d].
    rope_pos [Bt][2g] (with rope_theta > 0): committed keys are rotated."""
    L, Bt, S, Hkv, d = k_new.shape
    num_pages, P = k_cache.shape[1], k_cache.shape[3]
    rc = load_library().simsd_kv_commit(
        _dtype_code(k_new), _p(k_new), _p(v_new), L, _p(tau), _p(section), _p(rope_pos), float(rope_theta),
        _p(accepted_len), _p(k_cache),
        _p(v_cache), num_pages, _p(block_table), block_table.shape[1], P, _p(prefix_len), Bt, S // 2, Hkv, d,
        _p(err_word), _stream(stream))
    _check(rc, "simsd_kv_commit")


def simsd_debug_expire_next_wait(which, limit_us):
    """Test hook: the next attention (DEBUG_WAIT_ATTENTION) or acceptance
    (DEBUG_WAIT_ACCEPT) call of this thread waits for an arrival that never
    comes and gives up after limit_us."""
    _check(load_library().simsd_debug_expire_next_wait(int(which), int(limit_us)), "simsd_debug_expire_next_wait")


def simsd_check_error(err_word, stream=None):
    """Synchronises the stream; returns the device error word (int)."""
    w = ctypes.c_int32(0)
    rc = load_library().simsd_check_error(_p(err_word), ctypes.byref(w), _stream(stream))
    if rc not in (SIMSD_OK, SIMSD_ERR_DEVICE):
        _check(rc, "simsd_check_error")
    return int(w.value)


def simsd_accept_sampled_workspace_bytes(Bt, gamma, vocab) -> int:
    return int(load_library().simsd_accept_sampled_workspace_bytes(Bt, gamma, vocab))


def simsd_accept_sampled_ws(target_logits, draft_logits, draft, u_accept, u_sample, accepted_len, out_tokens,
                            workspace=None, temperature=1.0, err_word=None, stream=None):
    """simsd_accept_sampled with a caller workspace (uint8 device tensor of
    simsd_accept_sampled_workspace_bytes() bytes, or None when that is 0)."""
    Bt, rows, V = target_logits.shape
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    rc = load_library().simsd_accept_sampled_ws(_p(target_logits), _p(draft_logits), _p(draft), _p(u_accept),
                                                _p(u_sample), float(temperature), Bt, rows - 1, V, _p(accepted_len),
                                                _p(out_tokens), _p(workspace), nbytes, _p(err_word),
                                                _stream(stream))
    _check(rc, "simsd_accept_sampled_ws")
