"""Python front end of the fp64 CPU oracle (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  It builds ``simsd_oracle.c`` with the
host C compiler and calls it through ``ctypes`` on numpy arrays.  It imports
nothing from the CUDA package and shares no code with it.

Each function cites the passage of the SimSD paper it follows:

* :func:`build_mask` -- Sec. 3.1 "Temporal Attention Mask", Eq. (1), and
  "Position Encoding Alignment" (RoPE copy).
* :func:`verify_attention` -- Sec. 3.2 "Target Model Verification" with the
  KV cache of Sec. 3.3: exact masked softmax attention in fp64.
* :func:`accept` -- Sec. 3.2, Eq. (2) at temperature 0 (one-hot draft and
  target distributions): accept the longest prefix whose drafts equal the
  target argmax.
* :func:`kv_commit` -- Sec. 3.2 (commit of accepted tokens) and Sec. 3.3
  (KV cache reuse): append the accepted drafts' K/V to the paged cache.

Every function is pinned by ``tests/test_oracle_*.py`` against closed forms,
library routines, invariants and brute force on tiny inputs.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "simsd_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "libsimsd_oracle.so")
_lib = None
_lock = threading.Lock()

ERR_STEP_MAP = 1
ERR_PREFIX_LEN = 2
ERR_PAGE = 4
ERR_DRAFT = 8
ERR_ACCEPT_LEN = 32

SECT_D, SECT_DT, SECT_PAD = 0, 1, 255
# step-map codes besides the drafted labels 1..gamma (0 is padding)
STEP_UNDRAFTED, STEP_DECODED = -1, -2


def build(force: bool = False) -> str:
    """Compiles the oracle into ``oracle/_build/libsimsd_oracle.so``.

    IEEE semantics are kept (no fast-math, no FMA contraction) so that the
    oracle gives the same bits on x86-64 and aarch64 hosts.
    """
    os.makedirs(_OUT_DIR, exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i = ctypes.c_int
            lib.oracle_build_mask.argtypes = [P, P, i, i, P, P, P, P, P]
            lib.oracle_verify_attention.argtypes = [i, P, P, P, P, P, P, i, i, i, P, P, i, i, i, i, i,
                                                    ctypes.c_double, ctypes.c_double, i, P, i]
            lib.oracle_accept.argtypes = [P, P, i, i, i, P, P, P]
            lib.oracle_kv_commit.argtypes = [i, P, P, i, P, P, P, P, P, i, i, i, P, i, i, i, i,
                                             ctypes.c_double]
            lib.oracle_accept_sampled.argtypes = [P, P, P, P, P, ctypes.c_double, i, i, i, P, P, P, P]
            lib.oracle_accept_sampled.restype = ctypes.c_int
            lib.oracle_rope_rotate.argtypes = [P, i, i, ctypes.c_double, ctypes.c_double]
            lib.oracle_rope_rotate.restype = None
            for f in (lib.oracle_build_mask, lib.oracle_verify_attention, lib.oracle_accept,
                      lib.oracle_kv_commit, lib.oracle_max_threads):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def max_threads() -> int:
    """OpenMP threads the oracle uses by default (OMP_NUM_THREADS or all cores)."""
    return int(_load().oracle_max_threads())


def build_mask(step_map, prefix_len, gamma: int) -> dict:
    """Eq. (1) mask plus per-slot labels.

    step_map: int32 [Bt][gamma] or None for the identity map.  Entries:
    1..gamma drafted labels (distinct), 0 padding, STEP_UNDRAFTED (-1) a
    position that stays [MASK] (mask slot only, tau = gamma + 1),
    STEP_DECODED (-2) a clean token decoded earlier in the block (data slot
    only, tau = 0).  Returns tau, section, rope_pos ([Bt][2gamma]),
    mask_bits (uint64 [Bt][2gamma]), dense (uint8 [Bt][2gamma][2gamma]) and
    the error bits.
    """
    lib = _load()
    prefix_len = _c(prefix_len, np.int32)
    Bt = prefix_len.shape[0]
    S = 2 * gamma
    sm = None if step_map is None else _c(step_map, np.int32).reshape(Bt, gamma)
    tau = np.zeros((Bt, S), np.int32)
    sect = np.zeros((Bt, S), np.uint8)
    rope = np.zeros((Bt, S), np.int32)
    bits = np.zeros((Bt, S), np.uint64)
    dense = np.zeros((Bt, S, S), np.uint8)
    err = lib.oracle_build_mask(_ptr(sm), _ptr(prefix_len), Bt, gamma, _ptr(tau), _ptr(sect),
                                _ptr(rope), _ptr(bits), _ptr(dense))
    return dict(tau=tau, section=sect, rope_pos=rope, mask_bits=bits, dense=dense, err=int(err))


def _as_storage(x):
    """Returns (dtype code, contiguous array of the stored bits): code 0 for
    float32 values, 1 for bfloat16 bit patterns held in uint16."""
    if x.dtype == np.float32:
        return 0, np.ascontiguousarray(x)
    if x.dtype == np.uint16:
        return 1, np.ascontiguousarray(x)
    raise TypeError(f"oracle inputs must be float32 or bf16 bits (uint16), got {x.dtype}")


def verify_attention(q, k_new, v_new, k_cache, v_cache, block_table, prefix_len, step_map,
                     gamma: int, scale: float | None = None, threads: int = 0, rope_theta: float = 0.0,
                     rope_mode: int = 1):
    """Exact masked attention of the verification forward, in fp64.

    q [Bt][2g][Hq][d]; k_new, v_new [Bt][2g][Hkv][d];
    k_cache, v_cache [num_pages][Hkv][P][d]; block_table [Bt][max_pages];
    all float32 or all bf16 bit patterns (uint16).  rope_theta > 0: q and
    k_new are rotated first (rope_mode 1: aligned RoPE copy of Sec. 3.1,
    2: physical positions of the Table 4 ablation).  Returns (out float64
    [Bt][2g][Hq][d], error bits).
    """
    lib = _load()
    dt, q = _as_storage(q)
    dts = {dt}
    dk, k_new = _as_storage(k_new)
    dv, v_new = _as_storage(v_new)
    dkc, k_cache = _as_storage(k_cache)
    dvc, v_cache = _as_storage(v_cache)
    dts |= {dk, dv, dkc, dvc}
    if len(dts) != 1:
        raise TypeError("all attention inputs must share one storage type")
    Bt, S, Hq, d = q.shape
    assert S == 2 * gamma
    Hkv = k_new.shape[2]
    num_pages, _, P, _ = k_cache.shape
    block_table = _c(block_table, np.int32)
    max_pages = block_table.shape[1]
    prefix_len = _c(prefix_len, np.int32)
    sm = None if step_map is None else _c(step_map, np.int32)
    if scale is None:
        scale = 1.0 / float(np.sqrt(d))
    out = np.zeros((Bt, S, Hq, d), np.float64)
    err = lib.oracle_verify_attention(dt, _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache),
                                      _ptr(v_cache), _ptr(block_table), max_pages, P, num_pages,
                                      _ptr(prefix_len), _ptr(sm), Bt, gamma, Hq, Hkv, d,
                                      float(scale), float(rope_theta), int(rope_mode), _ptr(out),
                                      int(threads))
    return out, int(err)


def rope_rotate(x, pos: float, theta: float):
    """The oracle's rotary embedding of the rows of x [..., d] at one
    position (rotate-half layout); returns a float64 copy."""
    lib = _load()
    a = np.array(x, dtype=np.float64, copy=True, order="C")
    d = a.shape[-1]
    lib.oracle_rope_rotate(_ptr(a), int(a.size // d), d, float(pos), float(theta))
    return a


def accept(logits, draft, gamma: int):
    """Greedy longest-prefix acceptance.

    logits float32 [Bt][gamma+1][V]; draft int32 [Bt][gamma].  Returns
    (accepted_len [Bt], out_tokens [Bt][gamma+1], row_argmax [Bt][gamma+1],
    error bits).
    """
    lib = _load()
    logits = _c(logits, np.float32)
    Bt, rows, V = logits.shape
    assert rows == gamma + 1
    draft = _c(draft, np.int32).reshape(Bt, gamma)
    a = np.zeros(Bt, np.int32)
    ot = np.zeros((Bt, gamma + 1), np.int32)
    am = np.zeros((Bt, gamma + 1), np.int32)
    err = lib.oracle_accept(_ptr(logits), _ptr(draft), Bt, gamma, V, _ptr(a), _ptr(ot), _ptr(am))
    return a, ot, am, int(err)


def accept_sampled(target_logits, draft_logits, draft, u_accept, u_sample, gamma: int, temperature: float = 1.0):
    """Stochastic acceptance, Eq. (2): accept draft r iff u_accept[r] <
    min(1, p_theta(x_r) / p_phi(x_r)); at the first rejection draw from the
    residual max(0, p_theta - p_phi), after full acceptance from
    p_theta^(gamma), by inverse CDF with u_sample.

    target_logits float32 [Bt][gamma+1][V]; draft_logits float32
    [Bt][gamma][V]; draft int32 [Bt][gamma]; u_accept float32 [Bt][gamma];
    u_sample float32 [Bt].  Returns (accepted_len, out_tokens, alpha
    [Bt][gamma] float64, margin [Bt] float64, error bits).
    """
    lib = _load()
    tl = _c(target_logits, np.float32)
    Bt, rows, V = tl.shape
    assert rows == gamma + 1
    dl = _c(draft_logits, np.float32).reshape(Bt, gamma, V)
    dr = _c(draft, np.int32).reshape(Bt, gamma)
    ua = _c(u_accept, np.float32).reshape(Bt, gamma)
    us = _c(u_sample, np.float32).reshape(Bt)
    a = np.zeros(Bt, np.int32)
    ot = np.zeros((Bt, gamma + 1), np.int32)
    al = np.zeros((Bt, gamma), np.float64)
    mg = np.zeros(Bt, np.float64)
    err = lib.oracle_accept_sampled(_ptr(tl), _ptr(dl), _ptr(dr), _ptr(ua), _ptr(us), float(temperature), Bt, gamma,
                                    V, _ptr(a), _ptr(ot), _ptr(al), _ptr(mg))
    return a, ot, al, mg, int(err)


def kv_commit(k_new, v_new, step_map, accepted_len, k_cache, v_cache, block_table, prefix_len,
              gamma: int, rope_theta: float = 0.0):
    """Appends the accepted drafts' data-slot K/V to the paged cache.

    k_new, v_new [L][Bt][2g][Hkv][d]; k_cache, v_cache [L][num_pages][Hkv][P][d]
    (float32 or bf16 bits as uint16).  rope_theta > 0: k_new is not rotated
    yet and each committed key is rotated at its position n + k.  Works on
    copies; returns (k_cache, v_cache, prefix_len, error bits).
    """
    lib = _load()
    k_new = np.ascontiguousarray(k_new)
    v_new = np.ascontiguousarray(v_new)
    kc = np.array(k_cache, copy=True, order="C")
    vc = np.array(v_cache, copy=True, order="C")
    L, Bt, S, Hkv, d = k_new.shape
    assert S == 2 * gamma and kc.dtype == k_new.dtype
    num_pages, P = kc.shape[1], kc.shape[3]
    block_table = _c(block_table, np.int32)
    n = np.array(prefix_len, dtype=np.int32, copy=True)
    a = _c(accepted_len, np.int32)
    sm = None if step_map is None else _c(step_map, np.int32)
    err = lib.oracle_kv_commit(k_new.dtype.itemsize, _ptr(k_new), _ptr(v_new), L, _ptr(sm), _ptr(a),
                               _ptr(kc), _ptr(vc), _ptr(block_table), block_table.shape[1], P,
                               num_pages, _ptr(n), Bt, gamma, Hkv, d, float(rope_theta))
    return kc, vc, n, int(err)
