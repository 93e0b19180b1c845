"""Test infrastructure: ctypes wrapper around the fp64 CPU oracle.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  The CUDA library never calls it.

Every function takes and returns numpy arrays on the host.  Inputs that the
kernels see as bf16 / fp16 are passed as their raw ``uint16`` bit patterns so
that both sides read identical values.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "optr_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboptr_oracle.so")
_lock = threading.Lock()
_lib = None

D = 128
G = 32
P = 16
CHUNK = 1536  # record bytes per (page, KV head) with G = 32


def chunk_bytes(group: int = 32) -> int:
    """Record bytes per (page, KV head): 1536 for G = 32 (four scale/min
    pairs per slot), 1152 for the compact G = 128 record (one pair)."""
    return 1152 if group == 128 else 1536


def _layout_group(pool) -> int:
    """Group size implied by a pool's record size."""
    n = pool.shape[-1]
    if n not in (1152, 1536):
        raise ValueError(f"pool record of {n} bytes: expected 1536 or 1152")
    return 128 if n == 1152 else 32


def build(force: bool = False) -> str:
    """Compile the oracle shared library in-tree (gcc, OpenMP)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fopenmp",
           "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ctypes.CDLL(build())
            _declare(_lib)
    return _lib


_P = ctypes.c_void_p


def _declare(L):
    i, f = ctypes.c_int, ctypes.c_float
    L.oracle_quantize_group.argtypes = [_P, i, f, _P, _P, _P, _P]
    L.oracle_quantize_group.restype = i
    L.oracle_kv_append.argtypes = [_P, _P, i, _P, _P, _P, i, i, _P, i, i, _P,
                                   _P, _P, f, f, _P, i]
    L.oracle_kv_append.restype = i
    L.oracle_decode_attention.argtypes = [_P, _P, _P, i, i, _P, i, i, i, _P,
                                          _P, _P, _P, _P, i, _P, i]
    L.oracle_decode_attention.restype = i
    L.oracle_decode_attention_win.argtypes = [_P, _P, _P, i, i, _P, i, i, i,
                                              _P, _P, _P, _P, _P, i, i, i, _P,
                                              _P, _P, i, _P, i]
    L.oracle_decode_attention_win.restype = i
    L.oracle_window_write.argtypes = [_P, _P, i, _P, _P, i, _P, i, i, i, i, _P]
    L.oracle_window_write.restype = i
    L.oracle_attention_dense_win.argtypes = [_P, _P, _P, i, _P, _P, _P, i, f,
                                             f, i, i, _P, _P, i]
    L.oracle_attention_dense_win.restype = i
    L.oracle_attention_dense.argtypes = [_P, _P, _P, i, _P, _P, _P, i, f, f,
                                         _P, _P]
    L.oracle_attention_dense.restype = i
    L.oracle_rotate_quantize.argtypes = [_P, _P, f, _P, _P, _P, _P, _P]
    L.oracle_rotate_quantize.restype = i
    L.oracle_rotate_quantize_g.argtypes = [_P, _P, f, _P, _P, _P, _P, _P, i]
    L.oracle_rotate_quantize_g.restype = i
    L.oracle_read_slot.argtypes = [_P, i, i, i, i, _P, _P, i]
    L.oracle_read_slot.restype = i
    L.oracle_code_byte.argtypes = [i]
    L.oracle_code_byte.restype = i
    L.oracle_code_shift.argtypes = [i]
    L.oracle_code_shift.restype = i
    L.oracle_set_threads.argtypes = [i]
    L.oracle_set_threads.restype = None
    L.oracle_get_threads.argtypes = []
    L.oracle_get_threads.restype = i


def _c(a, dtype):
    """Contiguous array of the given dtype (no copy when already right)."""
    return np.ascontiguousarray(a, dtype=dtype)


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None else None


def set_threads(n: int) -> None:
    lib().oracle_set_threads(int(n))


def get_threads() -> int:
    return int(lib().oracle_get_threads())


def quantize_group(z, clip: float = 1.0):
    """Q2 on one group (any length): returns codes, scale bits, min bits, u,
    degenerate flag."""
    z = _c(z, np.float32)
    n = z.size
    codes = np.zeros(n, np.uint8)
    u = np.zeros(n, np.float32)
    s = np.zeros(1, np.uint16)
    m = np.zeros(1, np.uint16)
    deg = lib().oracle_quantize_group(_ptr(z), n, float(clip), _ptr(codes),
                                      _ptr(s), _ptr(m), _ptr(u))
    return codes, int(s[0]), int(m[0]), u, bool(deg)


def rotate_quantize(x, R, clip: float = 1.0, group: int = 32):
    """z = x R (fp64) and its per-group quantization for one 128-vector
    (groups of ``group`` = 32 or 128 channels; scale/min per 32-channel
    block of the stored layout)."""
    x = _c(x, np.float64)
    R = _c(R, np.float32)
    z = np.zeros(D, np.float64)
    codes = np.zeros(D, np.uint8)
    s = np.zeros(4, np.uint16)
    m = np.zeros(4, np.uint16)
    u = np.zeros(D, np.float32)
    rc = lib().oracle_rotate_quantize_g(_ptr(x), _ptr(R), float(clip), _ptr(z),
                                        _ptr(codes), _ptr(s), _ptr(m), _ptr(u),
                                        int(group))
    if rc != 0:
        raise ValueError("group size must be 32 or 128")
    return z, codes, s, m, u


def kv_append(k_bits, v_bits, cu_new, pos0, block_table, pool, R_k, R_v, mu,
              clip_k=1.0, clip_v=1.0, want_u=False, group=32):
    """Oracle cache write; ``pool`` (uint8 [num_pages][h_kv][chunk_bytes(group)])
    is modified in place.  Returns the pre-rounding values when want_u."""
    k_bits = _c(k_bits, np.uint16)
    v_bits = _c(v_bits, np.uint16)
    cu_new = _c(cu_new, np.int32)
    pos0 = _c(pos0, np.int32)
    bt = _c(block_table, np.int32)
    assert pool.dtype == np.uint8 and pool.flags["C_CONTIGUOUS"]
    assert pool.shape[-1] == chunk_bytes(group), "pool record size vs group"
    n_tok, h_kv = k_bits.shape[0], k_bits.shape[1]
    B = pos0.size
    max_pages = bt.shape[1]
    num_pages = pool.shape[0]
    u = np.zeros((n_tok, h_kv, 2, D), np.float32) if want_u else None
    rc = lib().oracle_kv_append(
        _ptr(k_bits), _ptr(v_bits), n_tok, _ptr(cu_new), _ptr(pos0), _ptr(bt),
        B, max_pages, _ptr(pool), num_pages, h_kv, _ptr(_c(R_k, np.float32)),
        _ptr(_c(R_v, np.float32)), _ptr(_c(mu, np.float32)), float(clip_k),
        float(clip_v), _ptr(u), int(group))
    if rc != 0:
        raise ValueError("oracle_kv_append: table entry or position out of range"
                         " (or group size not 32 / 128)")
    return u


def decode_attention(q_bits, block_table, seq_lens, pool, R_k, R_v, h_kv,
                     rows=None, want_p=False, win=None, win_slot=None, sink=0,
                     recent=0, mu=None):
    """Oracle decode (the pool's record size selects its layout: 1536 bytes
    for G = 32, 1152 for G = 128).  Returns float64 [B][h_q][128]; when ``rows`` (a list of
    (b, j)) is given only those rows are computed (others stay zero).  With
    ``sink`` / ``recent`` > 0 the BF16 window positions are read from ``win``
    (uint16 bf16 bits [n_slots][h_kv][2][sink + recent][128]) at the slots
    ``win_slot`` [B], and ``mu`` (float32 [h_kv][128]) centers their keys."""
    q_bits = _c(q_bits, np.uint16)
    bt = _c(block_table, np.int32)
    sl = _c(seq_lens, np.int32)
    B, h_q = q_bits.shape[0], q_bits.shape[1]
    out = np.zeros((B, h_q, D), np.float64)
    if rows:
        sb = np.array([r[0] for r in rows], np.int32)
        sj = np.array([r[1] for r in rows], np.int32)
        n_sel = len(rows)
    else:
        sb = sj = None
        n_sel = 0
    p = None
    if want_p:
        assert n_sel == 1
        p = np.zeros(int(sl[rows[0][0]]), np.float64)
    windows = sink > 0 or recent > 0
    if windows:
        win = _c(win, np.uint16)
        assert win.shape[1:] == (h_kv, 2, sink + recent, D)
        win_slot = _c(win_slot, np.int32)
        mu = _c(mu, np.float32)
        n_slots = win.shape[0]
    else:
        win = win_slot = mu = None
        n_slots = 0
    rc = lib().oracle_decode_attention_win(
        _ptr(q_bits), _ptr(bt), _ptr(sl), B, bt.shape[1], _ptr(pool),
        pool.shape[0], h_q, h_kv, _ptr(_c(R_k, np.float32)),
        _ptr(_c(R_v, np.float32)), _ptr(mu), _ptr(win), _ptr(win_slot),
        n_slots, int(sink), int(recent), _ptr(out), _ptr(sb), _ptr(sj), n_sel,
        _ptr(p), _layout_group(pool))
    if rc != 0:
        raise ValueError("oracle_decode_attention: table entry or window slot out of range")
    return (out, p) if want_p else out


def new_windows(n_slots, h_kv, sink, recent):
    """Zeroed window store (bf16 bits) for n_slots sequences."""
    return np.zeros((n_slots, h_kv, 2, sink + recent, D), np.uint16)


def window_write(k_bits, v_bits, cu_new, pos0, win, win_slot, sink, recent):
    """Window part of the oracle cache write; ``win`` is modified in place."""
    k_bits = _c(k_bits, np.uint16)
    v_bits = _c(v_bits, np.uint16)
    cu_new = _c(cu_new, np.int32)
    pos0 = _c(pos0, np.int32)
    win_slot = _c(win_slot, np.int32)
    assert win.dtype == np.uint16 and win.flags["C_CONTIGUOUS"]
    n_tok, h_kv = k_bits.shape[0], k_bits.shape[1]
    assert win.shape[1:] == (h_kv, 2, sink + recent, D)
    rc = lib().oracle_window_write(
        _ptr(k_bits), _ptr(v_bits), n_tok, _ptr(cu_new), _ptr(pos0), pos0.size,
        _ptr(win_slot), win.shape[0], h_kv, int(sink), int(recent), _ptr(win))
    if rc != 0:
        raise ValueError("oracle_window_write: window slot out of range")


def attention_dense(q, K, V, R_k, R_v, mu, quantize=True, clip_k=1.0,
                    clip_v=1.0, want_p=False, sink=0, recent=0, group=32):
    """Single-head dense statement in the inverse-rotation form; positions
    s < sink or s >= n - recent are BF16 window positions."""
    q = _c(q, np.float64)
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    n = K.shape[0]
    out = np.zeros(D, np.float64)
    p = np.zeros(max(n, 1), np.float64) if want_p else None
    lib().oracle_attention_dense_win(_ptr(q), _ptr(K), _ptr(V), n,
                                     _ptr(_c(R_k, np.float32)),
                                     _ptr(_c(R_v, np.float32)),
                                     _ptr(_c(mu, np.float64)),
                                     int(bool(quantize)), float(clip_k),
                                     float(clip_v), int(sink), int(recent),
                                     _ptr(out), _ptr(p), int(group))
    return (out, p[:n]) if want_p else out


def read_slot(pool, page, h, slot):
    """Dequantized rotated (khat, vhat) of one cache slot."""
    kh = np.zeros(D, np.float64)
    vh = np.zeros(D, np.float64)
    lib().oracle_read_slot(_ptr(pool), pool.shape[1], int(page), int(h),
                           int(slot), _ptr(kh), _ptr(vh), _layout_group(pool))
    return kh, vh


def code_byte(ch: int) -> int:
    return int(lib().oracle_code_byte(int(ch)))


def code_shift(ch: int) -> int:
    return int(lib().oracle_code_shift(int(ch)))
