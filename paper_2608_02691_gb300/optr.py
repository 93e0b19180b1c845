"""Thin ctypes binding of the C ABI in ``include/optr.h``.

Function names match the C entry points.  The binding only marshals
arguments: torch tensors become raw device pointers, the current torch CUDA
stream becomes the ``cudaStream_t``, and negative status codes raise
``OptrError``.  Every step of the computation runs in ``liboptr.so``; if the
library has not been built, the first call raises instead of falling back to
anything else.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

_lib = None
_lock = threading.Lock()

OPTR_VARIANT_DEFAULT = 0
OPTR_VARIANT_CUDA_CORE = 1
OPTR_VARIANT_TENSOR = 2
PAGE_HEAD_BYTES = 1536       # record bytes per (page, KV head), G = 32
PAGE_HEAD_BYTES_G128 = 1152  # the compact G = 128 record
HEAD_DIM = 128
# device error bits (optr_device_error)
OPTR_DEVERR_PAGE_ID = 1
OPTR_DEVERR_POSITION = 2
OPTR_DEVERR_SEQ_LEN = 4
OPTR_DEVERR_CU_NEW = 8
OPTR_DEVERR_FP16_RANGE = 16
OPTR_DEVERR_TIMEOUT = 32
OPTR_DEVERR_WIN_SLOT = 64


class OptrError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {optr_strerror(status)} (status {status})")
        self.status = status


class optr_config(ctypes.Structure):
    _fields_ = [("h_q", ctypes.c_int), ("h_kv", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("group", ctypes.c_int),
                ("page_size", ctypes.c_int), ("clip_k", ctypes.c_float),
                ("clip_v", ctypes.c_float), ("append_variant", ctypes.c_int),
                ("decode_variant", ctypes.c_int), ("sink", ctypes.c_int),
                ("recent", ctypes.c_int)]


class optr_calib_config(ctypes.Structure):
    _fields_ = [("g", ctypes.c_int), ("d_model", ctypes.c_int),
                ("T", ctypes.c_int), ("nt", ctypes.c_int),
                ("T_held", ctypes.c_int), ("nt_held", ctypes.c_int),
                ("steps", ctypes.c_int), ("select_every", ctypes.c_int),
                ("group", ctypes.c_int), ("sink", ctypes.c_int),
                ("recent", ctypes.c_int), ("lr", ctypes.c_double),
                ("lam", ctypes.c_double), ("clip_k", ctypes.c_double),
                ("clip_v", ctypes.c_double)]


_V = ctypes.c_void_p
_I = ctypes.c_int
_SIG = {
    "optr_params_create": (_I, [ctypes.POINTER(optr_config), _V, _V, _V,
                                ctypes.POINTER(_V)]),
    "optr_params_destroy": (None, [_V]),
    "optr_page_bytes": (ctypes.c_size_t, [_V]),
    "optr_kv_append": (_I, [_V, _V, _V, _I, _V, _V, _V, _I, _I, _V, _I, _V]),
    "optr_decode_workspace_size": (ctypes.c_size_t, [_V, _I, _I]),
    "optr_decode_attention": (_I, [_V, _V, _V, _V, _I, _I, _V, _I, _V, _V,
                                   ctypes.c_size_t, _V]),
    "optr_device_error": (_I, [_V, ctypes.POINTER(ctypes.c_uint32)]),
    "optr_strerror": (ctypes.c_char_p, [_I]),
    "optr_selftest_wait_timeout": (_I, [_V, ctypes.c_ulonglong, _V]),
    "optr_calib_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(optr_calib_config)]),
    "optr_calibrate_head": (_I, [ctypes.POINTER(optr_calib_config)] + [_V] * 17
                            + [ctypes.c_size_t, _V]),
    "optr_calib_loss_grad": (_I, [ctypes.POINTER(optr_calib_config), _I] + [_V] * 12
                             + [ctypes.c_size_t, _V]),
    "optr_decode_attention_noalloc": (_I, [_V, _V, _V, _V, _I, _I, _V, _I,
                                           _V, _V]),
    "optr_decode_step": (_I, [_V, _V, _V, _V, _I, _V, _V, _V, _V, _I, _I, _V,
                              _I, _V, _V, ctypes.c_size_t, _V]),
    "optr_window_bytes": (ctypes.c_size_t, [_V, _I]),
    "optr_kv_append_win": (_I, [_V, _V, _V, _I, _V, _V, _V, _I, _I, _V, _I,
                                _V, _V, _I, _V]),
    "optr_decode_attention_win": (_I, [_V, _V, _V, _V, _I, _I, _V, _I, _V,
                                       _V, _I, _V, _V, ctypes.c_size_t, _V]),
    "optr_decode_step_win": (_I, [_V, _V, _V, _V, _I, _V, _V, _V, _V, _I, _I,
                                  _V, _I, _V, _V, _I, _V, _V, ctypes.c_size_t,
                                  _V]),
    "optr_profile_enable": (_I, [_V, _I]),
    "optr_profile_last": (_I, [_V, ctypes.POINTER(ctypes.c_float)]),
}


def library_path() -> str:
    return _build.LIB


def lib():
    """The loaded ``liboptr.so``; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(
                    f"{path} is missing: build the CUDA library first "
                    "(python -c 'import __graft_entry__ as g; g.build()')")
            L = ctypes.CDLL(path)
            for name, (res, args) in _SIG.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def optr_strerror(status: int) -> str:
    return lib().optr_strerror(int(status)).decode()


def _check(status: int, what: str):
    if status != 0:
        raise OptrError(status, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


# per-step activations: CUDA tensors or pinned host tensors, which the
# kernels read or write in place
_IO = ("q", "k", "v", "out")


def _dev(t, dtype, name):
    where = t.is_cuda or (name in _IO and t.is_pinned())
    if not (where and t.dtype == dtype and t.is_contiguous()):
        kind = "CUDA or pinned host" if name in _IO else "CUDA"
        raise ValueError(f"{name} must be a contiguous {kind} {dtype} tensor")
    return t


class Params:
    """Owner of an ``optr_params*`` handle (destroyed with the object)."""

    def __init__(self, handle, cfg: optr_config):
        self.handle = handle
        self.cfg = cfg

    def __del__(self):
        h, self.handle = getattr(self, "handle", None), None
        if h and _lib is not None:
            _lib.optr_params_destroy(h)

    @property
    def h_q(self):
        return self.cfg.h_q

    @property
    def h_kv(self):
        return self.cfg.h_kv


def optr_params_create(R_k, R_v, mu, h_q: int, clip_k: float = 1.0,
                       clip_v: float = 1.0,
                       append_variant: int = OPTR_VARIANT_DEFAULT,
                       decode_variant: int = OPTR_VARIANT_DEFAULT,
                       sink: int = 0, recent: int = 0,
                       group: int = 32) -> Params:
    """R_k, R_v float32 [h_kv][128][128] and mu float32 [h_kv][128] (host
    tensors); the library copies them to the current CUDA device.  R_v may be
    None: the value rotation is folded into the model's W_V / W_O.  sink /
    recent > 0 keep BF16 windows (the *_win calls); group is the Q2 group
    size (32, or the paper's 128)."""
    R_k = R_k.detach().to("cpu", torch.float32).contiguous()
    if R_v is not None:
        R_v = R_v.detach().to("cpu", torch.float32).contiguous()
    mu = mu.detach().to("cpu", torch.float32).contiguous()
    h_kv = R_k.shape[0]
    if R_k.shape != (h_kv, 128, 128) or (R_v is not None and R_v.shape != R_k.shape) or \
            mu.shape != (h_kv, 128):
        raise ValueError("R_k, R_v must be [h_kv][128][128], mu [h_kv][128]")
    cfg = optr_config(h_q, h_kv, 128, group, 16, clip_k, clip_v, append_variant,
                      decode_variant, sink, recent)
    h = ctypes.c_void_p()
    _check(lib().optr_params_create(ctypes.byref(cfg), _ptr(R_k),
                                    None if R_v is None else _ptr(R_v),
                                    _ptr(mu), ctypes.byref(h)),
           "optr_params_create")
    return Params(h, cfg)


def optr_page_bytes(p: Params) -> int:
    return int(lib().optr_page_bytes(p.handle))


def optr_kv_append(p: Params, k, v, cu_new, pos0, block_table, pool,
                   stream=None) -> None:
    """k, v bf16 [n_tok][h_kv][128]; cu_new int32 [B+1]; pos0 int32 [B];
    block_table int32 [B][max_pages]; pool uint8 [num_pages][h_kv][1536]."""
    _dev(k, torch.bfloat16, "k")
    _dev(v, torch.bfloat16, "v")
    _dev(cu_new, torch.int32, "cu_new")
    _dev(pos0, torch.int32, "pos0")
    _dev(block_table, torch.int32, "block_table")
    _dev(pool, torch.uint8, "pool")
    B, max_pages = block_table.shape
    _check(lib().optr_kv_append(p.handle, _ptr(k), _ptr(v), k.shape[0],
                                _ptr(cu_new), _ptr(pos0), _ptr(block_table),
                                B, max_pages, _ptr(pool), pool.shape[0],
                                _stream(stream)),
           "optr_kv_append")


def optr_decode_workspace_size(p: Params, B: int, max_pages: int) -> int:
    return int(lib().optr_decode_workspace_size(p.handle, B, max_pages))


def optr_decode_attention(p: Params, q, block_table, seq_lens, pool, out,
                          workspace, stream=None) -> None:
    """q bf16 [B][h_q][128]; out float32 [B][h_q][128]; workspace uint8 of
    at least optr_decode_workspace_size bytes (256-byte aligned)."""
    _dev(q, torch.bfloat16, "q")
    _dev(block_table, torch.int32, "block_table")
    _dev(seq_lens, torch.int32, "seq_lens")
    _dev(pool, torch.uint8, "pool")
    _dev(out, torch.float32, "out")
    _dev(workspace, torch.uint8, "workspace")
    B, max_pages = block_table.shape
    _check(lib().optr_decode_attention(
        p.handle, _ptr(q), _ptr(block_table), _ptr(seq_lens), B, max_pages,
        _ptr(pool), pool.shape[0], _ptr(out), _ptr(workspace),
        workspace.numel(), _stream(stream)), "optr_decode_attention")


def optr_decode_step(p: Params, q, k, v, cu_new, pos0, block_table, seq_lens,
                     pool, out, workspace, stream=None) -> None:
    """optr_kv_append of the step's new tokens (k, v, cu_new, pos0) followed
    by optr_decode_attention over the updated cache; seq_lens counts the new
    tokens."""
    for t, dt, nm in ((q, torch.bfloat16, "q"), (k, torch.bfloat16, "k"),
                      (v, torch.bfloat16, "v"), (cu_new, torch.int32, "cu_new"),
                      (pos0, torch.int32, "pos0"),
                      (block_table, torch.int32, "block_table"),
                      (seq_lens, torch.int32, "seq_lens"),
                      (pool, torch.uint8, "pool"), (out, torch.float32, "out"),
                      (workspace, torch.uint8, "workspace")):
        _dev(t, dt, nm)
    B, max_pages = block_table.shape
    _check(lib().optr_decode_step(
        p.handle, _ptr(q), _ptr(k), _ptr(v), k.shape[0], _ptr(cu_new),
        _ptr(pos0), _ptr(block_table), _ptr(seq_lens), B, max_pages,
        _ptr(pool), pool.shape[0], _ptr(out), _ptr(workspace),
        workspace.numel(), _stream(stream)), "optr_decode_step")


def optr_window_bytes(p: Params, n_slots: int) -> int:
    return int(lib().optr_window_bytes(p.handle, n_slots))


def _win_args(p, win, win_slot):
    if win is None:
        return None, None, 0
    _dev(win, torch.bfloat16, "win")
    _dev(win_slot, torch.int32, "win_slot")
    rows = p.cfg.sink + p.cfg.recent
    if tuple(win.shape[1:]) != (p.h_kv, 2, rows, 128):
        raise ValueError("win must be [n_slots][h_kv][2][sink + recent][128]")
    return _ptr(win), _ptr(win_slot), win.shape[0]


def optr_kv_append_win(p: Params, k, v, cu_new, pos0, block_table, pool, win,
                       win_slot, stream=None) -> None:
    """optr_kv_append plus the BF16-window copy: win bf16
    [n_slots][h_kv][2][sink + recent][128], win_slot int32 [B]."""
    for t, dt, nm in ((k, torch.bfloat16, "k"), (v, torch.bfloat16, "v"),
                      (cu_new, torch.int32, "cu_new"), (pos0, torch.int32, "pos0"),
                      (block_table, torch.int32, "block_table"),
                      (pool, torch.uint8, "pool")):
        _dev(t, dt, nm)
    w, ws_, n_slots = _win_args(p, win, win_slot)
    B, max_pages = block_table.shape
    _check(lib().optr_kv_append_win(
        p.handle, _ptr(k), _ptr(v), k.shape[0], _ptr(cu_new), _ptr(pos0),
        _ptr(block_table), B, max_pages, _ptr(pool), pool.shape[0], w, ws_,
        n_slots, _stream(stream)), "optr_kv_append_win")


def optr_decode_attention_win(p: Params, q, block_table, seq_lens, pool, win,
                              win_slot, out, workspace, stream=None) -> None:
    """optr_decode_attention with the BF16 windows read from win."""
    for t, dt, nm in ((q, torch.bfloat16, "q"),
                      (block_table, torch.int32, "block_table"),
                      (seq_lens, torch.int32, "seq_lens"),
                      (pool, torch.uint8, "pool"), (out, torch.float32, "out"),
                      (workspace, torch.uint8, "workspace")):
        _dev(t, dt, nm)
    w, ws_, n_slots = _win_args(p, win, win_slot)
    B, max_pages = block_table.shape
    _check(lib().optr_decode_attention_win(
        p.handle, _ptr(q), _ptr(block_table), _ptr(seq_lens), B, max_pages,
        _ptr(pool), pool.shape[0], w, ws_, n_slots, _ptr(out), _ptr(workspace),
        workspace.numel(), _stream(stream)), "optr_decode_attention_win")


def optr_decode_step_win(p: Params, q, k, v, cu_new, pos0, block_table,
                         seq_lens, pool, win, win_slot, out, workspace,
                         stream=None) -> None:
    """optr_decode_step with BF16 windows: the step's window copies and the
    windowed decode."""
    for t, dt, nm in ((q, torch.bfloat16, "q"), (k, torch.bfloat16, "k"),
                      (v, torch.bfloat16, "v"), (cu_new, torch.int32, "cu_new"),
                      (pos0, torch.int32, "pos0"),
                      (block_table, torch.int32, "block_table"),
                      (seq_lens, torch.int32, "seq_lens"),
                      (pool, torch.uint8, "pool"), (out, torch.float32, "out"),
                      (workspace, torch.uint8, "workspace")):
        _dev(t, dt, nm)
    w, ws_, n_slots = _win_args(p, win, win_slot)
    B, max_pages = block_table.shape
    _check(lib().optr_decode_step_win(
        p.handle, _ptr(q), _ptr(k), _ptr(v), k.shape[0], _ptr(cu_new),
        _ptr(pos0), _ptr(block_table), _ptr(seq_lens), B, max_pages,
        _ptr(pool), pool.shape[0], w, ws_, n_slots, _ptr(out), _ptr(workspace),
        workspace.numel(), _stream(stream)), "optr_decode_step_win")


def new_windows(p: Params, n_slots: int, device="cuda") -> torch.Tensor:
    """A zero-filled window store [n_slots][h_kv][2][sink + recent][128]
    (bf16)."""
    return torch.zeros(n_slots, p.h_kv, 2, p.cfg.sink + p.cfg.recent, 128,
                       dtype=torch.bfloat16, device=device)


NOALLOC_SCRATCH_BYTES = 16 << 20


def optr_decode_attention_noalloc(p: Params, q, block_table, seq_lens, pool,
                                  out, stream=None) -> None:
    """Decode without a workspace argument: the library uses its own fixed
    16 MiB device scratch array, so this call allocates nothing.  Calls
    that overlap on the GPU share that array and must be serialised."""
    _dev(q, torch.bfloat16, "q")
    _dev(block_table, torch.int32, "block_table")
    _dev(seq_lens, torch.int32, "seq_lens")
    _dev(pool, torch.uint8, "pool")
    _dev(out, torch.float32, "out")
    B, max_pages = block_table.shape
    _check(lib().optr_decode_attention_noalloc(
        p.handle, _ptr(q), _ptr(block_table), _ptr(seq_lens), B, max_pages,
        _ptr(pool), pool.shape[0], _ptr(out), _stream(stream)),
        "optr_decode_attention_noalloc")


def optr_device_error(p: Params) -> int:
    flags = ctypes.c_uint32(0)
    _check(lib().optr_device_error(p.handle, ctypes.byref(flags)),
           "optr_device_error")
    return int(flags.value)


def optr_selftest_wait_timeout(p: Params, limit_ns: int, stream=None) -> None:
    """Launch the bounded-wait self-test (see include/optr.h); the timeout
    shows up in optr_device_error."""
    _check(lib().optr_selftest_wait_timeout(p.handle, int(limit_ns),
                                            _stream(stream)),
           "optr_selftest_wait_timeout")


def optr_profile_enable(p: Params, on: bool = True) -> None:
    _check(lib().optr_profile_enable(p.handle, int(bool(on))),
           "optr_profile_enable")


def optr_profile_last(p: Params) -> dict:
    """Durations (ms) of the stages of the most recent append / decode."""
    ms = (ctypes.c_float * 4)()
    _check(lib().optr_profile_last(p.handle, ms), "optr_profile_last")
    return {"append": ms[0], "qrot": ms[1], "partial": ms[2], "combine": ms[3]}


def new_pool(p: Params, num_pages: int, device="cuda") -> torch.Tensor:
    """A zero-filled pool tensor [num_pages][h_kv][record bytes] (uint8):
    1536 bytes per (page, KV head) for G = 32, 1152 for G = 128."""
    rec = PAGE_HEAD_BYTES_G128 if p.cfg.group == 128 else PAGE_HEAD_BYTES
    return torch.zeros(num_pages, p.h_kv, rec, dtype=torch.uint8, device=device)


def new_workspace(p: Params, B: int, max_pages: int, device="cuda"):
    n = optr_decode_workspace_size(p, B, max_pages)
    return torch.empty(n, dtype=torch.uint8, device=device)


# ------------------------------------------------------------ calibration

def calib_config(g, d_model, T, nt, T_held=0, nt_held=0, steps=80,
                 select_every=20, group=32, sink=0, recent=0, lr=0.02, lam=1.0,
                 clip_k=1.0, clip_v=1.0) -> optr_calib_config:
    return optr_calib_config(g, d_model, T, nt, T_held, nt_held, steps,
                             select_every, group, sink, recent, lr, lam, clip_k,
                             clip_v)


def optr_calib_workspace_size(cfg: optr_calib_config) -> int:
    return int(lib().optr_calib_workspace_size(ctypes.byref(cfg)))


def _calib_ws(cfg, device):
    n = optr_calib_workspace_size(cfg)
    if n == 0:
        raise OptrError(-1, "optr_calib_workspace_size")
    return torch.empty(n, dtype=torch.uint8, device=device)


def optr_calibrate_head(cfg: optr_calib_config, q, K, V, t_pos, W_O,
                        held=None, R0_K=None, R0_V=None, stream=None):
    """One KV head's calibration (see include/optr.h).  q [nt][g][128],
    K, V [T][128], W_O [g][d_model][128] float64 CUDA tensors, t_pos int32;
    held = (q, K, V, t_pos) of the held-out trace or None.  Returns R_K,
    R_V, mu, hist_k, hist_v (CUDA float64)."""
    dev = K.device
    d = 128
    R_K = torch.empty(d, d, dtype=torch.float64, device=dev)
    R_V = torch.empty_like(R_K)
    mu = torch.empty(d, dtype=torch.float64, device=dev)
    hk = torch.empty(max(cfg.steps, 1), dtype=torch.float64, device=dev)
    hv = torch.empty_like(hk)
    ws = _calib_ws(cfg, dev)
    h = held if held is not None else (None, None, None, None)
    _check(lib().optr_calibrate_head(
        ctypes.byref(cfg), _ptr(q), _ptr(K), _ptr(V), _ptr(t_pos), _ptr(W_O),
        _ptr(h[0]), _ptr(h[1]), _ptr(h[2]), _ptr(h[3]), _ptr(R0_K), _ptr(R0_V),
        _ptr(R_K), _ptr(R_V), _ptr(mu), _ptr(hk), _ptr(hv), _ptr(ws),
        ws.numel(), _stream(stream)), "optr_calibrate_head")
    return R_K, R_V, mu, hk[:cfg.steps], hv[:cfg.steps]


def optr_calib_loss_grad(cfg: optr_calib_config, which: int, q, K, V, t_pos,
                         W_O, mu, R0, A, R_K=None, grad=True, stream=None):
    """L_K (which 0) or L_V (which 1) at R = R0 exp(A - A^T) and its
    gradient with respect to A (None when grad is False)."""
    dev = K.device
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    dA = torch.empty(128, 128, dtype=torch.float64, device=dev) if grad else None
    ws = _calib_ws(cfg, dev)
    _check(lib().optr_calib_loss_grad(
        ctypes.byref(cfg), int(which), _ptr(q), _ptr(K), _ptr(V), _ptr(t_pos),
        _ptr(W_O), _ptr(mu), _ptr(R_K), _ptr(R0), _ptr(A), _ptr(loss), _ptr(dA),
        _ptr(ws), ws.numel(), _stream(stream)), "optr_calib_loss_grad")
    return loss, dA
