"""ctypes binding of libdard.so: argument marshalling only.

Each function takes torch CUDA tensors for device data and NumPy / Python integer
sequences for the per-sequence host metadata, fills the C argument struct declared in
``include/dard.h`` and calls the library entry point of the same name on the current torch
stream (or the given one). Every step of the computation runs in the library's CUDA
kernels; there is no fallback: a missing library raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdard.so")

DARD_F32, DARD_BF16 = 0, 1
ORDER_CONFIDENCE, ORDER_BIDIR, ORDER_L2R, ORDER_ENTROPY, ORDER_MARGIN = 0, 1, 2, 3, 4
STATUS_BAD_STATE, STATUS_BAD_SHADOW, STATUS_INVALID_ROW, STATUS_TIMEOUT = 0x1, 0x2, 0x4, 0x8
MAX_SEQS, MAX_BLOCK = 256, 128
SCORE_NOALLOC_MAX_ROWS = 8192

_I32P = ctypes.POINTER(ctypes.c_int32)


class AttnArgs(ctypes.Structure):
    _fields_ = [("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("o", ctypes.c_void_p), ("dtype", ctypes.c_int32), ("hq", ctypes.c_int32),
                ("hkv", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("num_seqs", ctypes.c_int32), ("n_orig", _I32P), ("block_start", _I32P),
                ("block_len", _I32P), ("shadow_len", _I32P), ("state", ctypes.c_void_p),
                ("prev_conf", ctypes.c_void_p), ("shadow_src", ctypes.c_void_p),
                ("scale", ctypes.c_float), ("status", ctypes.c_void_p),
                ("query_start", _I32P)]


class ScoreArgs(ctypes.Structure):
    _fields_ = [("logits_x", ctypes.c_void_p), ("logits_s", ctypes.c_void_p),
                ("dtype", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("row_stride", ctypes.c_int64), ("num_seqs", ctypes.c_int32),
                ("block_len", _I32P), ("state_in", ctypes.c_void_p),
                ("tau_c", ctypes.c_float), ("tau_u", ctypes.c_float),
                ("lambda_", ctypes.c_float), ("p0", ctypes.c_float),
                ("conf", ctypes.c_void_p), ("token", ctypes.c_void_p),
                ("state_out", ctypes.c_void_p), ("w_out", ctypes.c_void_p),
                ("counts", ctypes.c_void_p), ("status", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
                ("cur_token", ctypes.c_void_p), ("p_cur", ctypes.c_void_p),
                ("tokens", ctypes.c_void_p), ("mask_token", ctypes.c_int32),
                ("entropy", ctypes.c_void_p), ("margin", ctypes.c_void_p),
                ("order_key", ctypes.c_void_p), ("order_mode", ctypes.c_int32)]


class DardError(RuntimeError):
    def __init__(self, code: int, fn: str, message: str):
        super().__init__(f"{fn} failed: {status_string(code)}: {message}")
        self.code = code


_lib = None

# Exported entry points: name -> (restype, argtypes)
EXPORTS = {
    "dard_step_attention": (ctypes.c_int, [ctypes.POINTER(AttnArgs), ctypes.c_void_p]),
    "dard_score_and_transition": (ctypes.c_int, [ctypes.POINTER(ScoreArgs), ctypes.c_void_p]),
    "dard_score_and_transition_noalloc": (ctypes.c_int, [ctypes.POINTER(ScoreArgs),
                                                         ctypes.c_void_p]),
    "dard_score_workspace_size": (ctypes.c_size_t, [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]),
    "dard_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "dard_last_error": (ctypes.c_char_p, []),
    "dard_version": (ctypes.c_int32, []),
}


def lib(path: str | None = None) -> ctypes.CDLL:
    """Loads libdard.so once; raises if it has not been built."""
    global _lib
    if _lib is None:
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build it with paper_2608_26574_gb300.build.build()")
        L = ctypes.CDLL(p)
        for name, (res, args) in EXPORTS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def status_string(code: int) -> str:
    return lib().dard_status_string(code).decode()


def _check(code: int, fn: str):
    if code != 0:
        raise DardError(code, fn, lib().dard_last_error().decode())


def _ptr(t) -> int | None:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("device tensor expected")
    if not t.is_contiguous():
        raise ValueError("contiguous tensor expected")
    return t.data_ptr()


def _rows_ptr(t) -> int:
    """Device pointer of a 2-D tensor whose rows are contiguous (any row pitch)."""
    if not t.is_cuda:
        raise ValueError("device tensor expected")
    if t.dim() != 2 or (t.numel() > 0 and t.stride(1) != 1):
        raise ValueError("2-D tensor with contiguous rows expected")
    return t.data_ptr()


def _row_pitch(t) -> int:
    """Elements between rows (an empty tensor has no rows to step over: its width)."""
    return t.stride(0) if t.numel() > 0 else t.shape[1]


def _host_i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _stream(stream) -> int:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return DARD_BF16
    if t.dtype == torch.float32:
        return DARD_F32
    raise ValueError(f"unsupported dtype {t.dtype}")


def dard_step_attention(q, k, v, o, n_orig, block_start, block_len, shadow_len, state,
                        prev_conf, shadow_src, scale: float = 0.0, status=None, stream=None,
                        query_start=None):
    """Masked attention of one layer; q/o [rows, hq, d], k/v [rows, hkv, d] on the device.
    ``query_start`` (per sequence, optional): first query row; earlier rows are keys only."""
    n_orig, block_start = _host_i32(n_orig), _host_i32(block_start)
    qs = _host_i32(query_start) if query_start is not None else None
    block_len, shadow_len = _host_i32(block_len), _host_i32(shadow_len)
    a = AttnArgs()
    a.q, a.k, a.v, a.o = _ptr(q), _ptr(k), _ptr(v), _ptr(o)
    a.dtype = _dtype_code(q)
    a.hq, a.hkv, a.head_dim = q.shape[1], k.shape[1], q.shape[2]
    a.num_seqs = len(n_orig)
    a.n_orig = n_orig.ctypes.data_as(_I32P)
    a.block_start = block_start.ctypes.data_as(_I32P)
    a.block_len = block_len.ctypes.data_as(_I32P)
    a.shadow_len = shadow_len.ctypes.data_as(_I32P)
    a.state, a.prev_conf, a.shadow_src = _ptr(state), _ptr(prev_conf), _ptr(shadow_src)
    a.scale = scale
    a.status = _ptr(status)
    a.query_start = qs.ctypes.data_as(_I32P) if qs is not None else None
    _check(lib().dard_step_attention(ctypes.byref(a), _stream(stream)), "dard_step_attention")


def dard_score_workspace_size(rows: int, vocab: int, num_seqs: int) -> int:
    return int(lib().dard_score_workspace_size(rows, vocab, num_seqs))


def dard_score_and_transition(logits_x, logits_s, block_len, state_in, tau_c, tau_u, lam, p0,
                              conf, token, state_out, workspace, w_out=None, counts=None,
                              status=None, stream=None, cur_token=None, p_cur=None,
                              tokens=None, mask_token: int = 0, entropy=None, margin=None,
                              order_key=None, order_mode: int = ORDER_CONFIDENCE):
    """Scoring and transition of every block row; logits [rows, V] with contiguous rows and
    the same row pitch (``stride(0)``, at least V) in both tensors. Optional end of step:
    ``p_cur`` of ``cur_token``, and ``tokens`` (x^, or ``mask_token`` for rows ending in M);
    ``entropy``, ``margin`` and the next step's ``order_key`` for ``order_mode``."""
    block_len = _host_i32(block_len)
    if _row_pitch(logits_x) != _row_pitch(logits_s) or logits_x.shape != logits_s.shape:
        raise ValueError("logits_x and logits_s need the same shape and row pitch")
    a = ScoreArgs()
    a.logits_x, a.logits_s = _rows_ptr(logits_x), _rows_ptr(logits_s)
    a.dtype = _dtype_code(logits_s)
    a.vocab = logits_s.shape[1]
    a.row_stride = _row_pitch(logits_s)
    a.num_seqs = len(block_len)
    a.block_len = block_len.ctypes.data_as(_I32P)
    a.state_in = _ptr(state_in)
    a.tau_c, a.tau_u, a.lambda_, a.p0 = tau_c, tau_u, lam, p0
    a.conf, a.token, a.state_out = _ptr(conf), _ptr(token), _ptr(state_out)
    a.w_out, a.counts, a.status = _ptr(w_out), _ptr(counts), _ptr(status)
    a.workspace = _ptr(workspace)
    a.workspace_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    a.cur_token, a.p_cur, a.tokens = _ptr(cur_token), _ptr(p_cur), _ptr(tokens)
    a.mask_token = mask_token
    a.entropy, a.margin, a.order_key = _ptr(entropy), _ptr(margin), _ptr(order_key)
    a.order_mode = order_mode
    _check(lib().dard_score_and_transition(ctypes.byref(a), _stream(stream)),
           "dard_score_and_transition")


def dard_score_and_transition_noalloc(logits_x, logits_s, block_len, state_in, tau_c, tau_u,
                                      lam, p0, conf, token, state_out, w_out=None, counts=None,
                                      status=None, stream=None):
    """``dard_score_and_transition`` without a workspace: the library's built-in scratch
    (at most ``SCORE_NOALLOC_MAX_ROWS`` block rows; calls that overlap on one device race)."""
    block_len = _host_i32(block_len)
    if _row_pitch(logits_x) != _row_pitch(logits_s) or logits_x.shape != logits_s.shape:
        raise ValueError("logits_x and logits_s need the same shape and row pitch")
    a = ScoreArgs()
    a.logits_x, a.logits_s = _rows_ptr(logits_x), _rows_ptr(logits_s)
    a.dtype = _dtype_code(logits_s)
    a.vocab = logits_s.shape[1]
    a.row_stride = _row_pitch(logits_s)
    a.num_seqs = len(block_len)
    a.block_len = block_len.ctypes.data_as(_I32P)
    a.state_in = _ptr(state_in)
    a.tau_c, a.tau_u, a.lambda_, a.p0 = tau_c, tau_u, lam, p0
    a.conf, a.token, a.state_out = _ptr(conf), _ptr(token), _ptr(state_out)
    a.w_out, a.counts, a.status = _ptr(w_out), _ptr(counts), _ptr(status)
    _check(lib().dard_score_and_transition_noalloc(ctypes.byref(a), _stream(stream)),
           "dard_score_and_transition_noalloc")
