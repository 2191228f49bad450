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
                ("query_start", _I32P), ("rope_theta", ctypes.c_float),
                ("rope_style", ctypes.c_int32), ("k_rope", ctypes.c_void_p)]

DARD_ROPE_INTERLEAVED, DARD_ROPE_HALF = 0, 1


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

class AttnPlan(ctypes.Structure):
    _fields_ = [("kernel", ctypes.c_int32), ("ctas", ctypes.c_int64),
                ("tile_pairs", ctypes.c_int64), ("tile_pairs_skipped", ctypes.c_int64)]


# Exported entry points: name -> (restype, argtypes)
EXPORTS = {
    "dard_attention_plan": (ctypes.c_int, [ctypes.POINTER(AttnArgs), ctypes.POINTER(AttnPlan)]),
    "dard_step_attention": (ctypes.c_int, [ctypes.POINTER(AttnArgs), ctypes.c_void_p]),
    "dard_attention_kernel": (ctypes.c_int, [ctypes.POINTER(AttnArgs),
                                             ctypes.POINTER(ctypes.c_int32)]),
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


def _host_i32(a) -> np.ndarray:
    """An owned, contiguous int32 copy of a per-sequence host array."""
    return np.array(a, dtype=np.int32, copy=True).reshape(-1)


def _torch():
    import torch
    return torch


def _raw_stream(device_index: int) -> int:
    """cudaStream_t of the device's current torch stream."""
    torch = _torch()
    f = getattr(torch._C, "_cuda_getCurrentRawStream", None)
    if f is not None:
        return f(device_index)
    return torch.cuda.current_stream(device_index).cuda_stream


def _stream_handle(stream, device_index: int) -> int:
    """``stream`` as a raw handle: a torch stream, an int, or None for the current stream."""
    if stream is None:
        return _raw_stream(device_index)
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.bfloat16:
        return DARD_BF16
    if t.dtype == torch.float32:
        return DARD_F32
    raise ValueError(f"unsupported dtype {t.dtype}")


def _dev(t, name: str, n: int, dtype, device: int | None = None) -> int | None:
    """Device pointer of an optional contiguous tensor of ``dtype`` with at least ``n``
    elements (None for a missing tensor)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name}: device tensor expected")
    if not t.is_contiguous():
        raise ValueError(f"{name}: contiguous tensor expected")
    if t.dtype != dtype:
        raise ValueError(f"{name}: {dtype} expected, got {t.dtype}")
    if t.numel() < n:
        raise ValueError(f"{name}: at least {n} elements expected, got {t.numel()}")
    if device is not None and t.get_device() != device:
        raise ValueError(f"{name}: on device {t.get_device()}, expected {device}")
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


class AttentionCall:
    """``dard_step_attention`` with everything but q, k, v and o marshalled once.

    One step's per-sequence metadata and mask inputs (states, c_{t-1}, shadow sources) are
    the same for every layer, so a caller running many layers builds this once per step and
    calls it per layer. The host arrays are copied; the device tensors are referenced and
    must stay alive and unchanged in size while the object is used. Each call checks q, k,
    v and o against the row count the metadata implies (sum of n_orig + shadow_len), sets
    the four pointers and the stream, and calls the library.

    ``rope_theta`` > 0 makes the call apply RoPE (base theta, pairing ``rope_style``) to q
    and k, which then arrive before RoPE; every call then needs ``k_rope``, a tensor shaped
    like k that receives the rotated keys (k itself rotates k in place)."""

    def __init__(self, n_orig, block_start, block_len, shadow_len, state, prev_conf,
                 shadow_src, scale: float = 0.0, status=None, query_start=None,
                 rope_theta: float = 0.0, rope_style: int = DARD_ROPE_INTERLEAVED):
        torch = _torch()
        self._host = [_host_i32(x) for x in (n_orig, block_start, block_len, shadow_len)]
        self._qs = _host_i32(query_start) if query_start is not None else None
        n, b0, bl, sl = self._host
        ns = len(n)
        if any(len(x) != ns for x in self._host[1:]) or (self._qs is not None and
                                                        len(self._qs) != ns):
            raise ValueError("per-sequence arrays differ in length")
        self.rows = int(n.astype(np.int64).sum() + sl.astype(np.int64).sum())
        blk, sh = int(bl.astype(np.int64).sum()), int(sl.astype(np.int64).sum())
        self.device = state.get_device() if state is not None else None
        a = AttnArgs()
        a.num_seqs = ns
        a.n_orig, a.block_start, a.block_len, a.shadow_len = (
            x.ctypes.data_as(_I32P) for x in self._host)
        a.query_start = self._qs.ctypes.data_as(_I32P) if self._qs is not None else None
        a.state = _dev(state, "state", blk, torch.uint8)
        a.prev_conf = _dev(prev_conf, "prev_conf", blk, torch.float32, self.device)
        a.shadow_src = _dev(shadow_src, "shadow_src", sh, torch.int32, self.device)
        a.status = _dev(status, "status", 1, torch.int32, self.device)
        a.scale = scale
        a.rope_theta = rope_theta
        a.rope_style = rope_style
        self.rope = rope_theta != 0.0
        self._keep = (state, prev_conf, shadow_src, status)
        self._args = a
        self._ref = ctypes.byref(a)
        self._fn = lib().dard_step_attention

    def __call__(self, q, k, v, o, stream=None, k_rope=None):
        """Masked attention of one layer; q/o [rows, hq, d], k/v [rows, hkv, d]; with RoPE,
        ``k_rope`` (like k) receives the rotated keys."""
        dev = self._bind(q, k, v, o, k_rope)
        _check(self._fn(self._ref, _stream_handle(stream, dev)), "dard_step_attention")

    def kernel(self, q, k, v, o) -> int:
        """The kernel a call on these tensors launches, without launching it: 1 or 2 (the
        tensor-core kernel with one or two query tiles per CTA), 4 (the CTA-pair kernel),
        3 (fp32 CUDA cores), 0 (no query rows)."""
        self._bind(q, k, v, o, k if self.rope else None)
        out = ctypes.c_int32(-1)
        _check(lib().dard_attention_kernel(self._ref, ctypes.byref(out)), "dard_attention_kernel")
        return int(out.value)

    def plan(self, q, k, v, o) -> dict:
        """The launch plan of a call on these tensors, without launching it: the kernel, its
        CTAs, and the (query tile, key tile) pairs it computes and skips."""
        self._bind(q, k, v, o, k if self.rope else None)
        out = AttnPlan()
        _check(lib().dard_attention_plan(self._ref, ctypes.byref(out)), "dard_attention_plan")
        return {"kernel": int(out.kernel), "ctas": int(out.ctas),
                "tile_pairs": int(out.tile_pairs),
                "tile_pairs_skipped": int(out.tile_pairs_skipped)}

    def _bind(self, q, k, v, o, k_rope=None) -> int:
        """Checks q, k, v, o (and k_rope) against the metadata and sets their pointers;
        returns the device index."""
        if not (q.is_cuda and k.is_cuda and v.is_cuda and o.is_cuda):
            raise ValueError("q, k, v and o must be device tensors")
        if not (q.is_contiguous() and k.is_contiguous() and v.is_contiguous()
                and o.is_contiguous()):
            raise ValueError("q, k, v and o must be contiguous")
        qs, ks = q.shape, k.shape
        if (len(qs) != 3 or len(ks) != 3 or o.shape != qs or v.shape != ks or ks[2] != qs[2]
                or qs[0] < self.rows or ks[0] < self.rows):
            raise ValueError(f"q/o [>={self.rows}, hq, d] and k/v [>={self.rows}, hkv, d] "
                             f"expected, got {tuple(qs)}, {tuple(ks)}, {tuple(v.shape)}, "
                             f"{tuple(o.shape)}")
        dt = q.dtype
        if k.dtype != dt or v.dtype != dt or o.dtype != dt:
            raise ValueError("q, k, v and o need one dtype")
        dev = q.get_device()
        if (k.get_device() != dev or v.get_device() != dev or o.get_device() != dev
                or (self.device is not None and dev != self.device)):
            raise ValueError("q, k, v, o and the mask inputs need one device")
        if k_rope is not None and (not k_rope.is_cuda or k_rope.shape != ks or
                                   k_rope.dtype != dt or k_rope.get_device() != dev or
                                   not k_rope.is_contiguous()):
            raise ValueError("k_rope must be a contiguous device tensor like k")
        a = self._args
        a.q, a.k, a.v, a.o = q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr()
        a.k_rope = k_rope.data_ptr() if k_rope is not None else None
        a.dtype = _dtype_code(q)
        a.hq, a.hkv, a.head_dim = qs[1], ks[1], qs[2]
        return dev


def dard_step_attention(q, k, v, o, n_orig, block_start, block_len, shadow_len, state,
                        prev_conf, shadow_src, scale: float = 0.0, status=None, stream=None,
                        query_start=None, rope_theta: float = 0.0,
                        rope_style: int = DARD_ROPE_INTERLEAVED, k_rope=None):
    """Masked attention of one layer; q/o [rows, hq, d], k/v [rows, hkv, d] on the device.
    ``query_start`` (per sequence, optional): first query row; earlier rows are keys only.
    ``rope_theta`` > 0: q and k arrive before RoPE, ``k_rope`` receives the rotated keys."""
    AttentionCall(n_orig, block_start, block_len, shadow_len, state, prev_conf, shadow_src,
                  scale=scale, status=status, query_start=query_start, rope_theta=rope_theta,
                  rope_style=rope_style)(q, k, v, o, stream, k_rope=k_rope)


def dard_attention_kernel(q, k, v, o, n_orig, block_start, block_len, shadow_len, state,
                          prev_conf, shadow_src, scale: float = 0.0, query_start=None) -> int:
    """The kernel dard_step_attention would launch for these arguments (see
    ``AttentionCall.kernel``), without launching anything."""
    return AttentionCall(n_orig, block_start, block_len, shadow_len, state, prev_conf,
                         shadow_src, scale=scale, query_start=query_start).kernel(q, k, v, o)


def dard_score_workspace_size(rows: int, vocab: int, num_seqs: int) -> int:
    return int(lib().dard_score_workspace_size(rows, vocab, num_seqs))


class ScoreCall:
    """``dard_score_and_transition`` with everything but the two logits tensors marshalled
    once: the block lengths, thresholds and every state and output buffer. A decode loop
    builds it once per block (or once, with in-place states) and calls it each step on that
    step's logits. The device tensors are referenced and must stay alive and unchanged in
    size while the object is used. ``workspace=None`` selects
    ``dard_score_and_transition_noalloc`` (the library's built-in scratch)."""

    def __init__(self, block_len, state_in, tau_c, tau_u, lam, p0, conf, token, state_out,
                 workspace, w_out=None, counts=None, status=None, cur_token=None, p_cur=None,
                 tokens=None, mask_token: int = 0, entropy=None, margin=None, order_key=None,
                 order_mode: int = ORDER_CONFIDENCE):
        torch = _torch()
        self._bl = _host_i32(block_len)
        ns = len(self._bl)
        self.rows = rows = int(self._bl.astype(np.int64).sum())
        self.device = dev = state_in.get_device() if state_in is not None else None
        f32, i32, u8 = torch.float32, torch.int32, torch.uint8
        a = ScoreArgs()
        a.num_seqs = ns
        a.block_len = self._bl.ctypes.data_as(_I32P)
        a.state_in = _dev(state_in, "state_in", rows, u8)
        a.tau_c, a.tau_u, a.lambda_, a.p0 = tau_c, tau_u, lam, p0
        a.conf = _dev(conf, "conf", rows, f32, dev)
        a.token = _dev(token, "token", rows, i32, dev)
        a.state_out = _dev(state_out, "state_out", rows, u8, dev)
        a.w_out = _dev(w_out, "w_out", rows, f32, dev)
        a.counts = _dev(counts, "counts", 3 * ns, i32, dev)
        a.status = _dev(status, "status", 1, i32, dev)
        a.cur_token = _dev(cur_token, "cur_token", rows, i32, dev)
        a.p_cur = _dev(p_cur, "p_cur", rows, f32, dev)
        a.tokens = _dev(tokens, "tokens", rows, i32, dev)
        a.mask_token = mask_token
        a.entropy = _dev(entropy, "entropy", rows, f32, dev)
        a.margin = _dev(margin, "margin", rows, f32, dev)
        a.order_key = _dev(order_key, "order_key", rows, f32, dev)
        a.order_mode = order_mode
        if workspace is not None:
            a.workspace = _dev(workspace, "workspace", 0, workspace.dtype, dev)
            a.workspace_bytes = workspace.numel() * workspace.element_size()
            self._fn, self._name = lib().dard_score_and_transition, "dard_score_and_transition"
        else:
            self._fn = lib().dard_score_and_transition_noalloc
            self._name = "dard_score_and_transition_noalloc"
        self._keep = (state_in, conf, token, state_out, w_out, counts, status, cur_token,
                      p_cur, tokens, entropy, margin, order_key, workspace)
        self._args = a
        self._ref = ctypes.byref(a)

    def __call__(self, logits_x, logits_s, stream=None):
        """Scores every block row; logits [rows, V] with contiguous rows and one row pitch
        (``stride(0)``, at least V) in both tensors."""
        shp = logits_s.shape
        if logits_x.shape != shp or len(shp) != 2 or shp[0] < self.rows:
            raise ValueError(f"logits_x and logits_s [>={self.rows}, V] of one shape expected, "
                             f"got {tuple(logits_x.shape)} and {tuple(shp)}")
        pitch = _row_pitch(logits_s)
        if _row_pitch(logits_x) != pitch:
            raise ValueError("logits_x and logits_s need the same row pitch")
        if logits_x.dtype != logits_s.dtype:
            raise ValueError("logits_x and logits_s need one dtype")
        a = self._args
        a.logits_x, a.logits_s = _rows_ptr(logits_x), _rows_ptr(logits_s)
        dev = logits_s.get_device()
        if logits_x.get_device() != dev or (self.device is not None and dev != self.device):
            raise ValueError("the logits and the state and output buffers need one device")
        a.dtype = _dtype_code(logits_s)
        a.vocab = shp[1]
        a.row_stride = pitch
        _check(self._fn(self._ref, _stream_handle(stream, dev)), self._name)


def dard_score_and_transition(logits_x, logits_s, block_len, state_in, tau_c, tau_u, lam, p0,
                              conf, token, state_out, workspace, w_out=None, counts=None,
                              status=None, stream=None, cur_token=None, p_cur=None,
                              tokens=None, mask_token: int = 0, entropy=None, margin=None,
                              order_key=None, order_mode: int = ORDER_CONFIDENCE):
    """Scoring and transition of every block row; logits [rows, V] with contiguous rows and
    the same row pitch (``stride(0)``, at least V) in both tensors. Optional end of step:
    ``p_cur`` of ``cur_token``, and ``tokens`` (x^, or ``mask_token`` for rows ending in M);
    ``entropy``, ``margin`` and the next step's ``order_key`` for ``order_mode``."""
    if workspace is None:
        raise ValueError("workspace is required (see dard_score_workspace_size)")
    ScoreCall(block_len, state_in, tau_c, tau_u, lam, p0, conf, token, state_out, workspace,
              w_out=w_out, counts=counts, status=status, cur_token=cur_token, p_cur=p_cur,
              tokens=tokens, mask_token=mask_token, entropy=entropy, margin=margin,
              order_key=order_key, order_mode=order_mode)(logits_x, logits_s, stream)


def dard_score_and_transition_noalloc(logits_x, logits_s, block_len, state_in, tau_c, tau_u,
                                      lam, p0, conf, token, state_out, w_out=None, counts=None,
                                      status=None, stream=None):
    """``dard_score_and_transition`` without a workspace: the library's built-in scratch
    (at most ``SCORE_NOALLOC_MAX_ROWS`` block rows; calls that overlap on one device race)."""
    ScoreCall(block_len, state_in, tau_c, tau_u, lam, p0, conf, token, state_out, None,
              w_out=w_out, counts=counts, status=status)(logits_x, logits_s, stream)
