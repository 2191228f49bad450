"""Device-side holder of one DARD step's inputs and outputs (torch for memory only).

``DeviceStep`` uploads a seeded ``workloads.Workload`` (one layer, or all layers) to the GPU,
owns the output tensors and the scoring workspace, and calls the two C-ABI entry points
through ``binding``. It is what the tests, ``bench.py`` and ``smoke()`` drive.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as B
from .workloads import Workload


def to_device(a: np.ndarray, dtype: str, device) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype == "bf16":
        t = t.to(torch.bfloat16)  # values are already bf16-exact: the conversion is exact
    return t.to(device)


class DeviceStep:
    def __init__(self, wl: Workload, device="cuda", layers=None, attention=True, scoring=True,
                 logit_pitch: int | None = None):
        self.wl = wl
        self.device = torch.device(device)
        dt = wl.dtype
        self.n_orig = np.array([s.n_orig for s in wl.seqs], dtype=np.int32)
        self.block_start = np.array([s.block_start for s in wl.seqs], dtype=np.int32)
        self.block_len = np.array([s.block_len for s in wl.seqs], dtype=np.int32)
        self.shadow_len = np.array([s.n_shadow for s in wl.seqs], dtype=np.int32)
        qs = np.array([s.query_start for s in wl.seqs], dtype=np.int32)
        self.query_start = qs if qs.any() else None
        dev = self.device
        self.state = torch.from_numpy(wl.state_all()).to(dev)
        self.prev_conf = torch.from_numpy(wl.prev_conf_all()).to(dev)
        sh = wl.shadow_src_all()
        self.shadow_src = torch.from_numpy(sh if len(sh) else np.zeros(1, np.int32)).to(dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self._attn_calls: dict[tuple, B.AttentionCall] = {}
        self._k_rope: dict[int, torch.Tensor] = {}
        self._score_calls: dict[tuple[bool, bool], B.ScoreCall] = {}
        self.layers = []
        if attention:
            idx = range(len(wl.q)) if layers is None else layers
            for li in idx:
                q = to_device(wl.q[li], dt, dev)
                k = to_device(wl.k[li], dt, dev)
                v = to_device(wl.v[li], dt, dev)
                self.layers.append((q, k, v, torch.empty_like(q)))
        self.rows = wl.total_block
        if scoring and wl.logits_s is not None:
            self.lx = to_device(wl.logits_x, dt, dev)
            self.ls = to_device(wl.logits_s, dt, dev)
            if logit_pitch is not None and logit_pitch != wl.vocab:
                # rows padded to `logit_pitch` elements; the padding holds a huge value that
                # must never be read
                for name in ("lx", "ls"):
                    t = getattr(self, name)
                    big = torch.full((t.shape[0], logit_pitch), 3.0e38, dtype=t.dtype, device=dev)
                    big[:, :wl.vocab] = t
                    setattr(self, name, big[:, :wl.vocab])
            nbytes = B.dard_score_workspace_size(self.rows, wl.vocab, len(wl.seqs))
            self.workspace = torch.zeros(max(nbytes, 16), dtype=torch.uint8, device=dev)
            r = max(self.rows, 1)
            self.conf = torch.empty(r, dtype=torch.float32, device=dev)
            self.token = torch.empty(r, dtype=torch.int32, device=dev)
            self.state_out = torch.empty(r, dtype=torch.uint8, device=dev)
            self.w_out = torch.empty(r, dtype=torch.float32, device=dev)
            self.counts = torch.empty(3 * len(wl.seqs), dtype=torch.int32, device=dev)

    def attention_call(self, scale: float = 0.0, rope=None) -> B.AttentionCall:
        """The prepared attention call of this step (metadata marshalled once per scale and
        RoPE setting; ``rope`` = (theta, style) or None)."""
        key = (scale, rope)
        c = self._attn_calls.get(key)
        if c is None:
            theta, style = rope if rope is not None else (0.0, B.DARD_ROPE_INTERLEAVED)
            c = B.AttentionCall(self.n_orig, self.block_start, self.block_len, self.shadow_len,
                                self.state, self.prev_conf, self.shadow_src, scale=scale,
                                status=self.status, query_start=self.query_start,
                                rope_theta=theta, rope_style=style)
            self._attn_calls[key] = c
        return c

    def k_rope(self, layer: int = 0) -> torch.Tensor:
        """The buffer that receives a layer's rotated keys when RoPE is applied."""
        t = self._k_rope.get(layer)
        if t is None:
            t = torch.empty_like(self.layers[layer][1])
            self._k_rope[layer] = t
        return t

    def attention(self, layer: int = 0, scale: float = 0.0, stream=None, out=None, rope=None):
        """One layer's attention; ``rope`` = (theta, style) applies RoPE in the call (the
        rotated keys land in ``k_rope(layer)``)."""
        q, k, v, o = self.layers[layer]
        o = o if out is None else out
        kr = self.k_rope(layer) if rope is not None else None
        self.attention_call(scale, rope)(q, k, v, o, stream, k_rope=kr)
        return o

    def score_call(self, w_out=True, counts=True, state_in=None) -> B.ScoreCall:
        """The prepared scoring call over this step's buffers (cached for the step's own
        states; a caller-given ``state_in`` gets a fresh one)."""
        key = (bool(w_out), bool(counts))
        c = self._score_calls.get(key) if state_in is None else None
        if c is None:
            wl = self.wl
            c = B.ScoreCall(self.block_len, self.state if state_in is None else state_in,
                            wl.tau_c, wl.tau_u, wl.lam, wl.p0, self.conf, self.token,
                            self.state_out, self.workspace, w_out=self.w_out if w_out else None,
                            counts=self.counts if counts else None, status=self.status)
            if state_in is None:
                self._score_calls[key] = c
        return c

    def score(self, stream=None, w_out=True, counts=True, state_in=None):
        self.score_call(w_out, counts, state_in)(self.lx, self.ls, stream)
