"""Seeded synthetic inputs for the DARD step (no DARD arithmetic lives here).

These generators are the one module that both the CUDA path's tests/bench and the CPU
oracle consume: they only draw random numbers (NumPy PCG64) and lay them out. Values that
the kernels read in bfloat16 are rounded to bfloat16 here (round to nearest even) and
returned as float32 arrays that hold exactly those values, so both sides see identical
inputs.

Workloads (shapes of the paper's setting: LLaDA-8B-class layers, 32 heads, head_dim 128,
vocab 126464, block decoding as in Appendix A.2):

  tiny        1 seq, 4 heads, d=64, prompt 32, block 32 (40/30/30 % M/C/U), fp32.
  8b          1 seq, 32 heads MHA, d=128, prompt 512, gen 256 in blocks of 32, block 3,
              50/25/25 %, bf16; logits 32 x 126464.
  gqa         1 seq, 28 query / 4 kv heads, d=128, prompt 4096, gen 1024 in blocks of 64,
              block 8, 30/40/30 %, bf16; logits 64 x 152064.
  ragged      32 seqs of the 8b shape, prompt ~ U{256..2048}, block index ~ U{0..7},
              masked fraction ~ U[0.2, 0.8], rest split evenly between C and U.
  mm          8 seqs, prompt 576 image + 128 text positions, gen 512 in blocks of 32,
              block 10, 20/60/20 %, 32 independent layers per step.

Shadow layouts: "paper" appends one shadow row per block position (the shadow sequence
restricted to the current block); "candidates" appends shadow rows for C positions only.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

STATE_M, STATE_C, STATE_U = 0, 1, 2

# (tau_c, tau_u) per workload, from the threshold grids of Appendix A.2.
TAUS = {"tiny": (0.4, 0.9), "8b": (0.5, 0.8), "gqa": (0.5, 0.8), "ragged": (0.5, 0.8),
        "mm": (0.4, 0.9)}
LAMBDA = 0.5 ** (1.0 / 8.0)
P0 = 0.1
SEED_BASE = 1000
CONFIG_INDEX = {"tiny": 0, "8b": 1, "gqa": 2, "ragged": 3, "mm": 4}


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32.
    Finite inputs only: the largest finite pattern plus the rounding bias stays below 2^32,
    so the sum is formed in uint32."""
    bits = np.array(a, dtype=np.float32, copy=True).view(np.uint32)
    bias = bits >> np.uint32(16)
    bias &= np.uint32(1)
    bias += np.uint32(0x7FFF)
    bits += bias
    bits &= np.uint32(0xFFFF0000)
    return bits.view(np.float32)


def state_counts(B: int, fractions: tuple[float, float, float]) -> list[int]:
    """Exact M/C/U counts by largest remainder; equal remainders favour the lower code."""
    raw = [B * f for f in fractions]
    base = [int(math.floor(x)) for x in raw]
    rem = [x - b for x, b in zip(raw, base)]
    left = B - sum(base)
    order = sorted(range(3), key=lambda s: (-rem[s], s))
    for s in order[:left]:
        base[s] += 1
    return base


@dataclass
class Seq:
    n_orig: int
    block_start: int
    state: np.ndarray       # uint8 [B]
    prev_conf: np.ndarray   # float32 [B]
    shadow_src: np.ndarray  # int32 [S]
    prompt: int = 0         # prompt length P0 (positions 0 .. P0-1)
    query_start: int = 0    # first query row (prefix caching: P0; 0 = every row is a query)

    @property
    def block_len(self) -> int:
        return int(len(self.state))

    @property
    def n_shadow(self) -> int:
        return int(len(self.shadow_src))

    @property
    def rows(self) -> int:
        return self.n_orig + self.n_shadow


@dataclass
class Workload:
    name: str
    dtype: str                    # "bf16" or "f32": the type the kernels read
    hq: int
    hkv: int
    head_dim: int
    vocab: int
    seqs: list
    tau_c: float
    tau_u: float
    lam: float = LAMBDA
    p0: float = P0
    layers: int = 1
    q: list = field(default_factory=list)   # per layer float32 [rows, hq, d]
    k: list = field(default_factory=list)   # per layer float32 [rows, hkv, d]
    v: list = field(default_factory=list)
    logits_x: np.ndarray | None = None      # float32 [sum B, vocab]
    logits_s: np.ndarray | None = None
    row_std: np.ndarray | None = None       # per-row std of Q, K and V
    logit_spec: tuple | None = None         # logits: (std, planted fraction, planted height)

    @property
    def total_rows(self) -> int:
        return sum(s.rows for s in self.seqs)

    @property
    def total_block(self) -> int:
        return sum(s.block_len for s in self.seqs)

    def row_offsets(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum([s.rows for s in self.seqs])]).astype(np.int64)

    def block_offsets(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum([s.block_len for s in self.seqs])]).astype(np.int64)

    def state_all(self) -> np.ndarray:
        return np.concatenate([s.state for s in self.seqs]).astype(np.uint8)

    def prev_conf_all(self) -> np.ndarray:
        return np.concatenate([s.prev_conf for s in self.seqs]).astype(np.float32)

    def shadow_src_all(self) -> np.ndarray:
        parts = [s.shadow_src for s in self.seqs]
        return (np.concatenate(parts) if parts else np.zeros(0)).astype(np.int32)


def _draw_states(rng, B: int, fractions, tau_c: float, tau_u: float):
    counts = state_counts(B, fractions)
    codes = np.repeat(np.array([STATE_M, STATE_C, STATE_U], dtype=np.uint8), counts)
    state = codes[rng.permutation(B)]
    conf = np.empty(B, dtype=np.float32)
    nm, nc, nu = (state == STATE_M).sum(), (state == STATE_C).sum(), (state == STATE_U).sum()
    # U ~ U(tau_u, 1], C ~ U(tau_c, tau_u], M ~ U[0, tau_c]
    conf[state == STATE_U] = tau_u + (1.0 - tau_u) * (1.0 - rng.random(nu))
    conf[state == STATE_C] = tau_c + (tau_u - tau_c) * (1.0 - rng.random(nc))
    conf[state == STATE_M] = tau_c * rng.random(nm)
    return state, conf


def _shadow(state: np.ndarray, b0: int, layout: str) -> np.ndarray:
    B = len(state)
    if layout == "paper":
        return (b0 + np.arange(B)).astype(np.int32)
    if layout == "candidates":
        return (b0 + np.flatnonzero(state == STATE_C)).astype(np.int32)
    raise ValueError(layout)


def _qkv(rng, seqs, hq, hkv, d, dtype, std_fn):
    rows = sum(s.rows for s in seqs)
    std = std_fn(rows)  # [rows] per-row std
    out = []
    for h in (hq, hkv, hkv):
        a = rng.standard_normal((rows, h, d), dtype=np.float32)
        a *= std[:, None, None].astype(np.float32)
        out.append(round_bf16(a) if dtype == "bf16" else a)
    return out


def _logits(rng, nrows, vocab, std, dtype, mode, plant_frac, plant_height):
    a = rng.standard_normal((nrows, vocab), dtype=np.float32)
    a *= np.float32(std)
    cols = rng.integers(0, vocab, size=nrows)
    if mode == "literal":
        n_plant = int(round(plant_frac * nrows))
        rows = rng.permutation(nrows)[:n_plant]
        a[rows, cols[rows]] += np.float32(plant_height)
    elif mode == "spanning":
        # Planted value around the log of the row's expected exp-mass, so that the
        # confidence of the planted token spans the thresholds: log(V) + std^2/2 is the
        # log of V * E[exp(N(0, std^2))].
        centre = math.log(vocab) + 0.5 * std * std
        a[np.arange(nrows), cols] = (centre + rng.uniform(-4.0, 4.6, size=nrows)).astype(np.float32)
    elif mode != "plain":
        raise ValueError(mode)
    return round_bf16(a) if dtype == "bf16" else a


def make(name: str, layout: str = "paper", logits: str = "literal", attention: bool = True,
         scoring: bool = True, layers: int | None = None, seed: int | None = None,
         prefix: bool = False) -> Workload:
    """Build one named workload. ``logits``: "literal" (the stated distribution and planted
    peaks), "spanning" (planted confidences spread across the thresholds) or "plain".
    ``prefix``: the prefix-cached variant, whose queries start after the prompt (the same
    inputs; only which rows are queries changes)."""
    if seed is None:
        seed = SEED_BASE + CONFIG_INDEX[name]
    rng = np.random.default_rng(np.random.PCG64(seed))
    tau_c, tau_u = TAUS[name]
    isd = 1.0 / math.sqrt(128.0)

    if name == "tiny":
        st, cf = _draw_states(rng, 32, (0.4, 0.3, 0.3), tau_c, tau_u)
        seqs = [Seq(64, 32, st, cf, _shadow(st, 32, layout), prompt=32)]
        wl = Workload(name, "f32", 4, 4, 64, 1024, seqs, tau_c, tau_u)
        std_fn = lambda rows: np.ones(rows)  # noqa: E731
        lspec = (2.0, 0.5, 6.0)
    elif name == "8b":
        b0 = 512 + 3 * 32
        st, cf = _draw_states(rng, 32, (0.5, 0.25, 0.25), tau_c, tau_u)
        seqs = [Seq(512 + 256, b0, st, cf, _shadow(st, b0, layout), prompt=512)]
        wl = Workload(name, "bf16", 32, 32, 128, 126464, seqs, tau_c, tau_u)
        std_fn = lambda rows: np.full(rows, isd)  # noqa: E731
        lspec = (3.0, 0.4, 6.0)
    elif name == "gqa":
        b0 = 4096 + 8 * 64
        st, cf = _draw_states(rng, 64, (0.3, 0.4, 0.3), tau_c, tau_u)
        seqs = [Seq(4096 + 1024, b0, st, cf, _shadow(st, b0, layout), prompt=4096)]
        wl = Workload(name, "bf16", 28, 4, 128, 152064, seqs, tau_c, tau_u)
        std_fn = lambda rows: np.full(rows, isd)  # noqa: E731
        lspec = (3.0, 0.0, 0.0)
    elif name == "ragged":
        seqs = []
        for _ in range(32):
            p0 = int(rng.integers(256, 2049))
            idx = int(rng.integers(0, 8))
            fm = float(rng.uniform(0.2, 0.8))
            st, cf = _draw_states(rng, 32, (fm, (1 - fm) / 2, (1 - fm) / 2), tau_c, tau_u)
            b0 = p0 + 32 * idx
            seqs.append(Seq(p0 + 256, b0, st, cf, _shadow(st, b0, layout), prompt=p0))
        wl = Workload(name, "bf16", 32, 32, 128, 126464, seqs, tau_c, tau_u)
        std_fn = lambda rows: np.full(rows, isd)  # noqa: E731
        lspec = (3.0, 0.4, 6.0)
    elif name == "mm":
        b0 = 704 + 10 * 32
        seqs = []
        for _ in range(8):
            st, cf = _draw_states(rng, 32, (0.2, 0.6, 0.2), tau_c, tau_u)
            seqs.append(Seq(704 + 512, b0, st, cf, _shadow(st, b0, layout), prompt=704))
        wl = Workload(name, "bf16", 32, 32, 128, 126464, seqs, tau_c, tau_u)
        wl.layers = 32 if layers is None else layers

        def std_fn(rows, _seqs=seqs):
            parts = []
            for s in _seqs:
                r = np.full(s.rows, isd)
                r[:576] = 1.5  # image-embedding positions
                parts.append(r)
            return np.concatenate(parts)
        lspec = (3.0, 0.4, 6.0)
    else:
        raise ValueError(name)

    if prefix:
        for sq in wl.seqs:
            sq.query_start = sq.prompt
    # the distributions, for callers that draw the bulk tensors elsewhere (on the device)
    wl.row_std = np.asarray(std_fn(sum(sq.rows for sq in wl.seqs)), dtype=np.float64)
    wl.logit_spec = lspec
    if attention:
        for _ in range(wl.layers):
            q, k, v = _qkv(rng, wl.seqs, wl.hq, wl.hkv, wl.head_dim, wl.dtype, std_fn)
            wl.q.append(q)
            wl.k.append(k)
            wl.v.append(v)
    if scoring:
        std, frac, height = lspec
        nrows = wl.total_block
        wl.logits_x = _logits(rng, nrows, wl.vocab, std, wl.dtype, logits, frac, height)
        wl.logits_s = _logits(rng, nrows, wl.vocab, std, wl.dtype, logits, frac, height)
    return wl


def attention_flops(wl: Workload) -> float:
    """Algorithmic attention FLOPs of one layer: every query row attends exactly N keys
    (one copy per original position), QK^T and PV each 2*d FLOPs per (row, key, head)."""
    return float(sum(4.0 * wl.head_dim * (s.rows - s.query_start) * s.n_orig * wl.hq
                     for s in wl.seqs))


def scoring_bytes(wl: Workload) -> float:
    """Algorithmic scoring bytes: the shadow logits of every block row plus the original
    logits of M rows, each read once."""
    esz = 2 if wl.dtype == "bf16" else 4
    n_m = sum(int((s.state == STATE_M).sum()) for s in wl.seqs)
    return float(wl.vocab * esz * (wl.total_block + n_m))


def custom(specs, hq: int, hkv: int, head_dim: int, dtype: str = "bf16", vocab: int = 0,
           seed: int = 0, qkv_std: float | None = None, probe: bool = False,
           logits: str = "spanning", logit_std: float = 3.0, tau=(0.5, 0.8)) -> Workload:
    """A seeded workload from explicit per-sequence specs (edge cases, small shapes).

    specs: list of dicts with n_orig, block_start, and either state (uint8 array) or
    fractions (M, C, U) with block_len; optional prev_conf (float32 array) and shadow
    ("paper", "candidates" or an explicit int array of original positions).
    probe=True draws Q = 0 (uniform attention over the attended keys) and K, V ~ N(0, 1), so
    that every attended key shows in the output with weight 1/N.
    """
    rng = np.random.default_rng(np.random.PCG64(seed))
    tau_c, tau_u = tau
    seqs = []
    for sp in specs:
        if "state" in sp:
            st = np.asarray(sp["state"], dtype=np.uint8)
            cf = np.empty(len(st), np.float32)
            for code, lo, hi in ((STATE_M, 0.0, tau_c), (STATE_C, tau_c, tau_u), (STATE_U, tau_u, 1.0)):
                sel = st == code
                cf[sel] = lo + (hi - lo) * (1.0 - rng.random(int(sel.sum())))
        else:
            st, cf = _draw_states(rng, sp["block_len"], sp["fractions"], tau_c, tau_u)
        if sp.get("prev_conf") is not None:
            cf = np.asarray(sp["prev_conf"], dtype=np.float32)
        shadow = sp.get("shadow", "paper")
        src = _shadow(st, sp["block_start"], shadow) if isinstance(shadow, str) else \
            np.asarray(shadow, dtype=np.int32)
        seqs.append(Seq(sp["n_orig"], sp["block_start"], st, cf, src,
                        query_start=int(sp.get("query_start", 0))))
    wl = Workload("custom", dtype, hq, hkv, head_dim, vocab, seqs, tau_c, tau_u)
    std = (1.0 / math.sqrt(head_dim)) if qkv_std is None else qkv_std
    rows = wl.total_rows
    if probe:
        q = np.zeros((rows, hq, head_dim), np.float32)
        k = rng.standard_normal((rows, hkv, head_dim), dtype=np.float32)
        v = rng.standard_normal((rows, hkv, head_dim), dtype=np.float32)
    else:
        q = rng.standard_normal((rows, hq, head_dim), dtype=np.float32) * np.float32(std)
        k = rng.standard_normal((rows, hkv, head_dim), dtype=np.float32) * np.float32(std)
        v = rng.standard_normal((rows, hkv, head_dim), dtype=np.float32) * np.float32(std)
    if dtype == "bf16":
        q, k, v = round_bf16(q), round_bf16(k), round_bf16(v)
    wl.q, wl.k, wl.v = [q], [k], [v]
    if vocab > 0:
        nrows = wl.total_block
        wl.logits_x = _logits(rng, nrows, vocab, logit_std, dtype, logits, 0.5, 6.0)
        wl.logits_s = _logits(rng, nrows, vocab, logit_std, dtype, logits, 0.5, 6.0)
    return wl
