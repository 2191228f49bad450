"""Plain CPU oracle for the per-step hot path of DARD (arXiv 2608.26574).

TEST INFRASTRUCTURE ONLY. This module is imported by ``tests/``, by
``__graft_entry__.smoke()`` and by ``bench.py`` (its ``cpu_baseline`` leg and its
``--impl reference`` arm). The product package ``paper_2608_26574_gb300`` never imports,
links or runs it, and it shares no code with the CUDA path.

Everything is written for a reader to check against the paper by eye:

* the state-specific attention mask over the augmented sequence x~_t = (x_t; s_t)
  (Sec. 3.1, Eq. 2; Sec. 3.2, query blocks 1-6 and Eq. 3),
* masked softmax attention in float64 (a library matmul is one step), optionally after
  the rotary position embedding of queries and keys, with each shadow row at the position
  it copies (Sec. 3.1),
* prediction / confidence (Sec. 3.1, Eq. 1), the verification-outcome kernel
  (Sec. 3.2, Eq. 5), the guidance weight (Eq. 6), logit mixing (Eq. 7) and the
  three-state transition (Eq. 8), taken in the order of Algorithm 1.

Precision: float64 throughout, except the mixed logits of Eq. 7, which decide an argmax
and are therefore formed in float32 exactly as the kernel forms them:
``mix = ls + w * (lx - ls)`` with each operation rounded to float32 (the paper's
``w*lx + (1-w)*ls`` regrouped; see ``mix_logits``).

Readings of points the paper leaves open (numbered as in the project's full list of
readings, whose other entries concern the workloads and the decoding driver):
  R1  keys of M positions seen by C queries and by M shadow queries come from s;
  R2  a shadow query s^i always sees its own shadow key s^i (no self leak), an original
      query x^i always sees x^i;
  R3  positions before the current block are U, positions after it are M and have no
      shadow row, so every query sees them in x; a block position without a shadow row
      is likewise seen in x by every query;
  R4  ties in the Eq. 3 order are literal (``<=`` on stored float32 confidences);
  R5  argmax ties go to the lowest vocabulary index;
  R6  a scored row is invalid when its softmax normaliser is not finite or is zero
      (NaN, +inf, or all -inf logits): confidence 0, token -1, state M;
  R7  a state byte above 2 is treated as M;
  R8  the attention scale is 1/sqrt(head_dim) unless given;
  R16 p_cur, reported beside c, is the probability the scored distribution (shadow logits
      for C and U positions, mixed logits for M positions) gives to the token currently at
      the position; 0 for a token outside the vocabulary or an invalid row;
  R17 the token update that closes a step of Algorithm 1: positions that end the step in
      M hold the mask token again, every other position holds its new prediction x^;
  R18 the ordering variants of the attention-mask ablation of Sec. 5 (bidirectional, l2r,
      entropy, margin) differ only in the key that Eq. 3 compares: bidirectional = equal
      keys (every C pair attends both ways), l2r = minus the block position (earlier
      positions rank higher), entropy = minus the entropy of the scored distribution (in
      nats; more certain ranks higher), margin = p(x^) minus the second-largest probability
      (a repeated maximum gives 0; a one-entry vocabulary gives 1). An invalid row (R6) has
      entropy 0 and margin 0;
  R20 the positional embedding is RoPE (the paper names none; its dLLMs use rotary
      positions), applied to queries and keys before the masked attention; original row r
      sits at position r and a shadow row at the position it copies (Sec. 3.1 only fixes
      that the two copies share one positional embedding). Both common pairings of the
      rotated elements are provided.

Parity pins: every function here is pinned by ``tests/test_oracle_pins.py`` except where
a docstring says "parity unpinned".
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

# State codes of the per-token state vector (Sec. 3.2: masked / candidate / unmasked).
M, C, U = 0, 1, 2

# Hyper-parameters fixed by Appendix A.2: lambda = 0.917, i.e. 0.5 ** (1/8), and p0 = 0.1.
LAMBDA_DEFAULT = 0.5 ** (1.0 / 8.0)
P0_DEFAULT = 0.1


# --------------------------------------------------------------------------------------
# Sequence layout
# --------------------------------------------------------------------------------------
@dataclass
class SeqLayout:
    """One sequence of the augmented input (Sec. 3.1; Appendix C.4 for block-only shadow).

    n_orig      N: original positions (prompt + full generation length).
    block_start b0: first position of the block being decoded.
    state       uint8[B]: state of each block position (M=0, C=1, U=2).
    prev_conf   float32[B]: c_{t-1} of each block position (orders C tokens, Eq. 3).
    shadow_src  int[S]: original position of each shadow row; shadow rows are stored after
                the N original rows, so row N+k is the shadow copy s^{shadow_src[k]}.
    """

    n_orig: int
    block_start: int
    state: np.ndarray
    prev_conf: np.ndarray
    shadow_src: np.ndarray

    @property
    def block_len(self) -> int:
        return int(len(self.state))

    @property
    def n_shadow(self) -> int:
        return int(len(self.shadow_src))

    @property
    def rows(self) -> int:
        return self.n_orig + self.n_shadow


def position_states(lay: SeqLayout) -> np.ndarray:
    """State of every original position j in [0, N) (reading R3, R7).

    Positions before the block are decoded context (U); the block carries its own states;
    positions after the block are still [Mask] (M).
    """
    st = np.empty(lay.n_orig, dtype=np.int64)
    b0, B = lay.block_start, lay.block_len
    st[:b0] = U
    blk = lay.state.astype(np.int64)
    blk = np.where(blk > 2, M, blk)  # R7
    st[b0:b0 + B] = blk
    st[b0 + B:] = M
    return st


def position_conf(lay: SeqLayout) -> np.ndarray:
    """c_{t-1} of every original position; only C positions are ever compared (Eq. 3)."""
    c = np.zeros(lay.n_orig, dtype=np.float32)
    c[lay.block_start:lay.block_start + lay.block_len] = lay.prev_conf
    return c


def shadow_row_of(lay: SeqLayout) -> np.ndarray:
    """For each original position j, the row index of s^j, or -1 when j has no shadow row."""
    sh = np.full(lay.n_orig, -1, dtype=np.int64)
    for k, j in enumerate(lay.shadow_src):
        sh[int(j)] = lay.n_orig + k
    return sh


# --------------------------------------------------------------------------------------
# Attention mask (Sec. 3.1 Eq. 2; Sec. 3.2 query blocks 1-6, Eq. 3)
# --------------------------------------------------------------------------------------
def query_identity(lay: SeqLayout, r: int) -> tuple[str, int]:
    """Row r of x~_t is the original copy x^r (r < N) or the shadow copy s^i, i = shadow_src."""
    if r < lay.n_orig:
        return "x", r
    return "s", int(lay.shadow_src[r - lay.n_orig])


def sees_shadow_copy(copy: str, i: int, st: np.ndarray, conf: np.ndarray) -> np.ndarray:
    """For the query (copy, i), whether it takes s^j (True) or x^j (False), for every j.

    Each branch restates one paragraph of Sec. 3.2; Eq. 2 makes "attends x^j" and
    "attends s^j" complementary, so one boolean per key position says everything.
    """
    n = len(st)
    j = np.arange(n)
    is_m, is_c, is_u = st == M, st == C, st == U
    si = int(st[i])
    out = np.zeros(n, dtype=bool)

    if si == U:
        # U verification (blocks 3 and 6): U keys in x; M and C keys in s. A shadow query
        # s^i does not see x^i. The original query x^i uses the same pattern.
        out = is_m | is_c
        if copy == "s":
            out = out | (j == i)
    elif si == C:
        # C verification (blocks 2 and 5): U keys in x; of the C keys only those with
        # c_{t-1}^i <= c_{t-1}^j in x (Eq. 3), the rest in s; M keys in s (R1).
        higher_or_equal = conf[i] <= conf  # float32 comparison, R4
        out = is_m | (is_c & ~higher_or_equal)
        if copy == "s":
            out = out | (j == i)  # R2
    else:
        if copy == "x":
            # M prediction from x (block 1): C and U keys in x; M keys in x as well, since
            # the original sequence is the plain dLLM context.
            out = np.zeros(n, dtype=bool)
        else:
            # M prediction from s (block 4): U keys in x; C keys in s (C treated as
            # masked); M keys in s (R1).
            out = is_m | is_c
    return out


def attention_mask(lay: SeqLayout, rows: np.ndarray | None = None) -> np.ndarray:
    """Boolean mask over the rows of x~_t: mask[a, kr] is True iff query row rows[a] (every
    row when ``rows`` is None) attends key row kr. Row/key order: the N original rows, then
    the S shadow rows.

    Eq. 2 holds by construction: for every position j exactly one of x^j and s^j is True.
    Where the rule picks s^j but j has no shadow row, x^j is taken (R3).
    """
    st = position_states(lay)
    conf = position_conf(lay)
    sh = shadow_row_of(lay)
    n = lay.n_orig
    rows = np.arange(lay.rows) if rows is None else np.asarray(rows)
    mask = np.zeros((len(rows), lay.rows), dtype=bool)
    j = np.arange(n)
    for a, r in enumerate(rows):
        copy, i = query_identity(lay, int(r))
        take_s = sees_shadow_copy(copy, i, st, conf) & (sh >= 0)
        mask[a, j[~take_s]] = True
        mask[a, sh[take_s]] = True
    return mask


# --------------------------------------------------------------------------------------
# Masked softmax attention (float64)
# --------------------------------------------------------------------------------------
def masked_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, mask: np.ndarray,
                     scale: float | None = None, rows: np.ndarray | None = None) -> np.ndarray:
    """O[r, h] = sum_kr softmax_kr(scale * <q[r,h], k[kr,g]>, over mask[r]) * v[kr, g].

    q: [R, Hq, d]; k, v: [R, Hkv, d]; g = h // (Hq // Hkv) (grouped-query heads share a
    key/value head). ``rows`` restricts the query rows computed (for sampled parity at full
    size); ``mask`` holds one row per computed query row ([R, R], or [len(rows), R]).
    Returns float64 [len(rows), Hq, d].
    """
    R, hq, d = q.shape
    hkv = k.shape[1]
    assert hq % hkv == 0
    group = hq // hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)  # R8
    if rows is None:
        rows = np.arange(R)
    assert mask.shape == (len(rows), k.shape[0])
    q64 = q[rows].astype(np.float64)
    k64 = k.astype(np.float64)
    v64 = v.astype(np.float64)
    out = np.empty((len(rows), hq, d), dtype=np.float64)
    for h in range(hq):
        g = h // group
        z = (q64[:, h, :] @ k64[:, g, :].T) * scale
        z = np.where(mask, z, -np.inf)
        z = z - z.max(axis=1, keepdims=True)
        p = np.exp(z)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v64[:, g, :]
    return out


# --------------------------------------------------------------------------------------
# Rotary position embedding of the augmented sequence (Sec. 3.1)
# --------------------------------------------------------------------------------------
ROPE_INTERLEAVED, ROPE_HALF = 0, 1


def row_positions(lay: SeqLayout) -> np.ndarray:
    """Position of every row of x~_t (R20): the original copy x^r sits at r, and the shadow
    copy s^j shares the positional embedding of x^j (Sec. 3.1), so shadow row N + k sits at
    shadow_src[k]."""
    return np.concatenate([np.arange(lay.n_orig, dtype=np.int64),
                           np.asarray(lay.shadow_src, dtype=np.int64)])


def rope(x: np.ndarray, positions: np.ndarray, theta: float,
         style: int = ROPE_INTERLEAVED) -> np.ndarray:
    """Rotary position embedding (Su et al., RoFormer, 2021) in float64 (R20).

    x: [R, H, d]; positions: [R]. For frequency index i < d/2, f_i = theta^(-2i/d), and the
    pair (a, b) of a row at position p becomes (a cos(p f_i) - b sin(p f_i),
    a sin(p f_i) + b cos(p f_i)) in every head. The pairs are elements (2i, 2i+1)
    (ROPE_INTERLEAVED) or (i, i + d/2) (ROPE_HALF). Returns float64 [R, H, d].
    """
    R, H, d = x.shape
    i = np.arange(d // 2, dtype=np.float64)
    freq = float(theta) ** (-2.0 * i / d)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * freq[None, :]  # [R, d/2]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x64 = x.astype(np.float64)
    if style == ROPE_INTERLEAVED:
        first, second = np.s_[..., 0::2], np.s_[..., 1::2]
    elif style == ROPE_HALF:
        first, second = np.s_[..., : d // 2], np.s_[..., d // 2:]
    else:
        raise ValueError(style)
    a, b = x64[first], x64[second]
    out = np.empty_like(x64)
    out[first] = a * cos - b * sin
    out[second] = a * sin + b * cos
    return out


# --------------------------------------------------------------------------------------
# Scoring: confidence, mixing weight, logit mixing, state transition
# --------------------------------------------------------------------------------------
def confidence(logits_row: np.ndarray) -> tuple[float, int, bool]:
    """Eq. 1: x^ = argmax_v p(v), c = p(x^), p = softmax of the logits, in float64.

    Ties go to the lowest index (R5). Returns (c, token, valid); an invalid row (R6) gives
    (0.0, -1, False).
    """
    x = logits_row.astype(np.float64)
    if np.isnan(x).any() or np.isposinf(x).any() or np.isneginf(x).all():
        return 0.0, -1, False
    m = x.max()
    token = int(np.flatnonzero(x == m)[0])
    z = np.exp(x - m).sum()
    return float(1.0 / z), token, True


def token_probability(logits_row: np.ndarray, tok: int) -> float:
    """R16: softmax(logits)[tok] in float64, i.e. exp(l_tok - max) / sum exp(l - max).

    0.0 for tok outside [0, V) or an invalid row (R6).
    """
    x = logits_row.astype(np.float64)
    if not (0 <= tok < len(x)):
        return 0.0
    if np.isnan(x).any() or np.isposinf(x).any() or np.isneginf(x).all():
        return 0.0
    m = x.max()
    return float(math.exp(x[tok] - m) / np.exp(x - m).sum())


def entropy(logits_row: np.ndarray) -> float:
    """R18: -sum_v p_v ln p_v of the softmax of the row (float64); 0 for an invalid row."""
    x = logits_row.astype(np.float64)
    if np.isnan(x).any() or np.isposinf(x).any() or np.isneginf(x).all():
        return 0.0
    p = np.exp(x - x.max())
    p /= p.sum()
    nz = p > 0
    return float(-(p[nz] * np.log(p[nz])).sum())


def margin(logits_row: np.ndarray) -> float:
    """R18: p(x^) minus the second-largest probability (float64); 0 for an invalid row."""
    x = logits_row.astype(np.float64)
    if np.isnan(x).any() or np.isposinf(x).any() or np.isneginf(x).all():
        return 0.0
    p = np.exp(x - x.max())
    p /= p.sum()
    if len(p) < 2:
        return float(p[0])
    top = np.sort(p)
    return float(top[-1] - top[-2])


# Ordering modes of R18 (the key Eq. 3 compares in the next step)
ORDER_CONFIDENCE, ORDER_BIDIR, ORDER_L2R, ORDER_ENTROPY, ORDER_MARGIN = 0, 1, 2, 3, 4


def order_key(mode: int, c: float, h: float, mg: float, i: int) -> float:
    """R18: the next step's ordering key of block position i."""
    return {ORDER_CONFIDENCE: c, ORDER_BIDIR: 0.0, ORDER_L2R: -float(i),
            ORDER_ENTROPY: -h, ORDER_MARGIN: mg}[mode]


def next_tokens(token: np.ndarray, state_out: np.ndarray, mask_token: int) -> np.ndarray:
    """R17, the last line of Algorithm 1's step: positions in C_{t+1} and U_{t+1} take the
    decoded token x^, positions in M_{t+1} keep the mask token."""
    return np.where(np.asarray(state_out) == M, mask_token, np.asarray(token)).astype(np.int64)


def next_state(c: float, tau_c: float, tau_u: float) -> int:
    """Eq. 8: c <= tau_c -> M; tau_c < c <= tau_u -> C; tau_u < c -> U."""
    if c <= tau_c:
        return M
    if c <= tau_u:
        return C
    return U


def mixing_weight(i: int, promoted: list[int], demoted: list[int],
                  lam: float, p0: float) -> tuple[float, float, float]:
    """Eq. 5 and Eq. 6 for one masked position i (float64).

    P_i = sum_{j in P} lam^|i-j|, D_i = sum_{j in D} lam^|i-j|, w = (P_i + p0)/(P_i + D_i + p0).
    Returns (w, P_i, D_i).
    """
    lam = float(lam)
    p_i = sum(lam ** abs(i - j) for j in promoted)
    d_i = sum(lam ** abs(i - j) for j in demoted)
    w = (p_i + p0) / (p_i + d_i + p0)
    return w, p_i, d_i


def mix_logits(lx: np.ndarray, ls: np.ndarray, w: np.float32) -> np.ndarray:
    """Eq. 7: logit_mix = w * logit(x) + (1 - w) * logit(s), regrouped as ls + w*(lx - ls).

    Formed in float32, one rounding per operation, so that the argmax it decides is taken
    in the same precision on both sides.
    """
    lx = lx.astype(np.float32)
    ls = ls.astype(np.float32)
    w = np.float32(w)
    diff = (lx - ls).astype(np.float32)
    return (ls + (w * diff).astype(np.float32)).astype(np.float32)


@dataclass
class ScoreResult:
    conf: np.ndarray       # float64 [B]
    token: np.ndarray      # int64 [B]
    state_out: np.ndarray  # uint8 [B]
    w: np.ndarray          # float32 [B], NaN for rows that are not M
    valid: np.ndarray      # bool [B]
    promoted: list
    demoted: list
    counts: np.ndarray     # int64 [3]: M, C, U after the transition
    p_cur: np.ndarray | None = None        # float64 [B] (R16), when cur_token is given
    tokens_next: np.ndarray | None = None  # int64 [B] (R17), when mask_token is given
    entropy: np.ndarray | None = None      # float64 [B] (R18) of each scored distribution
    margin: np.ndarray | None = None       # float64 [B] (R18)


def score_block(logits_x: np.ndarray, logits_s: np.ndarray, state_in: np.ndarray,
                tau_c: float, tau_u: float, lam: float = LAMBDA_DEFAULT,
                p0: float = P0_DEFAULT, cur_token: np.ndarray | None = None,
                mask_token: int | None = None) -> ScoreResult:
    """One block of Algorithm 1 after the forward pass (float64 except Eq. 7).

    logits_x / logits_s: [B, V] logits of x^i and s^i for every block position i.
    1. C and U positions: c and x^ from the shadow logits (Eq. 1).
    2. C positions move by Eq. 8; those that reach U form P, those that reach M form D.
    3. M positions: w from P and D (Eq. 5, 6), mixed logits (Eq. 7), c and x^ from them.
    4. M and U positions move by Eq. 8.
    Optional: p_cur of cur_token on each scored distribution (R16), and the next step's
    tokens (R17) when mask_token is given.
    """
    B = len(state_in)
    st = np.where(state_in > 2, M, state_in).astype(np.int64)  # R7
    conf = np.zeros(B, dtype=np.float64)
    ent = np.zeros(B, dtype=np.float64)
    mgn = np.zeros(B, dtype=np.float64)
    token = np.full(B, -1, dtype=np.int64)
    valid = np.zeros(B, dtype=bool)
    new = np.zeros(B, dtype=np.int64)
    w_out = np.full(B, np.nan, dtype=np.float32)
    p_cur = None if cur_token is None else np.zeros(B, dtype=np.float64)

    # 1-2: candidate and unmasked positions are verified from the shadow sequence.
    promoted, demoted = [], []
    for i in range(B):
        if st[i] == M:
            continue
        c, tok, ok = confidence(logits_s[i])
        conf[i], token[i], valid[i] = c, tok, ok
        ent[i], mgn[i] = entropy(logits_s[i]), margin(logits_s[i])
        if p_cur is not None:
            p_cur[i] = token_probability(logits_s[i], int(cur_token[i]))
        new[i] = next_state(c, tau_c, tau_u) if ok else M
        if st[i] == C:
            if new[i] == U:
                promoted.append(i)
            elif new[i] == M:
                demoted.append(i)

    # 3-4: masked positions mix the two predictions, weighted by nearby outcomes.
    for i in range(B):
        if st[i] != M:
            continue
        w, _, _ = mixing_weight(i, promoted, demoted, lam, p0)
        w32 = np.float32(w)
        w_out[i] = w32
        mixed = mix_logits(logits_x[i], logits_s[i], w32)
        c, tok, ok = confidence(mixed)
        conf[i], token[i], valid[i] = c, tok, ok
        ent[i], mgn[i] = entropy(mixed), margin(mixed)
        if p_cur is not None:
            p_cur[i] = token_probability(mixed, int(cur_token[i]))
        new[i] = next_state(c, tau_c, tau_u) if ok else M

    counts = np.array([(new == s).sum() for s in (M, C, U)], dtype=np.int64)
    tokens_next = None if mask_token is None else next_tokens(token, new, mask_token)
    return ScoreResult(conf, token, new.astype(np.uint8), w_out, valid, promoted, demoted,
                       counts, p_cur, tokens_next, ent, mgn)


def top2_gap(row: np.ndarray) -> float:
    """Difference between the two largest entries of a row (float64); inf if V < 2.

    Used to report near-ties separately: a position whose top-2 logits differ by under
    1e-3 may legitimately take either argmax under rounding.
    """
    x = np.sort(row.astype(np.float64))
    if len(x) < 2:
        return math.inf
    return float(x[-1] - x[-2])
