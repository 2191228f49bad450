"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test names the passage it follows. None of them re-calls the oracle's own formula to
produce its expectation: expectations come from closed forms, library routines (torch /
scipy softmax attention), brute force on tiny inputs, invariants the paper states, or the
paper's printed numbers (tests/golden).
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle as orc
from oracle import C, M, U, SeqLayout

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _layout(states, confs, prompt=3, future=2, shadow="paper"):
    B = len(states)
    b0 = prompt
    st = np.array(states, dtype=np.uint8)
    if shadow == "paper":
        src = b0 + np.arange(B)
    elif shadow == "candidates":
        src = b0 + np.flatnonzero(st == C)
    else:
        src = np.array(shadow, dtype=np.int64)
    return SeqLayout(prompt + B + future, b0, st, np.array(confs, dtype=np.float32),
                     np.asarray(src, dtype=np.int32))


def _rand_layout(rng, B=12, prompt=7, future=5, shadow="paper"):
    st = rng.integers(0, 3, size=B)
    cf = rng.choice(np.array([0.55, 0.6, 0.65, 0.7, 0.75], dtype=np.float32), size=B)
    return _layout(st, cf, prompt, future, shadow)


def _copy_of_key(lay, kr):
    """(copy, position) of key row kr."""
    if kr < lay.n_orig:
        return "x", kr
    return "s", int(lay.shadow_src[kr - lay.n_orig])


def _attended(lay, mask, r):
    return {_copy_of_key(lay, kr) for kr in np.flatnonzero(mask[r])}


# ---------------------------------------------------------------------------------------
# Mask: Eq. 2 and the query blocks of Sec. 3.2
# ---------------------------------------------------------------------------------------
@pytest.mark.parametrize("shadow", ["paper", "candidates"])
def test_eq2_exactly_one_copy_per_position(shadow):
    """Eq. 2: every query attends exactly one of x^j and s^j for every position j."""
    rng = np.random.default_rng(1)
    for _ in range(20):
        lay = _rand_layout(rng, shadow=shadow)
        mask = orc.attention_mask(lay)
        assert mask.shape == (lay.rows, lay.rows)
        for r in range(lay.rows):
            seen = _attended(lay, mask, r)
            positions = [j for _, j in seen]
            assert sorted(positions) == list(range(lay.n_orig)), (r, seen)
        assert (mask.sum(axis=1) == lay.n_orig).all()


def test_all_unmasked_reduces_to_full_bidirectional():
    """With every token U and no candidates, original queries see every original key:
    plain bidirectional attention over x (Sec. 3.2, U blocks: U keys are taken in x)."""
    lay = _layout([U] * 6, [0.95] * 6, prompt=4, future=0)
    mask = orc.attention_mask(lay)
    n = lay.n_orig
    assert mask[:n, :n].all()
    assert not mask[:n, n:].any()
    # shadow queries: all of x except their own position, which they see in s
    for k in range(lay.n_shadow):
        i = int(lay.shadow_src[k])
        assert _attended(lay, mask, n + k) == {("x", j) for j in range(n) if j != i} | {("s", i)}


def _paper_sets(lay, copy, i, st, cf):
    """Attended set of query (copy, i) assembled from the sentences of Sec. 3.2, as a set of
    (copy, position) pairs, for a layout where every block position has a shadow row."""
    n = lay.n_orig
    Ux = {("x", j) for j in range(n) if st[j] == U}
    Mx = {("x", j) for j in range(n) if st[j] == M}
    Cx = {("x", j) for j in range(n) if st[j] == C}
    Ms = {("s", j) for j in range(n) if st[j] == M}
    Cs = {("s", j) for j in range(n) if st[j] == C}
    if st[i] == U:       # blocks 3 and 6
        got = Ux | Ms | Cs
        if copy == "s":
            got = (got - {("x", i)}) | {("s", i)}
    elif st[i] == C:     # blocks 2 and 5 with Eq. 3
        hi = {("x", j) for j in range(n) if st[j] == C and cf[i] <= cf[j]}
        lo = {("s", j) for j in range(n) if st[j] == C and not cf[i] <= cf[j]}
        got = Ux | hi | lo | Ms
        if copy == "s":
            got = (got - {("x", i)}) | {("s", i)}
    else:
        if copy == "x":  # block 1
            got = Ux | Cx | Mx
        else:            # block 4
            got = Ux | Cs | Ms
    # positions outside the block have no shadow row: the s-copy falls back to x
    return {("x", j) if (c == "s" and not lay.block_start <= j < lay.block_start + lay.block_len)
            else (c, j) for c, j in got}


@pytest.mark.parametrize("B", [1, 2, 3, 4])
def test_mask_brute_force_against_paper_sets(B):
    """Every row's attended set equals the set the paper's rules list, for all 3^B state
    vectors and every order of confidences including ties (Sec. 3.2, Eq. 3)."""
    levels = [0.6, 0.7, 0.8]
    conf_choices = list(itertools.product(levels[:min(B, 3)], repeat=B))
    for states in itertools.product([M, C, U], repeat=B):
        for confs in conf_choices:
            lay = _layout(states, confs, prompt=2, future=1)
            mask = orc.attention_mask(lay)
            st = orc.position_states(lay)
            cf = orc.position_conf(lay)
            for r in range(lay.rows):
                copy, i = ("x", r) if r < lay.n_orig else ("s", int(lay.shadow_src[r - lay.n_orig]))
                assert _attended(lay, mask, r) == _paper_sets(lay, copy, i, st, cf), (states, confs, r)


def test_u_queries_never_see_candidates_in_x():
    """Sec. 3.2: U verification excludes uncertain C tokens from the context."""
    rng = np.random.default_rng(2)
    for _ in range(20):
        lay = _rand_layout(rng)
        mask = orc.attention_mask(lay)
        st = orc.position_states(lay)
        for r in range(lay.rows):
            copy, i = ("x", r) if r < lay.n_orig else ("s", int(lay.shadow_src[r - lay.n_orig]))
            if st[i] != U:
                continue
            for c, j in _attended(lay, mask, r):
                if st[j] == C:
                    assert c == "s"


def test_shadow_query_never_sees_own_original_key():
    """Sec. 3.2: a shadow query s^i is blocked from x^i (no leak of the token it verifies)."""
    rng = np.random.default_rng(3)
    for _ in range(20):
        lay = _rand_layout(rng)
        mask = orc.attention_mask(lay)
        for k in range(lay.n_shadow):
            i = int(lay.shadow_src[k])
            assert ("x", i) not in _attended(lay, mask, lay.n_orig + k)
            assert ("s", i) in _attended(lay, mask, lay.n_orig + k)


def test_confidence_order_is_autoregressive():
    """Eq. 4 / Appendix E: with distinct confidences, the shadow query of the k-th C token in
    descending-confidence order sees, among C tokens, exactly the x copies of the k-1 tokens
    before it."""
    rng = np.random.default_rng(4)
    for _ in range(20):
        B = 10
        st = rng.integers(0, 3, size=B)
        cf = rng.permutation(np.linspace(0.55, 0.75, B)).astype(np.float32)
        lay = _layout(st, cf, prompt=3, future=2)
        mask = orc.attention_mask(lay)
        b0 = lay.block_start
        cands = [b0 + p for p in range(B) if st[p] == C]
        order = sorted(cands, key=lambda j: -cf[j - b0])
        for k, i in enumerate(order):
            row = lay.n_orig + (i - b0)
            seen_c_in_x = {j for c, j in _attended(lay, mask, row) if c == "x" and j in cands}
            assert seen_c_in_x == set(order[:k])


def test_l2r_special_case():
    """Sec. 4.3 (l2r variant): when c_{t-1} decreases with position, the C-to-C part of
    Eq. 3 for original queries is left-to-right causal (x^j visible iff j <= i)."""
    B = 8
    st = [C] * B
    cf = np.linspace(0.79, 0.51, B).astype(np.float32)
    lay = _layout(st, cf, prompt=2, future=0)
    mask = orc.attention_mask(lay)
    b0 = lay.block_start
    for p in range(B):
        seen = {j for c, j in _attended(lay, mask, b0 + p) if c == "x" and j >= b0}
        assert seen == {b0 + q for q in range(p + 1)}


def test_masked_query_blocks_1_and_4():
    """Sec. 3.2: M queries in x see C and U keys in x; M queries in s see U keys in x and
    C keys in s."""
    rng = np.random.default_rng(5)
    for _ in range(20):
        lay = _rand_layout(rng)
        mask = orc.attention_mask(lay)
        st = orc.position_states(lay)
        b0, B = lay.block_start, lay.block_len
        for p in range(B):
            if st[b0 + p] != M:
                continue
            xs = _attended(lay, mask, b0 + p)
            ss = _attended(lay, mask, lay.n_orig + p)
            for j in range(lay.n_orig):
                if st[j] in (C, U):
                    assert ("x", j) in xs
                if st[j] == U:
                    assert ("x", j) in ss
                if st[j] == C:
                    assert ("s", j) in ss


def test_missing_shadow_row_falls_back_to_x():
    """Candidates-only shadow layout: a position without shadow row is seen in x by all."""
    lay = _layout([M, C, U, C, M], [0.1, 0.6, 0.9, 0.7, 0.2], prompt=2, future=1,
                  shadow="candidates")
    mask = orc.attention_mask(lay)
    for r in range(lay.rows):
        seen = _attended(lay, mask, r)
        for j in (2, 4, 6):  # block positions of the M, U, M tokens
            assert ("x", j) in seen


# ---------------------------------------------------------------------------------------
# Attention values
# ---------------------------------------------------------------------------------------
def _sdpa_torch(q, k, v, mask=None, scale=None):
    """Library softmax attention (torch CPU, float64); q [R,H,d], k/v [R,Hkv,d]."""
    hq, hkv = q.shape[1], k.shape[1]
    qt = torch.from_numpy(q.astype(np.float64)).permute(1, 0, 2)
    kt = torch.from_numpy(k.astype(np.float64)).permute(1, 0, 2).repeat_interleave(hq // hkv, 0)
    vt = torch.from_numpy(v.astype(np.float64)).permute(1, 0, 2).repeat_interleave(hq // hkv, 0)
    am = None if mask is None else torch.from_numpy(mask)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=am, scale=scale)
    return o.permute(1, 0, 2).numpy()


def test_identical_shadow_kv_equals_unmasked_attention():
    """If every shadow row carries the same key/value as its original row, each query sees
    one copy of every position and its output is plain attention over x (library SDPA)."""
    rng = np.random.default_rng(6)
    lay = _rand_layout(rng, B=10, prompt=9, future=6)
    R, n, hq, hkv, d = lay.rows, lay.n_orig, 4, 2, 16
    q = rng.standard_normal((R, hq, d))
    k = rng.standard_normal((R, hkv, d))
    v = rng.standard_normal((R, hkv, d))
    k[n:] = k[lay.shadow_src]
    v[n:] = v[lay.shadow_src]
    got = orc.masked_attention(q, k, v, orc.attention_mask(lay))
    want = _sdpa_torch(q, k[:n], v[:n])
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def test_masked_attention_matches_library_sdpa_with_dense_mask():
    """The fp64 masked softmax attention equals torch's SDPA given the same boolean mask,
    including grouped-query heads (Hq = 3 Hkv) and a non-default scale."""
    rng = np.random.default_rng(7)
    lay = _rand_layout(rng, B=9, prompt=5, future=4, shadow="candidates")
    R, hq, hkv, d = lay.rows, 6, 2, 8
    q = rng.standard_normal((R, hq, d))
    k = rng.standard_normal((R, hkv, d))
    v = rng.standard_normal((R, hkv, d))
    mask = orc.attention_mask(lay)
    for scale in (None, 0.3):
        got = orc.masked_attention(q, k, v, mask, scale=scale)
        want = _sdpa_torch(q, k, v, mask=mask, scale=scale)
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    rows = np.array([0, 3, R - 1])
    sub = orc.attention_mask(lay, rows=rows)
    assert (sub == mask[rows]).all()
    np.testing.assert_allclose(orc.masked_attention(q, k, v, sub, rows=rows),
                               orc.masked_attention(q, k, v, mask)[rows], atol=0)


def test_attention_rows_are_convex_combinations():
    """Softmax weights are positive and sum to one: every output coordinate lies within the
    range of the attended values."""
    rng = np.random.default_rng(8)
    lay = _rand_layout(rng)
    R, hq, d = lay.rows, 2, 8
    q = 3 * rng.standard_normal((R, hq, d))
    k = rng.standard_normal((R, hq, d))
    v = rng.standard_normal((R, hq, d))
    mask = orc.attention_mask(lay)
    o = orc.masked_attention(q, k, v, mask)
    for r in range(R):
        att = np.flatnonzero(mask[r])
        lo = v[att].min(axis=0) - 1e-12
        hi = v[att].max(axis=0) + 1e-12
        assert ((o[r] >= lo) & (o[r] <= hi)).all()


# ---------------------------------------------------------------------------------------
# RoPE of the augmented sequence (R20; Sec. 3.1: x^i and s^i share one position)
# ---------------------------------------------------------------------------------------
@pytest.mark.parametrize("style", [orc.ROPE_INTERLEAVED, orc.ROPE_HALF])
def test_rope_position_zero_is_identity(style):
    rng = np.random.default_rng(30)
    x = rng.standard_normal((5, 3, 16))
    assert np.array_equal(orc.rope(x, np.zeros(5, np.int64), 10000.0, style), x)


def test_rope_single_pair_closed_form():
    """d = 2: one pair at frequency theta^0 = 1, so position p turns (1, 0) into
    (cos p, sin p) and (0, 1) into (-sin p, cos p), a counter-clockwise rotation by p."""
    x = np.array([[[1.0, 0.0]], [[0.0, 1.0]], [[3.0, -2.0]]])
    for p in (1, 2, 7, 100, 4095):
        got = orc.rope(x, np.full(3, p), 500000.0)
        c, s = math.cos(p), math.sin(p)
        np.testing.assert_allclose(got[0, 0], [c, s], atol=1e-15)
        np.testing.assert_allclose(got[1, 0], [-s, c], atol=1e-15)
        np.testing.assert_allclose(got[2, 0], [3 * c + 2 * s, 3 * s - 2 * c], atol=1e-13)


@pytest.mark.parametrize("style", [orc.ROPE_INTERLEAVED, orc.ROPE_HALF])
def test_rope_frequency_of_each_pair(style):
    """d = 8, theta = 16: pair i turns at f_i = 16^(-2i/8) = 2^(-i) radians per position.
    A unit vector on the first element of pair i comes back as (cos(p 2^-i), sin(p 2^-i))
    on that pair's two elements (2i, 2i+1 interleaved; i, i+4 half) and zero elsewhere."""
    d, p = 8, 5
    for i in range(d // 2):
        a, b = (2 * i, 2 * i + 1) if style == orc.ROPE_INTERLEAVED else (i, i + d // 2)
        x = np.zeros((1, 1, d))
        x[0, 0, a] = 1.0
        want = np.zeros(d)
        want[a], want[b] = math.cos(p * 2.0 ** -i), math.sin(p * 2.0 ** -i)
        np.testing.assert_allclose(orc.rope(x, np.array([p]), 16.0, style)[0, 0], want,
                                   atol=1e-15)


@pytest.mark.parametrize("style", [orc.ROPE_INTERLEAVED, orc.ROPE_HALF])
def test_rope_preserves_every_pair_norm(style):
    rng = np.random.default_rng(31)
    d = 32
    x = rng.standard_normal((40, 2, d))
    pos = rng.integers(0, 1 << 20, size=40)
    y = orc.rope(x, pos, 10000.0, style)
    if style == orc.ROPE_INTERLEAVED:
        nx = x[..., 0::2] ** 2 + x[..., 1::2] ** 2
        ny = y[..., 0::2] ** 2 + y[..., 1::2] ** 2
    else:
        nx = x[..., :d // 2] ** 2 + x[..., d // 2:] ** 2
        ny = y[..., :d // 2] ** 2 + y[..., d // 2:] ** 2
    np.testing.assert_allclose(ny, nx, rtol=1e-12)


def test_rope_scores_depend_on_position_differences():
    """The defining property of RoPE, from complex arithmetic: with pair i read as
    z = x_2i + j x_2i+1, <rope(q, p1), rope(k, p2)> = Re sum_i z_q conj(z_k) e^(j (p1-p2) f_i)."""
    rng = np.random.default_rng(32)
    d, theta = 16, 10000.0
    q = rng.standard_normal((6, 1, d))
    k = rng.standard_normal((6, 1, d))
    p1 = rng.integers(0, 5000, size=6)
    p2 = rng.integers(0, 5000, size=6)
    got = (orc.rope(q, p1, theta) * orc.rope(k, p2, theta)).sum(-1)[:, 0]
    zq = q[:, 0, 0::2] + 1j * q[:, 0, 1::2]
    zk = k[:, 0, 0::2] + 1j * k[:, 0, 1::2]
    f = np.array([theta ** (-2.0 * i / d) for i in range(d // 2)])
    want = np.real((zq * np.conj(zk) * np.exp(1j * (p1 - p2)[:, None] * f)).sum(-1))
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-11)


def test_rope_half_pairing_is_a_permuted_interleaved_pairing():
    """Pairing (i, i + d/2) equals pairing (2i, 2i + 1) on the columns reordered as
    0, d/2, 1, d/2 + 1, ..."""
    rng = np.random.default_rng(33)
    d = 12
    x = rng.standard_normal((7, 3, d))
    pos = rng.integers(0, 3000, size=7)
    perm = np.ravel(np.column_stack([np.arange(d // 2), np.arange(d // 2) + d // 2]))
    inter = orc.rope(x[..., perm], pos, 500000.0, orc.ROPE_INTERLEAVED)
    back = np.empty_like(inter)
    back[..., perm] = inter
    np.testing.assert_allclose(orc.rope(x, pos, 500000.0, orc.ROPE_HALF), back, atol=1e-14)


def test_row_positions_put_shadow_rows_at_their_source():
    lay = _rand_layout(np.random.default_rng(34), B=10, prompt=6, future=3, shadow="candidates")
    pos = orc.row_positions(lay)
    assert np.array_equal(pos[:lay.n_orig], np.arange(lay.n_orig))
    assert np.array_equal(pos[lay.n_orig:], lay.shadow_src)


@pytest.mark.parametrize("style", [orc.ROPE_INTERLEAVED, orc.ROPE_HALF])
def test_rope_attention_with_shared_positions(style):
    """Two consequences pinned end to end. (1) Shifting every position by one constant
    leaves the RoPE attention unchanged. (2) Shadow rows that carry the keys and values of
    their source rows, rotated at their source positions, give plain RoPE attention over x
    (library SDPA on the rotated original rows), as with no RoPE."""
    rng = np.random.default_rng(35)
    lay = _rand_layout(rng, B=10, prompt=9, future=6)
    R, n, hq, hkv, d = lay.rows, lay.n_orig, 4, 2, 16
    q = rng.standard_normal((R, hq, d))
    k = rng.standard_normal((R, hkv, d))
    v = rng.standard_normal((R, hkv, d))
    pos = orc.row_positions(lay)
    mask = orc.attention_mask(lay)
    a = orc.masked_attention(orc.rope(q, pos, 100.0, style), orc.rope(k, pos, 100.0, style), v, mask)
    b = orc.masked_attention(orc.rope(q, pos + 777, 100.0, style),
                             orc.rope(k, pos + 777, 100.0, style), v, mask)
    np.testing.assert_allclose(a, b, atol=1e-12)
    k[n:] = k[lay.shadow_src]
    v[n:] = v[lay.shadow_src]
    qr, kr = orc.rope(q, pos, 100.0, style), orc.rope(k, pos, 100.0, style)
    got = orc.masked_attention(qr, kr, v, mask)
    want = _sdpa_torch(qr, kr[:n], v[:n])
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


# ---------------------------------------------------------------------------------------
# Scoring: Eq. 1, Eq. 5-8, Algorithm 1
# ---------------------------------------------------------------------------------------
def test_confidence_closed_forms():
    """Eq. 1 on rows with closed-form softmax maxima."""
    V = 1000
    c, tok, ok = orc.confidence(np.full(V, 2.5, dtype=np.float32))
    assert ok and tok == 0 and abs(c - 1.0 / V) < 1e-15
    a, b = 4.0, -1.0
    row = np.full(V, b, dtype=np.float32)
    row[637] = a
    c, tok, ok = orc.confidence(row)
    assert tok == 637 and abs(c - 1.0 / (1.0 + (V - 1) * math.exp(b - a))) < 1e-14
    # a row built as log-probabilities returns the planted probability
    p = np.full(V, 0.3 / (V - 1))
    p[5] = 0.7
    c, tok, ok = orc.confidence(np.log(p))
    assert tok == 5 and abs(c - 0.7) < 1e-12


def test_confidence_ties_lowest_index_and_bruteforce():
    rng = np.random.default_rng(9)
    row = rng.standard_normal(50).astype(np.float32)
    row[[7, 19, 33]] = row.max() + 1.0
    c, tok, ok = orc.confidence(row)
    assert tok == 7
    for _ in range(50):
        x = (rng.standard_normal(int(rng.integers(2, 12))) * 3).astype(np.float32)
        es = [math.exp(float(t)) for t in x]
        want = max(es) / math.fsum(es)
        c, tok, ok = orc.confidence(x)
        assert abs(c - want) < 1e-14
        assert tok == int(np.argmax(x))
        assert abs(c - scipy.special.softmax(x.astype(np.float64)).max()) < 1e-14


def test_confidence_invalid_rows():
    """Reading R6: non-finite normaliser -> (0, -1, invalid)."""
    for bad in ([1.0, np.nan, 0.0], [1.0, np.inf, 0.0], [-np.inf, -np.inf]):
        assert orc.confidence(np.array(bad, dtype=np.float32)) == (0.0, -1, False)
    c, tok, ok = orc.confidence(np.array([-np.inf, 0.0, -np.inf], dtype=np.float32))
    assert ok and tok == 1 and c == 1.0


def test_state_transition_boundaries():
    """Eq. 8 with its inclusive upper bounds."""
    tc, tu = 0.5, 0.8
    assert orc.next_state(0.5, tc, tu) == M
    assert orc.next_state(np.nextafter(0.5, 1.0), tc, tu) == C
    assert orc.next_state(0.8, tc, tu) == C
    assert orc.next_state(np.nextafter(0.8, 1.0), tc, tu) == U
    assert orc.next_state(0.0, tc, tu) == M
    assert orc.next_state(1.0, tc, tu) == U
    assert orc.next_state(0.6, 0.6, 0.6) == M and orc.next_state(0.61, 0.6, 0.6) == U


def test_paper_constants_golden():
    g = json.load(open(os.path.join(GOLDEN, "paper_constants.json")))
    assert abs(orc.LAMBDA_DEFAULT - g["lambda_printed"]) < 5e-4
    assert abs(orc.LAMBDA_DEFAULT ** 8 - 0.5) < 1e-15  # halves every 8 positions
    assert orc.P0_DEFAULT == g["p0"]


def test_mixing_weight_closed_forms():
    """Eq. 5-6 on cases with closed forms."""
    lam, p0 = orc.LAMBDA_DEFAULT, orc.P0_DEFAULT
    assert orc.mixing_weight(3, [], [], lam, p0)[0] == 1.0           # no outcomes -> w = 1
    assert orc.mixing_weight(3, [4], [], lam, p0)[0] == 1.0          # promotion only -> 1
    w, P, D = orc.mixing_weight(3, [], [4], lam, p0)
    assert P == 0 and abs(D - 0.5 ** (1 / 8)) < 1e-15
    assert abs(w - 0.1 / (0.5 ** (1 / 8) + 0.1)) < 1e-15            # 0.09833...
    w, P, D = orc.mixing_weight(10, [2], [18], lam, p0)              # symmetric outcomes
    x = 0.5 ** (8 / 8)
    assert abs(P - x) < 1e-15 and abs(D - x) < 1e-15
    assert abs(w - (x + p0) / (2 * x + p0)) < 1e-15
    # nearer demotion outweighs a farther promotion
    assert orc.mixing_weight(5, [13], [6], lam, p0)[0] < 0.5


def test_mixing_example_golden():
    """Appendix C.1 worked example (reading in tests/golden/mixing_example.json)."""
    g = json.load(open(os.path.join(GOLDEN, "mixing_example.json")))
    i, D = g["query_position"], g["demoted_in_window"]
    lam, p0 = orc.LAMBDA_DEFAULT, orc.P0_DEFAULT
    w_window = orc.mixing_weight(i, [], D, lam, p0)[0]
    assert abs(w_window - 0.1 / (lam ** 4 + lam + 0.1)) < 1e-15
    assert round(w_window, 2) != g["printed_w"]
    for dist in range(6, 16):
        w = orc.mixing_weight(i, [i + dist], D, lam, p0)[0]
        assert (round(w, 2) == g["printed_w"]) == (dist == 10), (dist, w)


def test_mix_logits_endpoints():
    """Eq. 7: w = 1 gives the original logits, w = 0 the shadow logits, and in between the
    float32 result is within one rounding of the exact convex combination."""
    rng = np.random.default_rng(10)
    lx = (rng.standard_normal(4096) * 3).astype(np.float32)
    ls = (rng.standard_normal(4096) * 3).astype(np.float32)
    # bf16-valued inputs make lx - ls exact, so the endpoints are exact
    lx = lx.astype(np.float32).view(np.uint32) & np.uint32(0xFFFF0000)
    ls = ls.astype(np.float32).view(np.uint32) & np.uint32(0xFFFF0000)
    lx, ls = lx.view(np.float32), ls.view(np.float32)
    assert (orc.mix_logits(lx, ls, np.float32(1.0)) == lx).all()
    assert (orc.mix_logits(lx, ls, np.float32(0.0)) == ls).all()
    for w in (0.25, 0.5, 0.917):
        exact = w * lx.astype(np.float64) + (1 - w) * ls.astype(np.float64)
        got = orc.mix_logits(lx, ls, np.float32(w)).astype(np.float64)
        assert np.abs(got - exact).max() <= 2 * np.abs(exact).max() * 2.0 ** -23


def _peaked_row(V, p, col):
    q = np.full(V, (1.0 - p) / (V - 1))
    q[col] = p
    return np.log(q).astype(np.float32)


def test_score_block_algorithm1_order():
    """Algorithm 1: C rows feed P (-> U) and D (-> M); a demoted U row is not in D; M rows
    use this step's P and D; counts are conserved."""
    V, tc, tu = 64, 0.5, 0.8
    state = np.array([C, C, U, M, U, M], dtype=np.uint8)
    target = [0.95, 0.2, 0.1, None, 0.6, None]  # c from the shadow logits
    ls = np.zeros((6, V), dtype=np.float32)
    lx = np.zeros((6, V), dtype=np.float32)
    for r, p in enumerate(target):
        if p is not None:
            ls[r] = _peaked_row(V, p, col=r + 1)
    # M rows: original logits peak at col 40 (p=0.9), shadow logits at col 50 (p=0.9)
    for r in (3, 5):
        lx[r] = _peaked_row(V, 0.9, 40)
        ls[r] = _peaked_row(V, 0.9, 50)
    res = orc.score_block(lx, ls, state, tc, tu)
    assert res.promoted == [0] and res.demoted == [1]       # row 2 (U -> M) not in D
    assert list(res.state_out[[0, 1, 2, 4]]) == [U, M, M, C]
    for r in (0, 1, 2, 4):
        assert abs(res.conf[r] - target[r]) < 1e-6 and res.token[r] == r + 1
    lam, p0 = orc.LAMBDA_DEFAULT, orc.P0_DEFAULT
    for r in (3, 5):
        w = (lam ** abs(r - 0) + p0) / (lam ** abs(r - 0) + lam ** abs(r - 1) + p0)
        assert abs(res.w[r] - np.float32(w)) == 0
        assert res.token[r] == (40 if w > 0.5 else 50)
    assert res.counts.sum() == 6
    assert set(res.promoted).isdisjoint(res.demoted)
    assert np.isnan(res.w[[0, 1, 2, 4]]).all()


def test_score_block_fixed_weight_special_cases():
    """With no C tokens (P = D = {}), w = 1 and M rows are decided by the original logits
    alone (Sec. 4.3, w = 1 variant)."""
    rng = np.random.default_rng(11)
    V = 128
    state = np.array([M, U, M, M], dtype=np.uint8)
    # bf16-valued logits, so that lx - ls and hence the w = 1 mixture are exact
    lx = ((rng.standard_normal((4, V)) * 2).astype(np.float32).view(np.uint32)
          & np.uint32(0xFFFF0000)).view(np.float32)
    ls = ((rng.standard_normal((4, V)) * 2).astype(np.float32).view(np.uint32)
          & np.uint32(0xFFFF0000)).view(np.float32)
    res = orc.score_block(lx, ls, state, 0.4, 0.9)
    for r in (0, 2, 3):
        assert res.w[r] == 1.0
        c, tok, _ = orc.confidence(lx[r])
        assert res.token[r] == tok and abs(res.conf[r] - c) < 1e-15


# ---------------------------------------------------------------- R16, R17 (p_cur, tokens)
def test_token_probability_closed_forms():
    """A uniform row gives 1/V to every token; a planted row gives p to the peak and
    (1 - p)/(V - 1) to the rest (float32 rounding of the log only)."""
    V = 50
    u = np.zeros(V, np.float32)
    for tok in (0, 17, V - 1):
        assert abs(orc.token_probability(u, tok) - 1.0 / V) < 1e-15
    row = _peaked_row(V, 0.73, col=9)
    assert abs(orc.token_probability(row, 9) - 0.73) < 1e-6
    assert abs(orc.token_probability(row, 3) - 0.27 / (V - 1)) < 1e-7


def test_token_probability_against_library_softmax():
    rng = np.random.default_rng(5)
    for V in (1, 2, 7, 300):
        row = (rng.standard_normal(V) * 3).astype(np.float32)
        ref = scipy.special.softmax(row.astype(np.float64))
        got = np.array([orc.token_probability(row, t) for t in range(V)])
        np.testing.assert_allclose(got, ref, rtol=1e-12, atol=0)
        c, tok, _ = orc.confidence(row)
        assert got[tok] == pytest.approx(c, rel=1e-12)   # Eq. 1: c = p(x^)


def test_token_probability_out_of_range_and_invalid_rows():
    row = np.zeros(8, np.float32)
    assert orc.token_probability(row, -1) == 0.0 and orc.token_probability(row, 8) == 0.0
    bad = row.copy()
    bad[2] = np.nan
    assert orc.token_probability(bad, 0) == 0.0
    assert orc.token_probability(np.full(8, -np.inf, np.float32), 0) == 0.0


def test_score_block_p_cur_uses_the_scored_distribution():
    """C/U rows: p_cur on the shadow logits; M rows: on the mixed logits (with no C rows,
    w = 1 and the mixture is the original logits)."""
    rng = np.random.default_rng(12)
    V = 96
    state = np.array([M, U, M, U], dtype=np.uint8)
    lx = ((rng.standard_normal((4, V)) * 2).astype(np.float32).view(np.uint32)
          & np.uint32(0xFFFF0000)).view(np.float32)
    ls = ((rng.standard_normal((4, V)) * 2).astype(np.float32).view(np.uint32)
          & np.uint32(0xFFFF0000)).view(np.float32)
    cur = np.array([3, 40, V, 0], np.int32)
    res = orc.score_block(lx, ls, state, 0.4, 0.9, cur_token=cur)
    assert res.p_cur[0] == pytest.approx(scipy.special.softmax(lx[0].astype(np.float64))[3], rel=1e-12)
    assert res.p_cur[1] == pytest.approx(scipy.special.softmax(ls[1].astype(np.float64))[40], rel=1e-12)
    assert res.p_cur[2] == 0.0                                   # token outside the vocabulary
    assert res.p_cur[3] == pytest.approx(scipy.special.softmax(ls[3].astype(np.float64))[0], rel=1e-12)


def test_next_tokens_fill_and_mask():
    """The last line of Algorithm 1's step: C and U positions take x^, M positions the mask."""
    tok = np.array([5, 7, 9, -1])
    st = np.array([M, C, U, M], np.uint8)
    assert list(orc.next_tokens(tok, st, 126336)) == [126336, 7, 9, 126336]
    V = 32
    rows = np.stack([_peaked_row(V, p, col=c) for p, c in ((0.95, 4), (0.6, 8), (0.1, 12))])
    res = orc.score_block(rows, rows, np.array([U, C, U], np.uint8), 0.5, 0.8, mask_token=-7)
    assert list(res.state_out) == [U, C, M]
    assert list(res.tokens_next) == [4, 8, -7]


# ---------------------------------------------------------------- R18 (ordering variants)
def test_entropy_and_margin_closed_forms():
    V = 40
    u = np.zeros(V, np.float32)
    assert orc.entropy(u) == pytest.approx(math.log(V), rel=1e-12)
    assert orc.margin(u) == 0.0
    p = 0.7
    row = _peaked_row(V, p, col=5)
    q = (1 - p) / (V - 1)
    assert orc.entropy(row) == pytest.approx(-p * math.log(p) - (1 - p) * math.log(q), rel=1e-6)
    assert orc.margin(row) == pytest.approx(p - q, rel=1e-6)
    two = np.zeros(V, np.float32)
    two[[3, 9]] = 4.0                               # a repeated maximum: margin 0
    assert orc.margin(two) == 0.0
    assert orc.entropy(np.zeros(1, np.float32)) == 0.0 and orc.margin(np.zeros(1, np.float32)) == 1.0
    bad = u.copy()
    bad[0] = np.nan
    assert orc.entropy(bad) == 0.0 and orc.margin(bad) == 0.0


def test_entropy_and_margin_against_library():
    rng = np.random.default_rng(8)
    for V in (2, 17, 500):
        row = (rng.standard_normal(V) * 2.5).astype(np.float32)
        p = scipy.special.softmax(row.astype(np.float64))
        assert orc.entropy(row) == pytest.approx(float(scipy.stats.entropy(p)), rel=1e-10)
        srt = np.sort(p)
        assert orc.margin(row) == pytest.approx(srt[-1] - srt[-2], rel=1e-10)


def test_order_keys_reproduce_the_ablation_orderings():
    """Eq. 3 with the R18 keys: equal keys make every C pair mutual (bidirectional); minus
    the position gives left-to-right causal order among C positions."""
    B = 6
    st = np.full(B, C, np.uint8)
    for mode, want in ((orc.ORDER_BIDIR, lambda i, j: True), (orc.ORDER_L2R, lambda i, j: j <= i)):
        keys = np.array([orc.order_key(mode, 0.5, 1.0, 0.2, i) for i in range(B)], np.float32)
        for i in range(B):
            sees_shadow = orc.sees_shadow_copy("x", i, st, keys)
            for j in range(B):
                if j != i:
                    assert (not sees_shadow[j]) == want(i, j), (mode, i, j)
    assert orc.order_key(orc.ORDER_CONFIDENCE, 0.7, 2.0, 0.1, 3) == 0.7
    assert orc.order_key(orc.ORDER_ENTROPY, 0.7, 2.0, 0.1, 3) == -2.0
    assert orc.order_key(orc.ORDER_MARGIN, 0.7, 2.0, 0.1, 3) == 0.1


# ---------------------------------------------------------------- near-tie gap, reading R7
def test_top2_gap_closed_forms():
    """The near-tie exclusion of the parity checks (reading R5: argmax ties go to the lowest
    index, so a gap under rounding may flip it): the gap is the largest entry minus the
    second largest, a repeated maximum gives 0, a single entry gives inf."""
    assert orc.top2_gap(np.array([1.0, 5.0, 3.0], np.float32)) == 2.0
    assert orc.top2_gap(np.array([-4.0, -1.5, -9.0, -2.0], np.float32)) == 0.5
    assert orc.top2_gap(np.array([3.0, 7.0, 7.0], np.float32)) == 0.0
    assert orc.top2_gap(np.array([7.0, 1.0, 7.0, 7.0], np.float32)) == 0.0
    assert orc.top2_gap(np.array([2.5], np.float32)) == math.inf
    assert orc.top2_gap(np.array([-np.inf, 2.0], np.float32)) == math.inf
    # the gap is never negative, whatever the order of the entries
    assert orc.top2_gap(np.array([9.0, 8.0, 1.0], np.float32)) == 1.0


def test_top2_gap_brute_force():
    """Against the definition over all pairs: max over i != j of x_i - x_j restricted to
    i = an argmax, i.e. the maximum minus the largest entry at any other index."""
    rng = np.random.default_rng(41)
    for _ in range(200):
        V = int(rng.integers(2, 9))
        x = rng.integers(-3, 4, size=V).astype(np.float32) * np.float32(0.25)
        a = int(np.argmax(x))
        others = [float(x[j]) for j in range(V) if j != a]
        assert orc.top2_gap(x) == float(x[a]) - max(others)


@pytest.mark.parametrize("bad", [3, 7, 255])
def test_state_byte_above_two_is_masked(bad):
    """Reading R7: a state byte above 2 behaves exactly as M, in the mask (every query's
    attended set, Sec. 3.2) and in scoring (Algorithm 1: the row is mixed and decided as an
    M row and counted as M)."""
    rng = np.random.default_rng(43 + bad)
    for shadow in ("paper", "candidates"):
        lay = _rand_layout(rng, B=10, shadow=shadow)
        st = lay.state.copy()
        m_rows = np.flatnonzero(st == M)
        if len(m_rows) == 0:
            st[0] = M
            m_rows = np.array([0])
        ref = SeqLayout(lay.n_orig, lay.block_start, st, lay.prev_conf,
                        np.asarray(lay.shadow_src, np.int32) if shadow == "paper"
                        else lay.block_start + np.flatnonzero(st == C).astype(np.int32))
        bad_st = st.copy()
        bad_st[m_rows] = bad
        odd = SeqLayout(ref.n_orig, ref.block_start, bad_st, ref.prev_conf, ref.shadow_src)
        assert np.array_equal(orc.attention_mask(odd), orc.attention_mask(ref))
    V = 96
    state = np.array([M, C, U, M, C, M], np.uint8)
    lx = rng.standard_normal((6, V)).astype(np.float32)
    ls = rng.standard_normal((6, V)).astype(np.float32)
    ls[1, 5] += 9.0   # promoted C row
    ls[4, 7] -= 0.0   # C row that stays low (demoted)
    want = orc.score_block(lx, ls, state, 0.4, 0.9)
    odd_state = state.copy()
    odd_state[[0, 5]] = bad
    got = orc.score_block(lx, ls, odd_state, 0.4, 0.9)
    assert np.array_equal(got.state_out, want.state_out)
    assert np.array_equal(got.token, want.token)
    assert np.array_equal(got.conf, want.conf)
    assert np.array_equal(got.w, want.w, equal_nan=True)
    assert list(got.counts) == list(want.counts)
    assert got.promoted == want.promoted and got.demoted == want.demoted
