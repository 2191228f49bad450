"""GPU parity of dard_step_attention against the CPU oracle (Eq. 2-3, Sec. 3.2 blocks 1-6)."""
import numpy as np
import pytest
import torch

from paper_2608_26574_gb300 import workloads as W
from paper_2608_26574_gb300.device import DeviceStep

from . import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(params=["1", "2", "4"])
def tc(request, monkeypatch):
    """Runs the test once per tensor-core kernel: one or two query tiles per CTA (1, 2), and
    the CTA-pair kernel (4, head_dim 128; head_dim 64 falls back to the model's choice)."""
    monkeypatch.setenv("DARD_ATTN_TC", request.param)
    return request.param


def _attend(wl, layer=0, scale=0.0):
    ds = DeviceStep(wl, layers=[layer], scoring=False)
    o = ds.attention(0, scale=scale)
    torch.cuda.synchronize()
    return ds, o.float().cpu().numpy()


@pytest.mark.parametrize("name,layout,sample", [
    ("tiny", "paper", None), ("tiny", "candidates", None),
    ("8b", "paper", None), ("8b", "candidates", None),
    ("gqa", "paper", 192), ("gqa", "candidates", 192),
    ("ragged", "paper", 48), ("mm", "paper", 64),
])
def test_attention_configs(name, layout, sample, tc):
    wl = W.make(name, layout=layout, scoring=False, layers=2 if name == "mm" else None)
    layers = [0, 1] if name == "mm" else [0]
    for li in layers:
        ds, o = _attend(wl, li)
        mx, mean, n = P.compare_attention(wl, li, o, sample=sample)
        print(name, layout, li, "max", mx, "mean", mean, "rows", n)
        assert mx <= P.ATT_MAX_ABS and mean <= P.ATT_MEAN_ABS
        assert int(ds.status.item()) == 0


def _probe_tol(wl):
    # Q = 0: every attended key has weight 1/N, so a single wrong key moves the output by
    # |v_a - v_b| / N >> this tolerance (bf16 output rounding and fp32 sums stay far below)
    n_min = min(s.n_orig for s in wl.seqs)
    return 0.25 / n_min


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("layout", ["paper", "candidates"])
def test_mask_probe_every_key(d, layout, tc):
    """Uniform attention (Q = 0) exposes every key selection of the in-kernel mask."""
    specs = [dict(n_orig=200, block_start=100, block_len=64, fractions=(0.3, 0.4, 0.3),
                  shadow=layout),
             dict(n_orig=131, block_start=0, block_len=37, fractions=(0.2, 0.5, 0.3), shadow=layout),
             dict(n_orig=97, block_start=60, block_len=37, fractions=(0.5, 0.3, 0.2), shadow=layout),
             dict(n_orig=300, block_start=172, block_len=128, fractions=(0.3, 0.4, 0.3),
                  shadow=layout)]
    wl = W.custom(specs, 4, 2, d, probe=True, seed=21 + d)
    ds, o = _attend(wl)
    mx, mean, n = P.compare_attention(wl, 0, o)
    print("probe", d, layout, mx, mean, n)
    assert mx <= _probe_tol(wl)


@pytest.mark.parametrize("d", [64, 128])
def test_mask_probe_last_tile_widths(d, tc):
    """Sequences whose last 128-key tile holds 1, 15, 16, 17, 48, 63, 64, 65, 100, 127 or
    128 keys (one tile only for the 100- and 17-row sequences): the keys past a sequence's
    end (the next sequence's rows, or past the tensor) must never be attended, and every
    key of the sequence exactly once (uniform attention, Q = 0)."""
    rows = [129, 271, 144, 145, 176, 319, 192, 321, 100, 255, 256, 17]
    specs = []
    for i, r in enumerate(rows):
        B = 8 if r < 64 else (16, 32)[i % 2]
        n = r - B  # "paper" layout: one shadow row per block position
        b0 = (n - B) if i % 3 == 0 else (n - B) // 2
        specs.append(dict(n_orig=n, block_start=b0, block_len=B, fractions=(0.3, 0.4, 0.3)))
    wl = W.custom(specs, 4, 2, d, probe=True, seed=61 + d)
    assert [s.n_orig + s.n_shadow for s in wl.seqs] == rows
    ds, o = _attend(wl)
    mx, mean, n = P.compare_attention(wl, 0, o)
    print("last tile widths", d, mx, mean, n)
    assert mx <= _probe_tol(wl)
    assert int(ds.status.item()) == 0


def test_attention_run_to_run_identical(tc):
    """Repeated launches on the same inputs give bit-identical outputs: the arithmetic has
    one fixed order, so any difference is a race in the pipeline (a buffer reused before
    its reader finished). A long multi-wave workload (GQA, 5184 rows, 41 key tiles per
    query tile) gives every barrier many phases."""
    wl = W.make("gqa", scoring=False, layers=1)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    q, k, v, _ = ds.layers[0]
    call = ds.attention_call()
    outs = []
    for _ in range(4):
        o = torch.full_like(q, float("nan"))
        call(q, k, v, o)
        torch.cuda.synchronize()
        outs.append(o)
    for o in outs[1:]:
        assert torch.equal(o, outs[0])
    assert int(ds.status.item()) == 0


@pytest.mark.parametrize("d", [64, 128])
def test_attention_fp32(d):
    """The fp32 CUDA-core kernel at both head dims: every key selection (uniform attention,
    Q = 0) and random values against the oracle, over two sequences with blocks, shadow rows
    in both layouts and grouped heads. fp32 throughout: the error stays near fp32 rounding."""
    specs = [dict(n_orig=150, block_start=60, block_len=40, fractions=(0.3, 0.4, 0.3)),
             dict(n_orig=70, block_start=0, block_len=33, fractions=(0.4, 0.3, 0.3),
                  shadow="candidates")]
    wl = W.custom(specs, 4, 2, d, dtype="f32", probe=True, seed=71 + d)
    _, o = _attend(wl)
    mx, _, _ = P.compare_attention(wl, 0, o)
    assert mx <= _probe_tol(wl)
    wl = W.custom(specs, 4, 2, d, dtype="f32", seed=81 + d, qkv_std=1.0)
    ds, o = _attend(wl)
    mx, mean, n = P.compare_attention(wl, 0, o)
    print("fp32", d, mx, mean, n)
    assert mx <= 2e-4
    assert int(ds.status.item()) == 0


def test_mask_probe_confidence_ties(tc):
    """Equal c_{t-1} among C tokens attend each other both ways (Eq. 3 uses <=)."""
    B = 48
    st = np.array([1] * 24 + [0] * 12 + [2] * 12, dtype=np.uint8)
    np.random.default_rng(0).shuffle(st)
    cf = np.where(st == 1, np.float32(0.65), np.float32(0.2)).astype(np.float32)
    cf[st == 2] = 0.95
    cf[np.flatnonzero(st == 1)[:8]] = 0.7
    specs = [dict(n_orig=160, block_start=70, state=st, prev_conf=cf)]
    wl = W.custom(specs, 2, 2, 128, probe=True, seed=5)
    _, o = _attend(wl)
    mx, _, _ = P.compare_attention(wl, 0, o)
    assert mx <= _probe_tol(wl)


@pytest.mark.parametrize("states", ["M", "C", "U"])
def test_mask_probe_uniform_states(states, tc):
    code = {"M": 0, "C": 1, "U": 2}[states]
    specs = [dict(n_orig=256, block_start=128, state=np.full(64, code, np.uint8))]
    wl = W.custom(specs, 2, 1, 128, probe=True, seed=code)
    _, o = _attend(wl)
    mx, _, _ = P.compare_attention(wl, 0, o)
    assert mx <= _probe_tol(wl)


@pytest.mark.parametrize("case", range(6))
def test_attention_fp32_random_shapes(case):
    """The fp32 CUDA-core kernel on seeded random ragged batches: sequences down to one row
    (key groups that see no key merge as empty), blocks anywhere, S = 0, grouped heads,
    both head dims, random query starts and score scales. fp32 throughout."""
    rng = np.random.default_rng(700 + case)
    specs = []
    for _ in range(int(rng.integers(1, 5))):
        n = int(rng.integers(1, 300))
        B_ = int(rng.integers(0, min(n, 64) + 1))
        b0 = int(rng.integers(0, n - B_ + 1))
        shadow = ["paper", "candidates", "none"][int(rng.integers(0, 3))]
        sp = dict(n_orig=n, block_start=b0, block_len=B_,
                  fractions=tuple(rng.dirichlet([1, 1, 1])))
        sp["shadow"] = np.zeros(0, np.int32) if shadow == "none" else shadow
        if rng.random() < 0.4:
            sp["query_start"] = int(rng.integers(0, n + 1))
        specs.append(sp)
    # a sequence of one to five rows: most key groups of its CTAs see no key
    specs.append(dict(n_orig=int(rng.integers(1, 6)), block_start=0, block_len=1,
                      fractions=(0.4, 0.3, 0.3)))
    hkv = int(rng.choice([1, 2]))
    hq = hkv * int(rng.choice([1, 3]))
    d = int(rng.choice([64, 128]))
    wl = W.custom(specs, hq, hkv, d, dtype="f32", seed=750 + case, qkv_std=float(rng.choice([0.2, 1.0])))
    scale = float(rng.choice([0.0, 0.3, 1.0]))
    ds, o = _attend(wl, scale=scale)
    if any(sq.query_start < sq.rows for sq in wl.seqs):
        mx, mean, n = P.compare_attention(wl, 0, o, scale=scale or None)
        vmax = max(1.0, float(np.abs(wl.v[0]).max()))
        print("fp32 random", case, [(sq.n_orig, sq.block_len, sq.n_shadow, sq.query_start)
                                    for sq in wl.seqs], hq, hkv, d, scale, mx, mean)
        assert mx <= 2e-4 * vmax
    assert int(ds.status.item()) == 0


@pytest.mark.parametrize("case", range(12))
def test_attention_random_shapes(case, tc):
    """Seeded random ragged batches: odd lengths, blocks at the start / end, S = 0,
    B = 1..128, grouped heads, larger scores (scale up to 1) to exercise the O rescale."""
    rng = np.random.default_rng(100 + case)
    specs = []
    for _ in range(int(rng.integers(1, 5))):
        n = int(rng.integers(1, 700))
        B = int(rng.integers(0, min(n, 128) + 1))
        b0 = int(rng.integers(0, n - B + 1))
        shadow = ["paper", "candidates", "none"][int(rng.integers(0, 3))]
        sp = dict(n_orig=n, block_start=b0, block_len=B,
                  fractions=tuple(rng.dirichlet([1, 1, 1])))
        sp["shadow"] = np.zeros(0, np.int32) if shadow == "none" else shadow
        specs.append(sp)
    hkv = int(rng.choice([1, 2, 4]))
    hq = hkv * int(rng.choice([1, 2, 3]))
    d = int(rng.choice([64, 128]))
    std = float(rng.choice([1.0 / np.sqrt(d), 0.5, 1.0]))
    wl = W.custom(specs, hq, hkv, d, seed=200 + case, qkv_std=std)
    scale = float(rng.choice([0.0, 0.3, 1.0]))
    ds, o = _attend(wl, scale=scale)
    mx, mean, n = P.compare_attention(wl, 0, o, scale=scale or None)
    print(case, [(s.n_orig, s.block_start, s.block_len, s.n_shadow) for s in wl.seqs],
          hq, hkv, d, std, scale, mx, mean)
    assert mx <= P.att_tol(wl) and mean <= P.ATT_MEAN_ABS


def test_attention_bad_shadow_rows_flagged(tc):
    """shadow_src outside the block or repeated: status bit, other rows still correct."""
    specs = [dict(n_orig=128, block_start=32, block_len=16, fractions=(0.4, 0.3, 0.3),
                  shadow=np.array([32, 33, 34, 34, 90, 35], np.int32))]
    wl = W.custom(specs, 2, 2, 128, seed=3)
    ds, o = _attend(wl)
    assert int(ds.status.item()) & 0x2
    # rows 0..127 of x: the oracle with the two bad shadow rows removed
    good = W.custom([dict(n_orig=128, block_start=32, state=wl.seqs[0].state,
                          prev_conf=wl.seqs[0].prev_conf, shadow=np.array([32, 33, 34, 35], np.int32))],
                    2, 2, 128, seed=3)
    keep = np.r_[0:128, 128, 129, 130, 133]
    good.q[0], good.k[0], good.v[0] = wl.q[0][keep], wl.k[0][keep], wl.v[0][keep]
    ref = P.oracle_attention(good, 0, 0)
    np.testing.assert_allclose(o[keep], ref, atol=P.ATT_MAX_ABS)


def _sentinel_out(ds):
    q = ds.layers[0][0]
    return torch.full_like(q, 7.0)


@pytest.mark.parametrize("name,sample", [("tiny", None), ("8b", None), ("gqa", 192),
                                         ("ragged", 48), ("mm", 64)])
def test_attention_prefix_cached(name, sample, tc):
    """Prefix caching (queries from the prompt's end on): the kept rows match the oracle,
    and the output rows of the cached prompt are left untouched."""
    wl = W.make(name, prefix=True, scoring=False, layers=1 if name == "mm" else None)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    out = _sentinel_out(ds)
    ds.attention(0, out=out)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy()
    mx, mean, n = P.compare_attention(wl, 0, o, sample=sample)
    print(name, "prefix", "max", mx, "mean", mean, "rows", n)
    assert mx <= P.ATT_MAX_ABS and mean <= P.ATT_MEAN_ABS
    offs = wl.row_offsets()
    for si, s in enumerate(wl.seqs):
        assert s.query_start == s.prompt > 0
        assert np.all(o[offs[si]:offs[si] + s.query_start] == 7.0)
    assert int(ds.status.item()) == 0


@pytest.mark.parametrize("case", range(6))
def test_attention_random_query_start(case, tc):
    """Random per-sequence query starts, including none (all rows) and the end (no rows)."""
    rng = np.random.default_rng(700 + case)
    specs = []
    for si in range(int(rng.integers(1, 5))):
        n = int(rng.integers(1, 600))
        B = int(rng.integers(0, min(n, 128) + 1))
        b0 = int(rng.integers(0, n - B + 1))
        sp = dict(n_orig=n, block_start=b0, block_len=B, fractions=tuple(rng.dirichlet([1, 1, 1])))
        rows = n + B
        sp["query_start"] = int(rng.choice([0, rows, int(rng.integers(0, rows + 1))]))
        specs.append(sp)
    hkv = int(rng.choice([1, 2]))
    d = int(rng.choice([64, 128]))
    wl = W.custom(specs, hkv * 2, hkv, d, seed=800 + case)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    out = _sentinel_out(ds)
    ds.attention(0, out=out)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy()
    if any(s.query_start < s.rows for s in wl.seqs):
        mx, mean, n = P.compare_attention(wl, 0, o)
        assert mx <= P.att_tol(wl) and mean <= P.ATT_MEAN_ABS
    offs = wl.row_offsets()
    for si, s in enumerate(wl.seqs):
        assert np.all(o[offs[si]:offs[si] + s.query_start] == 7.0)


@pytest.mark.parametrize("mode", ["bidir", "l2r"])
def test_attention_ordering_keys(mode, tc):
    """The ablation's orderings enter the mask as the Eq. 3 key in prev_conf: equal keys
    (every C pair mutual) and minus the block position (left-to-right among C). Uniform
    attention (Q = 0) exposes every key selection."""
    B = 64
    rng = np.random.default_rng(3 if mode == "bidir" else 4)
    st = rng.choice(np.array([0, 1, 2], np.uint8), size=B, p=[0.3, 0.5, 0.2])
    key = np.zeros(B, np.float32) if mode == "bidir" else -np.arange(B, dtype=np.float32)
    specs = [dict(n_orig=300, block_start=150, state=st, prev_conf=key)]
    wl = W.custom(specs, 2, 2, 128, probe=True, seed=9)
    _, o = _attend(wl)
    mx, _, _ = P.compare_attention(wl, 0, o)
    assert mx <= _probe_tol(wl)


def test_attention_maximum_batch(tc):
    """DARD_MAX_SEQS sequences with full 128-position blocks and their shadow rows."""
    rng = np.random.default_rng(91)
    specs = []
    for _ in range(256):
        n = int(rng.integers(128, 300))
        b0 = int(rng.integers(0, n - 128 + 1))
        specs.append(dict(n_orig=n, block_start=b0, block_len=128,
                          fractions=tuple(rng.dirichlet([1, 1, 1]))))
    wl = W.custom(specs, 2, 1, 64, seed=92)
    ds, o = _attend(wl)
    # a sample of rows per sequence, every block and shadow row of a few sequences
    mx, mean, n = P.compare_attention(wl, 0, o, sample=8)
    assert mx <= P.att_tol(wl) and mean <= P.ATT_MEAN_ABS
    assert int(ds.status.item()) == 0


def test_attention_no_query_rows(tc):
    """query_start at the end of every sequence: nothing is launched, the output is untouched."""
    specs = [dict(n_orig=90, block_start=10, block_len=16, fractions=(0.3, 0.4, 0.3),
                  query_start=106) for _ in range(2)]
    wl = W.custom(specs, 2, 2, 128, seed=93)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    out = _sentinel_out(ds)
    ds.attention(0, out=out)
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())


@pytest.mark.parametrize("d", [64, 128])
def test_mask_probe_skipped_shadow_tiles(d, tc):
    """Long runs of rows after the block (original queries of M positions attend x copies
    only, Sec. 3.2 query block 1): their CTAs skip the key tiles that hold only shadow rows.
    Uniform attention (Q = 0) shows that nothing they should see was skipped, and the host
    plan reports the skipped pairs."""
    specs = [dict(n_orig=700, block_start=100, block_len=64, fractions=(0.3, 0.4, 0.3)),
             dict(n_orig=900, block_start=0, block_len=128, fractions=(0.4, 0.3, 0.3)),
             dict(n_orig=640, block_start=200, block_len=32, fractions=(0.2, 0.5, 0.3),
                  shadow="candidates")]
    wl = W.custom(specs, 4, 2, d, probe=True, seed=31 + d)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    q, k, v, o = ds.layers[0]
    plan = ds.attention_call().plan(q, k, v, o)
    assert plan["tile_pairs_skipped"] > 0, plan
    o = ds.attention(0).float().cpu().numpy()
    torch.cuda.synchronize()
    mx, mean, n = P.compare_attention(wl, 0, o)
    # a wrongly skipped tile drops up to 64 attended keys of ~700 and moves a row's mean of
    # N(0, 1) values by ~1e-2; the bf16 output rounding (half an ulp: at most 2^-8 of |O|)
    # stays below 1.5 times that bound
    tol = max(_probe_tol(wl), 1.5 * 2.0 ** -8 * float(abs(o).max()))
    print("skip probe", d, plan, mx, mean, n, tol)
    assert mx <= tol
    assert int(ds.status.item()) == 0
