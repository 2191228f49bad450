"""GPU parity of dard_step_attention with RoPE applied in the call (rope_theta > 0).

Q and K arrive before RoPE; the call rotates the keys once into k_rope and each attention
kernel rotates its query tiles as it loads them, original row r at position r and shadow
row N + k at shadow_src[k] (Sec. 3.1: x^i and s^i share one positional embedding). The
oracle rotates q and k in float64 (R20) and runs the same masked attention. Two checks:
the rotated keys against the oracle's within one rounding to the storage type, and the
output against the oracle given the rotated operands in the precision the attention takes
them (bf16 for the tensor-core kernels: the bf16-input contract, 2e-2 max / 1e-2 mean).
The distance to the all-float64 composition is printed beside it.
"""
import numpy as np
import pytest
import torch

from paper_2608_26574_gb300 import binding as B
from paper_2608_26574_gb300 import workloads as W
from paper_2608_26574_gb300.device import DeviceStep

from . import parity as P

pytestmark = pytest.mark.gpu

THETA = 500000.0  # the RoPE base of LLaDA-8B-class models
IL, HALF = B.DARD_ROPE_INTERLEAVED, B.DARD_ROPE_HALF


@pytest.fixture(params=["1", "2", "4"])
def tc(request, monkeypatch):
    """Once per tensor-core kernel (4: the CTA-pair kernel, head_dim 128)."""
    monkeypatch.setenv("DARD_ATTN_TC", request.param)
    return request.param


def _key_tol(ref, dtype):
    """The kernel rounds each rotated key once to the storage type (round to nearest: at
    most 2^-8 of the value for bf16's 8 significant bits, 2^-24 for fp32) after fp32
    arithmetic whose angle and cos/sin errors stay near 1e-6."""
    rel = 2.0 ** -8 if dtype == "bf16" else 2.0 ** -24
    return rel * np.abs(ref) + 4e-6 * (np.abs(ref).max() + 1.0)


def _check_keys(ds, wl, rope):
    got = ds.k_rope(0).float().cpu().numpy()
    ref = P.oracle_keys_rope(wl, 0, rope)
    err = np.abs(got - ref)
    assert np.all(err <= _key_tol(ref, wl.dtype)), float(err.max())
    return float(err.max())


@pytest.mark.parametrize("name,sample,style", [
    ("tiny", None, IL), ("tiny", None, HALF), ("8b", None, IL), ("8b", None, HALF),
    ("gqa", 192, IL), ("gqa", 192, HALF), ("ragged", 48, IL), ("mm", 64, HALF),
])
def test_rope_configs(name, sample, style, tc):
    """The five workloads with RoPE: outputs within the flat bf16 bound, keys within one
    rounding of the oracle's rotated keys."""
    if name == "tiny" and tc != "1":
        pytest.skip("fp32 workload: one CUDA-core kernel whatever DARD_ATTN_TC says")
    wl = W.make(name, scoring=False, layers=1 if name == "mm" else None)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    rope = (THETA, style)
    o = ds.attention(0, rope=rope)
    torch.cuda.synchronize()
    oh = o.float().cpu().numpy()
    mx, mean, n = P.compare_attention(wl, 0, oh, sample=sample, rope=rope)
    ex, emean, _ = P.compare_attention(wl, 0, oh, sample=sample, rope=rope, bf16_operands=False)
    kerr = _check_keys(ds, wl, rope)
    print(name, style, tc, "max", mx, "mean", mean, "rows", n, "key err", kerr,
          "vs all-fp64 max", ex, "mean", emean)
    tol = P.ATT_MAX_ABS if wl.dtype == "bf16" else 2e-4
    assert mx <= tol and mean <= P.ATT_MEAN_ABS
    assert emean <= P.ATT_MEAN_ABS
    assert int(ds.status.item()) == 0


@pytest.mark.parametrize("name,sample", [("8b", None), ("gqa", 192)])
def test_rope_prefix_cached(name, sample, tc):
    """Prefix caching with RoPE: query rows from the prompt's end on keep their positions
    (the row index), the cached prompt rows of the output stay untouched."""
    wl = W.make(name, prefix=True, scoring=False)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    out = torch.full_like(ds.layers[0][0], 7.0)
    rope = (10000.0, IL)
    ds.attention(0, out=out, rope=rope)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy()
    mx, mean, n = P.compare_attention(wl, 0, o, sample=sample, rope=rope)
    assert mx <= P.ATT_MAX_ABS and mean <= P.ATT_MEAN_ABS
    q0 = wl.seqs[0].query_start
    assert q0 > 0 and np.all(o[:q0] == 7.0)


@pytest.mark.parametrize("case", range(8))
def test_rope_random_shapes(case, tc):
    """Seeded random ragged batches with RoPE: both pairings, both head dims, grouped
    heads, blocks anywhere, S = 0, candidate-only shadow rows, and random query starts."""
    rng = np.random.default_rng(900 + case)
    specs = []
    for _ in range(int(rng.integers(1, 5))):
        n = int(rng.integers(1, 700))
        B_ = int(rng.integers(0, min(n, 128) + 1))
        b0 = int(rng.integers(0, n - B_ + 1))
        shadow = ["paper", "candidates", "none"][int(rng.integers(0, 3))]
        sp = dict(n_orig=n, block_start=b0, block_len=B_,
                  fractions=tuple(rng.dirichlet([1, 1, 1])))
        sp["shadow"] = np.zeros(0, np.int32) if shadow == "none" else shadow
        if rng.random() < 0.3:
            sp["query_start"] = int(rng.integers(0, n + 1))
        specs.append(sp)
    hkv = int(rng.choice([1, 2, 4]))
    hq = hkv * int(rng.choice([1, 2, 3]))
    d = int(rng.choice([64, 128]))
    wl = W.custom(specs, hq, hkv, d, seed=950 + case, qkv_std=float(rng.choice([0.09, 0.5])))
    rope = (float(rng.choice([10000.0, THETA])), int(rng.integers(0, 2)))
    ds = DeviceStep(wl, layers=[0], scoring=False)
    o = ds.attention(0, rope=rope)
    torch.cuda.synchronize()
    if any(s.query_start < s.rows for s in wl.seqs):
        mx, mean, n = P.compare_attention(wl, 0, o.float().cpu().numpy(), rope=rope)
        print(case, d, hq, hkv, rope, mx, mean)
        assert mx <= P.att_tol(wl) and mean <= P.ATT_MEAN_ABS
    _check_keys(ds, wl, rope)
    assert int(ds.status.item()) == 0


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("style", [IL, HALF])
def test_rope_fp32(d, style):
    """The fp32 CUDA-core kernel with RoPE: error near fp32 rounding against the oracle."""
    specs = [dict(n_orig=150, block_start=60, block_len=40, fractions=(0.3, 0.4, 0.3)),
             dict(n_orig=70, block_start=0, block_len=33, fractions=(0.4, 0.3, 0.3),
                  shadow="candidates")]
    wl = W.custom(specs, 4, 2, d, dtype="f32", seed=81 + d, qkv_std=1.0)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    rope = (10000.0, style)
    o = ds.attention(0, rope=rope)
    torch.cuda.synchronize()
    mx, mean, n = P.compare_attention(wl, 0, o.float().cpu().numpy(), rope=rope)
    print("fp32 rope", d, style, mx, mean)
    assert mx <= 2e-4
    _check_keys(ds, wl, rope)


def test_rope_keys_in_place(tc):
    """k_rope = k rotates the keys in place: the output and the rotated keys are
    bit-identical to a call with a separate k_rope buffer."""
    wl = W.make("8b", scoring=False)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    q, k, v, _ = ds.layers[0]
    call = ds.attention_call(rope=(THETA, HALF))
    o1, kr = torch.empty_like(q), torch.empty_like(k)
    call(q, k, v, o1, k_rope=kr)
    k2 = k.clone()
    o2 = torch.empty_like(q)
    call(q, k2, v, o2, k_rope=k2)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(k2, kr)
    assert not torch.equal(k2, k)


def test_rope_without_k_rope_is_rejected():
    wl = W.make("8b", scoring=False)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    q, k, v, o = ds.layers[0]
    call = ds.attention_call(rope=(THETA, IL))
    with pytest.raises(B.DardError) as err:
        call(q, k, v, o)
    assert err.value.code == 1  # DARD_ERR_NULL


def test_rope_run_to_run_identical(tc):
    """Repeated RoPE calls give bit-identical outputs (the key pass and the attention kernel
    are ordered by the programmatic dependency, never racing)."""
    wl = W.make("gqa", scoring=False, layers=1)
    ds = DeviceStep(wl, layers=[0], scoring=False)
    outs = []
    for _ in range(4):
        ds.k_rope(0).fill_(float("nan"))
        outs.append(ds.attention(0, rope=(THETA, IL), out=torch.full_like(ds.layers[0][0], float("nan"))))
        torch.cuda.synchronize()
    for o in outs[1:]:
        assert torch.equal(o, outs[0])
