"""The C-ABI library builds, loads, exports every symbol of include/dard.h, and rejects bad
arguments on the host before any launch (no GPU needed: nothing here reaches a kernel)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_26574_gb300 import binding as B
from paper_2608_26574_gb300 import build as BUILD

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    BUILD.build()
    return B.lib()


def _declared_symbols():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            text = open(os.path.join(ROOT, "include", f)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(dard_[a-z0-9_]+)\s*\(", text))
    return names


def test_exports_every_declared_symbol(lib):
    declared = _declared_symbols()
    assert {"dard_step_attention", "dard_score_and_transition"} <= declared
    for name in declared:
        assert hasattr(lib, name), name
    assert declared <= set(B.EXPORTS)


def test_host_only_entry_points(lib):
    assert lib.dard_version() >= 100
    assert B.status_string(0) == "DARD_OK"
    assert B.status_string(7) == "DARD_ERR_WORKSPACE"
    assert B.status_string(99) == "DARD_ERR_UNKNOWN"
    assert B.dard_score_workspace_size(32, 126464, 1) >= 32 + 4
    assert B.dard_score_workspace_size(4096, 126464, 8) > B.dard_score_workspace_size(32, 126464, 1)
    assert B.dard_score_workspace_size(-1, 10, 1) == 0
    assert B.dard_score_workspace_size(4, 10, 0) == 0


def _attn_args(**kw):
    n = np.array([64], np.int32)
    b0 = np.array([32], np.int32)
    bl = np.array([32], np.int32)
    sl = np.array([32], np.int32)
    a = B.AttnArgs()
    a.q = a.k = a.v = a.o = 0x10000
    a.dtype, a.hq, a.hkv, a.head_dim, a.num_seqs = B.DARD_BF16, 4, 4, 64, 1
    keep = {"n": kw.pop("n", n), "b0": kw.pop("b0", b0), "bl": kw.pop("bl", bl), "sl": kw.pop("sl", sl)}
    if "qs" in kw:
        keep["qs"] = kw.pop("qs")
        a.query_start = keep["qs"].ctypes.data_as(B._I32P)
    a.n_orig = keep["n"].ctypes.data_as(B._I32P)
    a.block_start = keep["b0"].ctypes.data_as(B._I32P)
    a.block_len = keep["bl"].ctypes.data_as(B._I32P)
    a.shadow_len = keep["sl"].ctypes.data_as(B._I32P)
    a.state = a.prev_conf = a.shadow_src = 0x20000
    a.scale = 0.0
    for k, v in kw.items():
        setattr(a, k, v)
    return a, keep


@pytest.mark.parametrize("change,code", [
    ({"q": None}, 1), ({"state": None}, 1), ({"shadow_src": None}, 1),
    ({"dtype": 7}, 3), ({"num_seqs": 0}, 2), ({"num_seqs": 257}, 2),
    ({"hq": 6, "hkv": 4}, 2), ({"head_dim": 96}, 4), ({"scale": -1.0}, 3),
    ({"scale": float("inf")}, 3), ({"q": 0x10008}, 6),
    ({"n": np.array([0], np.int32)}, 2), ({"bl": np.array([129], np.int32)}, 2),
    ({"b0": np.array([40], np.int32)}, 2), ({"sl": np.array([33], np.int32)}, 2),
    ({"b0": np.array([-1], np.int32)}, 2),
    ({"qs": np.array([97], np.int32)}, 2), ({"qs": np.array([-1], np.int32)}, 2),
    # RoPE in the call: theta 0 or >= 1, a known pairing, a 16-byte aligned k_rope, and at
    # most 2^20 positions per sequence
    ({"rope_theta": 0.5, "k_rope": 0x30000}, 3), ({"rope_theta": -1.0, "k_rope": 0x30000}, 3),
    ({"rope_theta": float("nan"), "k_rope": 0x30000}, 3),
    ({"rope_theta": float("inf"), "k_rope": 0x30000}, 3),
    ({"rope_theta": 1e4, "rope_style": 2, "k_rope": 0x30000}, 3),
    ({"rope_theta": 1e4}, 1), ({"rope_theta": 1e4, "k_rope": 0x30008}, 6),
    ({"rope_theta": 1e4, "k_rope": 0x30000, "n": np.array([(1 << 20) + 1], np.int32),
      "b0": np.array([0], np.int32)}, 2),
])
def test_attention_validation(lib, change, code):
    a, keep = _attn_args(**change)
    assert lib.dard_step_attention(ctypes.byref(a), None) == code
    assert lib.dard_last_error().decode() != ""


def test_attention_null_args(lib):
    assert lib.dard_step_attention(None, None) == 1


@pytest.mark.parametrize("change,code", [
    ({"q": None}, 1), ({"dtype": 7}, 3), ({"num_seqs": 0}, 2), ({"hq": 6, "hkv": 4}, 2),
    ({"head_dim": 96}, 4), ({"scale": -1.0}, 3), ({"q": 0x10008}, 6),
    ({"bl": np.array([129], np.int32)}, 2), ({"qs": np.array([97], np.int32)}, 2),
])
def test_attention_kernel_query_validates_like_the_launch(lib, change, code):
    """dard_attention_kernel runs the launch's host validation and returns its codes,
    leaving the output untouched."""
    a, keep = _attn_args(**change)
    out = ctypes.c_int32(-1)
    assert lib.dard_attention_kernel(ctypes.byref(a), ctypes.byref(out)) == code
    assert out.value == -1


def test_attention_kernel_query_null(lib):
    a, keep = _attn_args()
    assert lib.dard_attention_kernel(ctypes.byref(a), None) == 1
    assert lib.dard_attention_kernel(None, ctypes.byref(ctypes.c_int32())) == 1


def _kernel(lib, **kw):
    a, keep = _attn_args(**kw)
    out = ctypes.c_int32(-1)
    assert lib.dard_attention_kernel(ctypes.byref(a), ctypes.byref(out)) == 0
    return out.value


def test_attention_kernel_choice(lib, monkeypatch):
    """The launcher's choice, planned on the host (nothing is launched; the device pointers
    are never read). Cases whose answer holds at 148 or 152 SMs: the 8B layer (one wave of
    query-tile pairs) takes the two-tile kernel, a 5184-row GQA sequence (about eight waves
    of single tiles) the one-tile kernel, fp32 the CUDA-core kernel, and a batch without
    query rows no kernel; DARD_ATTN_TC forces either tensor-core kernel."""
    monkeypatch.delenv("DARD_ATTN_TC", raising=False)
    i32 = lambda *x: np.array(x, np.int32)  # noqa: E731
    layer_8b = dict(n=i32(768), b0=i32(608), bl=i32(32), sl=i32(32), hq=32, hkv=32,
                    head_dim=128)
    gqa = dict(n=i32(5120), b0=i32(4608), bl=i32(64), sl=i32(64), hq=28, hkv=4, head_dim=128)
    assert _kernel(lib, **layer_8b) == 2
    assert _kernel(lib, **gqa) == 1
    assert _kernel(lib, **layer_8b, dtype=B.DARD_F32) == 3
    assert _kernel(lib, **layer_8b, qs=i32(800)) == 0
    monkeypatch.setenv("DARD_ATTN_TC", "1")
    assert _kernel(lib, **layer_8b) == 1
    monkeypatch.setenv("DARD_ATTN_TC", "2")
    assert _kernel(lib, **gqa) == 2


def _score_args(**kw):
    bl = kw.pop("bl", np.array([32], np.int32))
    a = B.ScoreArgs()
    a.logits_x = a.logits_s = 0x10000
    a.dtype, a.vocab, a.row_stride, a.num_seqs = B.DARD_BF16, 1024, 1024, 1
    a.block_len = bl.ctypes.data_as(B._I32P)
    a.state_in = 0x20000
    a.tau_c, a.tau_u, a.lambda_, a.p0 = 0.5, 0.8, 0.917, 0.1
    a.conf = a.token = a.state_out = 0x30000
    a.workspace = 0x40000
    a.workspace_bytes = 1 << 20
    for k, v in kw.items():
        setattr(a, k, v)
    return a, bl


@pytest.mark.parametrize("change,code", [
    ({"logits_s": None}, 1), ({"conf": None}, 1), ({"state_in": None}, 1),
    ({"dtype": 3}, 3), ({"vocab": 0}, 2), ({"row_stride": 100}, 2),
    ({"tau_c": 0.9, "tau_u": 0.8}, 3), ({"tau_u": 1.5}, 3), ({"lambda_": 1.0}, 3),
    ({"lambda_": 0.0}, 3), ({"p0": 0.0}, 3), ({"num_seqs": 0}, 2),
    ({"bl": np.array([200], np.int32)}, 2), ({"workspace": None}, 7),
    ({"workspace_bytes": 16}, 7), ({"logits_x": 0x10002}, 6), ({"row_stride": 1025}, 6),
    ({"p_cur": 0x50000}, 1), ({"order_mode": 5}, 3), ({"order_mode": -1}, 3),
])
def test_score_validation(lib, change, code):
    a, keep = _score_args(**change)
    assert lib.dard_score_and_transition(ctypes.byref(a), None) == code


def test_binding_raises_without_library(tmp_path, monkeypatch):
    monkeypatch.setattr(B, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        B.lib(str(tmp_path / "libdard.so"))


def _plan(lib, **kw):
    a, keep = _attn_args(**kw)
    out = B.AttnPlan()
    assert lib.dard_attention_plan(ctypes.byref(a), ctypes.byref(out)) == 0
    return out


@pytest.mark.parametrize("tc", ["1", "2", "4"])
def test_attention_plan_counts_skipped_tile_pairs(lib, monkeypatch, tc):
    """The host-only plan counts the (query tile, key tile) pairs each tensor-core kernel
    computes and skips: a key tile holding only shadow rows is skipped for the rows a CTA
    (or CTA pair) handles when they are all original queries of positions after the block
    (Sec. 3.2, query block 1 attends x copies only). Expected counts are worked out from the
    layout of each case by hand."""
    monkeypatch.setenv("DARD_ATTN_TC", tc)
    i32 = lambda *x: np.array(x, np.int32)  # noqa: E731
    # 8B layer: 768 original rows, block [608, 640), 32 shadow rows -> 800 rows, 7 key tiles;
    # 7 query tiles per head. Query tile 5 (rows 640..767) is all future-block rows.
    p = _plan(lib, n=i32(768), b0=i32(608), bl=i32(32), sl=i32(32), hq=32, hkv=32,
              head_dim=128)
    assert p.kernel == int(tc)
    assert p.tile_pairs + p.tile_pairs_skipped == 7 * 7 * 32
    # one-tile units: tile 5 skips key tile 6; 256-row units [512, 768) hold prompt rows
    assert p.tile_pairs_skipped == (32 if tc == "1" else 0)
    # GQA layer: 5120 original rows, block [4608, 4672), 64 shadow rows -> 5184 rows, 41 key
    # tiles, 41 query tiles per head; rows 4672..5119 are future-block rows.
    p = _plan(lib, n=i32(5120), b0=i32(4608), bl=i32(64), sl=i32(64), hq=28, hkv=4,
              head_dim=128)
    assert p.tile_pairs + p.tile_pairs_skipped == 41 * 41 * 28
    # one-tile units 37, 38, 39 (rows 4736..5119); two-tile unit [4864, 5120) = 2 tiles
    assert p.tile_pairs_skipped == (3 * 28 if tc == "1" else 2 * 28)
    # no shadow rows: nothing to skip
    p = _plan(lib, n=i32(300), b0=i32(100), bl=i32(32), sl=i32(0), hq=4, hkv=4, head_dim=128)
    assert p.tile_pairs_skipped == 0 and p.tile_pairs == 3 * 3 * 4


def test_attention_plan_fp32_and_empty(lib, monkeypatch):
    monkeypatch.delenv("DARD_ATTN_TC", raising=False)
    p = _plan(lib, dtype=B.DARD_F32)
    assert p.kernel == 3 and p.ctas >= 1 and p.tile_pairs == 0 and p.tile_pairs_skipped == 0
    p = _plan(lib, qs=np.array([96], np.int32))  # every row before query_start: no launch
    assert p.kernel == 0 and p.ctas == 0 and p.tile_pairs == 0


def test_attention_plan_validates_like_the_launch(lib):
    a, keep = _attn_args(head_dim=96)
    out = B.AttnPlan()
    assert lib.dard_attention_plan(ctypes.byref(a), ctypes.byref(out)) == 4
    assert lib.dard_attention_plan(ctypes.byref(a), None) == 1
    assert lib.dard_attention_plan(None, ctypes.byref(out)) == 1
