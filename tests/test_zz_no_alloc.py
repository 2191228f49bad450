"""dard_score_and_transition_noalloc (scratch inside the library) against the workspace entry
point dard_score_and_transition. Collected last on purpose: it must pass both alone and after
every other test has used the library on the same device."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_26574_gb300 import binding as B
from paper_2608_26574_gb300 import build as BUILD
from paper_2608_26574_gb300 import workloads as W
from paper_2608_26574_gb300.device import DeviceStep

from . import parity as P


def _fake_args(block_len):
    a = B.ScoreArgs()
    a.logits_x = a.logits_s = 0x10000
    a.dtype, a.vocab, a.row_stride, a.num_seqs = B.DARD_BF16, 1024, 1024, len(block_len)
    a.block_len = block_len.ctypes.data_as(B._I32P)
    a.state_in = 0x20000
    a.tau_c, a.tau_u, a.lambda_, a.p0 = 0.5, 0.8, 0.917, 0.1
    a.conf = a.token = a.state_out = 0x30000
    a.workspace, a.workspace_bytes = None, 0
    return a


def test_noalloc_rejects_rows_beyond_its_scratch():
    """More block rows than the built-in scratch holds: DARD_ERR_WORKSPACE, before any launch
    (the pointers are fake; nothing reaches a GPU)."""
    BUILD.build()
    L = B.lib()
    bl = np.full(B.SCORE_NOALLOC_MAX_ROWS // B.MAX_BLOCK + 1, B.MAX_BLOCK, np.int32)
    a = _fake_args(bl)
    assert L.dard_score_and_transition_noalloc(ctypes.byref(a), None) == 7
    assert "built-in scratch" in L.dard_last_error().decode()
    # sizes the workspace entry point rejects keep its own status
    a = _fake_args(np.array([B.MAX_BLOCK + 1], np.int32))
    assert L.dard_score_and_transition_noalloc(ctypes.byref(a), None) == 2
    assert L.dard_score_and_transition_noalloc(None, None) == 1


def _outputs(ds):
    return [t.clone() for t in (ds.conf, ds.token, ds.state_out, ds.w_out, ds.counts)]


def _noalloc(ds):
    wl = ds.wl
    B.dard_score_and_transition_noalloc(ds.lx, ds.ls, ds.block_len, ds.state, wl.tau_c, wl.tau_u,
                                        wl.lam, wl.p0, ds.conf, ds.token, ds.state_out,
                                        w_out=ds.w_out, counts=ds.counts, status=ds.status)


def _same(want, got):
    conf_w, tok_w, st_w, w_w, cnt_w = [t.cpu().numpy() for t in want]
    conf_g, tok_g, st_g, w_g, cnt_g = [t.cpu().numpy() for t in got]
    assert np.array_equal(tok_w, tok_g)
    assert np.array_equal(st_w, st_g)
    assert np.array_equal(cnt_w, cnt_g)
    assert np.max(np.abs(conf_w - conf_g), initial=0.0) <= P.CONF_TOL
    both_nan = np.isnan(w_w) & np.isnan(w_g)
    assert np.all(both_nan | (np.abs(w_w - w_g) <= P.W_REL * np.abs(w_w)))


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_two_calls_in_a_row():
    """Two different problems back to back through the built-in scratch, each equal to the
    workspace entry point on the same inputs (and to the oracle)."""
    steps = []
    for name, mode in (("ragged", "spanning"), ("8b", "literal")):
        wl = W.make(name, logits=mode, attention=False)
        ds = DeviceStep(wl, attention=False)
        ds.score()
        torch.cuda.synchronize()
        steps.append((ds, _outputs(ds)))
        for t in (ds.conf, ds.w_out):
            t.fill_(float("nan"))
        ds.token.fill_(-7)
        ds.state_out.fill_(9)
        ds.counts.fill_(-1)
    for ds, _ in steps:
        _noalloc(ds)
    torch.cuda.synchronize()
    for ds, want in steps:
        got = _outputs(ds)
        _same(want, got)
        conf, token, st, w, counts = [t.cpu().numpy() for t in got]
        P.compare_scores(ds.wl, conf, token, st, w_out=w, counts=counts)
        assert int(ds.status.item()) == 0
