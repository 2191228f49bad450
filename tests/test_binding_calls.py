"""The binding's prepared calls (AttentionCall, ScoreCall): argument checks on the host, and on
the GPU the same results as the one-shot functions, reused across layers, logits and streams.
Every rejected case raises before the library is called, so nothing bad reaches a kernel."""
import numpy as np
import pytest
import torch

from paper_2608_26574_gb300 import binding as B
from paper_2608_26574_gb300 import build as BUILD
from paper_2608_26574_gb300 import workloads as W
from paper_2608_26574_gb300.device import DeviceStep


@pytest.fixture(scope="module", autouse=True)
def _built():
    BUILD.build()


def test_attention_call_checks_metadata_on_the_host():
    st = torch.zeros(4, dtype=torch.uint8)
    pc = torch.zeros(4, dtype=torch.float32)
    sh = torch.zeros(4, dtype=torch.int32)
    with pytest.raises(ValueError, match="differ in length"):
        B.AttentionCall([8, 8], [4], [4, 4], [4, 4], st, pc, sh)
    with pytest.raises(ValueError, match="differ in length"):
        B.AttentionCall([8], [4], [4], [4], st, pc, sh, query_start=[0, 0])
    with pytest.raises(ValueError, match="device tensor"):
        B.AttentionCall([8], [4], [4], [4], st, pc, sh)


def test_score_call_checks_buffers_on_the_host():
    st = torch.zeros(4, dtype=torch.uint8)
    f = torch.zeros(4, dtype=torch.float32)
    i = torch.zeros(4, dtype=torch.int32)
    with pytest.raises(ValueError, match="device tensor"):
        B.ScoreCall([4], st, 0.5, 0.8, 0.9, 0.1, f, i, st, None)
    with pytest.raises(ValueError, match="workspace is required"):
        B.dard_score_and_transition(f, f, [4], st, 0.5, 0.8, 0.9, 0.1, f, i, st, None)


def test_host_arrays_are_copied():
    a = np.array([3, 4], np.int32)
    c = B._host_i32(a)
    a[0] = 99
    assert c.dtype == np.int32 and c.flags.c_contiguous and list(c) == [3, 4]


@pytest.mark.gpu
def test_attention_call_matches_the_one_shot_call():
    """One prepared call over three layers, on the current stream, a side stream and a raw
    stream handle: bit-identical to one-shot calls (the same kernels on the same inputs)."""
    wl = W.make("tiny", layers=3)
    ds = DeviceStep(wl)
    call = ds.attention_call()
    side = torch.cuda.Stream()
    for li, (q, k, v, _) in enumerate(ds.layers):
        want = torch.empty_like(q)
        B.dard_step_attention(q, k, v, want, ds.n_orig, ds.block_start, ds.block_len,
                              ds.shadow_len, ds.state, ds.prev_conf, ds.shadow_src,
                              status=ds.status, query_start=ds.query_start)
        for stream in (None, side, side.cuda_stream):
            got = torch.full_like(q, float("nan"))
            torch.cuda.synchronize()
            call(q, k, v, got, stream)
            torch.cuda.synchronize()
            assert torch.equal(got, want), (li, stream)
    assert int(ds.status.item()) == 0


@pytest.mark.gpu
def test_attention_call_rejects_mismatched_tensors():
    wl = W.make("tiny")
    ds = DeviceStep(wl)
    q, k, v, o = ds.layers[0]
    call = ds.attention_call()
    rows, d = call.rows, q.shape[2]
    assert rows == int((ds.n_orig + ds.shadow_len).sum())
    bad = [
        (q[:rows - 1], k, v, o[:rows - 1]),                     # fewer rows than the metadata
        (q, k[:rows - 1], v[:rows - 1], o),
        (q, k, v, o[:, :1]),                                    # o shape differs from q
        (q, k, v.double(), o),                                  # mixed dtypes
        (q.transpose(0, 1), k, v, o.transpose(0, 1)),           # not contiguous
        (q.cpu(), k, v, o),                                     # host tensor
        (q[..., :d // 2].contiguous(), k, v, o[..., :d // 2].contiguous()),  # head dims differ
    ]
    for args in bad:
        with pytest.raises(ValueError):
            call(*args)
    for kw in ({"state": ds.state.int()}, {"prev_conf": ds.prev_conf.double()},
               {"shadow_src": ds.shadow_src.long()}, {"status": ds.status.long()},
               {"state": ds.state[:1]}):
        a = dict(state=ds.state, prev_conf=ds.prev_conf, shadow_src=ds.shadow_src,
                 status=ds.status)
        a.update(kw)
        with pytest.raises(ValueError):
            B.AttentionCall(ds.n_orig, ds.block_start, ds.block_len, ds.shadow_len, **a)


def _score_outputs(ds):
    return [t.clone() for t in (ds.conf, ds.token, ds.state_out, ds.w_out, ds.counts)]


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny", "ragged"])
def test_score_call_matches_the_one_shot_call(name):
    """One prepared scoring call on two logits sets: bit-identical to one-shot calls."""
    wl = W.make(name, logits="spanning", attention=False)
    ds = DeviceStep(wl, attention=False)
    call = B.ScoreCall(ds.block_len, ds.state, wl.tau_c, wl.tau_u, wl.lam, wl.p0, ds.conf,
                       ds.token, ds.state_out, ds.workspace, w_out=ds.w_out, counts=ds.counts,
                       status=ds.status)
    sets = [(ds.lx, ds.ls), (ds.ls.clone(), ds.lx.clone())]
    for lx, ls in sets:
        B.dard_score_and_transition(lx, ls, ds.block_len, ds.state, wl.tau_c, wl.tau_u, wl.lam,
                                    wl.p0, ds.conf, ds.token, ds.state_out, ds.workspace,
                                    w_out=ds.w_out, counts=ds.counts, status=ds.status)
        want = _score_outputs(ds)
        for t in (ds.conf, ds.w_out):
            t.fill_(float("nan"))
        for t in (ds.token, ds.counts):
            t.fill_(-7)
        ds.state_out.fill_(9)
        call(lx, ls)
        got = _score_outputs(ds)
        for w, g in zip(want, got):
            assert torch.equal(w.nan_to_num(-1.0), g.nan_to_num(-1.0))
    assert int(ds.status.item()) == 0


@pytest.mark.gpu
def test_score_call_rejects_mismatched_tensors():
    wl = W.make("tiny", logits="spanning", attention=False)
    ds = DeviceStep(wl, attention=False)
    args = (ds.block_len, ds.state, wl.tau_c, wl.tau_u, wl.lam, wl.p0)
    call = B.ScoreCall(*args, ds.conf, ds.token, ds.state_out, ds.workspace)
    rows = call.rows
    for lx, ls in ((ds.lx[:rows - 1], ds.ls[:rows - 1]),            # fewer rows than the blocks
                   (ds.lx, ds.ls[:, :-1]),                         # shapes differ
                   (ds.lx.double(), ds.ls),                        # dtypes differ
                   (ds.lx.t(), ds.ls.t()),                         # rows not contiguous
                   (ds.lx.cpu(), ds.ls.cpu())):                    # host tensors
        with pytest.raises(ValueError):
            call(lx, ls)
    with pytest.raises(ValueError):  # row pitches differ
        wide = torch.zeros(rows, wl.vocab + 8, dtype=ds.ls.dtype, device=ds.ls.device)
        call(ds.lx, wide[:, :wl.vocab])
    for kw in ({"conf": ds.conf[:rows - 1]}, {"token": ds.token.long()},
               {"state_out": ds.state_out.int()}, {"w_out": ds.w_out.half()},
               {"counts": ds.counts[:1]}):
        a = dict(conf=ds.conf, token=ds.token, state_out=ds.state_out)
        extra = {}
        for key, val in kw.items():
            (a if key in a else extra)[key] = val
        with pytest.raises(ValueError):
            B.ScoreCall(*args, a["conf"], a["token"], a["state_out"], ds.workspace, **extra)


@pytest.mark.gpu
def test_attention_kernel_query(monkeypatch):
    """The kernel the launcher picks, asked without launching: the two-tile kernel for the
    8B layer, the one-tile kernel for a long GQA sequence, the CUDA-core kernel for fp32,
    and what DARD_ATTN_TC forces."""
    monkeypatch.delenv("DARD_ATTN_TC", raising=False)
    for name, want in (("8b", 2), ("gqa", 1), ("tiny", 3)):
        wl = W.make(name, scoring=False, layers=1)
        ds = DeviceStep(wl, layers=[0], scoring=False)
        q, k, v, o = ds.layers[0]
        assert ds.attention_call().kernel(q, k, v, o) == want, name
        assert B.dard_attention_kernel(q, k, v, o, ds.n_orig, ds.block_start, ds.block_len,
                                       ds.shadow_len, ds.state, ds.prev_conf,
                                       ds.shadow_src) == want
        if want != 3:
            monkeypatch.setenv("DARD_ATTN_TC", str(3 - want))
            assert ds.attention_call().kernel(q, k, v, o) == 3 - want
            monkeypatch.delenv("DARD_ATTN_TC")
