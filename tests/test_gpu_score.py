"""GPU parity of dard_score_and_transition against the CPU oracle (Eq. 1, 5-8, Algorithm 1)."""
import numpy as np
import pytest
import torch

from paper_2608_26574_gb300 import binding as B
from paper_2608_26574_gb300 import workloads as W
from paper_2608_26574_gb300.device import DeviceStep

from . import parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True, params=["passes", "fused"])
def score_path(request, monkeypatch):
    """Every scoring test runs on both launch paths: the two PDL-chained passes (the
    default) and the one launch whose M rows wait for their block's C rows (used when the
    whole grid fits on the device at once; the passes otherwise)."""
    monkeypatch.setenv("DARD_SCORE_PATH", request.param)
    return request.param


def _run(wl, state_in=None, reps=1, pitch=None):
    ds = DeviceStep(wl, attention=False, logit_pitch=pitch)
    for _ in range(reps):
        ds.score(state_in=state_in)
    torch.cuda.synchronize()
    return ds, (ds.conf.cpu().numpy(), ds.token.cpu().numpy(), ds.state_out.cpu().numpy(),
                ds.w_out.cpu().numpy(), ds.counts.cpu().numpy())


def _check(wl, outs):
    conf, token, st, w, counts = outs
    rep = P.compare_scores(wl, conf, token, st, w_out=w, counts=counts)
    offs = wl.block_offsets()
    for si in range(len(wl.seqs)):
        want = np.bincount(st[offs[si]:offs[si + 1]], minlength=3)
        assert list(counts[3 * si:3 * si + 3]) == list(want)
    return rep


@pytest.mark.parametrize("name", ["tiny", "8b", "gqa", "ragged", "mm"])
@pytest.mark.parametrize("mode", ["literal", "spanning"])
def test_score_configs(name, mode):
    wl = W.make(name, logits=mode, attention=False)
    ds, outs = _run(wl)
    rep = _check(wl, outs)
    assert int(ds.status.item()) == 0
    print(name, mode, rep)


@pytest.mark.parametrize("name", ["8b", "ragged"])
def test_score_repeated_calls_identical(name):
    """The workspace counters return to zero and the merges have one fixed order: repeated
    calls give bit-identical outputs (the 1024-row batch spreads each row over many CTAs)."""
    wl = W.make(name, logits="spanning", attention=False)
    ds = DeviceStep(wl, attention=False)
    ds.score()
    first = [t.clone() for t in (ds.conf, ds.token, ds.state_out, ds.w_out, ds.counts)]
    for _ in range(3):
        ds.score()
        torch.cuda.synchronize()
        for a, b in zip(first, (ds.conf, ds.token, ds.state_out, ds.w_out, ds.counts)):
            assert torch.equal(a, b) or bool(((a == b) | (torch.isnan(a) & torch.isnan(b))).all())


@pytest.mark.parametrize("vocab", [1, 7, 8, 9, 1000, 2049, 8191, 65537])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_score_ragged_vocab_tails(vocab, dtype):
    specs = [dict(n_orig=40, block_start=8, block_len=24, fractions=(0.4, 0.3, 0.3))]
    wl = W.custom(specs, 1, 1, 64, dtype=dtype, vocab=vocab, seed=vocab, logit_std=2.0)
    per16 = 8 if dtype == "bf16" else 4   # row pitch rounded up to 16 bytes
    pitch = (vocab + per16 - 1) // per16 * per16
    _check(wl, _run(wl, pitch=pitch + (per16 if vocab % 2 else 0))[1])


def test_score_many_sequences_and_degenerate_blocks():
    specs = [dict(n_orig=300, block_start=100, block_len=B, fractions=f)
             for B, f in ((1, (0, 1, 0)), (7, (1, 0, 0)), (32, (0, 0, 1)), (64, (0, 1, 0)),
                          (128, (0.2, 0.5, 0.3)), (0, (1, 0, 0)), (5, (0.2, 0.4, 0.4)))]
    wl = W.custom(specs, 1, 1, 64, vocab=5000, seed=3)
    _check(wl, _run(wl)[1])


def test_score_exact_ties_lowest_index():
    specs = [dict(n_orig=64, block_start=0, block_len=16, fractions=(0.5, 0.25, 0.25))]
    wl = W.custom(specs, 1, 1, 64, vocab=4096, seed=5, logits="plain")
    # plant the same maximum at several columns of every row (bf16-exact values)
    for arr in (wl.logits_x, wl.logits_s):
        for r in range(arr.shape[0]):
            cols = np.sort(np.random.default_rng(r).choice(4096, size=4, replace=False))
            arr[r, cols] = 16.0
    conf, token, st, w, counts = _run(wl)[1]
    _check(wl, (conf, token, st, w, counts))


def test_score_nonfinite_rows_and_bad_states():
    specs = [dict(n_orig=64, block_start=16, state=[0, 1, 2, 0, 1, 2, 7, 1, 0, 2])]
    wl = W.custom(specs, 1, 1, 64, vocab=3000, seed=9)
    wl.logits_s[1, 17] = np.nan          # C row with a NaN -> invalid
    wl.logits_s[2, 5] = np.inf           # U row with +inf -> invalid
    wl.logits_s[4, :] = -np.inf          # C row all -inf -> invalid
    wl.logits_x[3, 100] = np.nan         # M row: NaN in the original logits
    wl.logits_s[5, :10] = -np.inf        # some -inf values are fine
    ds, outs = _run(wl)
    conf, token, st, w, counts = outs
    _check(wl, outs)
    for r in (1, 2, 3, 4):
        assert conf[r] == 0 and token[r] == -1 and st[r] == 0
    s = int(ds.status.item())
    assert s & 0x4 and s & 0x1   # invalid rows and the state byte 7


def test_score_threshold_edges():
    """tau_c == tau_u (two states only) and the extreme thresholds 0 and 1."""
    specs = [dict(n_orig=80, block_start=40, block_len=32, fractions=(0.4, 0.3, 0.3))]
    for tau in ((0.6, 0.6), (0.0, 1.0), (0.0, 0.0), (1.0, 1.0)):
        wl = W.custom(specs, 1, 1, 64, vocab=2000, seed=11, tau=tau, logit_std=1.0)
        _check(wl, _run(wl)[1])


def _end_of_step(ds, cur, mask_token, in_place):
    """Scores with p_cur of `cur` and next-step tokens; with in_place, state_out is the
    state_in buffer and tokens overwrite the cur_token buffer."""
    wl = ds.wl
    rows = ds.state.numel()
    p_cur = torch.full((rows,), -1.0, dtype=torch.float32, device=ds.state.device)
    if in_place:
        state_io = ds.state.clone()
        tokens = cur.clone()
        cur_in, st_out = tokens, state_io
    else:
        state_io, tokens, cur_in, st_out = ds.state, torch.empty_like(cur), cur, ds.state_out
    B.dard_score_and_transition(ds.lx, ds.ls, ds.block_len, state_io, wl.tau_c, wl.tau_u, wl.lam,
                                wl.p0, ds.conf, ds.token, st_out, ds.workspace, w_out=ds.w_out,
                                counts=ds.counts, status=ds.status, cur_token=cur_in,
                                p_cur=p_cur, tokens=tokens, mask_token=mask_token)
    torch.cuda.synchronize()
    return (p_cur.cpu().numpy(), tokens.cpu().numpy(), st_out.cpu().numpy())


@pytest.mark.parametrize("name", ["tiny", "8b", "gqa", "mm", "ragged"])
@pytest.mark.parametrize("in_place", [False, True])
def test_score_end_of_step(name, in_place):
    """p_cur of the current token on each row's scored distribution, the next step's tokens
    (x^, or the mask token for rows ending in M), with the state updated in place or not."""
    wl = W.make(name, logits="spanning", attention=False)
    ds = DeviceStep(wl, attention=False)
    rng = np.random.default_rng(31)
    rows = wl.total_block
    cur = rng.integers(-2, wl.vocab + 2, size=rows).astype(np.int32)
    # a third of the rows hold their current argmax, so that p_cur = c is exercised too
    for si, res in enumerate(P.oracle_scores(wl)):
        a = wl.block_offsets()[si]
        for i in range(0, len(res.token), 3):
            cur[a + i] = res.token[i]
    cur_d = torch.from_numpy(cur).to(ds.state.device)
    mask_token = 126336
    p_cur, tokens, st = _end_of_step(ds, cur_d, mask_token, in_place)
    conf, token, w, counts = (t.cpu().numpy() for t in (ds.conf, ds.token, ds.w_out, ds.counts))
    rep = P.compare_scores(wl, conf, token, st, w_out=w, counts=counts, cur_token=cur,
                           p_cur=p_cur, tokens_next=tokens, mask_token=mask_token)
    assert int(ds.status.item()) == 0
    print(name, in_place, rep)


@pytest.mark.parametrize("name", ["tiny", "8b", "gqa", "mm"])
@pytest.mark.parametrize("mode", [B.ORDER_CONFIDENCE, B.ORDER_BIDIR, B.ORDER_L2R,
                                  B.ORDER_ENTROPY, B.ORDER_MARGIN])
def test_score_ordering_outputs(name, mode):
    """Entropy and margin of every scored distribution, and the next step's ordering key
    (the ablation's orderings: confidence, bidirectional, left-to-right, entropy, margin)."""
    wl = W.make(name, logits="spanning", attention=False)
    ds = DeviceStep(wl, attention=False)
    rows = ds.state.numel()
    dev = ds.state.device
    ent, mg, key = (torch.full((rows,), 99.0, dtype=torch.float32, device=dev) for _ in range(3))
    B.dard_score_and_transition(ds.lx, ds.ls, ds.block_len, ds.state, wl.tau_c, wl.tau_u, wl.lam,
                                wl.p0, ds.conf, ds.token, ds.state_out, ds.workspace,
                                w_out=ds.w_out, counts=ds.counts, status=ds.status, entropy=ent,
                                margin=mg, order_key=key, order_mode=mode)
    torch.cuda.synchronize()
    out = [t.cpu().numpy() for t in (ds.conf, ds.token, ds.state_out, ds.w_out, ds.counts,
                                     ent, mg, key)]
    rep = P.compare_scores(wl, *out[:3], w_out=out[3], counts=out[4], entropy=out[5],
                           margin=out[6], order_key=out[7], order_mode=mode)
    assert int(ds.status.item()) == 0
    print(name, mode, rep)


def test_score_maximum_batch():
    """The largest call the ABI allows: DARD_MAX_SEQS sequences with blocks of
    DARD_MAX_BLOCK positions (32768 rows), a small vocabulary."""
    specs = [dict(n_orig=B.MAX_BLOCK + 3, block_start=2, block_len=B.MAX_BLOCK,
                  fractions=(0.4, 0.3, 0.3)) for _ in range(B.MAX_SEQS)]
    wl = W.custom(specs, 1, 1, 64, vocab=256, seed=77, logit_std=2.0)
    ds, outs = _run(wl)
    _check(wl, outs)
    assert int(ds.status.item()) == 0


def test_score_all_blocks_empty():
    """Every block empty: no pass runs, and the counts still come out as zeros."""
    specs = [dict(n_orig=40, block_start=5, block_len=0, fractions=(1, 0, 0)) for _ in range(3)]
    wl = W.custom(specs, 1, 1, 64, vocab=512, seed=1)
    ds = DeviceStep(wl, attention=False)
    ds.counts.fill_(-5)
    ds.score()
    torch.cuda.synchronize()
    assert ds.counts.cpu().tolist() == [0] * 9
