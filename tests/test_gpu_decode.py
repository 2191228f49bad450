"""The multi-step driver (Algorithm 1's outer loop on a random-weight model): its batch
layout (CPU), its steps against the oracle (GPU), and completion of whole blocks (GPU)."""
import math

import numpy as np
import pytest
import torch

import oracle as orc
from paper_2608_26574_gb300 import decode as D

from . import parity as P


def test_make_batch_layout():
    """x rows then shadow rows per sequence; shadow rows hold the mask token and take the
    positions of the block positions they copy."""
    cfg = D.ModelConfig(vocab=64)
    prompts = [np.arange(5, dtype=np.int32), np.arange(3, dtype=np.int32) + 10]
    gen = [np.full(8, cfg.mask_token, np.int32) for _ in prompts]
    gen[0][:4] = 7
    b = D.make_batch(prompts, 8, 4, 1, gen, cfg, "cpu")
    toks, pos = b.tokens.numpy(), b.pos.numpy()
    assert list(b.n_orig) == [13, 11] and list(b.block_start) == [9, 7]
    assert len(toks) == 13 + 4 + 11 + 4
    assert list(toks[:13]) == [0, 1, 2, 3, 4, 7, 7, 7, 7] + [cfg.mask_token] * 4
    assert list(toks[13:17]) == [cfg.mask_token] * 4 and list(pos[13:17]) == [9, 10, 11, 12]
    assert list(pos[17:28]) == list(range(11)) and list(pos[28:32]) == [7, 8, 9, 10]
    assert list(b.x_rows.numpy()) == [9, 10, 11, 12, 17 + 7, 17 + 8, 17 + 9, 17 + 10]
    assert list(b.s_rows.numpy()) == [13, 14, 15, 16, 28, 29, 30, 31]
    assert list(b.shadow_src.numpy()) == [9, 10, 11, 12, 7, 8, 9, 10]


def _np(t):
    return t.double().cpu().numpy()


def _cpu_forward(model, rec_tokens, batch, state, prev_conf):
    """The model in float64 on the host, attention by the oracle's mask (Sec. 3.2)."""
    cfg = model.cfg

    def rms(x):
        return x / np.sqrt((x * x).mean(-1, keepdims=True) + 1e-6)

    def rope(x, pos):
        return orc.rope(x, pos, cfg.rope_base, orc.ROPE_INTERLEAVED)

    pos = batch.pos.cpu().numpy().astype(np.int64)
    h = _np(model.emb)[rec_tokens]
    rows = len(rec_tokens)
    nB = int(batch.block_len[0])
    for L in model.layers:
        a = rms(h)
        q = rope((a @ _np(L["wq"])).reshape(rows, cfg.hq, cfg.head_dim), pos)
        k = rope((a @ _np(L["wk"])).reshape(rows, cfg.hkv, cfg.head_dim), pos)
        v = (a @ _np(L["wv"])).reshape(rows, cfg.hkv, cfg.head_dim)
        o = np.zeros_like(q)
        for si, base in enumerate(batch.row_base):
            N = int(batch.n_orig[si])
            sl = slice(base, base + N + nB)
            lay = orc.SeqLayout(N, int(batch.block_start[si]), state[si * nB:(si + 1) * nB],
                                prev_conf[si * nB:(si + 1) * nB],
                                batch.shadow_src.cpu().numpy()[si * nB:(si + 1) * nB])
            # the positions the library derives (R20) are the batch's
            assert np.array_equal(orc.row_positions(lay), pos[sl])
            o[sl] = orc.masked_attention(q[sl], k[sl], v[sl], orc.attention_mask(lay))
        h = h + o.reshape(rows, -1) @ _np(L["wo"])
        m = rms(h)
        g = m @ _np(L["w1"])
        h = h + ((g / (1 + np.exp(-g))) * (m @ _np(L["w3"]))) @ _np(L["w2"])
    h = rms(h)
    xr, sr = batch.x_rows.cpu().numpy(), batch.s_rows.cpu().numpy()
    head = _np(model.head)
    return h[xr] @ head * cfg.logit_scale, h[sr] @ head * cfg.logit_scale


@pytest.mark.gpu
def test_decode_steps_match_the_oracle():
    """fp32 model (CUDA-core attention): each step's scoring against the oracle on the
    logits the GPU produced (states, tokens, next-step tokens and ordering key); the first
    step's logits against the float64 host forward."""
    cfg = D.ModelConfig(vocab=256, d_model=256, n_layers=2, hq=2, hkv=2, head_dim=64, mlp=256,
                        dtype="f32", logit_scale=6.0)
    model = D.DLLM(cfg, seed=3)
    rng = np.random.default_rng(3)
    prompts = [rng.integers(0, cfg.vocab - 1, size=n).astype(np.int32) for n in (24, 17)]
    thr = (0.3, 0.6)
    gen, steps, us, recs = D.decode(model, prompts, 32, 16, thr=thr, max_steps=6,
                                    min_progress=True, record=True)
    assert len(recs) >= 4
    nB = 16
    checked = 0
    for t, r in enumerate(recs):
        for si in range(len(prompts)):
            sl = slice(si * nB, (si + 1) * nB)
            res = orc.score_block(r.logits_x[sl], r.logits_s[sl], r.state_in[sl],
                                  np.float32(thr[0]), np.float32(thr[1]))
            border = np.array([min(abs(c - thr[0]), abs(c - thr[1])) < P.BORDER for c in res.conf])
            if border.any():
                continue
            conf = r.conf[sl]
            assert np.max(np.abs(conf - res.conf)) <= P.CONF_TOL
            # Eq. 8, then the min-progress rule: with no new U position, the most confident
            # non-U position (by the kernel's confidences) becomes U
            want_st = res.state_out.copy()
            if (want_st == 2).sum() <= (r.state_in[sl] == 2).sum():
                cand = np.where(want_st != 2, conf, -1.0)
                if cand.max() >= 0:
                    want_st[int(np.argmax(cand))] = 2
            assert list(r.state_out[sl]) == list(want_st), (t, si)
            for i in range(nB):
                row = (r.logits_s[sl][i] if r.state_in[sl][i] != 0 else
                       orc.mix_logits(r.logits_x[sl][i], r.logits_s[sl][i], res.w[i]))
                if res.valid[i] and orc.top2_gap(row) >= P.NEAR_TIE:
                    assert r.token[sl][i] == res.token[i]
                    want = cfg.mask_token if want_st[i] == 0 else res.token[i]
                    assert r.tokens_out[sl][i] == want
            checked += 1
        if t + 1 < len(recs) and recs[t + 1].state_in is not None and steps[0] > t + 1:
            # the next step's ordering key is this step's confidence (DARD's ordering)
            np.testing.assert_allclose(recs[t + 1].prev_conf_in, r.conf, rtol=0, atol=0)
    assert checked > 0
    # first step's model forward against the host
    b = D.make_batch(prompts, 32, 16, 0, None, cfg, model.device)
    lx_ref, ls_ref = _cpu_forward(model, b.tokens.cpu().numpy(), b, recs[0].state_in,
                                  recs[0].prev_conf_in)
    assert np.max(np.abs(recs[0].logits_x - lx_ref)) < 2e-3
    assert np.max(np.abs(recs[0].logits_s - ls_ref)) < 2e-3


@pytest.mark.gpu
def test_decode_blocks_complete_with_min_progress():
    """bf16 model: every block reaches all-U and hands over to the next, and the generated
    tokens hold no mask token. A random-weight model's predictions change with the context,
    so re-scored U positions keep falling back under the paper's thresholds; low thresholds
    (0.01, 0.05) let the loop finish and exercise its mechanics."""
    cfg = D.ModelConfig(vocab=512, d_model=256, n_layers=2, hq=2, hkv=2, head_dim=128, mlp=512,
                        logit_scale=8.0)
    model = D.DLLM(cfg, seed=5)
    rng = np.random.default_rng(5)
    prompts = [rng.integers(0, cfg.vocab - 1, size=40).astype(np.int32) for _ in range(3)]
    gen, steps, us, _ = D.decode(model, prompts, 64, 32, thr=(0.01, 0.05), max_steps=96,
                                 min_progress=True)
    assert len(steps) == 2 and all(1 <= s < 96 for s in steps)
    assert not (gen == cfg.mask_token).any()
    assert all(math.isfinite(u) and u > 0 for u in us)
