"""Seeded input generators: shapes, exact state counts, bf16 rounding (no GPU)."""
import numpy as np
import torch

from paper_2608_26574_gb300 import workloads as W


def test_round_bf16_matches_torch():
    rng = np.random.default_rng(0)
    a = (rng.standard_normal(100000) * 10 ** rng.uniform(-6, 6, 100000)).astype(np.float32)
    want = torch.from_numpy(a).to(torch.bfloat16).to(torch.float32).numpy()
    assert (W.round_bf16(a).view(np.uint32) == want.view(np.uint32)).all()


def test_state_counts_largest_remainder():
    assert W.state_counts(32, (0.4, 0.3, 0.3)) == [13, 10, 9]
    assert W.state_counts(32, (0.5, 0.25, 0.25)) == [16, 8, 8]
    assert W.state_counts(64, (0.3, 0.4, 0.3)) == [19, 26, 19]
    assert W.state_counts(32, (0.2, 0.6, 0.2)) == [7, 19, 6]


def test_shapes_and_layouts():
    wl = W.make("tiny")
    s = wl.seqs[0]
    assert (s.n_orig, s.block_start, s.block_len, s.n_shadow) == (64, 32, 32, 32)
    assert wl.q[0].shape == (96, 4, 64) and wl.logits_x.shape == (32, 1024)
    assert [(s.state == c).sum() for c in (0, 1, 2)] == [13, 10, 9]
    wl = W.make("tiny", layout="candidates")
    assert wl.total_rows == 74
    wl = W.make("8b", attention=False)
    s = wl.seqs[0]
    assert (s.n_orig, s.block_start, s.rows) == (768, 608, 800)
    assert wl.logits_s.shape == (32, 126464)
    assert (W.round_bf16(wl.logits_s) == wl.logits_s).all()
    # prev_conf ranges follow the state (tau_c, tau_u) = (0.5, 0.8)
    st, cf = s.state, s.prev_conf
    assert (cf[st == 2] > 0.8).all() and (cf[st == 1] > 0.5).all() and (cf[st == 1] <= 0.8).all()
    wl = W.make("gqa", scoring=False, layout="candidates")
    assert wl.seqs[0].rows == 5146 and wl.q[0].shape == (5146, 28, 128) and wl.k[0].shape[1] == 4


def test_seeded_reproducible():
    a = W.make("tiny")
    b = W.make("tiny")
    assert (a.q[0] == b.q[0]).all() and (a.logits_s == b.logits_s).all()
    assert (a.seqs[0].state == b.seqs[0].state).all()


def test_algorithmic_work_closed_forms():
    """The roofline numerators, from each configuration's definition by hand: attention
    4·d·(rows − query_start)·N·Hq FLOPs, scoring V·esize·(B + |M|) bytes."""
    from paper_2608_26574_gb300 import workloads as W
    wl = W.make("8b", attention=False, scoring=False)
    assert W.attention_flops(wl) == 4 * 128 * 800 * 768 * 32 == 10_066_329_600
    wl = W.make("8b", layout="candidates", attention=False, scoring=False)
    assert W.attention_flops(wl) == 4 * 128 * (768 + 8) * 768 * 32  # 8 C positions
    wl = W.make("8b", prefix=True, attention=False, scoring=False)
    assert W.attention_flops(wl) == 4 * 128 * (800 - 512) * 768 * 32  # queries after the prompt
    wl = W.make("gqa", attention=False, scoring=False)
    assert W.attention_flops(wl) == 4 * 128 * 5184 * 5120 * 28 == 380_507_258_880
    wl = W.make("tiny", attention=False, scoring=False)
    assert W.attention_flops(wl) == 4 * 64 * 96 * 64 * 4
    wl = W.make("8b", attention=False)
    assert W.scoring_bytes(wl) == 126464 * 2 * (32 + 16) == 12_140_544  # 16 M rows, bf16
    wl = W.make("gqa", attention=False)
    assert W.scoring_bytes(wl) == 152064 * 2 * (64 + 19)  # 19 M rows
    wl = W.make("tiny", attention=False)
    assert W.scoring_bytes(wl) == 1024 * 4 * (32 + 13)  # fp32 logits, 13 M rows
