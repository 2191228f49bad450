"""Multi-step DARD decoding: the outer loop of Algorithm 1 on a small random-weight model.

This drives the library's two entry points the way a diffusion LLM would, step after step:

* ``DLLM`` is a bidirectional transformer with random (seeded) weights: token embedding,
  ``n_layers`` blocks of RMSNorm, Q/K/V projections, rotary positions, attention, output
  projection and a SwiGLU MLP, then a final RMSNorm and the LM head. The projections and the
  MLP are plain library GEMMs (torch / cuBLAS); every attention layer is
  ``dard_step_attention`` over the augmented sequence x~_t = (x_t; s_t) of Sec. 3.1. The
  shadow rows hold the mask token (s_t is fully masked) and take the positions of the
  block positions they copy (shared positional embedding).
* ``decode`` runs Algorithm 1 block by block (semi-autoregressive blocks of ``block_len``
  positions): each step builds the augmented input, runs the model, and calls
  ``dard_score_and_transition`` with the end-of-step outputs in place (states, the block's
  tokens, and the next step's ordering key as prev_conf), until the block holds no M or C
  position or ``max_steps`` is reached. The paper states no minimum-progress rule; an
  optional one (``min_progress``) moves the most confident non-U position to U whenever a
  step adds no U position.

Nothing here is on the measured hot path of ``bench.py``; it exists to run the path in its
setting and to time whole steps (``python -m paper_2608_26574_gb300.decode``).
"""
from __future__ import annotations

import argparse
import json
import math
import time
from dataclasses import dataclass, field

import numpy as np
import torch

from . import binding as B


@dataclass
class ModelConfig:
    vocab: int = 4096
    d_model: int = 512
    n_layers: int = 2
    hq: int = 4
    hkv: int = 4
    head_dim: int = 128
    mlp: int = 1024
    dtype: str = "bf16"           # "bf16" (tensor-core attention) or "f32" (CUDA-core)
    logit_scale: float = 4.0      # sharpens the random LM head so that some predictions
    rope_base: float = 10000.0    # are confident enough to cross the thresholds

    @property
    def mask_token(self) -> int:
        return self.vocab - 1


class DLLM:
    """Random-weight bidirectional transformer (weights drawn from a seeded generator)."""

    def __init__(self, cfg: ModelConfig, device="cuda", seed: int = 0):
        self.cfg = cfg
        self.device = torch.device(device)
        self.dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
        g = torch.Generator().manual_seed(seed)

        def w(*shape, fan_in):
            return (torch.randn(*shape, generator=g) / math.sqrt(fan_in)).to(self.device, self.dt)

        d, hd = cfg.d_model, cfg.head_dim
        self.emb = w(cfg.vocab, d, fan_in=1)
        self.layers = []
        for _ in range(cfg.n_layers):
            self.layers.append(dict(
                wq=w(d, cfg.hq * hd, fan_in=d), wk=w(d, cfg.hkv * hd, fan_in=d),
                wv=w(d, cfg.hkv * hd, fan_in=d), wo=w(cfg.hq * hd, d, fan_in=cfg.hq * hd),
                w1=w(d, cfg.mlp, fan_in=d), w3=w(d, cfg.mlp, fan_in=d),
                w2=w(cfg.mlp, d, fan_in=cfg.mlp)))
        self.head = w(d, cfg.vocab, fan_in=d)

    @staticmethod
    def rmsnorm(x):
        xf = x.float()
        return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + 1e-6)).to(x.dtype)

    def forward(self, batch: "Batch", need_attn_out: bool = False):
        """Logits of the block rows: (logits_x [sum B_i, V], logits_s [sum B_i, V])."""
        cfg = self.cfg
        rows = batch.tokens.numel()
        h = self.emb[batch.tokens.long()]
        attn_outs = []
        # one step's mask metadata serves every layer: marshalled once. RoPE runs inside the
        # call (pairs (2i, 2i+1), base rope_base): q and k go in before RoPE, each row at its
        # position and each shadow row at the position it copies; k_rope receives the keys.
        attention = B.AttentionCall(batch.n_orig, batch.block_start, batch.block_len,
                                    batch.shadow_len, batch.state, batch.prev_conf,
                                    batch.shadow_src, status=batch.status,
                                    rope_theta=cfg.rope_base,
                                    rope_style=B.DARD_ROPE_INTERLEAVED)
        for L in self.layers:
            a = self.rmsnorm(h)
            q = (a @ L["wq"]).view(rows, cfg.hq, cfg.head_dim).contiguous()
            k = (a @ L["wk"]).view(rows, cfg.hkv, cfg.head_dim).contiguous()
            v = (a @ L["wv"]).view(rows, cfg.hkv, cfg.head_dim).contiguous()
            o = torch.empty_like(q)
            k_rope = torch.empty_like(k)
            attention(q, k, v, o, k_rope=k_rope)
            if need_attn_out:
                attn_outs.append((q, k, v, o))
            h = h + o.view(rows, cfg.hq * cfg.head_dim) @ L["wo"]
            m = self.rmsnorm(h)
            h = h + (torch.nn.functional.silu(m @ L["w1"]) * (m @ L["w3"])) @ L["w2"]
        h = self.rmsnorm(h)
        hx = h[batch.x_rows]
        hs = h[batch.s_rows]
        lx = (hx @ self.head) * cfg.logit_scale
        ls = (hs @ self.head) * cfg.logit_scale
        return (lx.contiguous(), ls.contiguous(), attn_outs) if need_attn_out else \
            (lx.contiguous(), ls.contiguous())


@dataclass
class Batch:
    """Device state of one decoding step over a batch of sequences (paper layout: one
    shadow row per block position, shadow_src[k] = b0 + k)."""
    tokens: torch.Tensor      # int32 [rows]: x_t then s_t (mask tokens) per sequence
    pos: torch.Tensor         # int32 [rows]: positions (shadow rows: their source position),
                              # the ones dard_step_attention derives for RoPE
    n_orig: np.ndarray
    block_start: np.ndarray
    block_len: np.ndarray
    shadow_len: np.ndarray
    state: torch.Tensor       # uint8 [sum B]
    prev_conf: torch.Tensor   # float32 [sum B]: the Eq. 3 ordering key
    shadow_src: torch.Tensor  # int32 [sum S]
    x_rows: torch.Tensor      # int64 [sum B]: rows of the block's x copies
    s_rows: torch.Tensor      # int64 [sum B]: rows of the shadow copies
    block_tok: torch.Tensor   # int32 [sum B]: view of the block's x tokens (gathered)
    status: torch.Tensor
    row_base: list = field(default_factory=list)


def make_batch(prompts: list[np.ndarray], gen_len: int, block_len: int, block_index: int,
               tokens_gen: list[np.ndarray] | None, cfg: ModelConfig, device) -> Batch:
    """Augmented inputs for the current block of every sequence. tokens_gen[i] holds the
    generated positions decoded so far (mask tokens where still masked)."""
    dev = torch.device(device)
    toks, pos, n_orig, b0s, x_rows, s_rows, shadow_src, bases = [], [], [], [], [], [], [], []
    base = 0
    for i, pr in enumerate(prompts):
        P0 = len(pr)
        N = P0 + gen_len
        gen = tokens_gen[i] if tokens_gen is not None else np.full(gen_len, cfg.mask_token)
        b0 = P0 + block_index * block_len
        x = np.concatenate([pr, gen]).astype(np.int32)
        s = np.full(block_len, cfg.mask_token, np.int32)
        toks.append(np.concatenate([x, s]))
        pos.append(np.concatenate([np.arange(N), np.arange(b0, b0 + block_len)]).astype(np.int32))
        n_orig.append(N)
        b0s.append(b0)
        x_rows.append(base + b0 + np.arange(block_len))
        s_rows.append(base + N + np.arange(block_len))
        shadow_src.append(np.arange(b0, b0 + block_len, dtype=np.int32))
        bases.append(base)
        base += N + block_len
    nB = len(prompts) * block_len
    return Batch(
        tokens=torch.from_numpy(np.concatenate(toks)).to(dev),
        pos=torch.from_numpy(np.concatenate(pos)).to(dev),
        n_orig=np.array(n_orig, np.int32), block_start=np.array(b0s, np.int32),
        block_len=np.full(len(prompts), block_len, np.int32),
        shadow_len=np.full(len(prompts), block_len, np.int32),
        state=torch.zeros(nB, dtype=torch.uint8, device=dev),
        prev_conf=torch.zeros(nB, dtype=torch.float32, device=dev),
        shadow_src=torch.from_numpy(np.concatenate(shadow_src)).to(dev),
        x_rows=torch.from_numpy(np.concatenate(x_rows)).long().to(dev),
        s_rows=torch.from_numpy(np.concatenate(s_rows)).long().to(dev),
        block_tok=torch.empty(nB, dtype=torch.int32, device=dev),
        status=torch.zeros(1, dtype=torch.int32, device=dev), row_base=bases)


@dataclass
class StepRecord:
    state_in: np.ndarray
    prev_conf_in: np.ndarray
    tokens_in: np.ndarray
    logits_x: np.ndarray | None
    logits_s: np.ndarray | None
    state_out: np.ndarray
    conf: np.ndarray
    token: np.ndarray
    tokens_out: np.ndarray
    counts: np.ndarray
    gpu_us: float


def step(model: DLLM, batch: Batch, thr: tuple[float, float], lam: float, p0: float,
         order_mode: int, workspace, outs: dict, min_progress: bool, keep_logits=False):
    """One step of Algorithm 1 for the current block of every sequence, on the device."""
    cfg = model.cfg
    batch.block_tok.copy_(batch.tokens[batch.x_rows])
    lx, ls = model.forward(batch)
    state_before = batch.state.clone() if keep_logits else None
    n, blen = len(batch.n_orig), int(batch.block_len[0])
    u_before = (batch.state.view(n, blen) == 2).sum(1) if min_progress else None
    B.dard_score_and_transition(
        lx, ls, batch.block_len, batch.state, thr[0], thr[1], lam, p0, outs["conf"], outs["token"],
        batch.state, workspace, counts=outs["counts"], status=batch.status,
        tokens=batch.block_tok, mask_token=cfg.mask_token, order_key=batch.prev_conf,
        order_mode=order_mode)
    if min_progress:
        # a sequence whose step added no U position: its most confident non-U position
        # becomes U with its prediction
        st = batch.state.view(n, blen)
        stuck = (st == 2).sum(1) <= u_before
        cand = torch.where(st != 2, outs["conf"].view(n, blen), torch.full_like(outs["conf"].view(n, blen), -1.0))
        best = cand.argmax(1)
        promote = stuck & (cand.gather(1, best[:, None]).squeeze(1) >= 0)
        rows = torch.arange(n, device=best.device) * blen + best
        two = torch.full_like(batch.state[rows], 2)
        batch.state[rows] = torch.where(promote, two, batch.state[rows])
        batch.block_tok[rows] = torch.where(promote, outs["token"][rows], batch.block_tok[rows])
    batch.tokens[batch.x_rows] = batch.block_tok
    return (lx, ls, state_before) if keep_logits else None


def decode(model: DLLM, prompts: list[np.ndarray], gen_len: int, block_len: int,
           thr=(0.5, 0.8), lam=0.5 ** (1 / 8), p0=0.1, order_mode: int = B.ORDER_CONFIDENCE,
           max_steps: int = 64, min_progress: bool = False, record: bool = False):
    """Algorithm 1 block by block. Returns (generated tokens [n, gen_len], per-block steps,
    per-step GPU microseconds, step records if ``record``)."""
    dev = model.device
    n = len(prompts)
    gen = [np.full(gen_len, model.cfg.mask_token, np.int32) for _ in range(n)]
    nB = n * block_len
    outs = dict(conf=torch.empty(nB, dtype=torch.float32, device=dev),
                token=torch.empty(nB, dtype=torch.int32, device=dev),
                counts=torch.empty(3 * n, dtype=torch.int32, device=dev))
    ws = torch.zeros(B.dard_score_workspace_size(nB, model.cfg.vocab, n), dtype=torch.uint8,
                     device=dev)
    steps_per_block, step_us, records = [], [], []
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for blk in range(gen_len // block_len):
        batch = make_batch(prompts, gen_len, block_len, blk, gen, model.cfg, dev)
        done = 0
        for t in range(max_steps):
            rec_in = None
            if record:
                rec_in = (batch.state.cpu().numpy(), batch.prev_conf.cpu().numpy(),
                          batch.tokens[batch.x_rows].cpu().numpy())
            e0.record()
            res = step(model, batch, thr, lam, p0, order_mode, ws, outs, min_progress,
                       keep_logits=record)
            e1.record()
            counts = outs["counts"].cpu().numpy()  # synchronises
            step_us.append(e0.elapsed_time(e1) * 1e3)
            if record:
                lx, ls, _ = res
                records.append(StepRecord(rec_in[0], rec_in[1], rec_in[2],
                                          lx.float().cpu().numpy(), ls.float().cpu().numpy(),
                                          batch.state.cpu().numpy(), outs["conf"].cpu().numpy(),
                                          outs["token"].cpu().numpy(),
                                          batch.tokens[batch.x_rows].cpu().numpy(),
                                          counts.copy(), step_us[-1]))
            done = t + 1
            st = batch.state.cpu().numpy()
            if (st == 2).all():
                break
        steps_per_block.append(done)
        blk_tok = batch.tokens[batch.x_rows].cpu().numpy().reshape(n, block_len)
        for i in range(n):
            gen[i][blk * block_len:(blk + 1) * block_len] = blk_tok[i]
    return np.stack(gen), steps_per_block, step_us, records


def main():
    ap = argparse.ArgumentParser(description="DARD multi-step decoding on a random-weight model")
    ap.add_argument("--seqs", type=int, default=4)
    ap.add_argument("--prompt", type=int, default=512)
    ap.add_argument("--gen", type=int, default=128)
    ap.add_argument("--block", type=int, default=32)
    ap.add_argument("--layers", type=int, default=4)
    ap.add_argument("--d-model", type=int, default=4096)
    ap.add_argument("--heads", type=int, default=32)
    ap.add_argument("--vocab", type=int, default=126464)
    ap.add_argument("--mlp", type=int, default=12288)
    ap.add_argument("--logit-scale", type=float, default=24.0)
    ap.add_argument("--order", type=int, default=B.ORDER_CONFIDENCE)
    ap.add_argument("--min-progress", action="store_true")
    ap.add_argument("--tau", type=float, nargs=2, default=(0.5, 0.8), metavar=("TAU_C", "TAU_U"))
    ap.add_argument("--max-steps", type=int, default=64)
    ap.add_argument("--seed", type=int, default=0)
    args = ap.parse_args()
    from . import build as Bu
    Bu.build()
    cfg = ModelConfig(vocab=args.vocab, d_model=args.d_model, n_layers=args.layers,
                      hq=args.heads, hkv=args.heads, head_dim=128, mlp=args.mlp,
                      logit_scale=args.logit_scale)
    model = DLLM(cfg, seed=args.seed)
    rng = np.random.default_rng(args.seed)
    prompts = [rng.integers(0, cfg.vocab - 1, size=args.prompt).astype(np.int32)
               for _ in range(args.seqs)]
    t0 = time.perf_counter()
    _, steps, us, _ = decode(model, prompts, args.gen, args.block, thr=tuple(args.tau),
                             order_mode=args.order, max_steps=args.max_steps,
                             min_progress=args.min_progress)
    wall = time.perf_counter() - t0
    warm = us[1:] if len(us) > 1 else us
    print(json.dumps({"steps_per_block": steps, "steps": len(us),
                      "step_us_median": float(np.median(warm)), "wall_s": wall,
                      "config": vars(args)}))


if __name__ == "__main__":
    main()
