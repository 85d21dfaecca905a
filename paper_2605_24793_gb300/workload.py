"""Seeded synthetic workloads for one verify/arbitrate round.

This module only draws random inputs; it holds none of the method's
arithmetic, so both the CUDA path and the CPU oracle can consume what it
produces without sharing any computation.  Every tensor is drawn from a
generator seeded with ``config.index * 1000 + tensor_id``.

Shapes follow the model pairs of the paper's experiments (Sec. 4.1: a
Qwen3-32B / Qwen3-4B pair and a LLaMA-3.3-70B / LLaMA-3.1-8B pair): the
verify step of a Qwen3-8B-, Qwen3-32B- and Llama-3-8B-shaped target.  No
dataset or trained weight is used; Q/K/V stand for the per-layer projections
of a teacher-forced pass (Sec. 3.1, Eq. 2), already position-encoded.

Layouts (row-major, innermost last):
  q        bf16 [L, B, R, Hq, D]      query rows of the K+1 block positions
  k_blk    bf16 [L, B, R, Hkv, D]     block keys (staging, not yet committed)
  v_blk    bf16 [L, B, R, Hkv, D]
  k_pages  bf16 [L, num_pages, Hkv, P, D]   paged KV cache (committed prefix)
  v_pages  bf16 [L, num_pages, Hkv, P, D]
  page_table int32 [B, max_pages]  (-1 marks an unused entry)
  ctx_len  int32 [B]               committed context length C_b
  hidden   bf16 [B*R, d]           final hidden state of every block row
  w        bf16 [V, d]             LM-head weight (nn.Linear layout)
  mlp      fp32 w1 [H, 8], b1 [H], w2 [H], b2 []   arbitration MLP
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import numpy as np
import torch

# tensor ids used in the seed formula config.index * 1000 + id
_TID = dict(ctx=1, pages=2, q=3, k_blk=4, v_blk=5, k_pages=6, v_pages=7,
            hidden=8, w=9, mlp=10, drafts=11, sample=12, rl=13,
            draft_q=14, draft_pick=15)

NUM_FEATURES = 8


@dataclasses.dataclass(frozen=True)
class RoundConfig:
    name: str
    index: int
    batch: int
    ctx_lo: int
    ctx_hi: int
    k: int                 # draft length K; the block has R = K + 1 rows
    layers: int
    hidden: int            # model width d (LM-head contraction length)
    q_heads: int
    kv_heads: int
    head_dim: int
    vocab: int
    mlp_hidden: int
    mismatch_rate: float
    mismatch_topk: int     # >1: mismatched ids from the target's ranks 2..topk; 0: any other id
    shuffled_pages: bool
    qkv_std: float = 1.0
    w_std: float = 0.02
    h_std: float = 1.0
    page_size: int = 16
    lam: float = 0.6       # decision threshold, Sec. 4.1 default

    @property
    def rows(self) -> int:
        return self.k + 1

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    @property
    def m_rows(self) -> int:
        return self.batch * self.rows

    def replace(self, **kw) -> "RoundConfig":
        return dataclasses.replace(self, **kw)


CONFIGS: Dict[str, RoundConfig] = {}


def _add(c: RoundConfig) -> None:
    CONFIGS[c.name] = c


# Tiny verify round: one layer, vocab 4096, everything N(0, 0.02^2) except the
# hidden rows (N(0,1), a post-norm state), 70% of drafts equal the target argmax.
_add(RoundConfig("tiny", 0, batch=1, ctx_lo=256, ctx_hi=256, k=4, layers=1,
                 hidden=512, q_heads=8, kv_heads=2, head_dim=64, vocab=4096,
                 mlp_hidden=64, mismatch_rate=0.3, mismatch_topk=0,
                 shuffled_pages=False, qkv_std=0.02))
# Qwen3-8B-shaped target, batch 1, context 4096, K=5.
_add(RoundConfig("qwen3_8b_b1", 1, batch=1, ctx_lo=4096, ctx_hi=4096, k=5, layers=36,
                 hidden=4096, q_heads=32, kv_heads=8, head_dim=128, vocab=151936,
                 mlp_hidden=256, mismatch_rate=0.3, mismatch_topk=8,
                 shuffled_pages=False))
# Qwen3-8B-shaped target, batch 16, contexts U[2048, 8192], K=7, shuffled pages.
_add(RoundConfig("qwen3_8b_b16", 2, batch=16, ctx_lo=2048, ctx_hi=8192, k=7, layers=36,
                 hidden=4096, q_heads=32, kv_heads=8, head_dim=128, vocab=151936,
                 mlp_hidden=256, mismatch_rate=0.3, mismatch_topk=8,
                 shuffled_pages=True))
# Qwen3-32B-shaped target, batch 32, contexts U[2048, 16384], K=7.
_add(RoundConfig("qwen3_32b_b32", 3, batch=32, ctx_lo=2048, ctx_hi=16384, k=7, layers=64,
                 hidden=5120, q_heads=64, kv_heads=8, head_dim=128, vocab=151936,
                 mlp_hidden=256, mismatch_rate=0.25, mismatch_topk=8,
                 shuffled_pages=True))
# Llama-3-8B-shaped long-reasoning sweep, batch 64, contexts U[8192, 32768].
for _k in (3, 5, 7):
    for _rate in (0.1, 0.3, 0.6):
        _add(RoundConfig(f"llama3_8b_b64_k{_k}_mm{int(_rate * 100)}", 4, batch=64,
                         ctx_lo=8192, ctx_hi=32768, k=_k, layers=32, hidden=4096,
                         q_heads=32, kv_heads=8, head_dim=128, vocab=128256,
                         mlp_hidden=256, mismatch_rate=_rate, mismatch_topk=8,
                         shuffled_pages=True))


def seed_of(cfg: RoundConfig, tensor: str) -> int:
    return cfg.index * 1000 + _TID[tensor]


def context_lengths(cfg: RoundConfig) -> np.ndarray:
    """C_b ~ U[ctx_lo, ctx_hi] (integers, both ends included)."""
    rng = np.random.default_rng(seed_of(cfg, "ctx"))
    if cfg.ctx_lo == cfg.ctx_hi:
        return np.full(cfg.batch, cfg.ctx_lo, dtype=np.int32)
    return rng.integers(cfg.ctx_lo, cfg.ctx_hi + 1, size=cfg.batch).astype(np.int32)


def pages_needed(ctx: np.ndarray, rows: int, page_size: int) -> np.ndarray:
    """Pages that hold the committed prefix plus one block of ``rows`` tokens."""
    return ((ctx.astype(np.int64) + rows + page_size - 1) // page_size).astype(np.int64)


def page_table(cfg: RoundConfig, ctx: np.ndarray, extra_tokens: int = 0):
    """Return (page_table int32 [B, max_pages], num_pages).

    Every sequence owns ceil((C_b + R + extra) / P) pages of one shared pool.
    With ``shuffled_pages`` the pool is a random permutation, so consecutive
    logical pages of a sequence sit at scattered physical pages.
    """
    need = pages_needed(ctx + extra_tokens, cfg.rows, cfg.page_size)
    num_pages = int(need.sum())
    max_pages = int(need.max())
    order = np.arange(num_pages, dtype=np.int64)
    if cfg.shuffled_pages:
        order = np.random.default_rng(seed_of(cfg, "pages")).permutation(num_pages)
    table = np.full((cfg.batch, max_pages), -1, dtype=np.int32)
    start = 0
    for b in range(cfg.batch):
        table[b, : need[b]] = order[start: start + need[b]]
        start += int(need[b])
    return table, num_pages


# Tensors up to this many elements are drawn with NumPy's PCG64 generator on
# the host, so they are bit-identical on every machine; larger ones are drawn
# on the target device by torch's generator (same seed, device-specific stream).
HOST_DRAW_LIMIT = 1 << 25


def _gen(cfg: RoundConfig, tensor: str, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed_of(cfg, tensor))
    return g


class _Normal:
    """N(0, std^2) bf16 draws for one named tensor of a config."""

    def __init__(self, cfg: RoundConfig, tensor: str, total: int, device):
        self.host = total <= HOST_DRAW_LIMIT
        self.device = torch.device(device)
        if self.host:
            self.rng = np.random.default_rng(seed_of(cfg, tensor))
        else:
            self.g = _gen(cfg, tensor, self.device)

    def fill(self, out: torch.Tensor, std: float) -> torch.Tensor:
        if self.host:
            v = self.rng.standard_normal(tuple(out.shape), dtype=np.float32) * np.float32(std)
            out.copy_(torch.from_numpy(v).to(torch.bfloat16))
        else:
            out.normal_(0.0, std, generator=self.g)
        return out

    def new(self, shape, std: float) -> torch.Tensor:
        return self.fill(torch.empty(shape, dtype=torch.bfloat16, device=self.device), std)


def mlp_params(cfg: RoundConfig, hidden: Optional[int] = None):
    """Arbitration MLP weights drawn like ``nn.Linear``'s default init.

    Weight and bias of a layer with fan-in n are U(-1/sqrt(n), 1/sqrt(n)).
    Returns fp32 CPU tensors (w1 [H, 8], b1 [H], w2 [H], b2 [] ).
    """
    H = cfg.mlp_hidden if hidden is None else hidden
    g = _gen(cfg, "mlp", "cpu")
    a1 = 1.0 / math.sqrt(NUM_FEATURES)
    a2 = 1.0 / math.sqrt(H)
    w1 = (torch.rand(H, NUM_FEATURES, generator=g) * 2 - 1) * a1
    b1 = (torch.rand(H, generator=g) * 2 - 1) * a1
    w2 = (torch.rand(H, generator=g) * 2 - 1) * a2
    b2 = (torch.rand((), generator=g) * 2 - 1) * a2
    return w1.float(), b1.float(), w2.float(), b2.float()


def make_round_inputs(cfg: RoundConfig, device="cpu", extra_tokens: int = 0,
                      alias_layers: bool = False) -> Dict[str, object]:
    """Draw every input of one round except the draft ids (see ``synth_drafts``).

    ``alias_layers`` backs all layers with one KV pool (same bytes read per
    layer, a fraction of the memory) for workloads whose full cache would not
    fit; the caller must report that it was used.
    """
    device = torch.device(device)
    L, B, R = cfg.layers, cfg.batch, cfg.rows
    Hq, Hkv, D, P = cfg.q_heads, cfg.kv_heads, cfg.head_dim, cfg.page_size
    ctx = context_lengths(cfg)
    table, num_pages = page_table(cfg, ctx, extra_tokens)
    out: Dict[str, object] = dict(cfg=cfg, ctx_len_np=ctx, page_table_np=table,
                                  num_pages=num_pages, alias_layers=alias_layers)
    def draw(name, shape, std):
        return _Normal(cfg, name, int(np.prod(shape)), device).new(shape, std)

    out["q"] = draw("q", (L, B, R, Hq, D), cfg.qkv_std)
    out["k_blk"] = draw("k_blk", (L, B, R, Hkv, D), cfg.qkv_std)
    out["v_blk"] = draw("v_blk", (L, B, R, Hkv, D), cfg.qkv_std)
    Lp = 1 if alias_layers else L
    for name in ("k_pages", "v_pages"):
        pool = torch.empty((Lp, num_pages, Hkv, P, D), dtype=torch.bfloat16, device=device)
        src = _Normal(cfg, name, pool.numel(), device)
        for l in range(Lp):           # layer by layer keeps the temporary small
            src.fill(pool[l], cfg.qkv_std)
        out[name] = pool
    out["hidden"] = draw("hidden", (B * R, cfg.hidden), cfg.h_std)
    out["w"] = draw("w", (cfg.vocab, cfg.hidden), cfg.w_std)
    out["mlp"] = mlp_params(cfg)
    out["page_table"] = torch.from_numpy(table).to(device)
    out["ctx_len"] = torch.from_numpy(ctx).to(device)
    return out


def synth_drafts(cfg: RoundConfig, ranked_ids: np.ndarray, round_index: int = 0) -> np.ndarray:
    """Draft block y_hat [B, K] for a chain draft.

    ``ranked_ids`` [B, R, t] are, per block row, the target's top-t token ids
    in rank order (whoever computed them).  Draft position i (1-based) is
    checked against row i-1.  With probability 1 - mismatch_rate the draft is
    the rank-1 id; otherwise it is drawn uniformly from ranks 2..topk
    (``mismatch_topk`` > 1) or from all other ids (``mismatch_topk`` == 0).
    ``round_index`` selects an independent draw for each round of a
    multi-round run.
    """
    rng = np.random.default_rng(seed_of(cfg, "drafts") + 7919 * round_index)
    B, K = cfg.batch, cfg.k
    draft = np.empty((B, K), dtype=np.int32)
    for b in range(B):
        for i in range(K):
            top1 = int(ranked_ids[b, i, 0])
            if rng.random() >= cfg.mismatch_rate:
                draft[b, i] = top1
            elif cfg.mismatch_topk > 1:
                draft[b, i] = int(ranked_ids[b, i, rng.integers(1, cfg.mismatch_topk)])
            else:
                other = int(rng.integers(0, cfg.vocab - 1))
                draft[b, i] = other + (other >= top1)
    return draft


def sample_seed(cfg: RoundConfig, round_index: int = 0) -> int:
    """64-bit key of round ``round_index``'s sampling noise (stochastic
    decoding); both words vary with the round."""
    return (seed_of(cfg, "sample") + round_index) * 0x9E3779B97F4A7C15 % (1 << 63)


def draft_for_rows(draft: np.ndarray) -> np.ndarray:
    """Per block row r, the draft id whose target log-prob row r scores
    (y_hat_{r+1}); the bonus row r = K has none (-1).  Shape [B * R]."""
    B, K = draft.shape
    out = np.full((B, K + 1), -1, dtype=np.int32)
    out[:, :K] = draft
    return out.reshape(-1)


def rl_batch(seed: int, groups: int, rollouts: int, rounds: int, k: int,
             mismatch_rate: float = 0.3, keep_rate: float = 0.6, correct_rate: float = 0.5):
    """Synthetic rollout records for the RL stage: ``groups`` prompts with
    ``rollouts`` rollouts of 1..``rounds`` rounds each; per position a
    mismatch with probability ``mismatch_rate``, the draft kept at a mismatch
    with probability ``keep_rate``, log-probabilities -Exp(1.5), a correct
    rollout with probability ``correct_rate``.  NumPy arrays: group_off,
    correct, round_off, match, accept, ell."""
    rng = np.random.default_rng(seed)
    nr = rng.integers(1, rounds + 1, size=groups * rollouts)
    round_off = np.concatenate([[0], np.cumsum(nr)]).astype(np.int32)
    R = int(round_off[-1])
    match = (rng.random((R, k)) >= mismatch_rate).astype(np.uint8)
    accept = np.where(match == 1, 1, rng.random((R, k)) < keep_rate).astype(np.uint8)
    ell = (-rng.exponential(1.5, (R, k))).astype(np.float32)
    correct = (rng.random(groups * rollouts) < correct_rate).astype(np.uint8)
    group_off = (np.arange(groups + 1) * rollouts).astype(np.int32)
    return group_off, correct, round_off, match, accept, ell


def draft_distributions(cfg: RoundConfig, logits: np.ndarray, noise: float = 1.0,
                        temperature: float = 1.0, round_index: int = 0) -> np.ndarray:
    """A stand-in for the draft model's distributions at the K draft
    positions, for speculative sampling: q_i = softmax((x_{i-1} + noise * eps)
    / T) with eps ~ N(0, 1), where ``logits`` [B, R, V] are the target's
    logits of the block rows (whoever computed them) -- a draft that roughly
    agrees with the target.  ``round_index`` selects an independent draw for
    each round of a multi-round run.  Returns float32 [B, K, V]."""
    x = np.asarray(logits, dtype=np.float64)
    B, R, V = x.shape
    rng = np.random.default_rng(seed_of(cfg, "draft_q") + 7919 * round_index)
    z = (x[:, : R - 1] + noise * rng.standard_normal((B, R - 1, V))) / temperature
    z -= z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    return (e / e.sum(axis=-1, keepdims=True)).astype(np.float32)


def sample_from(cfg: RoundConfig, q: np.ndarray, round_index: int = 0) -> np.ndarray:
    """Draft ids y_hat_i ~ q_i (inverse transform), [B, K] int32."""
    q = np.asarray(q, dtype=np.float64)
    rng = np.random.default_rng(seed_of(cfg, "draft_pick") + 7919 * round_index)
    cdf = np.cumsum(q, axis=-1)
    r = rng.random(q.shape[:-1] + (1,)) * cdf[..., -1:]
    return np.minimum(np.sum(cdf < r, axis=-1), q.shape[-1] - 1).astype(np.int32)


# ------------------------------------------------------------------ replay
_BF16_KEYS = ("q", "k_blk", "v_blk", "k_pages", "v_pages", "hidden", "w")


def save_inputs(path: str, inp: Dict[str, object], draft: Optional[np.ndarray] = None) -> None:
    """Write one round's inputs (and optionally its draft ids) to ``path``
    as an uncompressed ``.npz``, bf16 tensors as their 16-bit patterns, so
    that a case (a failing parity shape, say) can be replayed bit for bit
    without its generator.  Nothing is computed; there is no model state to
    checkpoint, since every input of a round is one of these arrays."""
    import json
    arrays = {k: inp[k].detach().cpu().contiguous().view(torch.int16).numpy()
              for k in _BF16_KEYS}
    w1, b1, w2, b2 = inp["mlp"]
    arrays.update(mlp_w1=w1.cpu().numpy(), mlp_b1=b1.cpu().numpy(), mlp_w2=w2.cpu().numpy(),
                  mlp_b2=np.asarray(float(b2), dtype=np.float32),
                  ctx_len_np=np.asarray(inp["ctx_len_np"]), page_table_np=np.asarray(inp["page_table_np"]),
                  num_pages=np.asarray(int(inp["num_pages"])),
                  alias_layers=np.asarray(bool(inp.get("alias_layers", False))),
                  cfg_json=np.asarray(json.dumps(dataclasses.asdict(inp["cfg"]))))
    if draft is not None:
        arrays["draft"] = np.asarray(draft, dtype=np.int32)
    np.savez(path, **arrays)


def load_inputs(path: str, device="cpu"):
    """Read what ``save_inputs`` wrote: (inputs as ``make_round_inputs``
    returns them, on ``device``; the draft ids or None)."""
    import json
    device = torch.device(device)
    with np.load(path, allow_pickle=False) as z:
        out: Dict[str, object] = dict(
            cfg=RoundConfig(**json.loads(str(z["cfg_json"]))),
            ctx_len_np=z["ctx_len_np"].copy(), page_table_np=z["page_table_np"].copy(),
            num_pages=int(z["num_pages"]), alias_layers=bool(z["alias_layers"]))
        for k in _BF16_KEYS:
            out[k] = torch.from_numpy(z[k].copy()).view(torch.bfloat16).to(device)
        out["mlp"] = (torch.from_numpy(z["mlp_w1"].copy()), torch.from_numpy(z["mlp_b1"].copy()),
                      torch.from_numpy(z["mlp_w2"].copy()), torch.tensor(float(z["mlp_b2"])))
        out["page_table"] = torch.from_numpy(out["page_table_np"]).to(device)
        out["ctx_len"] = torch.from_numpy(out["ctx_len_np"]).to(device)
        draft = z["draft"].copy() if "draft" in z.files else None
    return out, draft
