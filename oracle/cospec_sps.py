"""Speculative-sampling acceptance of the exact-match baseline at a
temperature -- TEST INFRASTRUCTURE ONLY (imported by tests/, and by the
CPU-baseline leg of bench.py at most; no product path calls it).

The paper's distribution-preserving baselines at T = 1 use standard
speculative sampling with acceptance-ratio correction (Sec. 3.1 "Stochastic
decoding", App. C.3); the paper does not restate it, so this follows the
published algorithm (Leviathan, Kalman, Matias, ICML 2023; Chen et al.,
2023).  With the target distribution p_i = softmax(x_{i-1} / T) of block row
i - 1 and the draft's distribution q_i at draft position i (y_hat_i was drawn
from q_i):

  for i = 1..K: accept y_hat_i with probability min(1, p_i(y_hat_i) / q_i(y_hat_i));
  at the first rejection i*: emit a sample of the residual
      r(v) = max(0, p_{i*}(v) - q_{i*}(v)) / sum_w max(0, p_{i*}(w) - q_{i*}(w))
  and stop (s = i*); if every position is accepted, emit a sample of
  p_{K+1} = softmax(x_K / T), the bonus (s = K + 1).

The emitted token at each position is then distributed exactly as p (the
algorithm's defining property, pinned by tests/test_oracle_sps.py).

Randomness (Philox4x32-10, oracle/philox.py; key = the 64-bit seed split
into its low and high words):
  * acceptance uniform of sequence b, position i: counter (i - 1, b, 1, 0),
    output word 0, u = (floor(r / 2^9) + 0.5) / 2^23; y_hat_i is accepted
    iff u * q_i(y_hat_i) < p_i(y_hat_i);
  * the residual or bonus sample of block row m = b * (K + 1) + row is the
    Gumbel-max argmax_v (log w(v) + g_{m,v}) with w = r (residual, where
    r(v) > 0) or w = p (bonus) and g the Gumbel noise of row m (counter
    (v, m // 4, 0, 0), output m % 4), the same noise the temperature
    sampling of the LM head uses; lowest id among exact ties.  A residual
    with no positive entry (possible only through rounding) falls back to p.
"""
from __future__ import annotations

import numpy as np

from .philox import MASK, philox4x32_10, uniform23

F64 = np.float64


def acceptance_uniforms(seed: int, batch: int, k: int) -> np.ndarray:
    """u[b, i-1] in (0, 1): counter (i - 1, b, 1, 0), output word 0."""
    i = np.arange(k, dtype=np.uint64)
    u = np.empty((batch, k), dtype=F64)
    for b in range(batch):
        out = philox4x32_10(i, np.full(k, b, dtype=np.uint64), 1, 0, seed & MASK, (seed >> 32) & MASK)
        u[b] = uniform23(out[0])
    return u


def gumbel_row(seed: int, m: int, vocab: int) -> np.ndarray:
    """Gumbel noise g[m, :] of one row: counter (v, m // 4, 0, 0), output m % 4."""
    v = np.arange(vocab, dtype=np.uint64)
    out = philox4x32_10(v, np.full(vocab, m // 4, dtype=np.uint64), 0, 0, seed & MASK,
                        (seed >> 32) & MASK)
    return -np.log(-np.log(uniform23(out[m % 4])))


def softmax_rows(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, dtype=F64)
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def sps_round(x, q, draft, seed: int, temperature: float = 1.0):
    """One round of speculative sampling for a batch.

    x [B, K+1, V] target logits of the block rows; q [B, K, V] the draft's
    distributions; draft [B, K] the drafted ids; temperature T > 0.
    Returns a dict:
      target  int64 [B, K+1]: y_hat_i at accepted positions, the residual
              (or bonus) sample at row s - 1, -1 after it
      accept  uint8 [B, K]: 1 at accepted positions, 0 from the rejection on
      ratio   float64 [B, K]: min(1, p_i(y_hat_i) / q_i(y_hat_i)) at every position
      u       float64 [B, K]: the acceptance uniforms
      s       int64 [B]; emitted int64 [B, K+1] (-1 padded)
      margin  float64 [B]: |u - ratio| at the deciding position (the rejection,
              or the smallest over the accepted ones), and
      key_margin float64 [B]: gap between the two largest keys of the sample.
    """
    x = np.asarray(x, dtype=F64)
    q = np.asarray(q, dtype=F64)
    draft = np.asarray(draft).astype(np.int64)
    B, R, V = x.shape
    K = R - 1
    p = softmax_rows(x / temperature)                       # [B, R, V]
    u = acceptance_uniforms(seed, B, K)
    out = dict(target=np.full((B, R), -1, dtype=np.int64), accept=np.zeros((B, K), dtype=np.uint8),
               ratio=np.zeros((B, K)), u=u, s=np.zeros(B, dtype=np.int64),
               emitted=np.full((B, R), -1, dtype=np.int64), margin=np.full(B, np.inf),
               key_margin=np.zeros(B))
    for b in range(B):
        for i in range(1, K + 1):
            y = draft[b, i - 1]
            pi, qi = p[b, i - 1, y], q[b, i - 1, y]
            out["ratio"][b, i - 1] = 1.0 if qi <= 0.0 else min(1.0, pi / qi)
        s = K + 1
        for i in range(1, K + 1):
            y = draft[b, i - 1]
            dec = abs(u[b, i - 1] - out["ratio"][b, i - 1])
            out["margin"][b] = min(out["margin"][b], dec)
            if not (u[b, i - 1] * q[b, i - 1, y] < p[b, i - 1, y]):
                s = i
                break
            out["accept"][b, i - 1] = 1
        row = s - 1
        g = gumbel_row(seed, b * R + row, V)
        w = None
        if s <= K:
            w = np.maximum(p[b, row] - q[b, row], 0.0)
            if not np.any(w > 0.0):
                w = None
        if w is None:
            w = p[b, row]
        with np.errstate(divide="ignore"):
            keys = np.where(w > 0.0, np.log(w), -np.inf) + g
        tok = int(np.argmax(keys))                          # first occurrence = lowest id
        top2 = np.sort(keys)[-2:] if V > 1 else np.array([-np.inf, keys[0]])
        out["key_margin"][b] = top2[1] - top2[0]
        out["s"][b] = s
        out["target"][b, :row] = draft[b, :row]
        out["target"][b, row] = tok
        out["emitted"][b, :row] = draft[b, :row]
        out["emitted"][b, row] = tok
    return out
