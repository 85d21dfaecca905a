"""CPU oracle for one CoSpec verify/arbitrate round -- TEST INFRASTRUCTURE ONLY.

Plain, slow, float64 NumPy restatement of what the round computes, written
from the paper ("Beyond the Target: From Imitation to Collaboration in
Speculative Decoding", CoSpec).  It shares no code with the CUDA path and is
only imported by the test-suite, by ``__graft_entry__.smoke()`` and by the
CPU-baseline leg of ``bench.py``.  No product path calls it.

Every floating-point input arrives as bf16 values (exact in float64); all
arithmetic below is float64.

Pins (what fixes each function other than itself; see tests/test_oracle_*.py):
  verify_attention      brute force on tiny inputs, closed forms (two-key
                        3:1 weights, constant V, single visible key), GQA
                        head mapping, causality, paged == contiguous; the
                        full block mask against the arbitrator's hybrid mask
                        over a dense sequence (Sec. 3.3).
  lmhead_stats          closed forms (one-hot logits, uniform logits, two
                        classes), tie-break, torch float64 cross-check.
  row_stats_sampled     Philox4x32-10 known-answer vectors of the generator's
                        authors; Gumbel moments (Euler's constant, pi^2/6);
                        sample frequencies against softmax; T -> 0 gives the
                        argmax.
  arbitration_features  hand-derived golden case (tests/golden).
  arbitration_mlp       parity unpinned: the paper defines no feature MLP;
                        only a hand-computed 2-input example fixes the formula.
  arbitrate / accept_scan  golden cases derived by hand from Eq. 4 and
                        Eq. 15, exhaustive comparison with the sequential
                        procedure of App. F (Inference Procedure).
  commit_kv             byte equality of touched / untouched slots.
  cospec_round          a whole round built by hand (identity LM head, rows
                        with two live logits, one mismatch, a three-unit MLP,
                        a two-layer commit across a page boundary): which row
                        scores which draft token, the bonus row's NaN, the
                        rows each position's features read, s, the emitted
                        tokens, key margins, per-layer pools.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np

F64 = np.float64


def _f64(x) -> np.ndarray:
    """Convert a NumPy array or a torch tensor (any dtype, any device) to float64."""
    if hasattr(x, "detach"):
        x = x.detach().to("cpu")
        import torch  # local: the oracle itself needs only NumPy
        x = x.to(torch.float64).numpy()
    return np.asarray(x, dtype=F64)


def _i64(x) -> np.ndarray:
    if hasattr(x, "detach"):
        x = x.detach().to("cpu").numpy()
    return np.asarray(x).astype(np.int64)


# ---------------------------------------------------------------------------
# Step 1: verify attention (Sec. 3.1, Eq. 2)
# ---------------------------------------------------------------------------

def gather_context(pages, page_table_row, ctx_len: int, page_size: int) -> np.ndarray:
    """Contiguous view [C, Hkv, D] of one sequence's committed KV.

    Token t of the prefix lives in physical page page_table_row[t // P],
    slot t % P (pages laid out [num_pages, Hkv, P, D]).
    """
    t = np.arange(ctx_len)
    phys = np.asarray(page_table_row)[t // page_size]
    return np.asarray(pages)[phys, :, t % page_size, :]


def verify_attention(q, k_blk, v_blk, k_pages, v_pages, page_table, ctx_len,
                     page_size: int, scale: Optional[float] = None,
                     seqs: Optional[Sequence[int]] = None,
                     heads: Optional[Sequence[int]] = None,
                     block_mask: str = "causal") -> np.ndarray:
    """Attention of the block rows of one layer (teacher-forced verify, Eq. 2).

    q [B,R,Hq,D]; k_blk, v_blk [B,R,Hkv,D] (the block's own keys/values);
    k_pages, v_pages [num_pages,Hkv,P,D]; page_table [B,max_pages];
    ctx_len [B].  Block row j of sequence b sits at absolute position C_b + j
    and attends to the C_b committed positions and to block rows 0..j
    (``block_mask="causal"``), or to every block row (``"full"``: the
    draft/target region of the arbitrator input, Sec. 3.3, which sees the
    whole context and itself bidirectionally).  Query head h reads KV head
    floor(h / G), G = Hq / Hkv.  Returns o [B,R,Hq,D] float64; rows of
    sequences / heads not selected by ``seqs`` / ``heads`` are left at zero.
    """
    if block_mask not in ("causal", "full"):
        raise ValueError(block_mask)
    q = _f64(q); k_blk = _f64(k_blk); v_blk = _f64(v_blk)
    k_pages = _f64(k_pages); v_pages = _f64(v_pages)
    page_table = _i64(page_table); ctx_len = _i64(ctx_len)
    B, R, Hq, D = q.shape
    Hkv = k_blk.shape[2]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    out = np.zeros((B, R, Hq, D), dtype=F64)
    for b in (range(B) if seqs is None else seqs):
        C = int(ctx_len[b])
        keys = np.concatenate([gather_context(k_pages, page_table[b], C, page_size), k_blk[b]], axis=0)
        vals = np.concatenate([gather_context(v_pages, page_table[b], C, page_size), v_blk[b]], axis=0)
        # visible[j, t]: key position t is seen by block row j iff t <= C + j
        # (causal), every position (full)
        if block_mask == "causal":
            visible = np.arange(C + R)[None, :] <= (C + np.arange(R))[:, None]
        else:
            visible = np.ones((R, C + R), dtype=bool)
        for h in (range(Hq) if heads is None else heads):
            kvh = h // G
            s = (q[b, :, h, :] @ keys[:, kvh, :].T) * scale           # [R, C+R]
            s = np.where(visible, s, -np.inf)
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p = p / p.sum(axis=1, keepdims=True)
            out[b, :, h, :] = p @ vals[:, kvh, :]
    return out


def hybrid_mask(l_c: int, n_region: int) -> np.ndarray:
    """The arbitrator's attention pattern over q = [c, region] (Sec. 3.3):
    context positions attend causally within the context; region positions
    (the draft/target block with its separators) attend to the whole context
    and to the whole region; no context position attends to the region.
    Returns visible [l, l] (query, key), l = l_c + n_region."""
    l = l_c + n_region
    i = np.arange(l)[:, None]
    t = np.arange(l)[None, :]
    return np.where(i < l_c, t <= i, True)


def dense_masked_attention(q, k, v, visible, scale: Optional[float] = None) -> np.ndarray:
    """softmax(q k^T * scale, masked) v for one head over a dense sequence:
    q, k, v [l, D], visible [l, l] boolean.  float64."""
    q = _f64(q); k = _f64(k); v = _f64(v)
    if scale is None:
        scale = 1.0 / math.sqrt(q.shape[1])
    s = np.where(visible, (q @ k.T) * scale, -np.inf)
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    return (p / p.sum(axis=1, keepdims=True)) @ v


# ---------------------------------------------------------------------------
# Step 2: LM head, argmax and log-prob statistics (Sec. 3.1 Eq. 2, Eq. 23)
# ---------------------------------------------------------------------------

STAT_MAX, STAT_SECOND, STAT_LSE, STAT_ENTROPY, STAT_DRAFT = range(5)


def lmhead_logits(hidden, w, vocab_chunk: int = 16384) -> np.ndarray:
    """x[m, v] = <hidden_m, W_v> in float64, [M, V].

    Each logit is one independent dot product; the vocabulary is visited in
    chunks only to bound the float64 copy of W.
    """
    h = _f64(hidden)
    V = w.shape[0]
    x = np.empty((h.shape[0], V), dtype=F64)
    for v0 in range(0, V, vocab_chunk):
        x[:, v0:v0 + vocab_chunk] = h @ _f64(w[v0:v0 + vocab_chunk]).T
    return x


def row_stats(x: np.ndarray, draft_for_row) -> tuple:
    """Per-row statistics of logits x [M, V].

    argmax: target prediction y_tilde (lowest id among exact ties);
    max, second (largest logit over ids != argmax), lse = log sum_v e^{x_v},
    entropy H = -sum_v p_v log p_v = lse - sum_v p_v x_v,
    draft_logit = x[draft_for_row] (NaN where draft_for_row < 0).
    Returns (argmax int64 [M], stats float64 [M, 5]).
    """
    x = np.asarray(x, dtype=F64)
    M, V = x.shape
    d = _i64(draft_for_row)
    am = np.argmax(x, axis=1)                     # first occurrence = lowest id
    rows = np.arange(M)
    mx = x[rows, am]
    rest = x.copy()
    rest[rows, am] = -np.inf
    second = rest.max(axis=1) if V > 1 else np.full(M, -np.inf)
    lse = mx + np.log(np.exp(x - mx[:, None]).sum(axis=1))
    p = np.exp(x - lse[:, None])
    entropy = lse - (p * x).sum(axis=1)
    draft_logit = np.where(d >= 0, x[rows, np.clip(d, 0, V - 1)], np.nan)
    stats = np.stack([mx, second, lse, entropy, draft_logit], axis=1)
    return am.astype(np.int64), stats


def gumbel_keys(x: np.ndarray, seed: int, temperature: float = 1.0) -> np.ndarray:
    """Perturbed keys x_v / T + g_v of the Gumbel-max rule, g = -log(-log u) with
    u from the Philox4x32-10 stream of `seed` (oracle/philox.py), [M, V]."""
    from .philox import gumbel_noise
    x = np.asarray(x, dtype=F64)
    return x / temperature + gumbel_noise(seed, x.shape[0], x.shape[1])


def row_stats_sampled(x: np.ndarray, draft_for_row, seed: int, temperature: float = 1.0):
    """Stochastic decoding (Sec. 3.1 "Stochastic decoding", App. C.3): the
    target candidate is a sample of softmax(x / T), drawn as the argmax of the
    Gumbel-perturbed keys (lowest id among exact ties).  The statistics are
    those of the logits themselves (as in row_stats).
    Returns (sample int64 [M], stats float64 [M, 5])."""
    _, stats = row_stats(x, draft_for_row)
    return np.argmax(gumbel_keys(x, seed, temperature), axis=1).astype(np.int64), stats


def lmhead_stats_sampled(hidden, w, draft_for_row, seed: int, temperature: float = 1.0,
                         vocab_chunk: int = 16384):
    """LM-head contraction with a temperature-T sample in place of the argmax."""
    return row_stats_sampled(lmhead_logits(hidden, w, vocab_chunk), draft_for_row, seed, temperature)


def lmhead_stats(hidden, w, draft_for_row, vocab_chunk: int = 16384):
    """LM-head contraction fused with argmax and statistics (Eq. 2, Eq. 23)."""
    return row_stats(lmhead_logits(hidden, w, vocab_chunk), draft_for_row)


def topk_ids(x: np.ndarray, t: int) -> np.ndarray:
    """Ids of the t largest logits per row, in rank order (ties: lowest id first)."""
    order = np.argsort(-np.asarray(x, dtype=F64), axis=1, kind="stable")
    return order[:, :t]


# ---------------------------------------------------------------------------
# Step 3: arbitration (Sec. 3.3, Eq. 13, Eq. 14, Eq. 17)
# ---------------------------------------------------------------------------

def arbitration_features(draft, argmax, stats) -> np.ndarray:
    """Feature vector f_i, i = 1..K, of each draft position; shape [B, K, 8].

    The paper's arbitrator reads the context, the draft block and the target
    verification tokens (Eq. 9) and scores each draft position with a head on
    its hidden state (Eq. 11).  This build's reading replaces that LM by a
    feature MLP fed with quantities the paper names, all of which are
    independent of the round's actions (Eq. 9 holds no action), with
    r = i - 1 the block row that predicts position i:
      F0 = l_i = x_r[y_hat_i] - lse_r    target log-prob of the draft (Eq. 23)
      F1 = max_r - lse_r                 target log-prob of y_tilde_i
      F2 = max_r - second_r              top-1 / top-2 margin
      F3 = H_r                           target entropy at row r
      F4 = max_i - lse_i                 target confidence one row later,
                                         after reading y_hat_i (bonus row at i=K)
      F5 = l_{i+1} (0 at i = K)          log-prob of the next draft token
      F6 = i / K                         position in the block
      F7 = #{j < i : Delta_j = 1} / K    matches before position i (Eq. 3)
    draft [B,K]; argmax [B,K+1]; stats [B,K+1,5].
    """
    draft = _i64(draft)
    argmax = _i64(argmax)
    st = _f64(stats)
    B, K = draft.shape
    f = np.zeros((B, K, 8), dtype=F64)
    for b in range(B):
        delta = (draft[b] == argmax[b, :K]).astype(np.int64)
        for i in range(1, K + 1):
            r = i - 1
            mx, sec, lse, ent, dl = st[b, r]
            f[b, r, 0] = dl - lse
            f[b, r, 1] = mx - lse
            f[b, r, 2] = mx - sec
            f[b, r, 3] = ent
            f[b, r, 4] = st[b, i, STAT_MAX] - st[b, i, STAT_LSE]
            f[b, r, 5] = (st[b, i, STAT_DRAFT] - st[b, i, STAT_LSE]) if i < K else 0.0
            f[b, r, 6] = i / K
            f[b, r, 7] = delta[:r].sum() / K
    return f


def arbitration_mlp(f, w1, b1, w2, b2) -> np.ndarray:
    """z = w2 . ReLU(W1 f + b1) + b2 (one hidden layer), f [..., 8] -> z [...].

    Stands in for the head g_phi of Eq. 11 (parity unpinned: the paper gives
    no formula for a feature MLP).
    """
    f = _f64(f)
    hid = np.maximum(f @ _f64(w1).T + _f64(b1), 0.0)
    return hid @ _f64(w2) + float(_f64(b2))


POLICY_MLP, POLICY_TARGET, POLICY_DRAFT = 0, 1, 2


def sigmoid(z):
    z = np.asarray(z, dtype=F64)
    return 1.0 / (1.0 + np.exp(-z))


def arbitrate(draft, argmax, stats, w1, b1, w2, b2, lam: float, mode: int = POLICY_MLP):
    """Acceptance probability p_i and action a_i of every draft position.

    Delta_i = 1[y_hat_i = y_tilde_i] (Eq. 3).  Matches are forced accepted:
    z_tilde = +inf, so p_i = sigma(+inf) = 1 and a_i = 1 (Eq. 13-14).  At a
    mismatch p_i = sigma(z_i) with z_i from the MLP (mode 0), or the forced
    policies p_i = 0 ("always target", mode 1) and p_i = 1 ("always draft",
    mode 2); the deterministic rule is a_i = 1[p_i > lambda] (Eq. 17, strict).
    Returns p float64 [B,K], a uint8 [B,K].
    """
    draft = _i64(draft)
    argmax = _i64(argmax)
    B, K = draft.shape
    match = draft == argmax[:, :K]
    if mode == POLICY_MLP:
        z = arbitration_mlp(arbitration_features(draft, argmax, stats), w1, b1, w2, b2)
        p_mis = sigmoid(z)
    elif mode == POLICY_TARGET:
        p_mis = np.zeros((B, K))
    elif mode == POLICY_DRAFT:
        p_mis = np.ones((B, K))
    else:
        raise ValueError("unknown policy mode")
    p = np.where(match, 1.0, p_mis)
    a = np.where(match, 1, (p > lam).astype(np.int64)).astype(np.uint8)
    return p, a


# ---------------------------------------------------------------------------
# Step 4: accepted length and emitted tokens (Eq. 4, Eq. 15)
# ---------------------------------------------------------------------------

def accept_scan(draft, argmax, accept):
    """s = min{i : Delta_i = 0 and a_i = 0}, else K+1 (Eq. 15).

    The round emits y_hat_1..y_hat_{s-1} followed by y_tilde_s (y_tilde_{K+1},
    the bonus, when s = K+1).  Returns s int64 [B] and emitted int64 [B, K+1]
    padded with -1.
    """
    draft = _i64(draft)
    argmax = _i64(argmax)
    accept = _i64(accept)
    B, K = draft.shape
    s = np.full(B, K + 1, dtype=np.int64)
    emitted = np.full((B, K + 1), -1, dtype=np.int64)
    for b in range(B):
        rejected = [i for i in range(1, K + 1)
                    if draft[b, i - 1] != argmax[b, i - 1] and accept[b, i - 1] == 0]
        if rejected:
            s[b] = min(rejected)
        n = int(s[b])
        emitted[b, : n - 1] = draft[b, : n - 1]
        emitted[b, n - 1] = argmax[b, n - 1]
    return s, emitted


def strict_spd_length(draft, argmax) -> np.ndarray:
    """Exact-match speculative decoding length (Eq. 4): first mismatch, else K+1."""
    draft = _i64(draft)
    argmax = _i64(argmax)
    B, K = draft.shape
    s = np.full(B, K + 1, dtype=np.int64)
    for b in range(B):
        mism = [i for i in range(1, K + 1) if draft[b, i - 1] != argmax[b, i - 1]]
        if mism:
            s[b] = min(mism)
    return s


# ---------------------------------------------------------------------------
# Step 5: KV commit of the accepted prefix (round structure of Eq. 15)
# ---------------------------------------------------------------------------

def commit_kv(k_blk, v_blk, k_pages, v_pages, page_table, ctx_len, s, page_size: int):
    """Append block rows 0..s_b-1 of every layer to the paged cache.

    Block row t of sequence b becomes prefix position C_b + t: physical page
    page_table[b, (C_b + t) // P], slot (C_b + t) % P.  Rows the round did
    not make final never reach the cache.  k_blk, v_blk [L,B,R,Hkv,D];
    pages [L,num_pages,Hkv,P,D] (NumPy arrays, any dtype; copied, not
    modified).  Returns (k_pages', v_pages', ctx_len + s).
    """
    kp = np.array(k_pages, copy=True)
    vp = np.array(v_pages, copy=True)
    page_table = _i64(page_table)
    ctx = _i64(ctx_len)
    s = _i64(s)
    L = kp.shape[0]
    for b in range(len(ctx)):
        for t in range(int(s[b])):
            pos = int(ctx[b]) + t
            page = page_table[b, pos // page_size]
            slot = pos % page_size
            for l in range(L):
                kp[l, page, :, slot, :] = k_blk[l, b, t]
                vp[l, page, :, slot, :] = v_blk[l, b, t]
    return kp, vp, ctx + s


# ---------------------------------------------------------------------------
# A whole round
# ---------------------------------------------------------------------------

def cospec_round(inp: dict, draft, lam: float, mode: int = POLICY_MLP,
                 with_attention: bool = True, with_commit: bool = True,
                 sample_seed: Optional[int] = None, temperature: float = 1.0) -> dict:
    """All five steps on the inputs drawn by the workload generator.

    ``inp`` holds q, k_blk, v_blk, k_pages, v_pages (per layer, leading L),
    page_table_np, ctx_len_np, hidden, w, mlp, cfg.  With ``sample_seed`` the
    target candidates are temperature samples (stochastic decoding, Sec. 3.1)
    instead of the argmax; ``key_margin`` [B, R] is the gap between the two
    largest keys that decided each row's candidate (logit or perturbed key).
    """
    cfg = inp["cfg"]
    B, K, R = cfg.batch, cfg.k, cfg.rows
    out = {}
    if with_attention:
        out["attn"] = [verify_attention(inp["q"][l], inp["k_blk"][l], inp["v_blk"][l],
                                        inp["k_pages"][0 if inp.get("alias_layers") else l],
                                        inp["v_pages"][0 if inp.get("alias_layers") else l],
                                        inp["page_table_np"], inp["ctx_len_np"], cfg.page_size)
                       for l in range(cfg.layers)]
    d = np.asarray(draft).reshape(B, K)
    dfr = np.full((B, R), -1, dtype=np.int64)
    dfr[:, :K] = d
    x = lmhead_logits(inp["hidden"], inp["w"])
    if sample_seed is None:
        am, st = row_stats(x, dfr.reshape(-1))
        keys = x
    else:
        am, st = row_stats_sampled(x, dfr.reshape(-1), sample_seed, temperature)
        keys = gumbel_keys(x, sample_seed, temperature)
    top2 = np.sort(keys, axis=1)[:, -2:] if keys.shape[1] > 1 else np.concatenate(
        [np.full((keys.shape[0], 1), -np.inf), keys], axis=1)
    out["key_margin"] = (top2[:, 1] - top2[:, 0]).reshape(B, R)
    out["logits"] = x
    out["argmax"] = am.reshape(B, R)
    out["stats"] = st.reshape(B, R, 5)
    w1, b1, w2, b2 = inp["mlp"]
    p, a = arbitrate(d, out["argmax"], out["stats"], w1, b1, w2, b2, lam, mode)
    out["p"], out["a"] = p, a
    s, emitted = accept_scan(d, out["argmax"], a)
    out["s"], out["emitted"] = s, emitted
    if with_commit:
        kb = _to_np(inp["k_blk"]); vb = _to_np(inp["v_blk"])
        kp = _to_np(inp["k_pages"]); vp = _to_np(inp["v_pages"])
        out["k_pages"], out["v_pages"], out["ctx_len"] = commit_kv(
            kb, vb, kp, vp, inp["page_table_np"], inp["ctx_len_np"], s, cfg.page_size)
    return out


def _to_np(t):
    """Raw copy of a tensor's values (bf16 kept as its 16-bit pattern)."""
    if hasattr(t, "detach"):
        import torch
        t = t.detach().to("cpu")
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).numpy().copy()
        return t.numpy().copy()
    return np.array(t, copy=True)
