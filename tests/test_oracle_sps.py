"""Pins of the oracle's speculative-sampling acceptance (the exact-match
baseline at a temperature, Sec. 3.1 "Stochastic decoding", App. C.3).

What fixes it, other than its own formula:
  * distribution preservation, the algorithm's defining property: every
    emitted token is distributed as the target's p, whatever the draft's q
    (Monte Carlo over many independent sequences);
  * the acceptance probability of a position is sum_v min(p(v), q(v)), so
    with the same p and q at every position the accepted length follows a
    truncated geometric law;
  * a one-hot draft at a token p rarely picks leaves p renormalised over the
    other tokens as the residual;
  * at a vanishing temperature with one-hot (greedy) drafts it reduces to
    exact-match speculative decoding (Eq. 4) emitting the target argmax;
  * a draft equal to the target is always accepted.
"""
import numpy as np
import pytest

from oracle import cospec_oracle as O
from oracle import cospec_sps as S

P_ROW = np.array([0.4, 0.25, 0.2, 0.1, 0.05])
Q_ROW = np.array([0.1, 0.5, 0.1, 0.25, 0.05])
BETA = float(np.minimum(P_ROW, Q_ROW).sum())        # 0.6
V = len(P_ROW)


def _batch(B, K, p=P_ROW, q=Q_ROW, seed=0):
    x = np.broadcast_to(np.log(p), (B, K + 1, V)).copy()
    qq = np.broadcast_to(q, (B, K, V)).copy()
    rng = np.random.default_rng(seed)
    draft = np.array([[rng.choice(V, p=q) for _ in range(K)] for _ in range(B)])
    return x, qq, draft


def _freq(tokens):
    tokens = np.asarray(tokens)
    return np.bincount(tokens, minlength=V) / len(tokens)


def test_first_token_follows_the_target_distribution():
    B = 12000
    x, q, draft = _batch(B, 1)
    out = S.sps_round(x, q, draft, seed=11)
    np.testing.assert_allclose(_freq(out["emitted"][:, 0]), P_ROW, atol=0.02)
    # position 1 is accepted with probability sum_v min(p, q)
    assert abs(out["accept"][:, 0].mean() - BETA) < 0.02


def test_accepted_length_is_truncated_geometric_and_every_token_follows_p():
    B, K = 8000, 3
    x, q, draft = _batch(B, K, seed=1)
    out = S.sps_round(x, q, draft, seed=12)
    s = out["s"]
    law = [(1 - BETA) * BETA ** (j - 1) for j in range(1, K + 1)] + [BETA ** K]
    np.testing.assert_allclose(np.bincount(s, minlength=K + 2)[1:] / B, law, atol=0.02)
    np.testing.assert_allclose(_freq(out["emitted"][:, 0]), P_ROW, atol=0.02)
    second = out["emitted"][s >= 2, 1]
    np.testing.assert_allclose(_freq(second), P_ROW, atol=0.03)
    # accepted positions carry the draft, the stop row the sample, then -1
    for b in range(20):
        n = s[b]
        assert np.array_equal(out["target"][b, : n - 1], draft[b, : n - 1])
        assert np.all(out["target"][b, n:] == -1)
        assert out["accept"][b, : n - 1].all() and not out["accept"][b, n - 1:].any()


def test_one_hot_draft_leaves_the_renormalised_target_as_residual():
    B = 10000
    q = np.eye(V)[4]                                   # the draft always proposes token 4
    x, qq, draft = _batch(B, 1, q=q)
    out = S.sps_round(x, qq, draft, seed=13)
    rej = out["s"] == 1
    assert abs(1 - rej.mean() - P_ROW[4]) < 0.01    # accepted with probability p(4) / 1
    expect = np.append(P_ROW[:4], 0.0) / P_ROW[:4].sum()
    np.testing.assert_allclose(_freq(out["emitted"][rej, 0]), expect, atol=0.02)
    # the residual never proposes the rejected token
    assert not np.any(out["emitted"][rej, 0] == 4)


def test_temperature_scales_the_target():
    B, T = 12000, 2.0
    x, q, draft = _batch(B, 1)
    out = S.sps_round(x, q, draft, seed=14, temperature=T)
    pt = np.sqrt(P_ROW) / np.sqrt(P_ROW).sum()        # softmax(log p / 2)
    np.testing.assert_allclose(_freq(out["emitted"][:, 0]), pt, atol=0.02)


def test_vanishing_temperature_with_greedy_drafts_is_exact_match_decoding():
    rng = np.random.default_rng(5)
    B, K, Vb = 64, 6, 40
    x = rng.standard_normal((B, K + 1, Vb)) * 3
    am = np.argmax(x, axis=2)
    draft = np.where(rng.random((B, K)) < 0.7, am[:, :K], rng.integers(0, Vb, (B, K)))
    q = np.eye(Vb)[draft]                              # a greedy draft is one-hot
    out = S.sps_round(x, q, draft, seed=15, temperature=1e-4)
    s_ref = O.strict_spd_length(draft, am)             # Eq. 4
    assert np.array_equal(out["s"], s_ref)
    for b in range(B):
        n = s_ref[b]
        assert out["emitted"][b, n - 1] == am[b, n - 1]
        assert np.array_equal(out["emitted"][b, : n - 1], draft[b, : n - 1])


def test_draft_equal_to_target_is_always_accepted():
    B, K = 500, 4
    x, q, draft = _batch(B, K, q=P_ROW)
    out = S.sps_round(x, q, draft, seed=16)
    assert np.all(out["s"] == K + 1) and out["accept"].all()
    np.testing.assert_allclose(out["ratio"], 1.0)
    np.testing.assert_allclose(_freq(out["emitted"][:, K]), P_ROW, atol=0.06)


@pytest.mark.parametrize("seed", [0, 0x1234_5678_9ABC])
def test_acceptance_uniforms_depend_on_sequence_position_and_seed(seed):
    u = S.acceptance_uniforms(seed, 3, 4)
    assert np.all((u > 0) & (u < 1))
    assert len(np.unique(u)) == u.size
    assert not np.array_equal(u, S.acceptance_uniforms(seed + 1, 3, 4))


def test_bonus_is_the_lm_head_temperature_sample_of_row_k():
    # With every position accepted the round emits a sample of p_{K+1}; it
    # uses block row m = b (K + 1) + K's Gumbel noise, so it equals the
    # temperature sample the LM head draws for that row (same seed).
    rng = np.random.default_rng(8)
    B, K, Vb, T, seed = 6, 3, 50, 0.7, 0xABCDEF0123
    x = rng.standard_normal((B, K + 1, Vb)) * 2
    q = S.softmax_rows(x[:, :K] / T)                   # the draft equals the target
    draft = np.argmax(x[:, :K], axis=2)
    out = S.sps_round(x, q, draft, seed=seed, temperature=T)
    assert np.all(out["s"] == K + 1)
    sample, _ = O.row_stats_sampled(x.reshape(B * (K + 1), Vb), np.full(B * (K + 1), -1), seed, T)
    assert np.array_equal(out["emitted"][:, K], sample.reshape(B, K + 1)[:, K])
