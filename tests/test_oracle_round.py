"""Pin of the oracle's whole-round composition (``cospec_round``) on a case
built by hand.

The parts (attention, statistics, features, MLP, scan, commit) have pins of
their own; this case fixes how the round wires them together:
  * block row r scores the draft token y_hat_{r+1} (Eq. 2, Eq. 23:
    l_i = log p_T(y_hat_i | prefix) comes from the row that predicts
    position i), and the bonus row r = K scores nothing (NaN);
  * position i is compared with the argmax of row i-1 (Eq. 3);
  * the arbitration sees the statistics of rows i-1 and i (F0..F7);
  * the accepted length follows Eq. 15 and the round emits
    y_hat_1..y_hat_{s-1} then y_tilde_s;
  * the commit writes block rows 0..s-1 of every layer to positions
    C..C+s-1 through the page table;
  * layer l's attention reads layer l's pool.

Setup: one sequence, K = 3, vocabulary 4, hidden width 4 and W = I, so the
logits of row r are its hidden row.  Every row has two live logits (the other
two at -100, whose weight e^-100 is far below the tolerance), so with a gap
delta between them: lse = max + log(1 + e^-delta) and entropy
H = log(1 + e^-delta) + delta * e^-delta / (1 + e^-delta) (binary softmax).

  row 0  x = [-100, 2, 0, -100]   argmax 1, second 0   (delta 2)
  row 1  x = [1, -100, 2, -100]   argmax 2, second 1   (delta 1)
  row 2  x = [-100, -100, 0, 3]   argmax 3, second 0   (delta 3)
  row 3  x = [2, -100, -100, 1]   argmax 0, second 1   (delta 1, bonus row)
  draft y_hat = [1, 0, 3]: position 1 matches (row 0 -> 1), position 2 is a
  mismatch (row 1 -> 2), position 3 matches (row 2 -> 3).

Draft logits: row 0 -> x0[1] = 2, row 1 -> x1[0] = 1, row 2 -> x2[3] = 3,
row 3 -> NaN.  Features of the mismatch (i = 2, r = 1), with
L1 = log(1 + e^-1), L3 = log(1 + e^-3), q1 = e^-1 / (1 + e^-1):
  F0 = 1 - (2 + L1) = -1 - L1     F1 = -L1       F2 = 1    F3 = L1 + q1
  F4 = 3 - (3 + L3) = -L3         F5 = x2[y_hat_3] - lse2 = -L3
  F6 = 2/3                        F7 = 1/3 (position 1 matched)
MLP with three hidden units:
  unit 0: ReLU(F0 + 3)                  = 2 - L1
  unit 1: ReLU(3 F6 + 3 F7 - 2.5)       = 0.5   (0 if F6 or F7 were off by one)
  unit 2: ReLU(F1 + F2 + F3 + F4 + F5)  = 1 + q1 - 2 L3
  z = unit0 + 2 unit1 + unit2 - 3.25 = 0.75 - L1 + q1 - 2 L3 ~ 0.608,
  p = sigma(z) ~ 0.648.
So with lambda = 0.6 the mismatch is kept (a = 1) and s = K + 1 = 4, emitting
[1, 0, 3, 0]; with lambda = 0.7 it is rejected, s = 2, emitting [1, 2].
"""
import math
import types

import numpy as np
import pytest

from oracle import cospec_oracle as O

DEAD = -100.0
LOGITS = np.array([[DEAD, 2.0, 0.0, DEAD],
                   [1.0, DEAD, 2.0, DEAD],
                   [DEAD, DEAD, 0.0, 3.0],
                   [2.0, DEAD, DEAD, 1.0]])
DRAFT = np.array([[1, 0, 3]])
K, R, V = 3, 4, 4
CTX = 14                       # the commit crosses a page boundary (P = 16)
PAGE_TABLE = np.array([[1, 0]])
V_CONST = (1.5, -2.0)          # every value row of layer 0 / layer 1


def _lse_h(mx, delta):
    L = math.log1p(math.exp(-delta))
    q = math.exp(-delta) / (1.0 + math.exp(-delta))
    return mx + L, L + delta * q


def _inputs():
    L, Hkv, D, P, npages = 2, 1, 2, 16, 2
    rng = np.random.default_rng(0)
    q = rng.standard_normal((L, 1, R, 1, D))
    k_blk = np.arange(L * R * Hkv * D, dtype=np.float64).reshape(L, 1, R, Hkv, D) + 10.0
    v_blk = np.empty((L, 1, R, Hkv, D))
    k_pages = rng.standard_normal((L, npages, Hkv, P, D))
    v_pages = np.empty((L, npages, Hkv, P, D))
    for l in range(L):
        v_blk[l] = V_CONST[l]
        v_pages[l] = V_CONST[l]
    w1 = np.zeros((3, 8))
    w1[0, 0] = 1.0
    w1[1, 6] = 3.0
    w1[1, 7] = 3.0
    w1[2, 1:6] = 1.0
    mlp = (w1, np.array([3.0, -2.5, 0.0]), np.array([1.0, 2.0, 1.0]), np.array(-3.25))
    cfg = types.SimpleNamespace(batch=1, k=K, rows=R, layers=L, page_size=P)
    return dict(cfg=cfg, q=q, k_blk=k_blk, v_blk=v_blk, k_pages=k_pages, v_pages=v_pages,
                page_table_np=PAGE_TABLE, ctx_len_np=np.array([CTX]), hidden=LOGITS.copy(),
                w=np.eye(V), mlp=mlp)


def test_round_statistics_are_wired_row_by_row():
    out = O.cospec_round(_inputs(), DRAFT, lam=0.6)
    assert out["argmax"].tolist() == [[1, 2, 3, 0]]
    expect = []
    for mx, second, delta, dl in ((2.0, 0.0, 2.0, 2.0), (2.0, 1.0, 1.0, 1.0),
                                  (3.0, 0.0, 3.0, 3.0), (2.0, 1.0, 1.0, math.nan)):
        lse, h = _lse_h(mx, delta)
        expect.append([mx, second, lse, h, dl])
    np.testing.assert_allclose(out["stats"][0], np.array(expect), rtol=0, atol=1e-12)
    # the gap between the two largest logits decides each row's candidate
    np.testing.assert_allclose(out["key_margin"], [[2.0, 1.0, 3.0, 1.0]], atol=1e-12)


def test_round_arbitrates_the_mismatch_with_rows_i_minus_1_and_i():
    L1 = math.log1p(math.exp(-1.0))
    L3 = math.log1p(math.exp(-3.0))
    q1 = math.exp(-1.0) / (1.0 + math.exp(-1.0))
    p_mis = 1.0 / (1.0 + math.exp(-(0.75 - L1 + q1 - 2.0 * L3)))
    assert 0.6 + 0.04 < p_mis < 0.7 - 0.04          # both thresholds decide clearly
    out = O.cospec_round(_inputs(), DRAFT, lam=0.6)
    np.testing.assert_allclose(out["p"], [[1.0, p_mis, 1.0]], atol=1e-12)
    assert out["a"].tolist() == [[1, 1, 1]]
    assert out["s"].tolist() == [4]
    assert out["emitted"].tolist() == [[1, 0, 3, 0]]
    rej = O.cospec_round(_inputs(), DRAFT, lam=0.7)
    assert rej["a"].tolist() == [[1, 0, 1]]
    assert rej["s"].tolist() == [2]
    assert rej["emitted"].tolist() == [[1, 2, -1, -1]]


@pytest.mark.parametrize("mode,s,emitted", [(O.POLICY_TARGET, 2, [1, 2, -1, -1]),
                                            (O.POLICY_DRAFT, 4, [1, 0, 3, 0])])
def test_round_forced_policies(mode, s, emitted):
    out = O.cospec_round(_inputs(), DRAFT, lam=0.6, mode=mode)
    assert out["s"].tolist() == [s]
    assert out["emitted"].tolist() == [emitted]


def test_round_commits_the_accepted_rows_of_every_layer():
    inp = _inputs()
    out = O.cospec_round(inp, DRAFT, lam=0.7)          # s = 2: rows 0 and 1
    assert out["ctx_len"].tolist() == [CTX + 2]
    kp = out["k_pages"]
    # positions 14 and 15 are slots 14 and 15 of logical page 0 = physical page 1
    for l in range(2):
        np.testing.assert_array_equal(kp[l, 1, 0, 14], inp["k_blk"][l, 0, 0, 0])
        np.testing.assert_array_equal(kp[l, 1, 0, 15], inp["k_blk"][l, 0, 1, 0])
    untouched = np.ones(kp.shape, dtype=bool)
    untouched[:, 1, 0, 14:16] = False
    np.testing.assert_array_equal(kp[untouched], inp["k_pages"][untouched])
    out4 = O.cospec_round(_inputs(), DRAFT, lam=0.6)   # s = 4: rows 2, 3 cross to page 0
    for l in range(2):
        np.testing.assert_array_equal(out4["k_pages"][l, 0, 0, 0], inp["k_blk"][l, 0, 2, 0])
        np.testing.assert_array_equal(out4["k_pages"][l, 0, 0, 1], inp["k_blk"][l, 0, 3, 0])


def test_round_attention_reads_each_layers_own_pool():
    out = O.cospec_round(_inputs(), DRAFT, lam=0.6)
    # with every value row of a layer equal to c, the attention output is c
    for l, c in enumerate(V_CONST):
        np.testing.assert_allclose(out["attn"][l], c, atol=1e-12)
