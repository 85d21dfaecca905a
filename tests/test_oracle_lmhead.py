"""Pins of the oracle's LM-head statistics (Sec. 3.1 Eq. 2; Eq. 23 log-prob)
to closed forms, tie rules and an independent float64 torch computation."""
import math

import numpy as np
import pytest
import torch

from oracle import cospec_oracle as O


def _onehot_head(logits):
    """hidden = e_0 and W[:, 0] = logits, so x = logits exactly."""
    V = len(logits)
    w = np.zeros((V, 3)); w[:, 0] = logits
    h = np.zeros((1, 3)); h[0, 0] = 1.0
    return h, w


def test_closed_form_four_classes():
    x = [0.0, math.log(2), math.log(3), math.log(2)]
    h, w = _onehot_head(x)
    am, st = O.lmhead_stats(h, w, np.array([3]))
    assert am[0] == 2
    mx, sec, lse, ent, dl = st[0]
    assert mx == pytest.approx(math.log(3), abs=1e-15)
    assert sec == pytest.approx(math.log(2), abs=1e-15)
    assert lse == pytest.approx(3 * math.log(2), abs=1e-14)          # log(1+2+3+2)
    p = [1 / 8, 2 / 8, 3 / 8, 2 / 8]
    assert ent == pytest.approx(-sum(v * math.log(v) for v in p), abs=1e-14)
    assert dl == pytest.approx(math.log(2), abs=1e-15)
    # l_i of Eq. 23 is the log-probability of the draft id: log(2/8)
    assert dl - lse == pytest.approx(math.log(0.25), abs=1e-14)


def test_uniform_logits():
    V = 1000
    h, w = _onehot_head([0.75] * V)
    am, st = O.lmhead_stats(h, w, np.array([-1]))
    assert am[0] == 0                                  # lowest id among ties
    assert st[0, O.STAT_SECOND] == 0.75
    assert st[0, O.STAT_LSE] == pytest.approx(0.75 + math.log(V), abs=1e-12)
    assert st[0, O.STAT_ENTROPY] == pytest.approx(math.log(V), abs=1e-12)
    assert math.isnan(st[0, O.STAT_DRAFT])


def test_tie_breaks_to_lowest_id_and_second_equals_top():
    h, w = _onehot_head([1.0, 5.0, 5.0, 2.0])
    am, st = O.lmhead_stats(h, w, np.array([2]))
    assert am[0] == 1
    assert st[0, O.STAT_MAX] == 5.0 and st[0, O.STAT_SECOND] == 5.0
    assert st[0, O.STAT_DRAFT] == 5.0


def test_two_classes_binary_entropy():
    a, b = 1.25, -0.5
    h, w = _onehot_head([a, b])
    am, st = O.lmhead_stats(h, w, np.array([1]))
    p = 1 / (1 + math.exp(-(a - b)))
    assert am[0] == 0
    assert st[0, O.STAT_LSE] == pytest.approx(math.log(math.exp(a) + math.exp(b)), abs=1e-14)
    assert st[0, O.STAT_ENTROPY] == pytest.approx(-(p * math.log(p) + (1 - p) * math.log(1 - p)), abs=1e-14)
    assert st[0, O.STAT_SECOND] == b


def test_matches_torch_float64_on_random_rows():
    g = torch.Generator().manual_seed(7)
    M, d, V = 6, 64, 3000
    hidden = torch.randn(M, d, generator=g).to(torch.bfloat16)
    w = (torch.randn(V, d, generator=g) * 0.3).to(torch.bfloat16)
    dfr = np.array([5, 17, -1, 2999, 0, 123])
    am, st = O.lmhead_stats(hidden, w, dfr, vocab_chunk=700)
    x = hidden.double() @ w.double().T
    assert np.array_equal(am, torch.argmax(x, dim=1).numpy())
    lse = torch.logsumexp(x, dim=1)
    np.testing.assert_allclose(st[:, O.STAT_LSE], lse.numpy(), rtol=1e-13)
    logp = torch.log_softmax(x, dim=1)
    ent = -(logp.exp() * logp).sum(dim=1)
    np.testing.assert_allclose(st[:, O.STAT_ENTROPY], ent.numpy(), rtol=1e-11, atol=1e-12)
    top2 = torch.topk(x, 2, dim=1).values
    np.testing.assert_allclose(st[:, O.STAT_MAX], top2[:, 0].numpy(), rtol=0, atol=0)
    np.testing.assert_allclose(st[:, O.STAT_SECOND], top2[:, 1].numpy(), rtol=0, atol=0)
    for m in range(M):
        if dfr[m] >= 0:
            assert st[m, O.STAT_DRAFT] == x[m, dfr[m]].item()


def test_feature_bounds_on_random_logits():
    rng = np.random.default_rng(8)
    x = rng.standard_normal((20, 500)) * 3
    d = rng.integers(0, 500, 20)
    am, st = O.row_stats(x, d)
    l = st[:, O.STAT_DRAFT] - st[:, O.STAT_LSE]
    top = st[:, O.STAT_MAX] - st[:, O.STAT_LSE]
    assert np.all(l <= top + 1e-12) and np.all(top <= 0)
    assert np.all(st[:, O.STAT_ENTROPY] >= -1e-12)
    assert np.all(st[:, O.STAT_ENTROPY] <= math.log(500) + 1e-12)


def test_topk_ids_rank_order():
    x = np.array([[0.1, 3.0, 2.0, 3.0, -1.0]])
    assert O.topk_ids(x, 3).tolist() == [[1, 3, 2]]
