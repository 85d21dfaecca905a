"""Pins of the oracle's arbitration, acceptance scan and KV commit
(Sec. 3.3 Eq. 13-15, Eq. 17; Sec. 3.1 Eq. 4; App. F Inference Procedure)."""
import itertools
import math
import os

import numpy as np
import pytest

from oracle import cospec_oracle as O


def _load_accept_cases(golden_dir):
    cases = []
    with open(os.path.join(golden_dir, "accept_cases.txt")) as fh:
        for line in fh:
            if not line.strip() or line.startswith("#"):
                continue
            cols = [c.split() for c in line.split("|")]
            K = int(cols[0][0])
            cases.append(dict(K=K, draft=[int(v) for v in cols[1]], target=[int(v) for v in cols[2]],
                              a=[int(v) for v in cols[3]], s=int(cols[4][0]),
                              emitted=[int(v) for v in cols[5]], s_strict=int(cols[6][0])))
    return cases


def test_golden_accept_cases(golden_dir):
    cases = _load_accept_cases(golden_dir)
    assert len(cases) >= 9
    for c in cases:
        K = c["K"]
        draft = np.array(c["draft"], dtype=np.int64).reshape(1, K)
        target = np.array(c["target"], dtype=np.int64).reshape(1, K + 1)
        a = np.array(c["a"], dtype=np.int64).reshape(1, K)
        s, em = O.accept_scan(draft, target, a)
        assert s[0] == c["s"], c
        assert em[0, : s[0]].tolist() == c["emitted"], c
        assert np.all(em[0, s[0]:] == -1)
        assert O.strict_spd_length(draft, target)[0] == c["s_strict"], c


def _sequential_round(draft, target, a):
    """App. F read literally: walk the block, keep matched or accepted drafts,
    stop at the first rejected mismatch with the target token, else add the bonus."""
    out = []
    for i, (d, t) in enumerate(zip(draft, target[:-1])):
        if d == t or a[i] == 1:
            out.append(d)
        else:
            out.append(t)
            return out
    out.append(target[-1])
    return out


@pytest.mark.parametrize("K", [0, 1, 2, 3, 5, 7])
def test_exhaustive_actions_match_sequential_procedure(K):
    rng = np.random.default_rng(K)
    for _ in range(6):
        target = rng.integers(0, 4, K + 1)
        draft = np.where(rng.random(K) < 0.5, target[:K], rng.integers(0, 4, K))
        for acts in itertools.product([0, 1], repeat=K):
            a = np.array(acts, dtype=np.int64).reshape(1, K)
            s, em = O.accept_scan(draft.reshape(1, K), target.reshape(1, K + 1), a)
            seq = _sequential_round(list(draft), list(target), acts)
            assert s[0] == len(seq) and 1 <= s[0] <= K + 1
            assert em[0, : s[0]].tolist() == seq


def _random_stats(rng, B, R, V=50):
    x = rng.standard_normal((B * R, V)) * 2
    am, st = O.row_stats(x, rng.integers(0, V, B * R))
    return x, am.reshape(B, R), st.reshape(B, R, 5)


def _mlp(rng, H=16):
    return (rng.standard_normal((H, 8)), rng.standard_normal(H), rng.standard_normal(H), 0.1)


def test_forced_policies_reduce_to_spd_and_full_block():
    rng = np.random.default_rng(11)
    B, K = 64, 6
    _, am, st = _random_stats(rng, B, K + 1)
    draft = np.where(rng.random((B, K)) < 0.6, am[:, :K], rng.integers(0, 50, (B, K)))
    w1, b1, w2, b2 = _mlp(rng)
    # always target -> exact-match SPD (Eq. 4)
    p, a = O.arbitrate(draft, am, st, w1, b1, w2, b2, 0.6, O.POLICY_TARGET)
    s, em = O.accept_scan(draft, am, a)
    np.testing.assert_array_equal(s, O.strict_spd_length(draft, am))
    # always draft -> the whole block plus the bonus token
    p, a = O.arbitrate(draft, am, st, w1, b1, w2, b2, 0.6, O.POLICY_DRAFT)
    s, em = O.accept_scan(draft, am, a)
    assert np.all(s == K + 1)
    np.testing.assert_array_equal(em[:, :K], draft)
    np.testing.assert_array_equal(em[:, K], am[:, K])


def test_block_size_one_is_greedy():
    rng = np.random.default_rng(12)
    x, am, st = _random_stats(rng, 5, 1)
    draft = np.zeros((5, 0), dtype=np.int64)
    p, a = O.arbitrate(draft, am, st, *_mlp(rng), 0.6)
    s, em = O.accept_scan(draft, am, a)
    assert np.all(s == 1)
    np.testing.assert_array_equal(em[:, 0], np.argmax(x, axis=1))


def test_matches_forced_even_with_minus_infinite_score():
    rng = np.random.default_rng(13)
    B, K = 16, 5
    _, am, st = _random_stats(rng, B, K + 1)
    draft = np.where(rng.random((B, K)) < 0.5, am[:, :K], (am[:, :K] + 1) % 50)
    w1, b1, w2, _ = _mlp(rng)
    p, a = O.arbitrate(draft, am, st, w1 * 0, b1 * 0, w2 * 0, -np.inf, 0.6)
    match = draft == am[:, :K]
    assert np.all(a[match] == 1) and np.all(p[match] == 1.0)
    assert np.all(a[~match] == 0) and np.all(p[~match] == 0.0)
    s, _ = O.accept_scan(draft, am, a)
    np.testing.assert_array_equal(s, O.strict_spd_length(draft, am))


def test_threshold_is_strict():
    rng = np.random.default_rng(14)
    _, am, st = _random_stats(rng, 1, 2)
    draft = ((am[:, :1] + 1) % 50)                 # one mismatch
    H = 4
    zero = (np.zeros((H, 8)), np.zeros(H), np.zeros(H))
    # z = b2 = logit(0.6)  ->  p == 0.6 exactly in float64? use p = 0.5 at lambda 0.5
    p, a = O.arbitrate(draft, am, st, *zero, 0.0, 0.5)
    assert p[0, 0] == 0.5 and a[0, 0] == 0
    p, a = O.arbitrate(draft, am, st, *zero, 1e-9, 0.5)
    assert a[0, 0] == 1


def test_golden_features(golden_dir):
    rows, feats = [], []
    with open(os.path.join(golden_dir, "features_case.txt")) as fh:
        for line in fh:
            parts = line.split()
            if not parts or parts[0].startswith("#"):
                continue
            if parts[0] == "draft":
                draft = np.array([int(v) for v in parts[1:]]).reshape(1, -1)
            elif parts[0] == "argmax":
                am = np.array([int(v) for v in parts[1:]]).reshape(1, -1)
            elif parts[0] == "row":
                rows.append([float(v) for v in parts[1:]])
            elif parts[0] == "feat":
                feats.append([float(v) for v in parts[1:]])
    st = np.array(rows).reshape(1, -1, 5)
    f = O.arbitration_features(draft, am, st)
    np.testing.assert_allclose(f[0], np.array(feats), rtol=0, atol=1e-15)


def test_mlp_hand_example():
    # two hidden units: pre-activations [1.5, -1.75] -> ReLU [1.5, 0] -> z = 2*1.5 - 1 = 2
    w1 = np.zeros((2, 8)); w1[0, 0] = 1.0; w1[1, 1] = -1.0
    b1 = np.array([0.5, 0.25]); w2 = np.array([2.0, 3.0])
    f = np.zeros(8); f[0] = 1.0; f[1] = 2.0
    z = O.arbitration_mlp(f, w1, b1, w2, -1.0)
    assert z == 2.0
    assert O.sigmoid(z) == pytest.approx(1 / (1 + math.exp(-2.0)), abs=1e-16)


def test_commit_writes_only_accepted_rows():
    rng = np.random.default_rng(15)
    L, B, R, Hkv, D, P = 2, 3, 5, 2, 4, 4
    ctx = np.array([6, 0, 3])
    need = (ctx + R + P - 1) // P
    num = int(need.sum())
    perm = rng.permutation(num)
    table = np.full((B, need.max()), -1)
    st = 0
    for b in range(B):
        table[b, :need[b]] = perm[st:st + need[b]]; st += need[b]
    kp = rng.integers(-1000, 1000, (L, num, Hkv, P, D)).astype(np.int16)
    vp = rng.integers(-1000, 1000, (L, num, Hkv, P, D)).astype(np.int16)
    kb = rng.integers(-1000, 1000, (L, B, R, Hkv, D)).astype(np.int16)
    vb = rng.integers(-1000, 1000, (L, B, R, Hkv, D)).astype(np.int16)
    s = np.array([3, 5, 1])
    kp2, vp2, ctx2 = O.commit_kv(kb, vb, kp, vp, table, ctx, s, P)
    np.testing.assert_array_equal(ctx2, ctx + s)
    touched = np.zeros((num, P), dtype=bool)
    for b in range(B):
        for t in range(s[b]):
            pos = ctx[b] + t
            pg, sl = table[b, pos // P], pos % P
            touched[pg, sl] = True
            np.testing.assert_array_equal(kp2[:, pg, :, sl], kb[:, b, t])
            np.testing.assert_array_equal(vp2[:, pg, :, sl], vb[:, b, t])
    for pg in range(num):
        for sl in range(P):
            if not touched[pg, sl]:
                np.testing.assert_array_equal(kp2[:, pg, :, sl], kp[:, pg, :, sl])
                np.testing.assert_array_equal(vp2[:, pg, :, sl], vp[:, pg, :, sl])
    assert touched.sum() == s.sum()


def test_commit_hand_case_across_a_page_boundary():
    # Page size 4.  Sequence 0 holds 3 tokens (pages 5, 2, 7 in that order)
    # and keeps 3 block rows: positions 3, 4, 5 -> page 5 slot 3, page 2
    # slots 0 and 1.  Sequence 1 holds 4 tokens (pages 0, 3, 1) and keeps 2:
    # positions 4, 5 -> page 3 slots 0 and 1.  Row t of sequence b carries
    # the value 10*b + t + 1 (K) and its negation (V); the pool starts at 0.
    L, B, R, Hkv, D, P, num = 1, 2, 4, 1, 1, 4, 8
    table = np.array([[5, 2, 7], [0, 3, 1]])
    ctx = np.array([3, 4])
    s = np.array([3, 2])
    kb = np.zeros((L, B, R, Hkv, D), dtype=np.int16)
    for b in range(B):
        for t in range(R):
            kb[0, b, t, 0, 0] = 10 * b + t + 1
    vb = -kb
    kp = np.zeros((L, num, Hkv, P, D), dtype=np.int16)
    kp2, vp2, ctx2 = O.commit_kv(kb, vb, kp, kp.copy(), table, ctx, s, P)
    expect = np.zeros((num, P), dtype=np.int16)
    expect[5, 3], expect[2, 0], expect[2, 1] = 1, 2, 3       # sequence 0, rows 0..2
    expect[3, 0], expect[3, 1] = 11, 12                      # sequence 1, rows 0..1
    np.testing.assert_array_equal(kp2[0, :, 0, :, 0], expect)
    np.testing.assert_array_equal(vp2[0, :, 0, :, 0], -expect)
    np.testing.assert_array_equal(ctx2, [6, 6])
