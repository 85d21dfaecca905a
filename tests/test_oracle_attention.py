"""Pins of the oracle's verify attention (Sec. 3.1, Eq. 2) to closed forms,
brute force and layout invariants -- no CUDA involved."""
import math

import numpy as np
import pytest

from oracle import cospec_oracle as O

pytestmark = pytest.mark.filterwarnings("ignore")


def _contiguous_pages(ctx_list, R, Hkv, P, D, rng):
    """Random contiguous caches and an identity page table."""
    B = len(ctx_list)
    need = [(c + R + P - 1) // P for c in ctx_list]
    num = sum(need)
    kp = rng.standard_normal((num, Hkv, P, D))
    vp = rng.standard_normal((num, Hkv, P, D))
    table = np.full((B, max(need)), -1, dtype=np.int64)
    s = 0
    for b in range(B):
        table[b, :need[b]] = np.arange(s, s + need[b])
        s += need[b]
    return kp, vp, table


def test_two_keys_three_to_one():
    # one context key and the row's own block key; q.k * D^-1/2 = ln 3 and 0
    D = 4
    q = np.zeros((1, 1, 1, D)); q[0, 0, 0, 0] = 2 * math.log(3.0)      # scale 1/2
    kp = np.zeros((1, 1, 4, D)); kp[0, 0, 0, 0] = 1.0
    vp = np.zeros((1, 1, 4, D)); vp[0, 0, 0] = [4, 0, 8, 0]
    kb = np.zeros((1, 1, 1, D)); kb[0, 0, 0, 1] = 1.0
    vb = np.zeros((1, 1, 1, D)); vb[0, 0, 0] = [0, 4, 0, 8]
    o = O.verify_attention(q, kb, vb, kp, vp, np.array([[0]]), np.array([1]), page_size=4)
    np.testing.assert_allclose(o[0, 0, 0], [3.0, 1.0, 6.0, 2.0], rtol=0, atol=1e-12)


def test_gqa_head_mapping_uses_floor_division():
    rng = np.random.default_rng(1)
    B, R, Hq, Hkv, D, P, C = 1, 3, 4, 2, 8, 4, 5
    kp, vp, table = _contiguous_pages([C], R, Hkv, P, D, rng)
    kb = rng.standard_normal((B, R, Hkv, D))
    vb = np.zeros((B, R, Hkv, D))
    for kvh in range(Hkv):
        vp[:, kvh] = kvh + 1.0
        vb[:, :, kvh] = kvh + 1.0
    q = rng.standard_normal((B, R, Hq, D))
    o = O.verify_attention(q, kb, vb, kp, vp, table, np.array([C]), P)
    for h in range(Hq):
        np.testing.assert_allclose(o[0, :, h], h // (Hq // Hkv) + 1.0, atol=1e-12)


def test_constant_values_give_that_value():
    rng = np.random.default_rng(2)
    B, R, Hq, Hkv, D, P = 2, 4, 4, 1, 8, 4
    ctx = [7, 0]
    kp, vp, table = _contiguous_pages(ctx, R, Hkv, P, D, rng)
    vp[:] = 0.375
    vb = np.full((B, R, Hkv, D), 0.375)
    o = O.verify_attention(rng.standard_normal((B, R, Hq, D)), rng.standard_normal((B, R, Hkv, D)),
                           vb, kp, vp, table, np.array(ctx), P)
    np.testing.assert_allclose(o, 0.375, atol=1e-12)


def test_causal_inside_block():
    rng = np.random.default_rng(3)
    B, R, Hq, Hkv, D, P = 1, 4, 2, 1, 8, 4
    kp, vp, table = _contiguous_pages([0], R, Hkv, P, D, rng)
    q = rng.standard_normal((B, R, Hq, D))
    kb = rng.standard_normal((B, R, Hkv, D))
    vb = rng.standard_normal((B, R, Hkv, D))
    o = O.verify_attention(q, kb, vb, kp, vp, table, np.array([0]), P)
    # row 0 of an empty context sees only its own key: o = v_blk[0]
    np.testing.assert_allclose(o[0, 0, 0], vb[0, 0, 0], atol=1e-12)
    kb2, vb2 = kb.copy(), vb.copy()
    kb2[0, 2:] = rng.standard_normal(kb2[0, 2:].shape)
    vb2[0, 2:] = rng.standard_normal(vb2[0, 2:].shape)
    o2 = O.verify_attention(q, kb2, vb2, kp, vp, table, np.array([0]), P)
    np.testing.assert_array_equal(o2[0, :2], o[0, :2])      # rows 0,1 never read rows >= 2
    assert np.abs(o2[0, 2:] - o[0, 2:]).max() > 1e-3


def test_paged_equals_contiguous_bitwise():
    rng = np.random.default_rng(4)
    B, R, Hq, Hkv, D, P = 3, 5, 8, 2, 16, 4
    ctx = [9, 0, 13]
    kp, vp, table = _contiguous_pages(ctx, R, Hkv, P, D, rng)
    q = rng.standard_normal((B, R, Hq, D))
    kb = rng.standard_normal((B, R, Hkv, D))
    vb = rng.standard_normal((B, R, Hkv, D))
    ref = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P)
    perm = rng.permutation(kp.shape[0])                  # physical page of logical page p
    kp2 = np.empty_like(kp); vp2 = np.empty_like(vp)
    kp2[perm] = kp; vp2[perm] = vp
    table2 = np.where(table >= 0, perm[np.clip(table, 0, None)], -1)
    got = O.verify_attention(q, kb, vb, kp2, vp2, table2, np.array(ctx), P)
    np.testing.assert_array_equal(got, ref)


def _brute(q, kb, vb, kp, vp, table, ctx, P):
    B, R, Hq, D = q.shape
    Hkv = kb.shape[2]
    G = Hq // Hkv
    out = np.zeros_like(q)
    for b in range(B):
        for h in range(Hq):
            g = h // G
            for j in range(R):
                keys, vals = [], []
                for t in range(ctx[b]):
                    pg = table[b][t // P]
                    keys.append(kp[pg, g, t % P]); vals.append(vp[pg, g, t % P])
                for t in range(j + 1):
                    keys.append(kb[b, t, g]); vals.append(vb[b, t, g])
                sc = [sum(q[b, j, h, e] * k[e] for e in range(D)) / math.sqrt(D) for k in keys]
                m = max(sc)
                wts = [math.exp(s - m) for s in sc]
                tot = sum(wts)
                for e in range(D):
                    out[b, j, h, e] = sum(w * v[e] for w, v in zip(wts, vals)) / tot
    return out


def test_brute_force_tiny_random():
    rng = np.random.default_rng(5)
    B, R, Hq, Hkv, D, P = 2, 3, 4, 2, 4, 4
    ctx = [6, 0]
    kp, vp, table = _contiguous_pages(ctx, R, Hkv, P, D, rng)
    q = rng.standard_normal((B, R, Hq, D)) * 2       # N(0,1)-scale scores, far from uniform
    kb = rng.standard_normal((B, R, Hkv, D))
    vb = rng.standard_normal((B, R, Hkv, D))
    got = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P)
    ref = _brute(q, kb, vb, kp, vp, table, ctx, P)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_selected_rows_only():
    rng = np.random.default_rng(6)
    B, R, Hq, Hkv, D, P = 3, 2, 4, 2, 8, 4
    ctx = [3, 5, 2]
    kp, vp, table = _contiguous_pages(ctx, R, Hkv, P, D, rng)
    q = rng.standard_normal((B, R, Hq, D))
    kb = rng.standard_normal((B, R, Hkv, D)); vb = rng.standard_normal((B, R, Hkv, D))
    full = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P)
    part = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P, seqs=[1], heads=[3])
    np.testing.assert_array_equal(part[1, :, 3], full[1, :, 3])
    assert not part[0].any() and not part[2].any()
