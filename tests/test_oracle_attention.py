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


# --- the arbitrator's hybrid mask (Sec. 3.3): region rows see the context and
# --- the whole region; the context never sees the region

def test_hybrid_mask_shape_and_rules():
    m = O.hybrid_mask(3, 4)
    assert m.shape == (7, 7)
    # context rows: causal, never the region
    for i in range(3):
        assert list(m[i]) == [t <= i for t in range(7)]
    # region rows: everything
    assert m[3:].all()


def test_full_block_mask_equals_dense_hybrid_attention():
    """The region rows of the dense hybrid-masked attention equal the paged
    block attention with the full block mask: context as the cache, region as
    the block."""
    rng = np.random.default_rng(11)
    l_c, n, Hq, Hkv, D, P = 13, 7, 4, 2, 8, 4
    q = rng.standard_normal((l_c + n, Hq, D)) * 1.5
    k = rng.standard_normal((l_c + n, Hkv, D))
    v = rng.standard_normal((l_c + n, Hkv, D))
    mask = O.hybrid_mask(l_c, n)
    dense = np.stack([O.dense_masked_attention(q[:, h], k[:, h // 2], v[:, h // 2], mask)
                      for h in range(Hq)], axis=1)                      # [l, Hq, D]
    # the same tokens as one sequence: context in pages, region as the block
    npages = (l_c + n + P - 1) // P
    kp = np.zeros((npages, Hkv, P, D)); vp = np.zeros((npages, Hkv, P, D))
    for t in range(l_c):
        kp[t // P, :, t % P] = k[t]; vp[t // P, :, t % P] = v[t]
    table = np.arange(npages)[None, :]
    got = O.verify_attention(q[None, l_c:], k[None, l_c:], v[None, l_c:], kp, vp, table,
                             np.array([l_c]), P, block_mask="full")
    np.testing.assert_allclose(got[0], dense[l_c:], rtol=1e-12, atol=1e-12)
    # and the context rows of the dense pass are plain causal attention over the context
    causal = np.stack([O.dense_masked_attention(q[:l_c, h], k[:l_c, h // 2], v[:l_c, h // 2],
                                                np.tril(np.ones((l_c, l_c), dtype=bool)))
                       for h in range(Hq)], axis=1)
    np.testing.assert_allclose(dense[:l_c], causal, rtol=1e-12, atol=1e-12)


def test_full_and_causal_block_agree_on_the_last_row_only():
    rng = np.random.default_rng(12)
    B, R, Hq, Hkv, D, P = 2, 5, 4, 2, 8, 4
    ctx = [9, 0]
    kp, vp, table = _contiguous_pages(ctx, R, Hkv, P, D, rng)
    q = rng.standard_normal((B, R, Hq, D)) * 2
    kb = rng.standard_normal((B, R, Hkv, D)); vb = rng.standard_normal((B, R, Hkv, D))
    full = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P, block_mask="full")
    causal = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P)
    np.testing.assert_allclose(full[:, R - 1], causal[:, R - 1], rtol=1e-12, atol=1e-12)
    assert np.abs(full[:, 0] - causal[:, 0]).max() > 1e-3


def test_full_block_brute_force():
    rng = np.random.default_rng(13)
    B, R, Hq, Hkv, D, P = 2, 3, 4, 2, 4, 4
    ctx = [5, 2]
    kp, vp, table = _contiguous_pages(ctx, R, Hkv, P, D, rng)
    q = rng.standard_normal((B, R, Hq, D)) * 2
    kb = rng.standard_normal((B, R, Hkv, D)); vb = rng.standard_normal((B, R, Hkv, D))
    got = O.verify_attention(q, kb, vb, kp, vp, table, np.array(ctx), P, block_mask="full")
    G = Hq // Hkv
    for b in range(B):
        for j in range(R):
            for h in range(Hq):
                keys, vals = [], []
                for t in range(ctx[b]):
                    keys.append(kp[table[b][t // P], h // G, t % P]); vals.append(vp[table[b][t // P], h // G, t % P])
                for jj in range(R):                     # every block row, before or after j
                    keys.append(kb[b, jj, h // G]); vals.append(vb[b, jj, h // G])
                sc = [sum(qe * ke for qe, ke in zip(q[b, j, h], kk)) / math.sqrt(D) for kk in keys]
                mx = max(sc)
                w = [math.exp(x - mx) for x in sc]
                ref = [sum(wi * vv[e] for wi, vv in zip(w, vals)) / sum(w) for e in range(D)]
                np.testing.assert_allclose(got[b, j, h], ref, rtol=1e-12, atol=1e-12)
