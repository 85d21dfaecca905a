"""Parity of the CUDA path (through the C ABI) with the CPU oracle on seeded
inputs small enough for the oracle, spanning several tiles, ragged tails and
the degenerate cases (empty context, K = 0, single / many KV splits)."""
import math

import numpy as np
import pytest
import torch

from oracle import cospec_oracle as O
from paper_2605_24793_gb300 import build as BLD
from paper_2605_24793_gb300 import cospec as C
from paper_2605_24793_gb300 import workload as W
from paper_2605_24793_gb300.round import VerifyRound

from .parity_util import assert_close, report_ties, tie_positions

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    C.load_library(BLD.build())
    torch.cuda.set_device(0)
    assert C.get_device_error() == 0
    yield
    assert C.get_device_error() == 0


def bf16(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).cuda()


def host(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def _paged_case(rng, B, R, Hq, Hkv, D, ctx, shuffled, std=1.0, spare_pages=0):
    P = 16
    need = [(c + R + P - 1) // P for c in ctx]
    num = sum(need) + spare_pages
    order = rng.permutation(num) if shuffled else np.arange(num)
    table = np.full((B, max(need)), -1, dtype=np.int32)
    s = 0
    for b in range(B):
        table[b, :need[b]] = order[s:s + need[b]]
        s += need[b]
    mk = lambda *shape: rng.standard_normal(shape).astype(np.float32) * std
    return dict(q=bf16(mk(B, R, Hq, D)), k_blk=bf16(mk(B, R, Hkv, D)), v_blk=bf16(mk(B, R, Hkv, D)),
                k_pages=bf16(mk(num, Hkv, P, D)), v_pages=bf16(mk(num, Hkv, P, D)),
                page_table=torch.from_numpy(table).cuda(),
                ctx_len=torch.tensor(ctx, dtype=torch.int32).cuda(), table_np=table,
                ctx_np=np.array(ctx))


ATTN_CASES = [
    # B, R, Hq, Hkv, D, contexts, shuffled pages
    (1, 6, 32, 8, 128, [4096], False),              # Qwen3-8B-like, many KV splits
    (4, 8, 64, 8, 128, [0, 17, 1000, 3333], True),  # G*R = 64 rows, empty and ragged contexts
    (1, 5, 8, 2, 64, [256], False),                 # head_dim 64
    (3, 3, 4, 4, 128, [5, 64, 65], True),           # G = 1, R = 3 -> 3 rows (one 16-row tile)
    (2, 16, 64, 8, 128, [100, 2000], True),         # G*R = 128 rows: one full row group
    (2, 8, 128, 8, 64, [31, 700], False),           # G = 16 -> 128 rows at head_dim 64
    (2, 1, 32, 8, 128, [0, 1], False),              # K = 0: one row per sequence
    (5, 4, 32, 8, 128, [8191, 40, 63, 64, 2049], True),
    (1, 26, 32, 8, 128, [4096], False),             # K = 25 (the paper's default): 104 rows, one group
    (2, 32, 128, 8, 64, [300, 1500], True),         # 512 rows per KV head: 4 row groups of 128
    (2, 2, 128, 1, 128, [500, 1200], True),         # G = 128 (one KV head): 256 rows, mma.sync
]


def expected_kernel(R, Hq, Hkv, D):
    """More than 32 query rows per KV head (G <= 64, head_dim 64 or 128):
    the tcgen05 kernel (row groups of up to 128 rows); otherwise the
    mma.sync kernel."""
    G = Hq // Hkv
    if G > 64 or D not in (64, 128):
        return C.ATTN_MMA_SYNC
    jb = 128 // G
    return C.ATTN_TCGEN05 if G * min(R, jb) > 32 else C.ATTN_MMA_SYNC

# Batches with a (sequence, KV head, row group) per SM and more than 32 query
# rows per group select the tcgen05 kernel.
_ctx = lambda n, seed: list(np.random.default_rng(seed).integers(0, 700, n))
# Batches above 64 sequences are taken in index order, not longest first.
ATTN_CASES += [
    (80, 6, 32, 8, 128, _ctx(80, 12), True),        # 24 rows: mma.sync kernel
    (70, 16, 32, 8, 128, _ctx(70, 13), True),       # 64 rows: tcgen05 kernel
    (64, 4, 32, 8, 128, _ctx(64, 15), True),        # 64 sequences: the largest batch ranked
    (65, 4, 32, 8, 128, _ctx(65, 16), True),        # 65: the smallest taken in index order
]
ATTN_TC_CASES = [
    (24, 8, 64, 8, 128, [0, 1, 63, 64, 65, 127, 128, 129] + _ctx(16, 1), True),  # G = 8: 64 rows
    (20, 4, 128, 8, 64, _ctx(20, 2), True),         # head_dim 64, G = 16: 64 rows
    (10, 8, 128, 8, 128, _ctx(10, 3), True),        # 128 rows: one full row group
    (20, 8, 40, 8, 128, _ctx(20, 4), False),        # G = 5: 40 rows
    (20, 16, 32, 8, 128, [2000] + _ctx(19, 5), True),  # G = 4, 16 block rows: 64 rows, longer context
    (3, 64, 8, 8, 128, [0, 100, 1500], True),        # R = 64, the largest block: 64 rows
    (2, 64, 16, 8, 64, [50, 700], True),             # R = 64, G = 2: 128 rows, head_dim 64
    (16, 26, 32, 8, 128, _ctx(16, 11), True),        # K = 25 at batch 16: 104 rows, one group
    (2, 32, 32, 8, 128, [600, 129], True),           # K = 31: exactly 128 rows
    (2, 33, 32, 8, 128, [300, 50], True),            # 132 rows: groups of 32 and 1 block rows
    (1, 16, 32, 8, 64, [2000], False),               # head_dim 64 at batch 1: a split of 8
    (2, 3, 64, 1, 128, [400, 1000], True),           # G = 64, the largest: row groups of 2 and 1 block rows
    (3, 11, 24, 8, 128, [129, 700, 0], True),        # G = 3: 33 rows, one past the mma.sync kernel
    (64, 8, 64, 8, 128, _ctx(64, 14), True),         # 64 sequences, ranked longest first
]


@pytest.mark.parametrize("case", ATTN_CASES, ids=lambda c: f"B{c[0]}R{c[1]}G{c[2]//c[3]}D{c[4]}")
def test_verify_attention_matches_oracle(case):
    B, R, Hq, Hkv, D, ctx, shuffled = case
    rng = np.random.default_rng(B * 1000 + R * 100 + Hq + D + sum(ctx))
    t = _paged_case(rng, B, R, Hq, Hkv, D, ctx, shuffled)
    max_ctx = max(ctx)
    assert C.verify_attn_plan(t["q"], t["k_pages"], t["page_table"], max_ctx)[0] == \
        expected_kernel(R, Hq, Hkv, D)
    out = torch.empty_like(t["q"])
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out, max_ctx)
    ref = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                             host(t["v_pages"]), t["table_np"], t["ctx_np"], 16)
    assert_close(host(out), ref, "attention")
    # a second call gives the same bits
    out2 = torch.empty_like(out)
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out2, max_ctx)
    assert torch.equal(out, out2)


@pytest.mark.parametrize("case", ATTN_TC_CASES, ids=lambda c: f"B{c[0]}R{c[1]}G{c[2] // c[3]}D{c[4]}")
def test_verify_attention_tcgen05_matches_oracle(case):
    B, R, Hq, Hkv, D, ctx, shuffled = case
    rng = np.random.default_rng(B * 1000 + R * 100 + Hq + D + int(sum(ctx)))
    t = _paged_case(rng, B, R, Hq, Hkv, D, ctx, shuffled)
    max_ctx = int(max(ctx))
    assert C.verify_attn_plan(t["q"], t["k_pages"], t["page_table"], max_ctx)[0] == C.ATTN_TCGEN05
    out = torch.empty_like(t["q"])
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out, max_ctx)
    ref = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                             host(t["v_pages"]), t["table_np"], t["ctx_np"], 16)
    assert_close(host(out), ref, "attention (tcgen05)")
    out2 = torch.empty_like(out)
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out2, max_ctx)
    assert torch.equal(out, out2)


# The tcgen05 kernel splits a (sequence, head, row group)'s KV range over a
# cluster when the batch has fewer units than SMs, and when a context passes
# 256 tiles of 128 keys: 2, 4 and 8 splits merged through distributed shared
# memory, with most sequences far shorter than the split.
ATTN_TC_SPLIT_CASES = [
    # B, R, Hq, Hkv, D, contexts, shuffled, expected splits
    (12, 8, 64, 8, 128, [6000] + _ctx(11, 8), True, 2),           # 96 units
    (6, 8, 64, 8, 128, [9000, 3000] + _ctx(4, 9), True, 4),       # 48 units
    (1, 8, 64, 8, 128, [6000], False, 12),                        # one wave of 12-CTA clusters
    (20, 8, 64, 8, 128, [33000, 9000] + _ctx(18, 10), False, 2),  # a context past 256 tiles
]


@pytest.mark.parametrize("case", ATTN_TC_SPLIT_CASES, ids=lambda c: f"B{c[0]}R{c[1]}S{c[7]}")
def test_verify_attention_tcgen05_split_matches_oracle(case):
    B, R, Hq, Hkv, D, ctx, shuffled, splits = case
    rng = np.random.default_rng(B * 1000 + R * 100 + Hq + D + int(sum(ctx)))
    t = _paged_case(rng, B, R, Hq, Hkv, D, ctx, shuffled)
    max_ctx = int(max(ctx))
    assert C.verify_attn_plan(t["q"], t["k_pages"], t["page_table"], max_ctx) == (C.ATTN_TCGEN05, splits)
    out = torch.empty_like(t["q"])
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out, max_ctx)
    ref = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                             host(t["v_pages"]), t["table_np"], t["ctx_np"], 16)
    assert_close(host(out), ref, "attention (tcgen05, split)")


# The arbitrator's draft/target region (Sec. 3.3): 2K+3 block rows that see
# the whole block; K = 7 gives 17 rows, K = 25 (the paper's default) 53.
ATTN_FULL_CASES = [
    # B, R, Hq, Hkv, D, contexts, shuffled, expected kernel
    (1, 17, 32, 8, 128, [4096], False, 1),          # K = 7 region on a Qwen3-4B-like arbitrator
    (3, 53, 32, 8, 128, [0, 300, 2500], True, 1),   # K = 25 region: 212 rows in groups of 128 and 84
    (2, 4, 128, 1, 128, [700, 90], True, 0),        # G = 128: 512 rows in 64-row groups, mma.sync
    (2, 9, 16, 8, 64, [100, 33], True, 0),          # head_dim 64, K = 3 region
    (20, 53, 8, 8, 128, _ctx(20, 6), True, 1),      # G = 1, 53 rows per group: tcgen05 kernel
    (24, 17, 32, 8, 128, _ctx(24, 7), True, 1),     # G = 4, 68 rows in one group: tcgen05 kernel
    (2, 64, 8, 8, 128, [300, 0], True, 1),          # a 64-row region, the largest block
]


@pytest.mark.parametrize("case", ATTN_FULL_CASES, ids=lambda c: f"B{c[0]}R{c[1]}G{c[2] // c[3]}D{c[4]}")
def test_verify_attention_full_block_matches_oracle(case):
    B, R, Hq, Hkv, D, ctx, shuffled, kernel = case
    rng = np.random.default_rng(B * 1000 + R * 100 + Hq + D + int(sum(ctx)) + 77)
    t = _paged_case(rng, B, R, Hq, Hkv, D, ctx, shuffled)
    max_ctx = int(max(ctx))
    assert C.verify_attn_plan(t["q"], t["k_pages"], t["page_table"], max_ctx)[0] == kernel
    out = torch.empty_like(t["q"])
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out, max_ctx, block_full=True)
    ref = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                             host(t["v_pages"]), t["table_np"], t["ctx_np"], 16, block_mask="full")
    assert_close(host(out), ref, "attention (full block)")
    # the causal call on the same inputs still matches the causal oracle
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out, max_ctx)
    ref_c = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                               host(t["v_pages"]), t["table_np"], t["ctx_np"], 16)
    assert_close(host(out), ref_c, "attention (causal, long block)")


def test_verify_attention_split_count_does_not_change_result_beyond_tolerance():
    rng = np.random.default_rng(3)
    t = _paged_case(rng, 2, 6, 32, 8, 128, [3000, 5000], True)
    ref = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                             host(t["v_pages"]), t["table_np"], t["ctx_np"], 16)
    for max_ctx in (5000, t["table_np"].shape[1] * 16):     # different split plans
        out = torch.empty_like(t["q"])
        C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                      t["ctx_len"], out, max_ctx)
        assert_close(host(out), ref, f"attention max_ctx={max_ctx}")


def test_verify_attention_constant_values():
    # closed form: constant V gives that constant whatever the scores
    rng = np.random.default_rng(4)
    t = _paged_case(rng, 2, 6, 32, 8, 128, [777, 3], True)
    t["v_pages"].fill_(0.375)
    t["v_blk"].fill_(0.375)
    out = torch.empty_like(t["q"])
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  t["ctx_len"], out, 777)
    assert torch.all(out.float() == 0.375)


def test_verify_attention_concurrent_host_threads():
    # Calls from several host threads (ctypes releases the GIL), each on its
    # own stream and with its own block size, so that first launches race to
    # set each variant's shared-memory limit: every result equals the same
    # call made alone.
    import threading
    rng = np.random.default_rng(11)
    shapes = [(2, 4, 32, 8, 128, [900, 40]), (1, 20, 32, 8, 128, [1500]),
              (2, 40, 16, 8, 128, [300, 700]), (3, 8, 64, 8, 128, [100, 2000, 5])]
    cases = [_paged_case(rng, *sh, True) for sh in shapes]
    refs = []
    for sh, t in zip(shapes, cases):
        out = torch.empty_like(t["q"])
        C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                      t["ctx_len"], out, max(sh[5]))
        refs.append(out)
    torch.cuda.synchronize()
    outs = [torch.empty_like(t["q"]) for t in cases]
    errors = []

    def worker(i):
        try:
            s = torch.cuda.Stream()
            t = cases[i]
            for _ in range(20):
                C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                              t["ctx_len"], outs[i], max(shapes[i][5]), stream=s)
            s.synchronize()
        except Exception as e:  # noqa: BLE001 - reported below
            errors.append(e)

    threads = [threading.Thread(target=worker, args=(i,)) for i in range(len(cases))]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    assert not errors, errors
    for ref, out in zip(refs, outs):
        assert torch.equal(ref, out)


LM_CASES = [
    # M, d, V, weight std
    (1, 64, 128, 0.1),
    (5, 512, 4096, 0.02),
    (6, 4096, 151936, 0.02),      # Qwen3-8B LM head, batch 1, K = 5
    (17, 256, 1000, 0.1),         # vocabulary not a multiple of the 128-row tile
    (128, 1024, 3000, 0.05),
    (300, 128, 2048, 0.1),        # two passes of 160 and 140 rows
    (256, 5120, 1280, 0.02),
    (384, 256, 3000, 0.05),       # two equal passes of 192 rows (the Llama K = 5 round)
    (512, 256, 2000, 0.05),       # two full 256-row passes
    (520, 128, 1500, 0.1),        # three passes of 176, 176 and 168 rows
]


@pytest.mark.parametrize("case", LM_CASES, ids=lambda c: f"M{c[0]}d{c[1]}V{c[2]}")
def test_lmhead_matches_oracle(case):
    M, d, V, wstd = case
    rng = np.random.default_rng(M * 7 + d + V)
    hidden = bf16(rng.standard_normal((M, d)))
    w = bf16(rng.standard_normal((V, d)) * wstd)
    dfr = rng.integers(0, V, M).astype(np.int32)
    dfr[::3] = -1
    dfr_t = torch.from_numpy(dfr).cuda()
    am = torch.empty(M, dtype=torch.int32, device="cuda")
    st = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    ws = C.new_lmhead_workspace(M, d, V)
    C.lmhead_argmax_features(hidden, w, dfr_t, am, st, ws)
    ref_am, ref_st = O.lmhead_stats(host(hidden), host(w), dfr)
    assert_close(st.cpu().numpy(), ref_st, "lm-head stats")
    margin = ref_st[:, 0] - ref_st[:, 1]
    clear = margin >= 1e-3
    assert np.array_equal(am.cpu().numpy()[clear], ref_am[clear])
    print(f"lm-head {case}: tie rows {(~clear).sum()}")


def test_lmhead_exact_ties_pick_lowest_id():
    rng = np.random.default_rng(11)
    M, d, V = 8, 256, 700
    hidden = rng.standard_normal((M, d))
    w = rng.standard_normal((V, d)) * 0.01
    w[[3, 130, 699]] = hidden[0] * 0.5          # three identical top rows for row 0
    w[[257, 258]] = hidden[1] * 0.5             # two identical top rows for row 1
    hidden_t, w_t = bf16(hidden), bf16(w)
    am = torch.empty(M, dtype=torch.int32, device="cuda")
    st = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    C.lmhead_argmax_features(hidden_t, w_t, torch.full((M,), -1, dtype=torch.int32, device="cuda"),
                             am, st, C.new_lmhead_workspace(M, d, V))
    am = am.cpu().numpy()
    st = st.cpu().numpy()
    assert am[0] == 3 and am[1] == 257
    assert st[0, 0] == st[0, 1] and st[1, 0] == st[1, 1]      # second == max on a tie
    assert np.all(np.isnan(st[:, 4]))


def _stats_case(rng, B, K, V=64):
    x = rng.standard_normal((B * (K + 1), V)) * 2.0
    top1 = np.argmax(x, axis=1).reshape(B, K + 1)
    draft = np.where(rng.random((B, K)) < 0.5, top1[:, :K], rng.integers(0, V, (B, K))).astype(np.int32)
    dfr = np.full((B, K + 1), -1)
    dfr[:, :K] = draft
    am, st = O.row_stats(x, dfr.reshape(-1))
    return draft, am.reshape(B, K + 1).astype(np.int32), st.reshape(B, K + 1, 5)


@pytest.mark.parametrize("K", [1, 3, 7, 31])
@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("lam", [0.4, 0.6, 0.8])
def test_arbitrate_matches_oracle(K, mode, lam):
    rng = np.random.default_rng(K * 100 + mode * 10 + int(lam * 10))
    B, H = 37, 256
    draft, am, st = _stats_case(rng, B, K)
    w1 = (rng.random((H, 8)) * 2 - 1) / math.sqrt(8)
    b1 = (rng.random(H) * 2 - 1) / math.sqrt(8)
    w2 = (rng.random(H) * 2 - 1) / math.sqrt(H)
    b2 = 0.05
    ref_p, ref_a = O.arbitrate(draft, am, st, w1, b1, w2, b2, lam, mode)
    p = torch.empty((B, K), dtype=torch.float32, device="cuda")
    a = torch.empty((B, K), dtype=torch.uint8, device="cuda")
    f32 = lambda v: torch.tensor(np.asarray(v, dtype=np.float32)).cuda()
    C.arbitrate(torch.from_numpy(draft).cuda(), torch.from_numpy(am).cuda(),
                f32(st), f32(w1), f32(b1), f32(w2), b2, lam, mode, p, a)
    p = p.cpu().numpy()
    a = a.cpu().numpy()
    assert_close(p, ref_p, "policy probability")
    clear = np.abs(ref_p - lam) >= 1e-3
    assert np.array_equal(a[clear], ref_a[clear])
    assert np.all(a[draft == am[:, :K]] == 1)


def test_features_feed_the_mlp_as_the_oracle_builds_them():
    # a one-hot first layer exposes each feature in turn through z
    rng = np.random.default_rng(21)
    B, K = 9, 7
    draft, am, st = _stats_case(rng, B, K)
    feats = O.arbitration_features(draft, am, st)
    mism = draft != am[:, :K]
    for k in range(8):
        w1 = np.zeros((2, 8)); w1[0, k] = 1.0; w1[1, k] = -1.0
        b1 = np.zeros(2); w2 = np.array([1.0, -1.0])           # z = relu(f) - relu(-f) = f_k
        p = torch.empty((B, K), dtype=torch.float32, device="cuda")
        a = torch.empty((B, K), dtype=torch.uint8, device="cuda")
        f32 = lambda v: torch.tensor(np.asarray(v, dtype=np.float32)).cuda()
        C.arbitrate(torch.from_numpy(draft).cuda(), torch.from_numpy(am).cuda(), f32(st), f32(w1),
                    f32(b1), f32(w2), 0.0, 0.5, 0, p, a)
        z = -np.log(1.0 / np.clip(p.cpu().numpy().astype(np.float64), 1e-30, 1 - 1e-7) - 1.0)
        assert_close(z[mism], feats[..., k][mism], f"feature F{k}", abs_tol=1e-3, rel_tol=1e-3)


@pytest.mark.parametrize("K,L,B", [(0, 3, 6), (1, 3, 6), (5, 3, 6), (7, 3, 6), (7, 64, 32)])
def test_accept_commit_matches_oracle(K, L, B):
    # (7, 64, 32): the commit grid of the Qwen3-32B-shaped round (64 layers x
    # 32 sequences, one CTA each), with short contexts
    rng = np.random.default_rng(40 + K + L)
    R, Hkv, D, P = K + 1, 8, 128, 16
    ctx = rng.integers(0, 200, B).astype(np.int32)
    need = (ctx + R + P - 1) // P
    num = int(need.sum())
    perm = rng.permutation(num)
    table = np.full((B, need.max()), -1, dtype=np.int32)
    s0 = 0
    for b in range(B):
        table[b, :need[b]] = perm[s0:s0 + need[b]]
        s0 += need[b]
    V = 50
    am = rng.integers(0, V, (B, R)).astype(np.int32)
    draft = np.where(rng.random((B, K)) < 0.6, am[:, :K], rng.integers(0, V, (B, K))).astype(np.int32)
    acc = (rng.random((B, K)) < 0.5).astype(np.uint8)
    acc[draft == am[:, :K]] = 1
    kb = bf16(rng.standard_normal((L, B, R, Hkv, D)))
    vb = bf16(rng.standard_normal((L, B, R, Hkv, D)))
    kp = bf16(rng.standard_normal((L, num, Hkv, P, D)))
    vp = bf16(rng.standard_normal((L, num, Hkv, P, D)))
    bits = lambda t: t.cpu().view(torch.int16).numpy()
    kp0, vp0 = bits(kp), bits(vp)
    ctx_t = torch.from_numpy(ctx).cuda()
    alen = torch.empty(B, dtype=torch.int32, device="cuda")
    em = torch.empty((B, R), dtype=torch.int32, device="cuda")
    C.accept_commit(torch.from_numpy(draft.reshape(B, K)).cuda(), torch.from_numpy(am).cuda(),
                    torch.from_numpy(acc.reshape(B, K)).cuda(), kb, vb, kp, vp,
                    torch.from_numpy(table).cuda(), ctx_t, alen, em)
    s, emitted = O.accept_scan(draft.reshape(B, K), am, acc.reshape(B, K))
    kp_ref, vp_ref, ctx_ref = O.commit_kv(bits(kb), bits(vb), kp0, vp0, table, ctx, s, P)
    assert np.array_equal(alen.cpu().numpy(), s)
    assert np.array_equal(em.cpu().numpy(), emitted)
    assert np.array_equal(ctx_t.cpu().numpy(), ctx_ref)
    assert np.array_equal(bits(kp), kp_ref) and np.array_equal(bits(vp), vp_ref)


def _tiny_round(mode, lam, cfg_name="tiny", **over):
    cfg = W.CONFIGS[cfg_name].replace(**over) if over else W.CONFIGS[cfg_name]
    inp = W.make_round_inputs(cfg, device="cuda")
    hostinp = {k: (v.cpu() if torch.is_tensor(v) else v) for k, v in inp.items()}
    x = O.lmhead_logits(hostinp["hidden"], hostinp["w"])
    draft = W.synth_drafts(cfg, O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8))
    ref = O.cospec_round(hostinp, draft, lam, mode)
    rnd = VerifyRound(inp, draft, lam, mode, keep_attn=True)
    rnd.run(restore=False)
    torch.cuda.synchronize()
    return cfg, draft, ref, rnd


def _check_round(cfg, draft, ref, rnd, lam):
    for l in range(cfg.layers):
        assert_close(host(rnd.attn_out[l]), ref["attn"][l], f"attention layer {l}")
    B, R, K = cfg.batch, cfg.rows, cfg.k
    st = rnd.stats.cpu().numpy().reshape(B, R, 5)
    assert_close(st, ref["stats"], "lm-head stats")
    s_gpu = rnd.accept_len.cpu().numpy()
    ties = tie_positions(ref["stats"], draft, ref["argmax"], ref["p"], ref["s"], s_gpu, lam)
    report_ties("round parity", f"{cfg.name} K={K} lambda={lam}", ties)
    tie = ties > 0
    ok = ~tie
    am = rnd.argmax.cpu().numpy().reshape(B, R)
    assert np.array_equal(am[ok], ref["argmax"][ok])
    if K > 0:
        assert_close(rnd.p.cpu().numpy()[ok], ref["p"][ok], "policy probability")
        assert np.array_equal(rnd.accept.cpu().numpy()[ok], ref["a"][ok])
    assert np.array_equal(s_gpu[ok], ref["s"][ok])
    assert np.array_equal(rnd.emitted.cpu().numpy()[ok], ref["emitted"][ok])
    assert np.array_equal(rnd.ctx_len.cpu().numpy()[ok], ref["ctx_len"][ok])
    kp = rnd.k_pages.cpu().view(torch.int16).numpy()
    vp = rnd.v_pages.cpu().view(torch.int16).numpy()
    table = rnd.inp["page_table_np"]
    for b in np.nonzero(ok)[0]:
        pages = table[b][table[b] >= 0]
        assert np.array_equal(kp[:, pages], ref["k_pages"][:, pages])
        assert np.array_equal(vp[:, pages], ref["v_pages"][:, pages])
    return int(tie.sum())


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_tiny_round_matches_oracle(mode):
    cfg, draft, ref, rnd = _tiny_round(mode, 0.6)
    assert _check_round(cfg, draft, ref, rnd, 0.6) == 0
    if mode == 1:
        assert np.array_equal(ref["s"], O.strict_spd_length(draft, ref["argmax"]))
    if mode == 2:
        assert np.all(ref["s"] == cfg.k + 1)


def test_small_batched_round_with_n01_inputs():
    # several sequences, three layers, shuffled pages, N(0,1) attention inputs
    cfg, draft, ref, rnd = _tiny_round(0, 0.6, batch=6, ctx_lo=0, ctx_hi=700, layers=3,
                                       qkv_std=1.0, shuffled_pages=True, k=7, mismatch_rate=0.5)
    ties = _check_round(cfg, draft, ref, rnd, 0.6)
    print(f"tie-affected sequences: {ties} of {cfg.batch}")


def test_packed_step_buffers_give_the_same_round():
    # The packed host-facing buffers rebind the inputs and results as views;
    # a replayed graph over them must reproduce the unpacked round bit for bit.
    cfg = W.CONFIGS["tiny"].replace(batch=5, ctx_lo=0, ctx_hi=900, layers=2, k=7,
                                    shuffled_pages=True, mismatch_rate=0.5)
    inp_ref = W.make_round_inputs(cfg, device="cuda")
    x = O.lmhead_logits(inp_ref["hidden"].cpu(), inp_ref["w"].cpu())
    draft = W.synth_drafts(cfg, O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8))
    plain = VerifyRound(inp_ref, draft, 0.6, 0, keep_attn=True)
    plain.replay()
    packed = VerifyRound(W.make_round_inputs(cfg, device="cuda"), draft, 0.6, 0, keep_attn=True)
    packed.pack_step_io()
    assert packed.q.data_ptr() == packed.io_in.data_ptr()
    for name in ("q", "k_blk", "v_blk", "hidden", "draft", "draft_for_row"):
        t = getattr(packed, name)
        assert t.data_ptr() % 256 == 0 and torch.equal(t.cpu(), getattr(plain, name).cpu())
    packed.replay()
    packed.replay()         # the graph restores the context: a second replay is the same round
    torch.cuda.synchronize()
    assert packed.accept_len.data_ptr() == packed.io_out.data_ptr()
    for name in ("accept_len", "emitted", "argmax", "stats", "p", "accept", "ctx_len",
                 "attn_out", "k_pages", "v_pages"):
        a, b = getattr(plain, name).cpu(), getattr(packed, name).cpu()
        assert torch.equal(a.view(torch.uint8) if a.is_floating_point() else a,
                           b.view(torch.uint8) if b.is_floating_point() else b), name
    B, R = cfg.batch, cfg.rows
    lead = (B + 63) // 64 * 64
    out = packed.io_out.cpu()
    assert torch.equal(out[:B], plain.accept_len.cpu())
    assert torch.equal(out[lead:].view(B, R), plain.emitted.cpu())


def test_block_size_one_round_is_greedy():
    cfg, draft, ref, rnd = _tiny_round(0, 0.6, k=0, batch=3, ctx_lo=10, ctx_hi=300)
    assert np.all(rnd.accept_len.cpu().numpy() == 1)
    em = rnd.emitted.cpu().numpy()
    x = O.lmhead_logits(rnd.hidden.cpu(), rnd.w.cpu())
    assert np.array_equal(em[:, 0], np.argmax(x, axis=1))
    _check_round(cfg, draft, ref, rnd, 0.6)


def test_device_checks_set_error_bits_without_faulting():
    rng = np.random.default_rng(5)
    t = _paged_case(rng, 2, 6, 32, 8, 128, [100, 200], False)
    out = torch.empty_like(t["q"])
    bad = t["page_table"].clone()
    bad[1, 3] = 10 ** 6                                    # page id outside the pool
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], bad, t["ctx_len"],
                  out, 200)
    assert C.get_device_error() & C.DEVERR_PAGE
    long_ctx = torch.tensor([100, t["table_np"].shape[1] * 16 + 1], dtype=torch.int32, device="cuda")
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  long_ctx, out, 200)
    assert C.get_device_error() & C.DEVERR_CTX
    M, d, V = 4, 128, 256
    C.lmhead_argmax_features(bf16(rng.standard_normal((M, d))), bf16(rng.standard_normal((V, d))),
                             torch.tensor([0, V, -1, 5], dtype=torch.int32, device="cuda"),
                             torch.empty(M, dtype=torch.int32, device="cuda"),
                             torch.empty((M, 5), dtype=torch.float32, device="cuda"),
                             C.new_lmhead_workspace(M, d, V))
    assert C.get_device_error() == C.DEVERR_TOKEN
    assert C.get_device_error() == 0                       # reading clears the word


def test_tcgen05_attention_device_checks_skip_only_the_bad_sequence():
    # 64 query rows per KV head: the tcgen05 kernel.  A page id outside the
    # pool (clamped to page 0 for the copy) and a context past the page table
    # (no tiles at all) each set their bit; the other sequence's rows still
    # match the oracle.
    rng = np.random.default_rng(6)
    t = _paged_case(rng, 2, 16, 32, 8, 128, [700, 300], True)
    assert C.verify_attn_plan(t["q"], t["k_pages"], t["page_table"], 700)[0] == C.ATTN_TCGEN05
    ref = O.verify_attention(host(t["q"]), host(t["k_blk"]), host(t["v_blk"]), host(t["k_pages"]),
                             host(t["v_pages"]), t["table_np"], t["ctx_np"], 16)
    out = torch.empty_like(t["q"])
    bad = t["page_table"].clone()
    bad[1, 5] = 10 ** 6
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], bad, t["ctx_len"],
                  out, 700)
    assert C.get_device_error() == C.DEVERR_PAGE
    assert_close(host(out)[0], ref[0], "attention (tcgen05), the sequence with valid pages")
    long_ctx = torch.tensor([700, t["table_np"].shape[1] * 16 + 1], dtype=torch.int32, device="cuda")
    out.fill_(1.0)
    C.verify_attn(t["q"], t["k_blk"], t["v_blk"], t["k_pages"], t["v_pages"], t["page_table"],
                  long_ctx, out, 700)
    assert C.get_device_error() == C.DEVERR_CTX
    assert_close(host(out)[0], ref[0], "attention (tcgen05), the sequence with a valid context")
    assert torch.all(out[1] == 0)                          # the skipped sequence attends nothing


def test_accept_commit_device_checks_skip_only_the_bad_sequence():
    # Sequence 1 would run past its page table (ctx + s > capacity): its
    # context stays, nothing of it is written.  Sequence 2's commit page is
    # outside the pool: those cells are skipped.  Sequence 0 commits exactly
    # as the oracle does.
    rng = np.random.default_rng(41)
    B, K, L, Hkv, D, P = 3, 3, 2, 8, 128, 16
    R = K + 1
    pages_per_seq = 4
    table = rng.permutation(B * pages_per_seq).astype(np.int32).reshape(B, pages_per_seq)
    ctx = np.array([37, pages_per_seq * P - 2, 21], dtype=np.int32)
    table_bad = table.copy()
    table_bad[2, ctx[2] // P] = 10 ** 6
    V = 50
    am = rng.integers(0, V, (B, R)).astype(np.int32)
    draft = am[:, :K].copy()                               # every draft matches: s = K + 1
    acc = np.ones((B, K), dtype=np.uint8)
    num = B * pages_per_seq
    kb = bf16(rng.standard_normal((L, B, R, Hkv, D)))
    vb = bf16(rng.standard_normal((L, B, R, Hkv, D)))
    kp = bf16(rng.standard_normal((L, num, Hkv, P, D)))
    vp = bf16(rng.standard_normal((L, num, Hkv, P, D)))
    bits = lambda x: x.cpu().view(torch.int16).numpy()
    kp0, vp0 = bits(kp), bits(vp)
    ctx_t = torch.from_numpy(ctx).cuda()
    alen = torch.empty(B, dtype=torch.int32, device="cuda")
    em = torch.empty((B, R), dtype=torch.int32, device="cuda")
    C.accept_commit(torch.from_numpy(draft).cuda(), torch.from_numpy(am).cuda(),
                    torch.from_numpy(acc).cuda(), kb, vb, kp, vp, torch.from_numpy(table_bad).cuda(),
                    ctx_t, alen, em)
    assert C.get_device_error() == C.DEVERR_CTX | C.DEVERR_PAGE
    s, emitted = O.accept_scan(draft, am, acc)
    assert np.array_equal(alen.cpu().numpy(), s) and np.array_equal(em.cpu().numpy(), emitted)
    got_ctx = ctx_t.cpu().numpy()
    assert got_ctx[0] == ctx[0] + R and got_ctx[1] == ctx[1]
    # the oracle commit of sequence 0 alone
    only0 = np.array([R, 0, 0], dtype=np.int64)
    kp_ref, vp_ref, _ = O.commit_kv(bits(kb), bits(vb), kp0, vp0, table, ctx, only0, P)
    kp_got, vp_got = bits(kp), bits(vp)
    for b in range(B):                                     # sequence 2 wrote nothing either
        pages = table[b]
        assert np.array_equal(kp_got[:, pages], kp_ref[:, pages])
        assert np.array_equal(vp_got[:, pages], vp_ref[:, pages])


# ---------------------------------------------------------------------------
# Stochastic decoding: temperature sampling in the LM-head epilogue (Sec. 3.1)
# ---------------------------------------------------------------------------

def _key_margin(keys: np.ndarray) -> np.ndarray:
    top2 = np.sort(keys, axis=1)[:, -2:]
    return top2[:, 1] - top2[:, 0]


SAMPLE_CASES = [
    # M, d, V, weight std, temperature, seed
    (1, 64, 128, 0.1, 1.0, 0),
    (6, 4096, 151936, 0.02, 1.0, 0x0123456789ABCDEF),   # Qwen3-8B LM head, batch 1, K = 5
    (17, 256, 1000, 0.1, 0.5, 7),                      # ragged vocabulary tile, rows not 4-aligned
    (300, 128, 2048, 0.1, 1.0, 2 ** 40 + 3),           # two passes (160 + 140 rows)
    (64, 512, 4096, 0.3, 2.0, 99),
]


@pytest.mark.parametrize("case", SAMPLE_CASES, ids=lambda c: f"M{c[0]}V{c[2]}T{c[4]}")
def test_lmhead_sampling_matches_oracle(case):
    M, d, V, wstd, T, seed = case
    rng = np.random.default_rng(M * 13 + V)
    hidden = bf16(rng.standard_normal((M, d)))
    w = bf16(rng.standard_normal((V, d)) * wstd)
    dfr = rng.integers(-1, V, M).astype(np.int32)
    smp = torch.empty(M, dtype=torch.int32, device="cuda")
    st = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    seed_t = torch.tensor([seed], dtype=torch.int64, device="cuda")
    C.lmhead_sample_features(hidden, w, torch.from_numpy(dfr).cuda(), T, seed_t, smp, st,
                             C.new_lmhead_workspace(M, d, V))
    x = O.lmhead_logits(host(hidden), host(w))
    ref_s, ref_st = O.row_stats_sampled(x, dfr, seed, T)
    assert_close(st.cpu().numpy(), ref_st, "sampled lm-head stats")
    clear = _key_margin(O.gumbel_keys(x, seed, T)) >= 1e-3
    got = smp.cpu().numpy()
    assert np.array_equal(got[clear], ref_s[clear])
    assert np.all((got >= 0) & (got < V))
    # with this much noise the sample is often not the argmax
    if M >= 17:
        assert np.mean(got != np.argmax(x, axis=1)) > 0.2
    print(f"sampled lm-head {case}: tie rows {(~clear).sum()}")


def test_lmhead_sampling_reads_the_seed_when_the_graph_runs():
    M, d, V = 12, 256, 3000
    rng = np.random.default_rng(5)
    hidden = bf16(rng.standard_normal((M, d)))
    w = bf16(rng.standard_normal((V, d)) * 0.05)
    dfr = torch.full((M,), -1, dtype=torch.int32, device="cuda")
    smp = torch.empty(M, dtype=torch.int32, device="cuda")
    st = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    seed_t = torch.tensor([1], dtype=torch.int64, device="cuda")
    ws = C.new_lmhead_workspace(M, d, V)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        C.lmhead_sample_features(hidden, w, dfr, 1.0, seed_t, smp, st, ws)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        C.lmhead_sample_features(hidden, w, dfr, 1.0, seed_t, smp, st, ws)
    x = O.lmhead_logits(host(hidden), host(w))
    seen = []
    for seed in (3, 2 ** 33 + 5, 12345):
        seed_t.fill_(seed)
        g.replay()
        torch.cuda.synchronize()
        got = smp.cpu().numpy()
        ref, _ = O.row_stats_sampled(x, np.full(M, -1), seed, 1.0)
        clear = _key_margin(O.gumbel_keys(x, seed, 1.0)) >= 1e-3
        assert np.array_equal(got[clear], ref[clear])
        seen.append(got)
    assert not np.array_equal(seen[0], seen[1]) and not np.array_equal(seen[1], seen[2])


def test_lmhead_sampling_at_tiny_temperature_is_the_argmax():
    M, d, V = 40, 512, 5000
    rng = np.random.default_rng(8)
    hidden = bf16(rng.standard_normal((M, d)))
    w = bf16(rng.standard_normal((V, d)) * 0.05)
    dfr = torch.full((M,), -1, dtype=torch.int32, device="cuda")
    ws = C.new_lmhead_workspace(M, d, V)
    am = torch.empty(M, dtype=torch.int32, device="cuda")
    smp = torch.empty(M, dtype=torch.int32, device="cuda")
    st0 = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    st1 = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    C.lmhead_argmax_features(hidden, w, dfr, am, st0, ws)
    C.lmhead_sample_features(hidden, w, dfr, 1e-5, torch.tensor([77], dtype=torch.int64,
                             device="cuda"), smp, st1, ws)
    x = O.lmhead_logits(host(hidden), host(w))
    top2 = np.sort(x, axis=1)[:, -2:]
    clear = (top2[:, 1] - top2[:, 0]) >= 1e-3
    assert np.array_equal(smp.cpu().numpy()[clear], am.cpu().numpy()[clear])
    # the statistics do not depend on the sampling (up to the summation order on exact ties)
    torch.testing.assert_close(st0, st1, rtol=1e-6, atol=1e-6, equal_nan=True)


@pytest.mark.parametrize("T", [1.0, 0.6])
def test_tiny_sampled_round_matches_oracle(T):
    cfg = W.CONFIGS["tiny"].replace(batch=3, k=6, mismatch_rate=0.5, ctx_lo=30, ctx_hi=200,
                                    shuffled_pages=True)
    inp = W.make_round_inputs(cfg, device="cuda")
    hostd = {kk: (v.cpu() if torch.is_tensor(v) else v) for kk, v in inp.items()}
    x = O.lmhead_logits(hostd["hidden"], hostd["w"])
    ranked = O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8)
    draft = W.synth_drafts(cfg, ranked)
    seed = W.sample_seed(cfg, 0)
    rnd = VerifyRound(inp, draft, cfg.lam, C.POLICY_MLP, temperature=T, seed=seed)
    rnd.run()
    torch.cuda.synchronize()
    ref = O.cospec_round(hostd, draft, cfg.lam, with_attention=False, with_commit=False,
                         sample_seed=seed, temperature=T)
    s_gpu = rnd.accept_len.cpu().numpy()
    ties = tie_positions(ref["stats"], draft, ref["argmax"], ref["p"], ref["s"], s_gpu, cfg.lam,
                         margin=ref["key_margin"])
    report_ties("sampled round parity", f"{cfg.name} T={T}", ties)
    tie = ties > 0
    ok = ~tie
    assert np.array_equal(s_gpu[ok], ref["s"][ok])
    assert np.array_equal(rnd.emitted.cpu().numpy().reshape(cfg.batch, -1)[ok], ref["emitted"][ok])
    clear = ref["key_margin"] >= 1e-3
    assert np.array_equal(rnd.argmax.cpu().numpy().reshape(cfg.batch, -1)[clear],
                          ref["argmax"][clear])
    print(f"sampled round T={T}: s {s_gpu.tolist()} ties {int(tie.sum())}")


def test_lmhead_sampling_noise_only_at_huge_temperature():
    """At T = 1e6 the keys are the Gumbel noise alone (|x / T| < 1e-5), so each
    row's sample is the position of the largest of V noise values: the
    generator, the counter layout and the upper tail of g are checked against
    the oracle's float64 noise directly."""
    M, d, V, T, seed = 64, 256, 20000, 1e6, 0xDEADBEEF12345
    rng = np.random.default_rng(21)
    hidden = bf16(rng.standard_normal((M, d)))
    w = bf16(rng.standard_normal((V, d)) * 0.01)
    smp = torch.empty(M, dtype=torch.int32, device="cuda")
    st = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    C.lmhead_sample_features(hidden, w, torch.full((M,), -1, dtype=torch.int32, device="cuda"), T,
                             torch.tensor([seed], dtype=torch.int64, device="cuda"), smp, st,
                             C.new_lmhead_workspace(M, d, V))
    x = O.lmhead_logits(host(hidden), host(w))
    keys = O.gumbel_keys(x, seed, T)
    clear = _key_margin(keys) >= 1e-3
    assert clear.sum() >= M - 2
    assert np.array_equal(smp.cpu().numpy()[clear], np.argmax(keys, axis=1)[clear])
