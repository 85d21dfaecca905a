"""Speculative sampling, the exact-match baseline at a temperature (Sec. 3.1
"Stochastic decoding", App. C.3), on the device against the oracle: the LM
head's logits mode, the acceptance kernels, a whole round with its commit,
and the distribution-preservation property of the kernels themselves."""
import numpy as np
import pytest
import torch

from oracle import cospec_oracle as O
from oracle import cospec_sps as S
from paper_2605_24793_gb300 import build as BLD
from paper_2605_24793_gb300 import cospec as C
from paper_2605_24793_gb300 import workload as W
from paper_2605_24793_gb300.round import VerifyRound

from .parity_util import TIE, assert_close, report_ties

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    C.load_library(BLD.build())
    torch.cuda.set_device(0)


def _bf16(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16).cuda()


def _lmhead_logits(hidden, w, dfr, T):
    M, V = hidden.shape[0], w.shape[0]
    argmax = torch.empty(M, dtype=torch.int32, device="cuda")
    stats = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    logits = torch.empty((M, V), dtype=torch.float32, device="cuda")
    ws = C.new_lmhead_workspace(M, hidden.shape[1], V)
    C.lmhead_logits_features(hidden, w, dfr, T, argmax, stats, logits, ws)
    return argmax, stats, logits


@pytest.mark.parametrize("M,d,V,T", [(13, 256, 5000, 1.0), (40, 512, 4099, 0.7),
                                     (300, 256, 3000, 1.3)])
def test_lmhead_logits_mode_matches_oracle(M, d, V, T):
    rng = np.random.default_rng(M + V)
    hidden = _bf16(rng.standard_normal((M, d)))
    w = _bf16(rng.standard_normal((V, d)) * 0.05)
    dfr_np = rng.integers(-1, V, M).astype(np.int32)
    dfr = torch.from_numpy(dfr_np).cuda()
    x = O.lmhead_logits(hidden.cpu(), w.cpu()) / T
    ref_am, ref_st = O.row_stats(x, dfr_np)
    am, st, logits = _lmhead_logits(hidden, w, dfr, T)
    torch.cuda.synchronize()
    assert C.get_device_error() == 0
    assert_close(logits.cpu().numpy(), x, "scaled logits")
    assert_close(st.cpu().numpy(), ref_st, "statistics of the scaled logits")
    clear = (ref_st[:, 0] - ref_st[:, 1]) >= TIE
    assert np.array_equal(am.cpu().numpy()[clear], ref_am[clear])


def _sps_case(B, K, V, T, noise, d=256, seed=0x5EED_0000_1234):
    cfg = W.CONFIGS["tiny"].replace(batch=B, k=K, vocab=V, hidden=d)
    R = K + 1
    rng = np.random.default_rng(B * 131 + K * 7 + V)
    hidden = _bf16(rng.standard_normal((B * R, d)))
    w = _bf16(rng.standard_normal((V, d)) * 0.08)
    x = O.lmhead_logits(hidden.cpu(), w.cpu()).reshape(B, R, V)
    q = W.draft_distributions(cfg, x, noise=noise, temperature=T)
    draft = W.sample_from(cfg, q)
    return cfg, hidden, w, x, q, draft, seed


@pytest.mark.parametrize("B,K,V,T,noise", [(16, 4, 3000, 1.0, 1.0), (8, 7, 5000, 0.8, 2.0),
                                           (32, 1, 2000, 1.0, 0.5), (4, 31, 1500, 1.0, 1.0),
                                           (5, 0, 1000, 1.0, 1.0), (3, 5, 151936, 1.0, 1.0)])
def test_sps_accept_matches_oracle(B, K, V, T, noise):
    cfg, hidden, w, x, q, draft, seed = _sps_case(B, K, V, T, noise)
    R = K + 1
    ref = S.sps_round(x, q.astype(np.float64), draft, seed, T)
    dfr = torch.from_numpy(W.draft_for_rows(draft)).cuda()
    _, st, logits = _lmhead_logits(hidden, w, dfr, T)
    target = torch.full((B * R,), -7, dtype=torch.int32, device="cuda")
    accept = torch.full((B, K), 7, dtype=torch.uint8, device="cuda")
    ratio = torch.empty((B, K), dtype=torch.float32, device="cuda")
    seed_t = torch.tensor([seed], dtype=torch.int64, device="cuda")
    C.sps_accept(torch.from_numpy(draft).cuda(), st, logits, torch.from_numpy(q).cuda(), seed_t,
                 target, accept, ratio, C.new_sps_workspace(B))
    torch.cuda.synchronize()
    assert C.get_device_error() == 0
    assert_close(ratio.cpu().numpy(), ref["ratio"], "acceptance ratio min(1, p/q)")
    ties = ((ref["margin"] < TIE) | (ref["key_margin"] < TIE)).astype(np.int64)
    report_ties("speculative-sampling parity", f"B={B} K={K} V={V} T={T}", ties)
    ok = ties == 0
    assert ok.sum() >= (B + 1) // 2
    assert np.array_equal(accept.cpu().numpy()[ok], ref["accept"][ok])
    assert np.array_equal(target.cpu().numpy().reshape(B, R)[ok], ref["target"][ok])


def test_sps_accept_rejects_a_draft_id_outside_the_vocabulary():
    # The acceptance kernel checks the draft ids itself: an id outside
    # [0, V) sets the token bit, reads no q or p for it, and is rejected;
    # the other sequences decide as the oracle does.
    B, K, V, T = 6, 4, 2000, 1.0
    cfg, hidden, w, x, q, draft, seed = _sps_case(B, K, V, T, 1.0)
    R = K + 1
    ref = S.sps_round(x, q.astype(np.float64), draft, seed, T)
    dfr = torch.from_numpy(W.draft_for_rows(draft)).cuda()    # the LM head sees valid ids
    _, st, logits = _lmhead_logits(hidden, w, dfr, T)
    bad = draft.copy()
    bad[2, 0] = V + 5
    target = torch.full((B * R,), -7, dtype=torch.int32, device="cuda")
    accept = torch.full((B, K), 7, dtype=torch.uint8, device="cuda")
    ratio = torch.empty((B, K), dtype=torch.float32, device="cuda")
    seed_t = torch.tensor([seed], dtype=torch.int64, device="cuda")
    C.sps_accept(torch.from_numpy(bad).cuda(), st, logits, torch.from_numpy(q).cuda(), seed_t,
                 target, accept, ratio, C.new_sps_workspace(B))
    torch.cuda.synchronize()
    assert C.get_device_error() == C.DEVERR_TOKEN
    acc = accept.cpu().numpy()
    assert acc[2, 0] == 0
    tgt = target.cpu().numpy().reshape(B, R)
    assert np.all((tgt[2] >= -1) & (tgt[2] < V))
    ties = ((ref["margin"] < TIE) | (ref["key_margin"] < TIE)).astype(np.int64)
    ok = ties == 0
    ok[2] = False
    assert np.array_equal(acc[ok], ref["accept"][ok])
    assert np.array_equal(tgt[ok], ref["target"][ok])


def test_sps_round_with_commit_matches_oracle():
    """A whole round: attention, LM head with logits, speculative-sampling
    acceptance, accept/commit, against the oracle's round and commit."""
    cfg = W.CONFIGS["tiny"].replace(batch=6, k=5, ctx_lo=30, ctx_hi=400, qkv_std=1.0,
                                    shuffled_pages=True)
    inp = W.make_round_inputs(cfg, device="cuda")
    host = {k: (v.cpu() if torch.is_tensor(v) else v) for k, v in inp.items()}
    x = O.lmhead_logits(host["hidden"], host["w"]).reshape(cfg.batch, cfg.rows, cfg.vocab)
    q = W.draft_distributions(cfg, x, noise=1.0)
    draft = W.sample_from(cfg, q)
    seed = W.sample_seed(cfg, 3)
    ref = S.sps_round(x, q.astype(np.float64), draft, seed, 1.0)
    kp, vp, ctx = O.commit_kv(O._to_np(inp["k_blk"]), O._to_np(inp["v_blk"]), O._to_np(inp["k_pages"]),
                              O._to_np(inp["v_pages"]), inp["page_table_np"], inp["ctx_len_np"],
                              ref["s"], cfg.page_size)
    rnd = VerifyRound(inp, draft, seed=seed, sps_q=torch.from_numpy(q).cuda())
    rnd.capture()
    rnd.replay()
    torch.cuda.synchronize()
    assert C.get_device_error() == 0
    ties = ((ref["margin"] < TIE) | (ref["key_margin"] < TIE)).astype(np.int64)
    report_ties("speculative-sampling round", cfg.name, ties)
    ok = ties == 0
    assert np.array_equal(rnd.accept_len.cpu().numpy()[ok], ref["s"][ok])
    assert np.array_equal(rnd.emitted.cpu().numpy()[ok], ref["emitted"][ok])
    assert np.array_equal(rnd.ctx_len.cpu().numpy()[ok], ctx[ok])
    gk = rnd.k_pages.cpu().view(torch.int16).numpy()
    gv = rnd.v_pages.cpu().view(torch.int16).numpy()
    for b in np.nonzero(ok)[0]:
        pages = inp["page_table_np"][b][inp["page_table_np"][b] >= 0]
        assert np.array_equal(gk[:, pages], kp[:, pages])
        assert np.array_equal(gv[:, pages], vp[:, pages])


def test_kernels_preserve_the_target_distribution():
    """The defining property of speculative sampling, checked on the device
    alone: over many independent sequences with the same target p and draft
    q, the first emitted token follows p and position 1 is accepted with
    probability sum_v min(p, q)."""
    B, K, V, d = 8192, 1, 8, 64
    p = np.array([0.3, 0.2, 0.15, 0.1, 0.1, 0.08, 0.05, 0.02])
    q = np.array([0.05, 0.4, 0.05, 0.2, 0.1, 0.1, 0.05, 0.05])
    logit = torch.from_numpy(np.log(p)).to(torch.bfloat16)
    pb = np.exp(logit.double().numpy())
    pb /= pb.sum()                                         # the target the bf16 logits define
    w = torch.zeros((V, d), dtype=torch.bfloat16)
    w[:, :V] = torch.eye(V)
    hidden = torch.zeros((B * (K + 1), d), dtype=torch.bfloat16)
    hidden[:, :V] = logit
    rng = np.random.default_rng(77)
    draft = rng.choice(V, size=(B, K), p=q).astype(np.int32)
    dfr = torch.from_numpy(W.draft_for_rows(draft)).cuda()
    _, st, logits = _lmhead_logits(hidden.cuda(), w.cuda(), dfr, 1.0)
    target = torch.empty(B * (K + 1), dtype=torch.int32, device="cuda")
    accept = torch.empty((B, K), dtype=torch.uint8, device="cuda")
    ratio = torch.empty((B, K), dtype=torch.float32, device="cuda")
    qd = torch.from_numpy(np.broadcast_to(q, (B, K, V)).astype(np.float32).copy()).cuda()
    C.sps_accept(torch.from_numpy(draft).cuda(), st, logits, qd,
                 torch.tensor([0xC0FFEE], dtype=torch.int64, device="cuda"), target, accept, ratio,
                 C.new_sps_workspace(B))
    torch.cuda.synchronize()
    t = target.cpu().numpy().reshape(B, K + 1)
    a = accept.cpu().numpy()[:, 0]
    first = np.where(a == 1, draft[:, 0], t[:, 0])
    freq = np.bincount(first, minlength=V) / B
    np.testing.assert_allclose(freq, pb, atol=0.02)
    assert abs(a.mean() - np.minimum(pb, q).sum()) < 0.02


def test_sps_rounds_match_oracle_round_by_round():
    """Several speculative-sampling rounds in a row from one graph (fresh
    seed, draft distribution and drafts per round): each round's accepted
    length and tokens, the growing context and the committed cache."""
    from paper_2605_24793_gb300.decode import MultiRoundDecoder
    k, rounds = 5, 4
    cfg = W.CONFIGS["tiny"].replace(k=k, batch=3, ctx_lo=40, ctx_hi=300, qkv_std=1.0,
                                    shuffled_pages=True)
    inp = W.make_round_inputs(cfg, device="cuda", extra_tokens=rounds * cfg.rows)
    host = {kk: (v.cpu() if torch.is_tensor(v) else v) for kk, v in inp.items()}
    dec = MultiRoundDecoder(cfg, rounds, inputs=inp, sps=True, temperature=1.0, draft_noise=0.5)
    res = dec.run()
    assert res["device_error"] == 0
    s_gpu = dec.s_hist.cpu().numpy()
    em_gpu = dec.emitted_hist.cpu().numpy()
    x = O.lmhead_logits(host["hidden"], host["w"]).reshape(cfg.batch, cfg.rows, cfg.vocab)
    kp, vp = O._to_np(inp["k_pages"]), O._to_np(inp["v_pages"])
    ctx = inp["ctx_len_np"].astype(np.int64)
    tie = np.zeros(cfg.batch, dtype=bool)
    for r in range(rounds):
        q = dec.q_table[r].cpu().numpy().astype(np.float64)
        ref = S.sps_round(x, q, dec.drafts_np[r], W.sample_seed(cfg, r), 1.0)
        ties = ((ref["margin"] < TIE) | (ref["key_margin"] < TIE)).astype(np.int64)
        report_ties("speculative-sampling rounds", f"{cfg.name} round {r}", ties)
        tie |= ties > 0
        ok = ~tie
        assert np.array_equal(s_gpu[r][ok], ref["s"][ok]), f"round {r}"
        assert np.array_equal(em_gpu[r][ok], ref["emitted"][ok]), f"round {r}"
        kp, vp, ctx = O.commit_kv(O._to_np(inp["k_blk"]), O._to_np(inp["v_blk"]), kp, vp,
                                  inp["page_table_np"], ctx, ref["s"], cfg.page_size)
    ok = ~tie
    assert np.array_equal(dec.rnd.ctx_len.cpu().numpy()[ok], ctx[ok])
    gk = dec.rnd.k_pages.cpu().view(torch.int16).numpy()
    for b in np.nonzero(ok)[0]:
        pages = inp["page_table_np"][b][inp["page_table_np"][b] >= 0]
        assert np.array_equal(gk[:, pages], kp[:, pages])
    assert res["tau"] == pytest.approx(float(s_gpu.mean()))
