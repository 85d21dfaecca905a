"""Parity at the full per-layer sizes of the benchmark workloads, in the
launch configuration bench.py times (graph-captured rounds).  The oracle
checks sampled (layer, sequence) attention blocks in full, every LM-head row,
and every discrete output of the round.  The two largest workloads keep
their per-layer shapes but run two layers (attention is one launch per
layer, so the launch configuration is unchanged)."""
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
    yield


def _gather_seq(inp, l, b):
    """Host copy of sequence b's pages of layer l, relabelled 0..n-1."""
    table = inp["page_table_np"][b]
    pages = table[table >= 0]
    lp = 0 if inp["k_pages"].shape[0] == 1 else l
    idx = torch.from_numpy(pages.astype(np.int64)).cuda()
    kp = inp["k_pages"][lp].index_select(0, idx).float().cpu().numpy()
    vp = inp["v_pages"][lp].index_select(0, idx).float().cpu().numpy()
    return kp, vp, np.arange(len(pages))[None, :]


CASES = [("qwen3_8b_b1", None, 3), ("qwen3_8b_b16", None, 4), ("qwen3_32b_b32", 2, 4)] + [
    (f"llama3_8b_b64_k{k}_mm{r}", 2, 3) for k in (3, 5, 7) for r in (10, 30, 60)]


@pytest.mark.parametrize("name,layers,nseq", CASES, ids=[c[0] for c in CASES])
def test_full_size_round(name, layers, nseq):
    cfg = W.CONFIGS[name]
    if layers:
        cfg = cfg.replace(layers=layers)
    inp = W.make_round_inputs(cfg, device="cuda")
    x = O.lmhead_logits(inp["hidden"].cpu(), inp["w"].cpu())
    draft = W.synth_drafts(cfg, O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8))
    B, R, K = cfg.batch, cfg.rows, cfg.k
    dfr = np.full((B, R), -1)
    dfr[:, :K] = draft
    ref_am, ref_st = O.row_stats(x, dfr.reshape(-1))
    del x
    ref_am = ref_am.reshape(B, R)
    ref_st = ref_st.reshape(B, R, 5)
    w1, b1, w2, b2 = inp["mlp"]
    ref_p, ref_a = O.arbitrate(draft, ref_am, ref_st, w1, b1, w2, b2, cfg.lam)
    ref_s, ref_em = O.accept_scan(draft, ref_am, ref_a)

    rng = np.random.default_rng(cfg.index)
    seqs = sorted(rng.choice(B, size=min(nseq, B), replace=False).tolist())
    lays = sorted({0, cfg.layers - 1, cfg.layers // 2})
    pre = {(l, b): _gather_seq(inp, l, b) for l in lays for b in seqs}
    ctx0 = inp["ctx_len_np"].copy()

    rnd = VerifyRound(inp, draft, cfg.lam, keep_attn=True)
    rnd.capture()
    rnd.replay()
    rnd.replay()                                  # a second replay restarts from the same context
    torch.cuda.synchronize()
    assert C.get_device_error() == 0

    for (l, b), (kp, vp, table) in pre.items():
        q = rnd.q[l, b:b + 1].float().cpu().numpy()
        kb = rnd.k_blk[l, b:b + 1].float().cpu().numpy()
        vb = rnd.v_blk[l, b:b + 1].float().cpu().numpy()
        ref = O.verify_attention(q, kb, vb, kp, vp, table, ctx0[b:b + 1], cfg.page_size)
        got = rnd.attn_out[l, b:b + 1].float().cpu().numpy()
        assert_close(got, ref, f"attention layer {l} seq {b}")

    st = rnd.stats.cpu().numpy().reshape(B, R, 5)
    assert_close(st, ref_st, "lm-head stats")
    s_gpu = rnd.accept_len.cpu().numpy()
    ties = tie_positions(ref_st, draft, ref_am, ref_p, ref_s, s_gpu, cfg.lam)
    report_ties("test_full_size_round", name, ties)
    tie = ties > 0
    ok = ~tie
    assert np.array_equal(rnd.argmax.cpu().numpy().reshape(B, R)[ok], ref_am[ok])
    assert_close(rnd.p.cpu().numpy()[ok], ref_p[ok], "policy probability")
    assert np.array_equal(rnd.accept.cpu().numpy()[ok], ref_a[ok])
    assert np.array_equal(s_gpu[ok], ref_s[ok])
    assert np.array_equal(rnd.emitted.cpu().numpy()[ok], ref_em[ok])
    assert np.array_equal(rnd.ctx_len.cpu().numpy()[ok], (ctx0 + ref_s)[ok])
    # committed rows of the sampled sequences: slots C..C+s-1 hold block rows 0..s-1
    kp_all = rnd.k_pages
    for b in seqs:
        if tie[b]:
            continue
        for t in range(int(ref_s[b])):
            pos = int(ctx0[b]) + t
            page = int(inp["page_table_np"][b, pos // cfg.page_size])
            for l in lays:
                lp = 0 if kp_all.shape[0] == 1 else l
                assert torch.equal(kp_all[lp, page, :, pos % cfg.page_size], rnd.k_blk[l, b, t])
                assert torch.equal(rnd.v_pages[lp, page, :, pos % cfg.page_size], rnd.v_blk[l, b, t])
    assert ok.sum() >= B // 2, "most sequences must be checked bit for bit"
