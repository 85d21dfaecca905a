"""Several rounds in a row on the device (App. F inference loop) against the
oracle applied round by round to its own committed cache: accepted lengths,
emitted tokens, the growing context and the committed cache bytes."""
import numpy as np
import pytest
import torch

from oracle import cospec_oracle as O
from paper_2605_24793_gb300 import build as BLD
from paper_2605_24793_gb300 import cospec as C
from paper_2605_24793_gb300 import workload as W
from paper_2605_24793_gb300.decode import MultiRoundDecoder

from .parity_util import report_ties, tie_positions

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    C.load_library(BLD.build())
    torch.cuda.set_device(0)


@pytest.mark.parametrize("k,rounds,lam", [(4, 4, 0.6), (25, 3, 0.4), (7, 5, 0.8)])
def test_rounds_match_oracle_round_by_round(k, rounds, lam):
    cfg = W.CONFIGS["tiny"].replace(k=k, batch=3, ctx_lo=40, ctx_hi=300, mismatch_rate=0.5,
                                    qkv_std=1.0, shuffled_pages=True)
    inp = W.make_round_inputs(cfg, device="cuda", extra_tokens=rounds * cfg.rows)
    host = {kk: (v.cpu() if torch.is_tensor(v) else v) for kk, v in inp.items()}
    x = O.lmhead_logits(host["hidden"], host["w"])
    ranked = O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8)
    drafts = np.stack([W.synth_drafts(cfg, ranked, r) for r in range(rounds)])

    dec = MultiRoundDecoder(cfg, rounds, lam, inputs=inp, drafts=drafts)
    res = dec.run()
    assert res["device_error"] == 0
    s_gpu = dec.s_hist.cpu().numpy()
    em_gpu = dec.emitted_hist.cpu().numpy()

    state = dict(host)
    tie_seqs = np.zeros(cfg.batch, dtype=bool)
    for r in range(rounds):
        ref = O.cospec_round(state, drafts[r], lam, with_attention=False)
        ties = tie_positions(ref["stats"], drafts[r], ref["argmax"], ref["p"], ref["s"], s_gpu[r], lam)
        report_ties("multi-round parity", f"{cfg.name} K={k} lambda={lam} round {r}", ties)
        tie_seqs |= ties > 0
        ok = ~tie_seqs
        assert np.array_equal(s_gpu[r][ok], ref["s"][ok]), f"round {r}"
        assert np.array_equal(em_gpu[r][ok], ref["emitted"][ok]), f"round {r}"
        state = dict(state)
        state["k_pages"] = torch.from_numpy(ref["k_pages"]).view(torch.bfloat16)
        state["v_pages"] = torch.from_numpy(ref["v_pages"]).view(torch.bfloat16)
        state["ctx_len_np"] = ref["ctx_len"].astype(np.int32)
    ok = ~tie_seqs
    assert np.array_equal(dec.rnd.ctx_len.cpu().numpy()[ok], state["ctx_len_np"][ok])
    kp = dec.rnd.k_pages.cpu().view(torch.int16).numpy()
    vp = dec.rnd.v_pages.cpu().view(torch.int16).numpy()
    table = inp["page_table_np"]
    for b in np.nonzero(ok)[0]:
        pages = table[b][table[b] >= 0]
        assert np.array_equal(kp[:, pages], state["k_pages"].view(torch.int16).numpy()[:, pages])
        assert np.array_equal(vp[:, pages], state["v_pages"].view(torch.int16).numpy()[:, pages])
    # Eq. 5: tau is the mean accepted length over the rounds
    assert res["tau"] == pytest.approx(float(s_gpu.mean()))
    assert 1.0 <= res["tau"] <= k + 1
    print(f"K={k} lambda={lam}: tau {res['tau']:.2f} over {rounds} rounds, ties {int(tie_seqs.sum())}")


def test_sampled_rounds_match_oracle_round_by_round():
    """Stochastic decoding (Sec. 3.1): a fresh seed per round from the device
    table; each round's sampled candidates and outcome match the oracle."""
    k, rounds, lam, T = 5, 4, 0.6, 1.0
    cfg = W.CONFIGS["tiny"].replace(k=k, batch=3, ctx_lo=40, ctx_hi=300, mismatch_rate=0.5,
                                    qkv_std=1.0, shuffled_pages=True)
    inp = W.make_round_inputs(cfg, device="cuda", extra_tokens=rounds * cfg.rows)
    host = {kk: (v.cpu() if torch.is_tensor(v) else v) for kk, v in inp.items()}
    x = O.lmhead_logits(host["hidden"], host["w"])
    ranked = O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8)
    drafts = np.stack([W.synth_drafts(cfg, ranked, r) for r in range(rounds)])
    dec = MultiRoundDecoder(cfg, rounds, lam, inputs=inp, drafts=drafts, temperature=T)
    res = dec.run()
    assert res["device_error"] == 0
    s_gpu = dec.s_hist.cpu().numpy()
    em_gpu = dec.emitted_hist.cpu().numpy()
    state = dict(host)
    tie_seqs = np.zeros(cfg.batch, dtype=bool)
    for r in range(rounds):
        ref = O.cospec_round(state, drafts[r], lam, with_attention=False,
                             sample_seed=W.sample_seed(cfg, r), temperature=T)
        ties = tie_positions(ref["stats"], drafts[r], ref["argmax"], ref["p"], ref["s"],
                             s_gpu[r], lam, margin=ref["key_margin"])
        report_ties("sampled multi-round parity", f"{cfg.name} K={k} T={T} round {r}", ties)
        tie_seqs |= ties > 0
        ok = ~tie_seqs
        assert np.array_equal(s_gpu[r][ok], ref["s"][ok]), f"round {r}"
        assert np.array_equal(em_gpu[r][ok], ref["emitted"][ok]), f"round {r}"
        state = dict(state)
        state["k_pages"] = torch.from_numpy(ref["k_pages"]).view(torch.bfloat16)
        state["v_pages"] = torch.from_numpy(ref["v_pages"]).view(torch.bfloat16)
        state["ctx_len_np"] = ref["ctx_len"].astype(np.int32)
    ok = ~tie_seqs
    assert np.array_equal(dec.rnd.ctx_len.cpu().numpy()[ok], state["ctx_len_np"][ok])
    # the rounds see different samples of the same logits
    assert len({tuple(e.reshape(-1)) for e in em_gpu}) > 1
    print(f"T={T}: tau {res['tau']:.2f} over {rounds} rounds, ties {int(tie_seqs.sum())}")
