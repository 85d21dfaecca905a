"""The seeded synthetic input recipe (CPU): context lengths, the paged pool
and its page table, tensor shapes and reproducibility, the arbitration MLP's
initialisation law, the draft synthesis and the RL rollout records."""
import math

import numpy as np
import pytest
import torch

from paper_2605_24793_gb300 import workload as W


def _tiny(**over):
    return W.CONFIGS["tiny"].replace(**over) if over else W.CONFIGS["tiny"]


def test_context_lengths_are_uniform_in_range_and_seeded():
    cfg = _tiny(batch=4000, ctx_lo=10, ctx_hi=50)
    c = W.context_lengths(cfg)
    assert c.dtype == np.int32 and c.min() >= 10 and c.max() <= 50
    assert c.min() == 10 and c.max() == 50            # both ends are drawn
    assert abs(c.mean() - 30) < 1.0
    assert np.array_equal(c, W.context_lengths(cfg))
    assert np.all(W.context_lengths(_tiny(batch=3, ctx_lo=77, ctx_hi=77)) == 77)


@pytest.mark.parametrize("shuffled", [False, True])
def test_page_table_gives_each_sequence_its_own_pages(shuffled):
    cfg = _tiny(batch=7, ctx_lo=0, ctx_hi=300, shuffled_pages=shuffled)
    ctx = W.context_lengths(cfg)
    table, num = W.page_table(cfg, ctx, extra_tokens=5)
    P, R = cfg.page_size, cfg.rows
    need = (ctx + 5 + R + P - 1) // P
    assert table.shape == (cfg.batch, need.max()) and num == need.sum()
    used = []
    for b in range(cfg.batch):
        assert np.all(table[b, :need[b]] >= 0) and np.all(table[b, need[b]:] == -1)
        assert need[b] * P >= ctx[b] + 5 + R               # room for the context and a block
        used.extend(table[b, :need[b]].tolist())
    assert sorted(used) == list(range(num))                # every pool page exactly once
    if not shuffled:
        assert used == list(range(num))                    # identity layout
    else:
        assert used != list(range(num))


def test_round_inputs_shapes_types_and_reproducibility():
    cfg = _tiny(batch=3, layers=2)
    a = W.make_round_inputs(cfg)
    b = W.make_round_inputs(cfg)
    L, B, R = cfg.layers, cfg.batch, cfg.rows
    Hq, Hkv, D, P = cfg.q_heads, cfg.kv_heads, cfg.head_dim, cfg.page_size
    assert tuple(a["q"].shape) == (L, B, R, Hq, D)
    assert tuple(a["k_blk"].shape) == tuple(a["v_blk"].shape) == (L, B, R, Hkv, D)
    assert tuple(a["k_pages"].shape) == (L, a["num_pages"], Hkv, P, D)
    assert tuple(a["hidden"].shape) == (B * R, cfg.hidden)
    assert tuple(a["w"].shape) == (cfg.vocab, cfg.hidden)
    for name in ("q", "k_blk", "v_blk", "k_pages", "v_pages", "hidden", "w"):
        assert a[name].dtype == torch.bfloat16
        assert torch.equal(a[name], b[name]), name
    assert a["page_table"].dtype == torch.int32 and a["ctx_len"].dtype == torch.int32
    # different tensors come from different streams
    assert not torch.equal(a["k_blk"], a["v_blk"])
    alias = W.make_round_inputs(cfg, alias_layers=True)
    assert alias["k_pages"].shape[0] == 1 and alias["alias_layers"]


def test_qkv_scale_follows_the_config():
    cfg = _tiny(batch=8, layers=1, qkv_std=1.0)
    q = W.make_round_inputs(cfg)["q"].float()
    assert abs(q.std().item() - 1.0) < 0.05 and abs(q.mean().item()) < 0.05


def test_mlp_init_is_the_linear_default_law():
    cfg = _tiny()
    H = 4096
    w1, b1, w2, b2 = W.mlp_params(cfg, hidden=H)
    assert tuple(w1.shape) == (H, 8) and tuple(b1.shape) == (H,) and tuple(w2.shape) == (H,)
    a1, a2 = 1 / math.sqrt(8), 1 / math.sqrt(H)
    assert w1.abs().max() <= a1 and b1.abs().max() <= a1
    assert w2.abs().max() <= a2 and abs(float(b2)) <= a2
    # U(-a, a) has variance a^2 / 3
    assert abs(w1.var().item() - a1 * a1 / 3) < 0.05 * a1 * a1


def _ranked(cfg, t=8):
    rng = np.random.default_rng(0)
    B, R = cfg.batch, cfg.rows
    return np.stack([np.stack([rng.permutation(cfg.vocab)[:t] for _ in range(R)]) for _ in range(B)])


def test_drafts_follow_the_mismatch_law():
    cfg = _tiny(batch=400, k=7, mismatch_rate=0.3, mismatch_topk=8)
    ranked = _ranked(cfg)
    d = W.synth_drafts(cfg, ranked)
    top1 = ranked[:, :cfg.k, 0]
    mism = d != top1
    assert abs(mism.mean() - 0.3) < 0.03
    # a mismatched id is one of the target's ranks 2..8
    for b, i in zip(*np.nonzero(mism)):
        assert d[b, i] in ranked[b, i, 1:8]
    assert np.array_equal(d, W.synth_drafts(cfg, ranked))
    assert not np.array_equal(d, W.synth_drafts(cfg, ranked, round_index=1))
    # the two extremes
    assert np.array_equal(W.synth_drafts(cfg.replace(mismatch_rate=0.0), ranked), top1)
    assert np.all(W.synth_drafts(cfg.replace(mismatch_rate=1.0), ranked) != top1)


def test_drafts_from_the_whole_vocabulary():
    cfg = _tiny(batch=200, k=5, mismatch_rate=1.0, mismatch_topk=0)
    ranked = _ranked(cfg)
    d = W.synth_drafts(cfg, ranked)
    assert np.all(d != ranked[:, :cfg.k, 0]) and d.min() >= 0 and d.max() < cfg.vocab


def test_draft_for_rows_layout():
    d = np.array([[5, 6, 7], [8, 9, 10]], dtype=np.int32)
    assert W.draft_for_rows(d).tolist() == [5, 6, 7, -1, 8, 9, 10, -1]


def test_sample_seeds_differ_per_round():
    cfg = _tiny()
    seeds = [W.sample_seed(cfg, r) for r in range(100)]
    assert len(set(seeds)) == 100 and all(0 <= s < (1 << 63) for s in seeds)


def test_rl_batch_records():
    g, c, ro, m, a, ell = W.rl_batch(3, groups=5, rollouts=4, rounds=6, k=7)
    assert g.tolist() == [0, 4, 8, 12, 16, 20] and len(c) == 20
    assert ro[0] == 0 and np.all(np.diff(ro) >= 1) and np.all(np.diff(ro) <= 6)
    assert m.shape == a.shape == ell.shape == (ro[-1], 7)
    assert np.all(a[m == 1] == 1) and np.all(ell <= 0)


def test_saved_inputs_replay_bit_for_bit(tmp_path):
    # a round's inputs and drafts written to .npz and read back are the same
    # bits, and the oracle's round on them gives the same result
    from oracle import cospec_oracle as O
    cfg = W.CONFIGS["tiny"].replace(batch=2, k=3, ctx_lo=20, ctx_hi=70, shuffled_pages=True)
    inp = W.make_round_inputs(cfg)
    x = O.lmhead_logits(inp["hidden"], inp["w"])
    draft = W.synth_drafts(cfg, O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8))
    path = str(tmp_path / "round.npz")
    W.save_inputs(path, inp, draft)
    got, got_draft = W.load_inputs(path)
    assert got["cfg"] == cfg and got["num_pages"] == inp["num_pages"]
    assert np.array_equal(got_draft, draft)
    assert np.array_equal(got["ctx_len_np"], inp["ctx_len_np"])
    assert np.array_equal(got["page_table_np"], inp["page_table_np"])
    for k in ("q", "k_blk", "v_blk", "k_pages", "v_pages", "hidden", "w"):
        assert got[k].dtype == torch.bfloat16 and torch.equal(got[k].view(torch.int16), inp[k].view(torch.int16))
    for a, b in zip(got["mlp"], inp["mlp"]):
        assert torch.equal(a, b)
    ref = O.cospec_round(inp, draft, 0.6)
    rep = O.cospec_round(got, got_draft, 0.6)
    for k in ("s", "emitted", "p"):
        assert np.array_equal(np.asarray(rep[k]), np.asarray(ref[k]), equal_nan=True), k
