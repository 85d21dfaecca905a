"""Multi-round CoSpec decoding on the device (App. F, Inference Procedure:
draft, verify, arbitrate, stop at the first rejected mismatch, commit,
repeat) and the mean accepted length tau = (1/R) sum_r s^(r) (Sec. 3.1, Eq. 5).
With a temperature, target candidates are drawn by sampling (stochastic
decoding, Sec. 3.1) with a fresh seed per round from a device table.  With
``sps`` the rounds are those of the exact-match baseline with speculative
sampling at that temperature (the paper's distribution-preserving comparison
at T = 1): each round's drafts are drawn from a synthetic draft distribution
(the target's logits plus Gaussian noise), kept in a device table with them.

The rounds reuse one CUDA graph: every replay copies that round's draft ids
from a device table (selected by a device-side round counter), runs the
round on a context that grows by the accepted length s, and records s.  The
draft ids are synthetic (the target's rank-1 id with probability 1 - rate,
else ranks 2..8), drawn independently per round; the verify inputs of the
block (Q, block K/V, hidden rows) are the workload's synthetic tensors.

  python -m paper_2605_24793_gb300.decode --config qwen3_8b_b1 --rounds 64
  python -m paper_2605_24793_gb300.decode --sweep        # K and lambda sweep
  python -m paper_2605_24793_gb300.decode --temperature 1
  python -m paper_2605_24793_gb300.decode --temperature 1 --sps   # the baseline
"""
from __future__ import annotations

import argparse
import json
from typing import Dict, Optional

import numpy as np
import torch

from . import cospec as C
from . import workload as W
from .round import VerifyRound


def target_logits(cfg: W.RoundConfig, hidden: torch.Tensor, w: torch.Tensor) -> np.ndarray:
    """fp32 logits of the block rows on the device, [B, R, V] on the host, used
    only to synthesise draft distributions."""
    h = hidden.float()
    out = [(h[r0:r0 + 64] @ w.float().T).cpu() for r0 in range(0, h.shape[0], 64)]
    return torch.cat(out).numpy().reshape(cfg.batch, cfg.rows, -1)


def target_ranked_ids(cfg: W.RoundConfig, hidden: torch.Tensor, w: torch.Tensor, t: int = 8):
    """Ranked top-t ids of each block row's logits (fp32 on the device), used
    only to synthesise draft ids."""
    h = hidden.float()
    out = []
    for r0 in range(0, h.shape[0], 64):
        out.append(torch.topk(h[r0:r0 + 64] @ w.float().T, t, dim=1).indices.cpu())
    return torch.cat(out).numpy().reshape(cfg.batch, cfg.rows, t)


class MultiRoundDecoder:
    def __init__(self, cfg: W.RoundConfig, rounds: int, lam: Optional[float] = None,
                 mode: int = C.POLICY_MLP, device="cuda", inputs: Optional[Dict] = None,
                 drafts: Optional[np.ndarray] = None, temperature: Optional[float] = None,
                 sps: bool = False, draft_noise: float = 1.0):
        self.cfg, self.rounds = cfg, rounds
        self.lam = cfg.lam if lam is None else lam
        self.inp = inputs if inputs is not None else W.make_round_inputs(
            cfg, device=device, extra_tokens=rounds * cfg.rows)
        dev = self.inp["q"].device
        self.sps = sps
        self.q_table = None
        if sps:
            if temperature is None:
                temperature = 1.0
            x = target_logits(cfg, self.inp["hidden"], self.inp["w"])
            qs = [W.draft_distributions(cfg, x, draft_noise, temperature, r) for r in range(rounds)]
            if drafts is None:
                drafts = np.stack([W.sample_from(cfg, q, r) for r, q in enumerate(qs)])
            self.q_table = torch.from_numpy(np.stack(qs)).to(dev)
            del x, qs
        if drafts is None:
            ranked = target_ranked_ids(cfg, self.inp["hidden"], self.inp["w"])
            drafts = np.stack([W.synth_drafts(cfg, ranked, r) for r in range(rounds)])
        self.drafts_np = drafts
        max_ctx = int(self.inp["ctx_len_np"].max()) + rounds * cfg.rows
        self.temperature = temperature
        self.seeds_np = np.array([W.sample_seed(cfg, r) for r in range(rounds)], dtype=np.int64)
        self.rnd = VerifyRound(self.inp, drafts[0], self.lam, mode, max_ctx=max_ctx,
                               temperature=temperature, seed=int(self.seeds_np[0]),
                               sps_q=None if self.q_table is None else self.q_table[0].clone())
        B, K, R = cfg.batch, cfg.k, cfg.rows
        dfr = np.full((rounds, B, R), -1, dtype=np.int32)
        dfr[:, :, :K] = drafts
        self.drafts = torch.from_numpy(np.ascontiguousarray(drafts, dtype=np.int32)).to(dev)
        self.dfr = torch.from_numpy(dfr.reshape(rounds, B * R)).to(dev)
        self.seeds = torch.from_numpy(self.seeds_np).to(dev)
        self.idx = torch.zeros(1, dtype=torch.int64, device=dev)
        self.s_hist = torch.zeros((rounds, B), dtype=torch.int32, device=dev)
        self.emitted_hist = torch.full((rounds, B, R), -1, dtype=torch.int32, device=dev)
        self.graph: Optional[torch.cuda.CUDAGraph] = None

    def _round(self):
        B, K = self.cfg.batch, self.cfg.k
        torch.index_select(self.drafts, 0, self.idx, out=self.rnd.draft.view(1, B, K))
        torch.index_select(self.dfr, 0, self.idx, out=self.rnd.draft_for_row.view(1, -1))
        if self.temperature is not None:
            torch.index_select(self.seeds, 0, self.idx, out=self.rnd.seed)
        if self.q_table is not None:
            torch.index_select(self.q_table, 0, self.idx,
                               out=self.rnd.draft_q.view((1,) + tuple(self.rnd.draft_q.shape)))
        self.rnd.run(restore=False)
        self.s_hist.index_copy_(0, self.idx, self.rnd.accept_len.view(1, B))
        self.emitted_hist.index_copy_(0, self.idx, self.rnd.emitted.view(1, B, -1))
        self.idx += 1

    def capture(self):
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self._round()                # warm-up on round 0, then rewind
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.reset()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self._round()
        self.graph = g
        self.reset()

    def reset(self):
        """Rewind to round 0 on the initial context (committed rows beyond
        the initial context are simply overwritten by the next run)."""
        self.idx.zero_()
        self.rnd.restore_context()
        self.s_hist.zero_()

    def run(self) -> Dict[str, float]:
        if self.graph is None:
            self.capture()
        self.reset()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(self.rounds):
            self.graph.replay()
        e1.record()
        e1.synchronize()
        ms = e0.elapsed_time(e1)
        s = self.s_hist.cpu().numpy()
        cfg = self.cfg
        return {"rounds": self.rounds, "tau": float(s.mean()),
                "tau_per_seq": s.mean(axis=0).tolist(),
                "ms_per_round": ms / self.rounds,
                "emitted_tokens_per_s": float(s.sum()) / (ms * 1e-3),
                "block_tokens_per_s": cfg.batch * cfg.rows * self.rounds / (ms * 1e-3),
                "device_error": C.get_device_error()}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--config", default="qwen3_8b_b1", choices=sorted(W.CONFIGS))
    ap.add_argument("--rounds", type=int, default=64)
    ap.add_argument("--k", type=int, default=None)
    ap.add_argument("--lam", type=float, default=None)
    ap.add_argument("--temperature", type=float, default=None,
                    help="sample target candidates at this temperature (default: greedy)")
    ap.add_argument("--sps", action="store_true",
                    help="the exact-match baseline with speculative sampling (T = 1 by default)")
    ap.add_argument("--draft-noise", type=float, default=1.0,
                    help="std of the noise added to the target logits to form the draft (--sps)")
    ap.add_argument("--sweep", action="store_true",
                    help="K in {15, 20, 25} at lambda 0.6, then lambda in {0.4, 0.6, 0.8} at K 25")
    args = ap.parse_args()
    from . import build as B
    C.load_library(B.build())
    base = W.CONFIGS[args.config]
    points = []
    if args.sweep:
        points = [(k, 0.6) for k in (15, 20, 25)] + [(25, lam) for lam in (0.4, 0.8)]
    else:
        points = [(args.k if args.k is not None else base.k, args.lam if args.lam is not None else base.lam)]
    for k, lam in points:
        cfg = base.replace(k=k)
        dec = MultiRoundDecoder(cfg, args.rounds, lam, temperature=args.temperature, sps=args.sps,
                                draft_noise=args.draft_noise)
        res = dec.run()
        res.update({"workload": cfg.name, "k": k, "lambda": lam, "batch": cfg.batch,
                    "temperature": dec.temperature,
                    "method": "exact-match, speculative sampling" if args.sps else "CoSpec",
                    "draft_noise": args.draft_noise if args.sps else None})
        print(json.dumps(res), flush=True)
        del dec
        torch.cuda.empty_cache()


if __name__ == "__main__":
    main()
