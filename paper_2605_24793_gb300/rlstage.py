"""Timing of the RL stage's reward shaping and advantages (Sec. 3.4) on a
synthetic rollout batch, through ``cospec_rl_advantages``.

  python -m paper_2605_24793_gb300.rlstage --groups 256 --rollouts 8 --rounds 64 --k 25
"""
from __future__ import annotations

import argparse
import json

import torch

from . import cospec as C
from . import workload as W


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--groups", type=int, default=256)
    ap.add_argument("--rollouts", type=int, default=8)
    ap.add_argument("--rounds", type=int, default=64)
    ap.add_argument("--k", type=int, default=25)
    ap.add_argument("--steps", type=int, default=50)
    args = ap.parse_args()
    from . import build as B
    C.load_library(B.build())
    arrs = W.rl_batch(W.seed_of(W.CONFIGS["tiny"], "rl"), args.groups, args.rollouts, args.rounds,
                      args.k)
    go, co, ro, ma, ac, el = [torch.from_numpy(a).cuda() for a in arrs]
    R = ma.shape[0]
    obj = [torch.rand((R, args.k), device="cuda") * 0.9 + 0.05 for _ in range(3)]
    for _ in range(3):
        C.rl_advantages(go, co, ro, ma, ac, el, None, *obj)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    for _ in range(args.steps):
        C.rl_advantages(go, co, ro, ma, ac, el, None, *obj)
    e1.record()
    e1.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    print(json.dumps({"groups": args.groups, "rollouts": args.groups * args.rollouts, "rounds": R,
                      "k": args.k, "decisions": R * args.k, "ms_per_call": ms,
                      "note": "per call incl. output allocation in the binding",
                      "device_error": C.get_device_error()}))


if __name__ == "__main__":
    main()
