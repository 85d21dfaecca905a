"""Timing of the arbitrator's attention for one round (Sec. 3.3).

The arbitrator LM reads q = [c, SEP, draft block, SEP, target block, SEP]
with a hybrid mask: the context is causal (and, decoding round after round,
already cached), the 2K+3 region tokens see the whole context and each other.
So each of its layers, per round, is one ``cospec_verify_attn`` call with the
region as a full-mask block (COSPEC_ATTN_BLOCK_FULL) over the paged context.
This module times those L calls, replayed from a CUDA graph, on synthetic
inputs shaped like the paper's draft/arbitrator backbones.

  python -m paper_2605_24793_gb300.arbitrator --k 25 --batch 1 --context 4096
"""
from __future__ import annotations

import argparse
import json

import numpy as np
import torch

from . import cospec as C
from . import workload as W

# Qwen3-4B-like backbone (the paper's draft for Qwen3-32B): 36 layers, 32 query /
# 8 KV heads, head_dim 128; the vocabulary plays no part here.
BACKBONE = dict(layers=36, hidden=2560, q_heads=32, kv_heads=8, head_dim=128)


def region_config(k: int, batch: int, context: int, layers: int) -> W.RoundConfig:
    """A workload whose block is the arbitrator's region: 2K+3 rows."""
    bb = dict(BACKBONE)
    bb["layers"] = layers
    return W.RoundConfig(f"arbitrator_k{k}_b{batch}_c{context}", 5, batch=batch, ctx_lo=context,
                         ctx_hi=context, k=2 * k + 2, vocab=1024, mlp_hidden=64, mismatch_rate=0.3,
                         mismatch_topk=8, shuffled_pages=batch > 1, **bb)


def time_region_attention(cfg: W.RoundConfig, steps: int = 50, warmup: int = 5) -> dict:
    inp = W.make_round_inputs(cfg, device="cuda")
    q, kb, vb = inp["q"], inp["k_blk"], inp["v_blk"]
    kp, vp = inp["k_pages"], inp["v_pages"]
    out = torch.empty_like(q[0])
    max_ctx = int(np.max(inp["ctx_len_np"]))

    def layers():
        for l in range(cfg.layers):
            pl = 0 if kp.shape[0] == 1 else l
            C.verify_attn(q[l], kb[l], vb[l], kp[pl], vp[pl], inp["page_table"], inp["ctx_len"], out,
                          max_ctx, kv_stable=l > 0, block_full=True)

    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        layers()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        layers()
    for _ in range(warmup):
        g.replay()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(s)
    with torch.cuda.stream(s):
        for _ in range(steps):
            g.replay()
    e1.record(s)
    e1.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / (steps * cfg.layers)
    ctx = inp["ctx_len_np"].astype(np.int64)
    kv_bytes = float(ctx.sum()) * 2 * cfg.kv_heads * cfg.head_dim * 2
    blk_bytes = 2.0 * cfg.batch * cfg.rows * (cfg.kv_heads + cfg.q_heads) * cfg.head_dim * 2
    kernel, splits = C.verify_attn_plan(q[0], kp[0], inp["page_table"], max_ctx)
    return {"workload": cfg.name, "region_rows": cfg.rows, "batch": cfg.batch,
            "context": int(ctx.max()), "layers": cfg.layers, "us_per_layer": us,
            "gbs": (kv_bytes + blk_bytes) / (us * 1e-6) / 1e9,
            "kernel": C.ATTN_KERNEL_NAMES[kernel], "splits": splits,
            "device_error": C.get_device_error()}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--k", type=int, nargs="+", default=[7, 25])
    ap.add_argument("--batch", type=int, nargs="+", default=[1, 16])
    ap.add_argument("--context", type=int, default=4096)
    ap.add_argument("--layers", type=int, default=BACKBONE["layers"])
    args = ap.parse_args()
    from . import build as B
    C.load_library(B.build())
    for k in args.k:
        for b in args.batch:
            res = time_region_attention(region_config(k, b, args.context, args.layers))
            print(json.dumps(res), flush=True)
            torch.cuda.empty_cache()


if __name__ == "__main__":
    main()
