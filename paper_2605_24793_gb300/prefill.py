"""Causal prefill of a context through the verify-attention call, in chunks.

The arbitrator reads q = [c, SEP, draft block, SEP, target block, SEP] with a
hybrid mask whose context part is causal (Sec. 3.3); decoding round after
round that context is cached, so a request prefills it once and every round
then attends its region with COSPEC_ATTN_BLOCK_FULL.  This driver builds the
cache: a chunk of up to 32 context tokens is a block whose rows attend
causally to the committed prefix and to the chunk's earlier rows
(cospec_verify_attn), after which all of its rows are committed into the
paged cache of every layer (cospec_accept_commit with every drafted token
equal to the target's, so the accepted length is the chunk's length).  Chunk
after chunk this is exactly causal self-attention over the context.  It uses
only the round's own calls; it is a functional path for a request's prefill,
not a tuned prefill kernel.

  python -m paper_2605_24793_gb300.prefill --context 4096 --layers 36
"""
from __future__ import annotations

import argparse
import json

import numpy as np
import torch

from . import cospec as cs

CHUNK = 32          # rows per chunk: the commit call accepts at most 31 drafted tokens + 1


class ChunkedPrefill:
    """Prefill of B contexts of C tokens each into a paged cache of L layers
    (page size 16, each sequence's pages contiguous in the pool)."""

    def __init__(self, layers: int, batch: int, context: int, q_heads: int, kv_heads: int,
                 head_dim: int, chunk: int = CHUNK, extra_tokens: int = 0, device="cuda"):
        if not 1 <= chunk <= CHUNK:
            raise ValueError(f"chunk must be in [1, {CHUNK}]")
        self.L, self.B, self.C = layers, batch, context
        self.Hq, self.Hkv, self.D, self.chunk = q_heads, kv_heads, head_dim, chunk
        P = 16
        per_seq = (context + extra_tokens + chunk + P - 1) // P
        dev = torch.device(device)
        self.k_pages = torch.zeros((layers, batch * per_seq, kv_heads, P, head_dim),
                                   dtype=torch.bfloat16, device=dev)
        self.v_pages = torch.zeros_like(self.k_pages)
        table = np.arange(batch * per_seq, dtype=np.int32).reshape(batch, per_seq)
        self.page_table = torch.from_numpy(table).to(dev)
        self.ctx_len = torch.zeros(batch, dtype=torch.int32, device=dev)
        self.max_ctx = context

    def run(self, q: torch.Tensor, k: torch.Tensor, v: torch.Tensor) -> torch.Tensor:
        """q [L, B, C, Hq, D], k / v [L, B, C, Hkv, D] (bf16): the context's
        per-layer projections.  Commits the context's K/V into the cache and
        returns the attention output [L, B, C, Hq, D]."""
        L, B, C = self.L, self.B, self.C
        if tuple(q.shape) != (L, B, C, self.Hq, self.D) or tuple(k.shape) != (L, B, C, self.Hkv, self.D):
            raise ValueError("q / k / v must be [L, B, C, H, D] with the prefill's shape")
        dev = q.device
        out = torch.empty_like(q)
        self.ctx_len.zero_()
        for c0 in range(0, C, self.chunk):
            R = min(self.chunk, C - c0)
            qc = q[:, :, c0:c0 + R].contiguous()
            kc = k[:, :, c0:c0 + R].contiguous()
            vc = v[:, :, c0:c0 + R].contiguous()
            oc = torch.empty((B, R, self.Hq, self.D), dtype=torch.bfloat16, device=dev)
            for l in range(L):
                cs.verify_attn(qc[l], kc[l], vc[l], self.k_pages[l], self.v_pages[l],
                              self.page_table, self.ctx_len, oc, self.max_ctx)
                out[l, :, c0:c0 + R] = oc
            # every row is kept: the "drafts" equal the "targets" (all zeros)
            draft = torch.zeros((B, R - 1), dtype=torch.int32, device=dev)
            tokens = torch.zeros(B * R, dtype=torch.int32, device=dev)
            accept = torch.ones((B, R - 1), dtype=torch.uint8, device=dev)
            s = torch.empty(B, dtype=torch.int32, device=dev)
            emitted = torch.empty((B, R), dtype=torch.int32, device=dev)
            cs.accept_commit(draft, tokens, accept, kc, vc, self.k_pages, self.v_pages,
                            self.page_table, self.ctx_len, s, emitted)
        return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--context", type=int, default=4096)
    ap.add_argument("--layers", type=int, default=36)
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--q-heads", type=int, default=32)
    ap.add_argument("--kv-heads", type=int, default=8)
    ap.add_argument("--head-dim", type=int, default=128)
    args = ap.parse_args()
    from . import build as B
    cs.load_library(B.build())
    g = torch.Generator(device="cuda")
    g.manual_seed(5000)
    L, Bt, T = args.layers, args.batch, args.context
    q = torch.empty((L, Bt, T, args.q_heads, args.head_dim), dtype=torch.bfloat16, device="cuda")
    k = torch.empty((L, Bt, T, args.kv_heads, args.head_dim), dtype=torch.bfloat16, device="cuda")
    v = torch.empty_like(k)
    for t in (q, k, v):
        t.normal_(0.0, 1.0, generator=g)
    pf = ChunkedPrefill(L, Bt, T, args.q_heads, args.kv_heads, args.head_dim)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        pf.run(q, k, v)                  # warm-up (also fills the library's plan caches)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    pf.run(q, k, v)
    e1.record()
    e1.synchronize()
    eager_ms = e0.elapsed_time(e1)
    # the same launches replayed from one CUDA graph: the device-side cost
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        pf.run(q, k, v)
    graph.replay()
    torch.cuda.synchronize()
    e0.record()
    graph.replay()
    e1.record()
    e1.synchronize()
    graph_ms = e0.elapsed_time(e1)
    launches = -(-T // CHUNK) * (L + 1)
    # cached K/V the verify calls read: chunk at c0 reads c0 committed positions
    kv_bytes = L * Bt * sum(range(0, T, CHUNK)) * args.kv_heads * args.head_dim * 2 * 2
    print(json.dumps({"context": T, "layers": L, "batch": Bt, "chunk": CHUNK,
                      "verify_and_commit_calls": launches, "eager_ms": eager_ms,
                      "cached_kv_gb_read": kv_bytes / 1e9,
                      "graph_kv_gbs": kv_bytes / (graph_ms * 1e-3) / 1e9,
                      "graph_ms": graph_ms, "tokens_per_s_eager": Bt * T / (eager_ms * 1e-3),
                      "tokens_per_s_graph": Bt * T / (graph_ms * 1e-3),
                      "device_error": cs.get_device_error()}))


if __name__ == "__main__":
    main()
