"""Causal prefill of a context through the round's own calls.

The arbitrator reads q = [c, SEP, draft block, SEP, target block, SEP] with a
hybrid mask whose context part is causal (Sec. 3.3); decoding round after
round that context is cached, so a request prefills it once and every round
then attends its region with COSPEC_ATTN_BLOCK_FULL.  Both drivers here build
that cache and the context's own attention output, cutting the context into
chunks of up to 32 tokens; a chunk is a block whose rows attend causally to
the cached positions before it and to the chunk's earlier rows
(cospec_verify_attn), and its K/V rows are committed into the paged cache of
every layer (cospec_accept_commit with every drafted token equal to the
target's, so the accepted length is the chunk's length).

* ``BlockPrefill`` commits every chunk's K/V first, in one call whose
  "sequences" are the chunks (each with its sequence's page-table row and its
  start as context length), and then attends all chunks of a layer in one
  verify-attention launch: chunk k sees exactly the positions before it.
* ``ChunkedPrefill`` walks the chunks one after another (attention of every
  layer, then the commit), the plain reference for the block driver.

  python -m paper_2605_24793_gb300.prefill --context 4096 --layers 36
"""
from __future__ import annotations

import argparse
import json

import numpy as np
import torch

from . import cospec as cs

CHUNK = 32          # rows per chunk: the commit call accepts at most 31 drafted tokens + 1


class BlockPrefill:
    """Prefill of B contexts of C tokens each into a paged cache of L layers
    (page size 16, each sequence's pages contiguous in the pool), every chunk
    of a layer attended in one launch."""

    def __init__(self, layers: int, batch: int, context: int, q_heads: int, kv_heads: int,
                 head_dim: int, chunk: int = CHUNK, extra_tokens: int = 0, device="cuda"):
        if not 1 <= chunk <= CHUNK:
            raise ValueError(f"chunk must be in [1, {CHUNK}]")
        self.L, self.B, self.C = layers, batch, context
        self.Hq, self.Hkv, self.D, self.chunk = q_heads, kv_heads, head_dim, chunk
        self.nck = max(1, -(-context // chunk))          # chunks per sequence
        P = 16
        # room for the padding rows of a ragged last chunk (never committed)
        per_seq = (self.nck * chunk + extra_tokens + P - 1) // P
        dev = torch.device(device)
        self.k_pages = torch.zeros((layers, batch * per_seq, kv_heads, P, head_dim),
                                   dtype=torch.bfloat16, device=dev)
        self.v_pages = torch.zeros_like(self.k_pages)
        table = np.arange(batch * per_seq, dtype=np.int32).reshape(batch, per_seq)
        self.page_table = torch.from_numpy(table).to(dev)
        self.ctx_len = torch.zeros(batch, dtype=torch.int32, device=dev)
        self.max_ctx = context
        # The chunk "sequences", latest chunks first (a batch this large is
        # attended in index order): b' = i * B + b is chunk nck - 1 - i of
        # sequence b, starts there, reads its sequence's pages and keeps its
        # valid rows (a ragged last chunk rejects the draft at its first
        # padding row, so the scan stops there).
        B2, R = batch * self.nck, chunk
        self.table2 = torch.from_numpy(np.tile(table, (self.nck, 1))).to(dev)
        starts = np.repeat((self.nck - 1 - np.arange(self.nck, dtype=np.int32)) * chunk, batch)
        self.start = torch.from_numpy(starts).to(dev)
        self.ctx2 = torch.empty(B2, dtype=torch.int32, device=dev)
        valid = np.minimum(chunk, context - starts)
        draft = np.zeros((B2, R - 1), dtype=np.int32)
        accept = np.ones((B2, R - 1), dtype=np.uint8)
        for i, v in enumerate(valid):
            if v < R:                    # position v mismatches and is rejected: s = v
                draft[i, v - 1] = 1
                accept[i, v - 1] = 0
        self.draft = torch.from_numpy(draft).to(dev)
        self.accept = torch.from_numpy(accept).to(dev)
        self.tokens = torch.zeros(B2 * R, dtype=torch.int32, device=dev)
        self.s = torch.empty(B2, dtype=torch.int32, device=dev)
        self.emitted = torch.empty((B2, R), dtype=torch.int32, device=dev)
        # projections in chunk-sequence order: [L, nck, B, chunk, H, D]
        self.qp = torch.zeros((layers, self.nck, batch, chunk, q_heads, head_dim),
                              dtype=torch.bfloat16, device=dev)
        self.kp = torch.zeros((layers, self.nck, batch, chunk, kv_heads, head_dim),
                              dtype=torch.bfloat16, device=dev)
        self.vp = torch.zeros_like(self.kp)
        self.outp = torch.empty_like(self.qp)

    def load(self, q: torch.Tensor, k: torch.Tensor, v: torch.Tensor) -> None:
        """q [L, B, C, Hq, D], k / v [L, B, C, Hkv, D] (bf16): the context's
        per-layer projections, placed into the chunk-padded buffers."""
        L, B, C = self.L, self.B, self.C
        if tuple(q.shape) != (L, B, C, self.Hq, self.D) or tuple(k.shape) != (L, B, C, self.Hkv, self.D):
            raise ValueError("q / k / v must be [L, B, C, H, D] with the prefill's shape")
        for c in range(self.nck):
            i, c0 = self.nck - 1 - c, c * self.chunk
            n = min(self.chunk, C - c0)
            self.qp[:, i, :, :n].copy_(q[:, :, c0:c0 + n])
            self.kp[:, i, :, :n].copy_(k[:, :, c0:c0 + n])
            self.vp[:, i, :, :n].copy_(v[:, :, c0:c0 + n])

    def step(self) -> None:
        """The prefill itself, from the loaded buffers: one commit, then one
        attention launch per layer (all launches, no host synchronisation)."""
        L, B2, R = self.L, self.B * self.nck, self.chunk
        kc = self.kp.view(L, B2, R, self.Hkv, self.D)
        vc = self.vp.view(L, B2, R, self.Hkv, self.D)
        self.ctx2.copy_(self.start)
        cs.accept_commit(self.draft, self.tokens, self.accept, kc, vc, self.k_pages, self.v_pages,
                         self.table2, self.ctx2, self.s, self.emitted)
        qc = self.qp.view(L, B2, R, self.Hq, self.D)
        oc = self.outp.view(L, B2, R, self.Hq, self.D)
        for l in range(L):
            cs.verify_attn(qc[l], kc[l], vc[l], self.k_pages[l], self.v_pages[l], self.table2,
                           self.start, oc[l], self.max_ctx)
        self.ctx_len.fill_(self.C)

    def run(self, q: torch.Tensor, k: torch.Tensor, v: torch.Tensor) -> torch.Tensor:
        """Commits the context's K/V into the cache and returns the attention
        output [L, B, C, Hq, D]."""
        self.load(q, k, v)
        self.step()
        out = torch.empty_like(q)
        for c in range(self.nck):
            i, c0 = self.nck - 1 - c, c * self.chunk
            n = min(self.chunk, self.C - c0)
            out[:, :, c0:c0 + n] = self.outp[:, i, :, :n]
        return out


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
    ap.add_argument("--method", choices=["block", "chunked"], default="block")
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
    if args.method == "block":
        pf = BlockPrefill(L, Bt, T, args.q_heads, args.kv_heads, args.head_dim)
        pf.load(q, k, v)                 # the projections, in the chunk-padded layout
        work = pf.step
        launches = 1 + L
    else:
        pf = ChunkedPrefill(L, Bt, T, args.q_heads, args.kv_heads, args.head_dim)
        work = lambda: pf.run(q, k, v)
        launches = -(-T // CHUNK) * (L + 1)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        work()                           # warm-up (also fills the library's plan caches)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    work()
    e1.record()
    e1.synchronize()
    eager_ms = e0.elapsed_time(e1)
    # the same launches replayed from one CUDA graph: the device-side cost
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        work()
    graph.replay()
    torch.cuda.synchronize()
    e0.record()
    graph.replay()
    e1.record()
    e1.synchronize()
    graph_ms = e0.elapsed_time(e1)
    # cached K/V the verify calls read: chunk at c0 reads c0 committed positions
    kv_bytes = L * Bt * sum(range(0, T, CHUNK)) * args.kv_heads * args.head_dim * 2 * 2
    # attention flops: every query head's causal row over the context
    flops = 4.0 * L * Bt * args.q_heads * args.head_dim * T * (T + 1) / 2
    print(json.dumps({"method": args.method, "context": T, "layers": L, "batch": Bt,
                      "chunk": CHUNK, "launches": launches, "eager_ms": eager_ms,
                      "graph_ms": graph_ms, "cached_kv_gb_read": kv_bytes / 1e9,
                      "attention_tflops": flops / (graph_ms * 1e-3) / 1e12,
                      "tokens_per_s_eager": Bt * T / (eager_ms * 1e-3),
                      "tokens_per_s_graph": Bt * T / (graph_ms * 1e-3),
                      "device_error": cs.get_device_error()}))


if __name__ == "__main__":
    main()
