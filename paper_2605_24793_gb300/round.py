"""One CoSpec verify/arbitrate round on the device (App. F, Inference
Procedure: verify the drafted block, arbitrate mismatches, stop at the first
rejection, commit), built from the four C-ABI calls.

``VerifyRound`` owns the scratch buffers of one workload and launches
L x verify_attn, the fused LM head, arbitration and accept/commit on one
stream.  Nothing in a round synchronises with the host, so a round can be
captured once into a CUDA graph and replayed (``capture`` / ``replay``).
"""
from __future__ import annotations

from typing import Dict, Optional

import numpy as np
import torch

from . import cospec as C


class VerifyRound:
    def __init__(self, inputs: Dict[str, object], draft: np.ndarray, lam: float = 0.6,
                 mode: int = C.POLICY_MLP, keep_attn: bool = False, max_ctx: Optional[int] = None,
                 temperature: Optional[float] = None, seed: int = 0,
                 sps_q: Optional[torch.Tensor] = None):
        """``temperature`` None: greedy target candidates (argmax).  Otherwise
        stochastic decoding (Sec. 3.1): candidates are Gumbel-max samples at
        that temperature, keyed by the device scalar ``self.seed``, which a
        caller may rewrite between replays of a captured round.

        ``sps_q`` [B, K, V] fp32 (the draft's distributions) turns the round
        into the exact-match baseline with speculative sampling at
        ``temperature`` (1 when None): the LM head writes the scaled logits,
        the acceptance step replaces arbitration, and the commit takes its
        tokens."""
        cfg = inputs["cfg"]
        self.cfg = cfg
        self.inp = inputs
        dev = inputs["q"].device
        B, K, R, L = cfg.batch, cfg.k, cfg.rows, cfg.layers
        self.lam, self.mode = float(lam), int(mode)
        self.q, self.k_blk, self.v_blk = inputs["q"], inputs["k_blk"], inputs["v_blk"]
        self.k_pages, self.v_pages = inputs["k_pages"], inputs["v_pages"]
        self.page_table, self.ctx_len = inputs["page_table"], inputs["ctx_len"]
        self.hidden, self.w = inputs["hidden"], inputs["w"]
        self.ctx0 = self.ctx_len.clone()
        self.max_ctx = int(max_ctx if max_ctx is not None else np.max(inputs["ctx_len_np"]))
        dfr = np.full((B, R), -1, dtype=np.int32)
        dfr[:, :K] = draft
        self.draft = torch.from_numpy(np.ascontiguousarray(draft, dtype=np.int32)).to(dev)
        self.draft_for_row = torch.from_numpy(dfr.reshape(-1)).to(dev)
        w1, b1, w2, b2 = inputs["mlp"]
        self.w1, self.b1, self.w2 = w1.to(dev), b1.to(dev), w2.to(dev)
        self.b2 = float(b2)
        self.dims = C.attn_dims(self.q[0], self.k_pages[0], self.page_table)
        M = B * R
        self.ws_lm = C.new_lmhead_workspace(M, cfg.hidden, cfg.vocab, dev)
        nout = L if keep_attn else 1
        self.attn_out = torch.empty((nout,) + tuple(self.q.shape[1:]), dtype=torch.bfloat16, device=dev)
        self.argmax = torch.empty(M, dtype=torch.int32, device=dev)
        self.stats = torch.empty((M, 5), dtype=torch.float32, device=dev)
        self.p = torch.empty((B, K), dtype=torch.float32, device=dev)
        self.accept = torch.empty((B, K), dtype=torch.uint8, device=dev)
        self.accept_len = torch.empty(B, dtype=torch.int32, device=dev)
        self.emitted = torch.empty((B, R), dtype=torch.int32, device=dev)
        self.temperature = None if temperature is None else float(temperature)
        self.seed = torch.tensor([int(seed)], dtype=torch.int64, device=dev)
        self.sps = sps_q is not None
        if self.sps:
            if self.temperature is None:
                self.temperature = 1.0
            if tuple(sps_q.shape) != (B, K, cfg.vocab):
                raise ValueError("sps_q must be [B, K, V]")
            self.draft_q = sps_q
            self.logits = torch.empty((M, cfg.vocab), dtype=torch.float32, device=dev)
            self.target = torch.empty(M, dtype=torch.int32, device=dev)
            self.ratio = torch.empty((B, K), dtype=torch.float32, device=dev)
            self.ws_sps = C.new_sps_workspace(B, dev)
        self.graph: Optional[torch.cuda.CUDAGraph] = None
        self.launches_per_round = self._count_launches()

    def pack_step_io(self) -> None:
        """Place the inputs a serving step receives from the host (Q and the
        block K/V of every layer, the hidden rows, the draft ids and, for
        speculative sampling, the draft's distributions) in one device
        buffer ``io_in`` and the results it hands back (accepted lengths,
        emitted tokens) in another, ``io_out``, so that a step moves each with
        a single copy.  The tensors become views of the buffers (each slice
        256-byte aligned); call before capturing a graph."""
        dev = self.q.device
        names = ("q", "k_blk", "v_blk", "hidden", "draft", "draft_for_row")
        if self.sps:
            names += ("draft_q",)            # the draft's distributions come with the drafts
        tensors = [getattr(self, n) for n in names]
        sizes = [t.numel() * t.element_size() for t in tensors]
        offs, total = [], 0
        for n in sizes:
            offs.append(total)
            total += (n + 255) // 256 * 256
        self.io_in = torch.empty(total, dtype=torch.uint8, device=dev)
        for name, t, off, n in zip(names, tensors, offs, sizes):
            view = self.io_in[off:off + n].view(t.dtype).view(t.shape)
            view.copy_(t)
            setattr(self, name, view)
        B, R = self.cfg.batch, self.cfg.rows
        lead = (B + 63) // 64 * 64                  # accepted lengths, then 256-byte aligned tokens
        self.io_out = torch.zeros(lead + B * R, dtype=torch.int32, device=dev)
        self.accept_len = self.io_out[:B]
        self.emitted = self.io_out[lead:].view(B, R)
        self.dims = C.attn_dims(self.q[0], self.k_pages[0], self.page_table)

    def _count_launches(self) -> int:
        """Kernels one round launches (attention: 1 per layer; LM head: a main
        and a merge kernel per 256-row pass; arbitration: 1 when K > 0;
        accept/commit: commit + scan)."""
        cfg = self.cfg
        passes = (cfg.m_rows + 255) // 256
        decide = 2 if self.sps else (1 if cfg.k > 0 else 0)
        return cfg.layers + 2 * passes + decide + 2

    def restore_context(self) -> None:
        """Reset ctx_len to the round's starting context (device copy)."""
        self.ctx_len.copy_(self.ctx0, non_blocking=True)

    def attention(self, l: int, kv_stable: Optional[bool] = None) -> torch.Tensor:
        """Layer l's verify attention.  ``kv_stable`` (default: l > 0) lets the
        launch stream its cache before the previous kernel ends."""
        pl = 0 if self.k_pages.shape[0] == 1 else l
        out = self.attn_out[l if self.attn_out.shape[0] > 1 else 0]
        # Layers after the first follow another attention launch, which writes
        # neither the context lengths, the page table nor the cached pages.
        return C.verify_attn(self.q[l], self.k_blk[l], self.v_blk[l], self.k_pages[pl],
                             self.v_pages[pl], self.page_table, self.ctx_len, out, self.max_ctx,
                             kv_stable=(l > 0) if kv_stable is None else kv_stable)

    def lmhead(self):
        if self.sps:
            return C.lmhead_logits_features(self.hidden, self.w, self.draft_for_row,
                                            self.temperature, self.argmax, self.stats,
                                            self.logits, self.ws_lm)
        if self.temperature is not None:
            return C.lmhead_sample_features(self.hidden, self.w, self.draft_for_row,
                                            self.temperature, self.seed, self.argmax, self.stats,
                                            self.ws_lm)
        return C.lmhead_argmax_features(self.hidden, self.w, self.draft_for_row, self.argmax,
                                        self.stats, self.ws_lm)

    def arbitrate(self):
        cfg = self.cfg
        if self.sps:
            return C.sps_accept(self.draft, self.stats, self.logits, self.draft_q, self.seed,
                                self.target, self.accept, self.ratio, self.ws_sps)
        return C.arbitrate(self.draft, self.argmax.view(cfg.batch, cfg.rows),
                           self.stats.view(cfg.batch, cfg.rows, 5), self.w1, self.b1, self.w2,
                           self.b2, self.lam, self.mode, self.p, self.accept)

    def commit(self):
        tokens = self.target if self.sps else self.argmax
        return C.accept_commit(self.draft, tokens, self.accept, self.k_blk, self.v_blk,
                               self.k_pages, self.v_pages, self.page_table, self.ctx_len,
                               self.accept_len, self.emitted)

    def run(self, restore: bool = True) -> None:
        """Queue one full round on the current stream."""
        if restore:
            self.restore_context()
        for l in range(self.cfg.layers):
            self.attention(l)
        self.lmhead()
        if self.cfg.k > 0 or self.sps:
            self.arbitrate()
        self.commit()

    def capture(self) -> torch.cuda.CUDAGraph:
        """Capture one round (with the context restore) into a CUDA graph."""
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.run()          # warm-up: kernel attributes and tensor maps settle
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run()
        self.graph = g
        return g

    def replay(self) -> None:
        if self.graph is None:
            self.capture()
        self.graph.replay()
