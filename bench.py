"""Benchmark of one CoSpec verify/arbitrate round on GB300.

A step is one full round -- L x verify attention, the fused LM head,
arbitration, accept/commit (with the context restore that lets every step
verify the same block) -- over one batch of the workload, replayed from a
CUDA graph.  Metric: verified block-tokens/s = batch * (K+1) / round time.
The default workload is the largest one: a Llama-3-8B-shaped target, batch
64, contexts U[8192, 32768], K = 7, 30 % draft mismatches, 32 layers.

  python bench.py [--config NAME] [--steps K] [--warmup W] [--gpus N]
  python bench.py --impl reference      # the CPU oracle on a bounded sample
  python bench.py --sweep               # the Llama-3-8B batch-64 points:
                                        # K in {3,5,7} x mismatch 10/30/60 %

One JSON line is printed by rank 0 (one per point with --sweep).  Under
torchrun every rank runs an independent replica of the workload (the round
shards by sequence and needs no collective); the host-side max over ranks of
the timed region gives the whole-job throughput.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2605_24793_gb300 import workload as W  # noqa: E402

METRIC = "verified block-tokens/s (device-timed)"
UNIT = "block-tokens/s"
DEFAULT_CONFIG = "llama3_8b_b64_k7_mm30"
SWEEP = [f"llama3_8b_b64_k{k}_mm{r}" for k in (3, 5, 7) for r in (10, 30, 60)]
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def peaks():
    try:
        with open(PEAKS_FILE) as fh:
            p = json.load(fh)
        return p, "measured"
    except (OSError, ValueError):
        return FALLBACK_PEAKS, "fallback"


# ------------------------------------------------------------------ work accounting
def attention_bytes(cfg, ctx: np.ndarray) -> float:
    """Algorithmic HBM bytes of one verify-attention launch: the cached K and
    V of every sequence (2 * Hkv * D * 2 bytes per position), the block K/V,
    Q and the output."""
    kv = float(np.sum(ctx.astype(np.int64))) * 2 * cfg.kv_heads * cfg.head_dim * 2
    blk = 2.0 * cfg.batch * cfg.rows * cfg.kv_heads * cfg.head_dim * 2
    qo = 2.0 * cfg.batch * cfg.rows * cfg.q_heads * cfg.head_dim * 2
    return kv + blk + qo


def attention_flops(cfg, ctx: np.ndarray) -> float:
    return 4.0 * cfg.rows * cfg.q_heads * cfg.head_dim * float(np.sum(ctx + cfg.rows))


def lmhead_bytes(cfg, logits: bool = False) -> float:
    """W streamed once plus the hidden rows and the per-row outputs (and the
    M x V fp32 logits when the LM head writes them, speculative sampling)."""
    b = 2.0 * cfg.vocab * cfg.hidden + 2.0 * cfg.m_rows * cfg.hidden + 24.0 * cfg.m_rows
    return b + (4.0 * cfg.m_rows * cfg.vocab if logits else 0.0)


def lmhead_flops(cfg) -> float:
    return 2.0 * cfg.m_rows * cfg.hidden * cfg.vocab


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.path = None
        self.gpu = gpu_index

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as fh:
            for line in fh:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": reasons,
                "samples": len(rows),
                "power_w_max": max((float(r[3]) for r in rows
                                    if r[3].replace(".", "").isdigit()), default=None)}


def throttled(clk: dict) -> bool:
    """A clock record that invalidates a timing: hw_slowdown,
    hw_thermal_slowdown or sw_thermal_slowdown active, or a median SM clock
    under 85 % of its maximum with no reason given (a leftover clock lock).
    sw_power_cap alone is kept."""
    reasons = set(clk.get("reasons") or [])
    if reasons & {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}:
        return True
    sm, smax = clk.get("sm_mhz"), clk.get("sm_max_mhz")
    return bool(sm and smax and not reasons and sm < 0.85 * smax)


# ------------------------------------------------------------------ drafts
def gpu_drafts(cfg, inp, with_top1: bool = False):
    """Draft ids for the benchmark, synthesised from the target's own top-8
    (fp32 logits of the bf16 operands, computed once before timing).  With
    ``with_top1`` also each row's fp32 top-1 id and its margin to the top-2
    logit, for the round's self-check."""
    h = inp["hidden"].float()
    ranked, margin = [], []
    for r0 in range(0, h.shape[0], 64):
        logits = h[r0:r0 + 64] @ inp["w"].float().T
        top = torch.topk(logits, 8, dim=1)
        ranked.append(top.indices.cpu())
        margin.append((top.values[:, 0] - top.values[:, 1]).cpu())
        del logits, top
    ranked = torch.cat(ranked).numpy().reshape(cfg.batch, cfg.rows, 8)
    draft = W.synth_drafts(cfg, ranked)
    if with_top1:
        return draft, ranked[..., 0].reshape(-1), torch.cat(margin).numpy()
    return draft


def self_check(cfg, rnd, top1, margin) -> dict:
    """The warm-up round checked on the host against what fixes it without
    the oracle: the LM head's argmax against the fp32 GEMM's top-1 (rows whose
    fp32 top-1/top-2 margin is below 1e-3 are near ties and may differ), and
    the accepted lengths and emitted tokens against the prefix rule (Eq. 15)
    applied to the round's own drafts, argmax and accept decisions: s is the
    first draft position whose token differs from the target's and was not
    accepted (K + 1 if none), the emitted tokens are the drafts before it and
    then the target's token at it."""
    am = rnd.argmax.cpu().numpy()
    draft = rnd.draft.cpu().numpy()
    acc = rnd.accept.cpu().numpy()
    s_gpu = rnd.accept_len.cpu().numpy()
    em = rnd.emitted.cpu().numpy()
    B, K, R = cfg.batch, cfg.k, cfg.rows
    amr = am.reshape(B, R)
    tie = margin < 1e-3
    diff = am != top1
    follows = True
    for b in range(B):
        sb = K + 1
        for i in range(1, K + 1):
            if draft[b, i - 1] != amr[b, i - 1] and acc[b, i - 1] == 0:
                sb = i
                break
        want = list(draft[b, :sb - 1]) + [amr[b, sb - 1]] + [-1] * (R - sb)
        follows &= int(s_gpu[b]) == sb and em[b].tolist() == [int(v) for v in want]
    return {"argmax_rows": int(am.size), "argmax_equal_fp32_top1": int((~diff).sum()),
            "argmax_differ_outside_near_ties": int((diff & ~tie).sum()),
            "near_ties": int(tie.sum()), "accepted_len_and_tokens_follow_eq15": bool(follows)}


def mismatch_stats(cfg, rnd) -> dict:
    """How the round's arbitration treated the draft/target mismatches
    (Sec. 3.3): positions i in 1..K whose draft token differs from the
    target's prediction, how many of them the policy accepted (a_i = 1),
    and how many of those accepted ones lie before the round's first
    rejection, i.e. reached the emitted block."""
    if cfg.k == 0:
        return {"mismatch_positions": 0, "mismatches_accepted": 0, "accepted_mismatch_fraction": None,
                "accepted_mismatches_emitted": 0}
    R = cfg.rows
    am = rnd.argmax.cpu().numpy().reshape(cfg.batch, R)[:, :cfg.k]
    draft = rnd.draft.cpu().numpy()
    acc = rnd.accept.cpu().numpy().astype(bool)
    s = rnd.accept_len.cpu().numpy()
    mism = draft != am
    kept = mism & acc
    before = np.arange(1, cfg.k + 1)[None, :] < s[:, None]      # positions i < s_b
    n = int(mism.sum())
    return {"mismatch_positions": n, "mismatches_accepted": int(kept.sum()),
            "accepted_mismatch_fraction": (float(kept.sum()) / n) if n else None,
            "accepted_mismatches_emitted": int((kept & before).sum())}


# ------------------------------------------------------------------ CPU oracle sample
class OracleSampler:
    """Times the CPU oracle on a bounded, seeded sample of one round.

    A round is L x B (layer, sequence) attention blocks and their KV commits,
    the LM head over all M = B * R rows, and the batch's arbitration and
    scan.  One sample step runs the oracle's verify attention and KV commit
    of one (layer, sequence) pair from a seeded list, one of L vocabulary
    slices of the LM head (with its statistics) for all M rows, and the
    arbitration and acceptance scan of the whole batch.  The full round is
    extrapolated, not run: the pairs' time per attended key position times
    the round's key positions (L x sum_b (C_b + R)), plus L x the mean slice
    time, plus the mean arbitration/scan time."""

    def __init__(self, cfg, inp, draft, pairs: int = 256, seed: int = 0):
        from oracle import cospec_oracle as O
        self.O = O
        self.cfg = cfg
        self.inp = inp
        self.draft = draft
        self.ctx = inp["ctx_len_np"].astype(np.int64)
        self.table = inp["page_table_np"]
        self.hidden = inp["hidden"].cpu()
        self.mlp = inp["mlp"]
        rng = np.random.default_rng(seed)
        self.pairs = list(zip(rng.integers(0, cfg.layers, pairs).tolist(),
                              rng.integers(0, cfg.batch, pairs).tolist()))
        self.n_slices = cfg.layers
        self.keypos_round = float(cfg.layers * np.sum(self.ctx + cfg.rows))
        self.rec = []            # per step: (pair seconds, pair key positions, slice s, tail s)
        self._held = None

    def _pair(self, l, b):
        """Host copies of layer l's inputs for sequence b (pages relabelled 0..n-1)."""
        if self._held is not None and self._held[0] == (l, b):
            return self._held[1]
        inp = self.inp
        row = self.table[b]
        pages = row[row >= 0].astype(np.int64)
        lp = 0 if inp["k_pages"].shape[0] == 1 else l
        idx = torch.from_numpy(pages).to(inp["k_pages"].device)
        d = dict(q=inp["q"][l, b:b + 1].cpu(), kb=inp["k_blk"][l, b:b + 1].cpu(),
                 vb=inp["v_blk"][l, b:b + 1].cpu(),
                 kp=inp["k_pages"][lp].index_select(0, idx).cpu(),
                 vp=inp["v_pages"][lp].index_select(0, idx).cpu(),
                 table=np.arange(len(pages))[None, :])
        self._held = ((l, b), d)
        return d

    def step(self, i):
        O, cfg = self.O, self.cfg
        l, b = self.pairs[i % len(self.pairs)]
        sl = i % self.n_slices
        d = self._pair(l, b)                                  # host copies: not timed
        V = cfg.vocab
        v0, v1 = (V * sl) // self.n_slices, (V * (sl + 1)) // self.n_slices
        wslice = self.inp["w"][v0:v1].cpu()
        P = cfg.page_size
        t0 = time.perf_counter()
        O.verify_attention(d["q"], d["kb"], d["vb"], d["kp"], d["vp"], d["table"],
                           self.ctx[b:b + 1], P)
        t1 = time.perf_counter()
        x = O.lmhead_logits(self.hidden, wslice)
        dfr = np.full((cfg.batch, cfg.rows), -1)
        dfr[:, :cfg.k] = self.draft
        dfr = np.where((dfr >= v0) & (dfr < v1), dfr - v0, -1)
        am, st = O.row_stats(x, dfr.reshape(-1))
        am = am.reshape(cfg.batch, cfg.rows) + v0
        st = st.reshape(cfg.batch, cfg.rows, 5)
        t2 = time.perf_counter()
        w1, b1, w2, b2 = self.mlp
        _, a = O.arbitrate(self.draft, am, st, w1, b1, w2, b2, cfg.lam)
        s, _ = O.accept_scan(self.draft, am, a)
        t3 = time.perf_counter()
        O.commit_kv(d["kb"].view(torch.int16).numpy()[None], d["vb"].view(torch.int16).numpy()[None],
                    d["kp"].view(torch.int16).numpy()[None], d["vp"].view(torch.int16).numpy()[None],
                    d["table"], self.ctx[b:b + 1], s[b:b + 1], P)
        t4 = time.perf_counter()
        self.rec.append(((t1 - t0) + (t4 - t3), float(self.ctx[b] + cfg.rows), t2 - t1, t3 - t2))
        return t4 - t0

    def round_seconds(self) -> float:
        r = np.array(self.rec)
        rate = float(np.mean(r[:, 0] / r[:, 1]))
        return rate * self.keypos_round + self.n_slices * float(np.mean(r[:, 2])) + float(np.mean(r[:, 3]))

    def describe(self, steps: int) -> str:
        cfg = self.cfg
        return (f"{steps} oracle steps, each: verify attention + KV commit of one seeded (layer, "
                f"sequence) pair, one of {self.n_slices} vocabulary slices of the LM head for all "
                f"{cfg.m_rows} rows, arbitration + scan of the whole batch; full round extrapolated "
                f"(not run) = pair time per key position x {self.keypos_round:.0f} key positions "
                f"+ {self.n_slices} x slice + arbitration/scan = {self.round_seconds():.2f} s")

    def run(self, budget_s: float, min_steps: int = 3):
        t_start = time.perf_counter()
        i = 0
        while i < min_steps or time.perf_counter() - t_start < budget_s:
            self.step(i)
            i += 1
        return i


def cpu_threads() -> int:
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 0) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count() or 1


def oracle_baseline(cfg, inp, draft, budget_s: float):
    sampler = OracleSampler(cfg, inp, draft)
    n = sampler.run(budget_s)
    round_s = sampler.round_seconds()
    return cfg.batch * cfg.rows / round_s, sampler.describe(n)


# ------------------------------------------------------------------ reference arm
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cfg = _config(args)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    inp = W.make_round_inputs(cfg, device=dev)
    if dev == "cuda":
        draft = gpu_drafts(cfg, inp)
    else:
        from oracle import cospec_oracle as O
        x = O.lmhead_logits(inp["hidden"], inp["w"])
        draft = W.synth_drafts(cfg, O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8))
    sampler = OracleSampler(cfg, inp, draft)
    for i in range(args.warmup):
        sampler.step(i)
    sampler.rec.clear()
    times = [sampler.step(args.warmup + i) for i in range(args.steps)]
    round_s = sampler.round_seconds()
    value = cfg.batch * cfg.rows / round_s
    sample = sampler.describe(args.steps)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * float(np.mean(times)), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg.name},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _config(args):
    cfg = W.CONFIGS[args.config]
    if args.layers:
        cfg = cfg.replace(layers=args.layers)
    if args.k is not None:
        cfg = cfg.replace(k=args.k)
    if args.batch:
        cfg = cfg.replace(batch=args.batch)
    return cfg


# ------------------------------------------------------------------ our arm
def measure(cfg, args, env, inp=None, with_cpu=True, with_e2e=True):
    """Time `cfg`'s round on this GPU; returns the JSON line (rank 0) or None.

    `env` = (world, rank, local_rank, dist).  The round's context is restored
    at the end, so the inputs can serve another measurement."""
    from paper_2605_24793_gb300 import cospec as C
    from paper_2605_24793_gb300 import replicas
    from paper_2605_24793_gb300.round import VerifyRound
    world, rank, local_rank, dist = env
    if inp is None:
        inp = W.make_round_inputs(cfg, device="cuda")
    sps_q = None
    if args.sps:
        # the exact-match baseline with speculative sampling: drafts drawn from
        # a synthetic draft distribution (the target's logits plus noise)
        from paper_2605_24793_gb300.decode import target_logits
        q = W.draft_distributions(cfg, target_logits(cfg, inp["hidden"], inp["w"]),
                                  args.draft_noise, args.temperature or 1.0)
        draft = W.sample_from(cfg, q)
        sps_q = torch.from_numpy(q).cuda()
        del q
    else:
        draft, top1, margin = gpu_drafts(cfg, inp, with_top1=True)
    rnd = VerifyRound(inp, draft, cfg.lam, temperature=args.temperature,
                      seed=W.sample_seed(cfg), sps_q=sps_q)
    rnd.pack_step_io()                    # one host->device and one device->host copy per step
    # layers after the first launch with the stable-cache promise (their plan
    # may differ from the first layer's and from an isolated launch's)
    attn_kernel, attn_splits = C.verify_attn_plan(inp["q"][0], inp["k_pages"][0], inp["page_table"],
                                                  rnd.max_ctx, kv_stable=True)
    _, iso_splits = C.verify_attn_plan(inp["q"][0], inp["k_pages"][0], inp["page_table"], rnd.max_ctx)
    lm_name = ("lmhead_logits_features" if args.sps else
               "lmhead_argmax_features" if args.temperature is None else "lmhead_sample_features")
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()

    # One graph per round is what a step replays.  Three more graphs of the
    # round's segments -- attention (L launches), LM head, tail (arbitration
    # + commit) -- replayed with events between them give the per-kernel
    # times of a second timed region.  Graphs of the LM head followed by one
    # attention launch that may not overlap it give the isolated launch time.
    def cap(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        return g

    with torch.cuda.stream(stream):
        rnd.run()                                     # eager warm-up, settles kernel attributes
    torch.cuda.synchronize()
    check = (self_check(cfg, rnd, top1, margin)
             if not args.sps and args.temperature is None else None)
    mism = mismatch_stats(cfg, rnd) if not args.sps else None
    g_attn = cap(lambda: ([rnd.restore_context()] + [rnd.attention(l) for l in range(cfg.layers)]))
    g_lm = cap(rnd.lmhead)

    def tail():
        if cfg.k > 0 or rnd.sps:
            rnd.arbitrate()
        rnd.commit()
    g_tail = cap(tail)
    g_all = cap(rnd.run)
    iso_layers = list(range(min(cfg.layers, 4)))
    g_iso = [cap(lambda l=l: (rnd.lmhead(), rnd.attention(l, kv_stable=False))) for l in iso_layers]

    def step():
        g_all.replay()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    stream.synchronize()
    if C.get_device_error(stream) != 0:
        raise RuntimeError("device error word set during warm-up")

    # pick a step count that keeps the timed region near 3 s when none is given
    steps = args.steps
    if steps is None:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record()
            for _ in range(5):
                step()
            e1.record()
        e1.synchronize()
        per = e0.elapsed_time(e1) / 5
        steps = int(max(20, min(20000, 3000.0 / max(per, 1e-3))))

    K = steps
    K2 = min(K, 400)                     # steps of the per-kernel region
    K3 = max(20, min(200, K2))           # pairs of the isolated-attention region
    e_all = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K2)]
    ei = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K3)]
    with torch.cuda.stream(stream):
        for _ in range(3):
            g_attn.replay()
            g_lm.replay()
            g_tail.replay()
        for g in g_iso:
            g.replay()
    def timed_regions():
        clocks = ClockSampler(local_rank)
        clocks.start()
        time.sleep(0.3)
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            e_all[0].record()
            for k in range(K):
                g_all.replay()
            e_all[1].record()
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        # second timed region: the same rounds, one graph per segment
        with torch.cuda.stream(stream):
            for k in range(K2):
                ev[k][0].record()
                g_attn.replay()
                ev[k][1].record()
                g_lm.replay()
                ev[k][2].record()
                g_tail.replay()
                ev[k][3].record()
        # third region: LM head alone, then LM head + one attention launch that
        # starts only after the LM head has ended (no stable-cache overlap); the
        # difference is the isolated attention launch (cycling over layers)
        with torch.cuda.stream(stream):
            for k in range(K3):
                ei[k][0].record()
                g_lm.replay()
                ei[k][1].record()
                g_iso[k % len(g_iso)].replay()
                ei[k][2].record()
        torch.cuda.synchronize()
        return clocks.stop()

    clk = timed_regions()
    # A region whose clock record shows a hardware or thermal slowdown, or SM
    # clocks well below their maximum with no reason given, is taken once
    # more (every rank, if any rank saw one); the line reports the second.
    if replicas.max_over_ranks(1.0 if throttled(clk) else 0.0, dist,
                               torch.device("cuda", local_rank)) > 0.0:
        first = clk
        clk = timed_regions()
        clk["remeasured_after"] = {k: first.get(k) for k in ("sm_mhz", "sm_max_mhz", "reasons")}
    total_ms = e_all[0].elapsed_time(e_all[1])
    attn_ms = float(np.mean([ev[k][0].elapsed_time(ev[k][1]) for k in range(K2)]))
    lm_ms = float(np.mean([ev[k][1].elapsed_time(ev[k][2]) for k in range(K2)]))
    tail_ms = float(np.mean([ev[k][2].elapsed_time(ev[k][3]) for k in range(K2)]))
    lm_alone = float(np.mean([ei[k][0].elapsed_time(ei[k][1]) for k in range(K3)]))
    lm_attn = float(np.mean([ei[k][1].elapsed_time(ei[k][2]) for k in range(K3)]))
    iso_ms = lm_attn - lm_alone
    total_ms = replicas.max_over_ranks(total_ms, dist, torch.device("cuda", local_rank))
    ms_per_step = total_ms / K
    value = replicas.job_throughput(cfg.batch * cfg.rows, ms_per_step * 1e-3, world)
    if C.get_device_error(stream) != 0:
        raise RuntimeError("device error word set during the timed region")
    s_mean = float(rnd.accept_len.float().mean().item())

    # ------------------------------------------------------------ roofline
    pk, pk_kind = peaks()
    ctx = inp["ctx_len_np"]
    a_bytes = attention_bytes(cfg, ctx)
    lm_bytes = lmhead_bytes(cfg, logits=rnd.sps)
    attn_launch_ms = attn_ms / cfg.layers
    hbm = float(pk["hbm_gbs"])
    tflops_peak = float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"]))
    lm_t_hbm = lm_bytes / (hbm * 1e9)
    lm_t_tc = lmhead_flops(cfg) / (tflops_peak * 1e12)
    seg = attn_ms + lm_ms + tail_ms
    kern = {
        "verify_attn": {"ms_per_launch": attn_launch_ms, "launches_per_step": cfg.layers,
                        "kernel": C.ATTN_KERNEL_NAMES[attn_kernel],
                        "splits": attn_splits,
                        "bytes_per_launch": a_bytes,
                        "gbs": a_bytes / (attn_launch_ms * 1e-3) / 1e9,
                        "frac_hbm": a_bytes / (attn_launch_ms * 1e-3) / 1e9 / hbm,
                        "share": attn_ms / seg,
                        "timing": ("average of the L launches of a round, back to back: each "
                                   "streams its cache while the previous layer computes")},
        "verify_attn_isolated": {"ms_per_launch": iso_ms, "bytes_per_launch": a_bytes,
                                 "splits": iso_splits,
                                 "gbs": a_bytes / (iso_ms * 1e-3) / 1e9,
                                 "frac_hbm": a_bytes / (iso_ms * 1e-3) / 1e9 / hbm,
                                 "layers": len(iso_layers), "pairs": K3,
                                 "timing": ("one launch after the LM head, with no overlap: "
                                            "time(LM head + attention) - time(LM head), "
                                            "each replayed as its own graph")},
        lm_name: {"ms_per_launch": lm_ms, "bytes_per_launch": lm_bytes,
                  "flops_per_launch": lmhead_flops(cfg),
                  "gbs": lm_bytes / (lm_ms * 1e-3) / 1e9,
                  "tflops": lmhead_flops(cfg) / (lm_ms * 1e-3) / 1e12,
                  "bound": "hbm" if lm_t_hbm >= lm_t_tc else "tensor",
                  "frac_roofline": max(lm_t_hbm, lm_t_tc) / (lm_ms * 1e-3),
                  "share": lm_ms / seg},
        ("sps_accept+accept_commit" if rnd.sps else "arbitrate+accept_commit"):
            {"ms_per_step": tail_ms, "share": tail_ms / seg},
    }
    if attn_ms >= lm_ms:
        dom = "verify_attn"
        achieved = a_bytes / (attn_launch_ms * 1e-3) / 1e9
        roof = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "traffic": None,
                "isolated": {"achieved": kern["verify_attn_isolated"]["gbs"],
                             "frac": kern["verify_attn_isolated"]["frac_hbm"]}}
    elif lm_t_hbm >= lm_t_tc:
        dom = lm_name
        achieved = lm_bytes / (lm_ms * 1e-3) / 1e9
        roof = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "traffic": None}
    else:
        dom = lm_name
        achieved = lmhead_flops(cfg) / (lm_ms * 1e-3) / 1e12
        roof = {"kernel": dom, "bound": "tensor", "achieved": achieved, "peak": tflops_peak,
                "unit": "TFLOP/s", "frac": achieved / tflops_peak, "traffic": None}
    roof["peak_source"] = f"{pk_kind} ({'MEASURED_PEAKS.json' if pk_kind == 'measured' else 'recipe fallback'})"
    if roof["unit"] == "GB/s":
        roof["frac_of_spec_8tbs"] = roof["achieved"] / 7900.0   # nominal HBM3e, for context
    traffic = TRAFFIC.get((cfg.name, dom))
    if traffic is not None:
        roof["traffic"] = traffic

    # ------------------------------------------------------------ end to end (host buffers)
    e2e = None
    if with_e2e:
        # a second set of step buffers (and graph), so that the next step's
        # inputs can be copied in while the current step computes
        rnd.restore_context()
        torch.cuda.synchronize()
        rnd2 = VerifyRound(inp, draft, cfg.lam, temperature=args.temperature,
                           seed=W.sample_seed(cfg), sps_q=sps_q)
        rnd2.pack_step_io()
        with torch.cuda.stream(stream):
            rnd2.run()
        torch.cuda.synchronize()
        g_all2 = cap(rnd2.run)
        e2e = end_to_end(cfg, [rnd, rnd2], [g_all, g_all2], stream, K if K <= 2000 else 2000, dist)
        if dist is None or rank == 0:
            e2e["value"] = world * e2e.pop("per_rank_value")
        del g_all2, rnd2

    cpu = None
    if rank == 0 and world == 1 and with_cpu:
        v, sample = oracle_baseline(cfg, inp, draft, args.cpu_budget)
        cpu = {"value": v, "unit": UNIT, "cores": cpu_threads(), "kind": "oracle", "sample": sample}
    rnd.restore_context()
    torch.cuda.synchronize()

    if rank != 0:
        return None
    return {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": cfg.name, "batch": cfg.batch, "k": cfg.k, "rows": cfg.rows,
                   "layers": cfg.layers, "context": [int(ctx.min()), int(ctx.max())],
                   "q_heads": cfg.q_heads, "kv_heads": cfg.kv_heads,
                   "head_dim": cfg.head_dim, "hidden": cfg.hidden, "vocab": cfg.vocab,
                   "page_size": cfg.page_size, "lambda": cfg.lam,
                   "mismatch_rate": cfg.mismatch_rate,
                   "decoding": (f"exact-match speculative sampling, T={rnd.temperature}, draft "
                                f"= target logits + N(0, {args.draft_noise}^2)" if rnd.sps else
                                "greedy" if args.temperature is None
                                else f"sampled, T={args.temperature}"),
                   "parallelism": f"replicas x{world}",
                   "l2": (f"inputs larger than L2: {(a_bytes * cfg.layers + lm_bytes) / 1e9:.2f}"
                          " GB streamed per step vs 129 MB L2"),
                   "graphs": ("one CUDA graph per step; per-kernel times from a second timed "
                              f"region of {K2} rounds replaying three graphs (attention, "
                              "LM head, arbitration+commit) with events between them")},
        "roofline": roof, "kernels": kernels_round(kern), "cpu_baseline": cpu, "e2e": e2e,
        "clocks": clk, "gpu_launches": K * rnd.launches_per_round,
        "accepted_len_mean": s_mean,
        "self_check": check,
        "mismatches": mism,
        "emitted_tokens_per_s": world * cfg.batch * s_mean / (ms_per_step * 1e-3),
        "accepted_len_of": ("the one synthetic round every step replays (same drafts, "
                            "context restored); python bench.py --sweep and python -m "
                            "paper_2605_24793_gb300.decode measure it over many rounds"),
    }


def run_sweep(args, env):
    """Every point of the Llama-3-8B batch-64 workload: K in {3, 5, 7} x draft
    mismatch rate {10, 30, 60} %.  Per point: the benchmark step (device-timed
    rounds, per-kernel fractions) and the mean accepted length tau over
    `--rounds` rounds decoded in a row (Eq. 5)."""
    from paper_2605_24793_gb300.decode import MultiRoundDecoder
    names = [n for n in SWEEP if args.points is None or n in args.points]
    by_k = {}
    for n in names:
        by_k.setdefault(W.CONFIGS[n].k, []).append(n)
    for k, group in by_k.items():
        base = W.CONFIGS[group[0]]
        if args.layers:
            base = base.replace(layers=args.layers)
        # one set of inputs per K (the mismatch rate changes only the drafts),
        # with page room for the decoded rounds
        inp = W.make_round_inputs(base, device="cuda", extra_tokens=args.rounds * base.rows)
        for n in group:
            cfg = W.CONFIGS[n].replace(layers=base.layers)
            inp["cfg"] = cfg
            line = measure(cfg, args, env, inp=inp, with_cpu=False, with_e2e=False)
            dec = MultiRoundDecoder(cfg, args.rounds, inputs=inp)
            res = dec.run()
            dec.reset()
            torch.cuda.synchronize()
            del dec
            if line is None:
                continue
            kk = line["kernels"]
            lm = kk.get("lmhead_argmax_features") or kk.get("lmhead_sample_features")
            print(json.dumps({
                "sweep": "llama3_8b_b64: K x draft mismatch rate",
                "workload": cfg.name, "k": cfg.k, "mismatch_rate": cfg.mismatch_rate,
                "batch": cfg.batch, "layers": cfg.layers,
                "tau": res["tau"], "rounds": res["rounds"],
                "mismatches_first_round": line.get("mismatches"),
                "decode_ms_per_round": res["ms_per_round"],
                "decode_emitted_tokens_per_s": res["emitted_tokens_per_s"],
                "block_tokens_per_s": line["value"], "ms_per_step": line["ms_per_step"],
                "steps": line["steps"],
                "attention_us_per_launch": 1e3 * kk["verify_attn"]["ms_per_launch"],
                "attention_frac_hbm": kk["verify_attn"]["frac_hbm"],
                "attention_isolated_frac_hbm": kk["verify_attn_isolated"]["frac_hbm"],
                "lmhead_us": 1e3 * lm["ms_per_launch"], "lmhead_bound": lm["bound"],
                "lmhead_frac_roofline": lm["frac_roofline"],
                "device_error": res["device_error"], "clocks": line["clocks"]}), flush=True)
        del inp
        torch.cuda.empty_cache()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--config", default=DEFAULT_CONFIG, choices=sorted(W.CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--layers", type=int, default=None, help="override the layer count")
    ap.add_argument("--batch", type=int, default=None,
                    help="override the batch (a smaller case of the same shapes)")
    ap.add_argument("--k", type=int, default=None,
                    help="override the draft length K (block rows K+1), e.g. 25 as in the paper")
    ap.add_argument("--temperature", type=float, default=None,
                    help="stochastic decoding: sample the target candidates at this temperature")
    ap.add_argument("--sps", action="store_true",
                    help="time the exact-match baseline with speculative sampling (T = 1 unless "
                         "--temperature) instead of the CoSpec round")
    ap.add_argument("--draft-noise", type=float, default=1.0,
                    help="--sps: std of the noise added to the target logits to form the draft")
    ap.add_argument("--sweep", action="store_true",
                    help="the Llama-3-8B batch-64 points (K x mismatch rate), one line each")
    ap.add_argument("--points", nargs="+", default=None, help="subset of the sweep's workloads")
    ap.add_argument("--rounds", type=int, default=32, help="decoded rounds per sweep point")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        if args.steps is None:
            args.steps = 10
        return run_reference(args)

    from paper_2605_24793_gb300 import replicas
    world, rank, local_rank = replicas.env_ranks()
    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))

    from paper_2605_24793_gb300 import build as BLD
    from paper_2605_24793_gb300 import cospec as C
    C.load_library(BLD.build())
    env = (world, rank, local_rank, dist)
    if args.sweep:
        run_sweep(args, env)
    else:
        line = measure(_config(args), args, env, with_cpu=not args.no_cpu_baseline,
                       with_e2e=not args.no_e2e)
        if line is not None:
            print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


# dram__bytes_read.sum + dram__bytes_write.sum per launch from one ncu capture
# (profiles/), keyed by (workload, kernel); an entry is removed when its
# kernel changes after the capture.  Llama batch 64: the mean of two
# full-size launches; Qwen3-32B: one launch of a two-layer run (the
# per-layer shapes of the full workload).
TRAFFIC = {
    ("llama3_8b_b64_k7_mm30", "verify_attn"): 5224868480.0,
    ("qwen3_8b_b1", "verify_attn"): 16918272.0,
    ("qwen3_32b_b32", "verify_attn"): 1362597120.0,
}


def kernels_round(k):
    out = {}
    for name, d in k.items():
        out[name] = {kk: (round(v, 6) if isinstance(v, float) else v) for kk, v in d.items()}
    return out


def end_to_end(cfg, rnds, graphs, stream, steps, dist):
    """The serving loop through host memory.  Every step copies its inputs
    from pinned host memory (Q and the block K/V of every layer, the hidden
    rows, the draft ids: one packed buffer), runs the round and copies the
    accepted lengths and emitted tokens (one packed buffer) back to pinned
    host memory, where the host reads them.  Two sets of step buffers
    alternate: step k+1's inputs are copied on a second stream while step k
    computes, and the host waits for step k-1's result while step k runs; the
    clock stops once the last step's result has been read."""
    pinned = rnds[0].io_in.cpu().pin_memory()
    backs = [torch.empty(r.io_out.shape, dtype=r.io_out.dtype, pin_memory=True) for r in rnds]
    h2d = pinned.numel() * pinned.element_size()
    d2h = backs[0].numel() * backs[0].element_size()
    cs = torch.cuda.Stream()
    h2d_done = [torch.cuda.Event() for _ in rnds]
    step_done = [torch.cuda.Event() for _ in rnds]
    checksum = 0

    def run(n):
        nonlocal checksum
        with torch.cuda.stream(cs):
            rnds[0].io_in.copy_(pinned, non_blocking=True)
            h2d_done[0].record(cs)
        for k in range(n):
            i, j = k % 2, (k + 1) % 2
            if k + 1 < n:
                if k >= 1:
                    cs.wait_event(step_done[j])        # step k-1 is done with buffer j
                with torch.cuda.stream(cs):
                    rnds[j].io_in.copy_(pinned, non_blocking=True)
                    h2d_done[j].record(cs)
            stream.wait_event(h2d_done[i])
            with torch.cuda.stream(stream):
                graphs[i].replay()
                backs[i].copy_(rnds[i].io_out, non_blocking=True)
                step_done[i].record(stream)
            if k >= 1:
                step_done[j].synchronize()             # the host reads step k-1's result
                checksum += int(backs[j][0])
        step_done[(n - 1) % 2].synchronize()
        checksum += int(backs[(n - 1) % 2][0])

    run(3)
    if dist:
        dist.barrier()
    t0 = time.perf_counter()
    run(steps)
    dt = time.perf_counter() - t0
    from paper_2605_24793_gb300 import replicas
    dt = replicas.max_over_ranks(dt, dist, torch.device("cuda", torch.cuda.current_device()))
    return {"per_rank_value": cfg.batch * cfg.rows * steps / dt, "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": 1e3 * dt / steps, "steps": steps,
            "timing": ("host wall clock over the steps: every step copies its inputs from pinned "
                       "host memory and its result back to pinned host memory, read by the host; "
                       "the next step's input copy overlaps the current step's compute (two "
                       "buffer sets)")}


if __name__ == "__main__":
    main()
