"""Benchmark of one CoSpec verify/arbitrate round on GB300.

A step is one full round -- L x verify attention, the fused LM head,
arbitration, accept/commit (with the context restore that lets every step
verify the same block) -- over one batch of the workload, replayed from CUDA
graphs.  Metric: verified block-tokens/s = batch * (K+1) / round time.

  python bench.py [--config qwen3_8b_b1] [--steps K] [--warmup W] [--gpus N]
  python bench.py --impl reference      # the CPU oracle on a bounded sample

One JSON line is printed by rank 0.  Under torchrun every rank runs an
independent replica of the workload (the round shards by sequence and needs
no collective); the host-side max over ranks of the timed region gives the
whole-job throughput.
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
DEFAULT_CONFIG = "qwen3_8b_b1"
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


def lmhead_bytes(cfg) -> float:
    """W streamed once plus the hidden rows and the per-row outputs."""
    return 2.0 * cfg.vocab * cfg.hidden + 2.0 * cfg.m_rows * cfg.hidden + 24.0 * cfg.m_rows


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


# ------------------------------------------------------------------ drafts
def gpu_drafts(cfg, inp) -> np.ndarray:
    """Draft ids for the benchmark, synthesised from the target's own top-8
    (fp32 logits of the bf16 operands, computed once before timing)."""
    h = inp["hidden"].float()
    ranked = []
    for r0 in range(0, h.shape[0], 64):
        logits = h[r0:r0 + 64] @ inp["w"].float().T
        ranked.append(torch.topk(logits, 8, dim=1).indices.cpu())
        del logits
    ranked = torch.cat(ranked).numpy().reshape(cfg.batch, cfg.rows, 8)
    return W.synth_drafts(cfg, ranked)


# ------------------------------------------------------------------ CPU oracle sample
class OracleSampler:
    """Times the CPU oracle on a bounded slice of the workload.

    One sample step runs, for one layer l (cycling), the oracle verify
    attention of every sequence, the oracle LM head over vocabulary slice l of
    L (logits and statistics), and the full arbitration, scan and commit of
    the round.  A full round is L such steps, so the full-round time is
    estimated as L x the mean step time."""

    def __init__(self, cfg, inp, draft, max_seqs: int = 64):
        from oracle import cospec_oracle as O
        self.O = O
        self.cfg = cfg
        self.draft = draft
        self.table = inp["page_table_np"]
        self.ctx = inp["ctx_len_np"]
        self.hidden = inp["hidden"].cpu()
        self.w = inp["w"]
        self.inp = inp
        self.mlp = inp["mlp"]
        self.B = cfg.batch
        self.layer_cache = {}
        # statistics of the full vocabulary for the arbitration inputs (not timed)
        self.argmax = None

    def _layer(self, l):
        if l not in self.layer_cache:
            inp, cfg = self.inp, self.cfg
            lp = 0 if inp["k_pages"].shape[0] == 1 else l
            pages = np.unique(self.table[self.table >= 0])
            remap = np.full(inp["num_pages"], -1, dtype=np.int64)
            remap[pages] = np.arange(len(pages))
            idx = torch.from_numpy(pages).to(inp["k_pages"].device)
            self.layer_cache = {l: dict(
                q=inp["q"][l].cpu(), kb=inp["k_blk"][l].cpu(), vb=inp["v_blk"][l].cpu(),
                kp=inp["k_pages"][lp].index_select(0, idx).cpu(),
                vp=inp["v_pages"][lp].index_select(0, idx).cpu(),
                table=np.where(self.table >= 0, remap[np.clip(self.table, 0, None)], -1))}
        return self.layer_cache[l]

    def step(self, l):
        O, cfg = self.O, self.cfg
        L = cfg.layers
        d = self._layer(l)
        V = cfg.vocab
        v0, v1 = (V * l) // L, (V * (l + 1)) // L
        wslice = self.w[v0:v1].cpu()
        t0 = time.perf_counter()
        O.verify_attention(d["q"], d["kb"], d["vb"], d["kp"], d["vp"], d["table"], self.ctx,
                           cfg.page_size)
        x = O.lmhead_logits(self.hidden, wslice)
        dfr = np.full((cfg.batch, cfg.rows), -1)
        dfr[:, :cfg.k] = self.draft
        dfr = np.where((dfr >= v0) & (dfr < v1), dfr - v0, -1)
        am, st = O.row_stats(x, dfr.reshape(-1))
        am = am.reshape(cfg.batch, cfg.rows) + v0
        st = st.reshape(cfg.batch, cfg.rows, 5)
        w1, b1, w2, b2 = self.mlp
        p, a = O.arbitrate(self.draft, am, st, w1, b1, w2, b2, cfg.lam)
        s, _ = O.accept_scan(self.draft, am, a)
        O.commit_kv(d["kb"].view(torch.int16).numpy()[None], d["vb"].view(torch.int16).numpy()[None],
                    d["kp"].view(torch.int16).numpy()[None], d["vp"].view(torch.int16).numpy()[None],
                    d["table"], self.ctx, s, cfg.page_size)
        return time.perf_counter() - t0

    def run(self, budget_s: float, min_steps: int = 1):
        times = []
        t_start = time.perf_counter()
        l = 0
        while len(times) < min_steps or time.perf_counter() - t_start < budget_s:
            times.append(self.step(l % self.cfg.layers))
            l += 1
            if len(times) >= self.cfg.layers and time.perf_counter() - t_start >= budget_s:
                break
        return times


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
    times = sampler.run(budget_s)
    round_s = cfg.layers * float(np.mean(times))
    value = cfg.batch * cfg.rows / round_s
    sample = (f"{len(times)} oracle steps of 1/{cfg.layers} of a round each (one layer's verify "
              f"attention for all {cfg.batch} sequences + a 1/{cfg.layers} vocabulary slice of the "
              f"LM head + arbitration and scan); full round = {cfg.layers} x mean step "
              f"= {round_s:.2f} s")
    return value, sample, times


# ------------------------------------------------------------------ reference arm
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cfg = W.CONFIGS[args.config]
    inp = W.make_round_inputs(cfg, device="cuda" if torch.cuda.is_available() else "cpu")
    draft = gpu_drafts(cfg, inp) if torch.cuda.is_available() else None
    if draft is None:
        from oracle import cospec_oracle as O
        x = O.lmhead_logits(inp["hidden"], inp["w"])
        draft = W.synth_drafts(cfg, O.topk_ids(x, 8).reshape(cfg.batch, cfg.rows, 8))
    sampler = OracleSampler(cfg, inp, draft)
    for i in range(args.warmup):
        sampler.step(i % cfg.layers)
    times = [sampler.step((args.warmup + i) % cfg.layers) for i in range(args.steps)]
    round_s = cfg.layers * float(np.mean(times))
    value = cfg.batch * cfg.rows / round_s
    sample = (f"each step: one layer's oracle verify attention for all {cfg.batch} sequences + a "
              f"1/{cfg.layers} vocabulary slice of the oracle LM head + arbitration and scan; "
              f"round time = {cfg.layers} x mean step")
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


# ------------------------------------------------------------------ our arm
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
    ap.add_argument("--k", type=int, default=None,
                    help="override the draft length K (block rows K+1), e.g. 25 as in the paper")
    ap.add_argument("--temperature", type=float, default=None,
                    help="stochastic decoding: sample the target candidates at this temperature")
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
    from paper_2605_24793_gb300.round import VerifyRound
    C.load_library(BLD.build())

    cfg = W.CONFIGS[args.config]
    if args.layers:
        cfg = cfg.replace(layers=args.layers)
    if args.k is not None:
        cfg = cfg.replace(k=args.k)
    inp = W.make_round_inputs(cfg, device="cuda")
    draft = gpu_drafts(cfg, inp)
    rnd = VerifyRound(inp, draft, cfg.lam, temperature=args.temperature,
                      seed=W.sample_seed(cfg))
    rnd.pack_step_io()                    # one host->device and one device->host copy per step
    attn_kernel, attn_splits = C.verify_attn_plan(inp["q"][0], inp["k_pages"][0], inp["page_table"],
                                                  rnd.max_ctx)
    lm_name = "lmhead_argmax_features" if args.temperature is None else "lmhead_sample_features"
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()

    # One graph per round is what a step replays.  Three more graphs of the
    # round's segments -- attention (L launches), LM head, tail (arbitration
    # + commit) -- replayed with events between them give the per-kernel
    # times of a second timed region.
    def cap(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        return g

    with torch.cuda.stream(stream):
        rnd.run()                                     # eager warm-up, settles kernel attributes
    torch.cuda.synchronize()
    g_attn = cap(lambda: ([rnd.restore_context()] + [rnd.attention(l) for l in range(cfg.layers)]))
    g_lm = cap(rnd.lmhead)

    def tail():
        if cfg.k > 0:
            rnd.arbitrate()
        rnd.commit()
    g_tail = cap(tail)
    g_all = cap(rnd.run)

    def step():
        g_all.replay()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    stream.synchronize()
    if C.get_device_error(stream) != 0:
        raise RuntimeError("device error word set during warm-up")

    # pick a step count that keeps the timed region near 3 s when none is given
    if args.steps is None:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record()
            for _ in range(5):
                step()
            e1.record()
        e1.synchronize()
        per = e0.elapsed_time(e1) / 5
        args.steps = int(max(20, min(20000, 3000.0 / max(per, 1e-3))))

    K = args.steps
    K2 = min(K, 400)                     # steps of the per-kernel region
    e_all = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K2)]
    with torch.cuda.stream(stream):
        for _ in range(3):
            g_attn.replay()
            g_lm.replay()
            g_tail.replay()
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
    torch.cuda.synchronize()
    clk = clocks.stop()
    total_ms = e_all[0].elapsed_time(e_all[1])
    attn_ms = float(np.mean([ev[k][0].elapsed_time(ev[k][1]) for k in range(K2)]))
    lm_ms = float(np.mean([ev[k][1].elapsed_time(ev[k][2]) for k in range(K2)]))
    tail_ms = float(np.mean([ev[k][2].elapsed_time(ev[k][3]) for k in range(K2)]))
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
    lm_bytes = lmhead_bytes(cfg)
    attn_launch_ms = attn_ms / cfg.layers
    hbm = float(pk["hbm_gbs"])
    tflops_peak = float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"]))
    lm_t_hbm = lm_bytes / (hbm * 1e9)
    lm_t_tc = lmhead_flops(cfg) / (tflops_peak * 1e12)
    kern = {
        "verify_attn": {"ms_per_launch": attn_launch_ms, "launches_per_step": cfg.layers,
                        "kernel": "tcgen05" if attn_kernel == C.ATTN_TCGEN05 else "mma.sync",
                        "splits": attn_splits,
                        "bytes_per_launch": a_bytes,
                        "gbs": a_bytes / (attn_launch_ms * 1e-3) / 1e9,
                        "frac_hbm": a_bytes / (attn_launch_ms * 1e-3) / 1e9 / hbm,
                        "share": attn_ms / (attn_ms + lm_ms + tail_ms)},
        lm_name: {"ms_per_launch": lm_ms, "bytes_per_launch": lm_bytes,
                                   "flops_per_launch": lmhead_flops(cfg),
                                   "gbs": lm_bytes / (lm_ms * 1e-3) / 1e9,
                                   "tflops": lmhead_flops(cfg) / (lm_ms * 1e-3) / 1e12,
                                   "bound": "hbm" if lm_t_hbm >= lm_t_tc else "tensor",
                                   "frac_roofline": max(lm_t_hbm, lm_t_tc) / (lm_ms * 1e-3),
                                   "share": lm_ms / (attn_ms + lm_ms + tail_ms)},
        "arbitrate+accept_commit": {"ms_per_step": tail_ms,
                                    "share": tail_ms / (attn_ms + lm_ms + tail_ms)},
    }
    if attn_ms >= lm_ms:
        dom = "verify_attn"
        achieved = a_bytes / (attn_launch_ms * 1e-3) / 1e9
        roof = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "traffic": None}
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
    if not args.no_e2e:
        e2e = end_to_end(cfg, rnd, step, stream, K if K <= 2000 else 2000, dist)
        if dist is None or rank == 0:
            e2e["value"] = world * e2e.pop("per_rank_value")

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, sample, _ = oracle_baseline(cfg, inp, draft, args.cpu_budget)
        cpu = {"value": v, "unit": UNIT, "cores": cpu_threads(), "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": cfg.name, "batch": cfg.batch, "k": cfg.k, "rows": cfg.rows,
                       "layers": cfg.layers, "context": [int(ctx.min()), int(ctx.max())],
                       "q_heads": cfg.q_heads, "kv_heads": cfg.kv_heads,
                       "head_dim": cfg.head_dim, "hidden": cfg.hidden, "vocab": cfg.vocab,
                       "page_size": cfg.page_size, "lambda": cfg.lam,
                       "decoding": ("greedy" if args.temperature is None
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
            "emitted_tokens_per_s": world * cfg.batch * s_mean / (ms_per_step * 1e-3),
            "accepted_len_of": ("the one synthetic round every step replays (same drafts, "
                                "context restored); python -m paper_2605_24793_gb300.decode "
                                "measures it over many rounds"),
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


# dram__bytes_read.sum + dram__bytes_write.sum per launch from one ncu capture
# (profiles/), keyed by (workload, kernel); an entry is removed when its
# kernel changes after the capture.  The attention entries (qwen3_8b_b1
# 16918528, qwen3_8b_b16 304239360, qwen3_32b_b32 1362598144 bytes) were
# removed when both attention kernels changed how they issue the cluster
# merge's copies; they come back with the next capture.
TRAFFIC = {
    ("qwen3_8b_b1", "lmhead_argmax_features"): 1248011008.0,
}


def kernels_round(k):
    out = {}
    for name, d in k.items():
        out[name] = {kk: (round(v, 6) if isinstance(v, float) else v) for kk, v in d.items()}
    return out


def end_to_end(cfg, rnd, step, stream, steps, dist):
    """Per step: copy the round's activations from pinned host memory (Q and
    the block K/V of every layer, the hidden rows, the draft ids; one packed
    buffer), run the round, read back the accepted lengths and emitted tokens
    (one packed buffer), synchronise."""
    srcs = [rnd.io_in]
    pinned = [t.cpu().pin_memory() for t in srcs]
    outs = [rnd.io_out]
    back = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs]
    h2d = sum(t.numel() * t.element_size() for t in pinned)
    d2h = sum(t.numel() * t.element_size() for t in back)

    def e2e_step():
        with torch.cuda.stream(stream):
            for dst, src in zip(srcs, pinned):
                dst.copy_(src, non_blocking=True)
            step()
            for dst, src in zip(back, outs):
                dst.copy_(src, non_blocking=True)
        stream.synchronize()

    for _ in range(3):
        e2e_step()
    if dist:
        dist.barrier()
    t0 = time.perf_counter()
    for _ in range(steps):
        e2e_step()
    dt = time.perf_counter() - t0
    from paper_2605_24793_gb300 import replicas
    dt = replicas.max_over_ranks(dt, dist, torch.device("cuda", torch.cuda.current_device()))
    return {"per_rank_value": cfg.batch * cfg.rows * steps / dt, "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": 1e3 * dt / steps, "steps": steps,
            "timing": "host wall clock around copies + round + read-back, stream synchronised each step"}


if __name__ == "__main__":
    main()
