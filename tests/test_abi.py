"""The C-ABI library builds for sm_103a, loads, exports every entry point of
include/cospec.h, and rejects bad arguments on the host before launching
anything (no GPU needed)."""
import ctypes
import os
import re
import shutil
import subprocess
import threading

import pytest
import torch

from paper_2605_24793_gb300 import build as B
from paper_2605_24793_gb300 import cospec as C

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    path = B.build()
    return C.load_library(path)


def _header_functions():
    text = open(os.path.join(ROOT, "include", "cospec.h")).read()
    return sorted(set(re.findall(r"COSPEC_API\s+[\w\s\*]+?\b(cospec_\w+)\s*\(", text)))


def test_header_declares_the_four_round_calls():
    names = _header_functions()
    for n in ("cospec_verify_attn", "cospec_lmhead_argmax_features", "cospec_arbitrate",
              "cospec_accept_commit"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    names = _header_functions()
    assert len(names) >= 8
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(C.EXPORTED)


def test_status_strings(lib):
    assert lib.cospec_status_string(0) == b"ok"
    assert lib.cospec_status_string(-1) == b"invalid argument"
    assert lib.cospec_status_string(-3) == b"workspace missing or too small"
    assert lib.cospec_status_string(123) == b"unknown status"
    # no CUDA error recorded on this thread yet
    assert lib.cospec_last_cuda_error() == b"cudaSuccess"


def _dims(**kw):
    d = dict(batch=2, rows=6, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16,
             max_pages_per_seq=300, num_pages=600, softmax_scale=0.0, flags=0)
    d.update(kw)
    return C.AttnDims(*d.values())


def test_attention_host_validation(lib):
    f = lib.cospec_verify_attn
    nul = None
    # null pointers are rejected before any CUDA call
    assert f(ctypes.byref(_dims()), 4096, *([nul] * 8), nul) == -1
    # shapes the kernels do not cover
    assert f(ctypes.byref(_dims(head_dim=96)), 4096, *([nul] * 8), nul) == -2
    assert f(ctypes.byref(_dims(page_size=32)), 4096, *([nul] * 8), nul) == -2
    assert f(ctypes.byref(_dims(rows=65)), 4096, *([nul] * 8), nul) == -2
    assert f(ctypes.byref(_dims(num_q_heads=30)), 4096, *([nul] * 8), nul) == -1
    assert f(ctypes.byref(_dims(softmax_scale=float("nan"))), 4096, *([nul] * 8), nul) == -1
    # max_ctx beyond the page-table row
    assert f(ctypes.byref(_dims()), 300 * 16 + 1, *([nul] * 8), nul) == -1
    # unknown flag bits
    assert f(ctypes.byref(_dims(flags=4)), 4096, *([nul] * 8), nul) == -1
    # empty batch is a no-op
    assert f(ctypes.byref(_dims(batch=0)), 0, *([nul] * 8), nul) == 0


def test_attention_plan_host_validation(lib):
    f = lib.cospec_verify_attn_plan
    k, sp = ctypes.c_int(), ctypes.c_int()
    assert f(ctypes.byref(_dims(head_dim=96)), 4096, ctypes.byref(k), ctypes.byref(sp)) == -2
    assert f(ctypes.byref(_dims()), 4096, None, None) == -1
    assert f(ctypes.byref(_dims()), 300 * 16 + 1, ctypes.byref(k), ctypes.byref(sp)) == -1


# Clusters of S CTAs resident at once on a GB300 (152 SMs), from
# cudaOccupancyMaxActiveClusters for every attention variant and S = 1..16:
# two CTAs per SM for the mma.sync kernel with <= 32 block keys, one otherwise
# (and for the tcgen05 kernel).
_GB300_TWO_PER_SM = dict(enumerate([304, 152, 97, 74, 58, 46, 38, 36, 30, 28, 23, 23, 19, 14, 14,
                                    14], start=1))
_GB300_ONE_PER_SM = dict(enumerate([152, 76, 46, 36, 28, 23, 15, 15, 15, 13, 8, 8, 7, 7, 7, 7],
                                   start=1))


def _gb300_resident(kernel, rows, block_rows, splits):
    table = _GB300_TWO_PER_SM if kernel == 0 and block_rows <= 32 else _GB300_ONE_PER_SM
    return table.get(splits, 0)


# (batch, rows, Hq, Hkv, head_dim, longest context, stable-cache flag) ->
# (kernel, splits): the planner's choice for each workload shape, which is
# also the fastest of the splits timed on a GB300 (Qwen3-8B batch 16: 4 splits
# against 2 and 8; Llama-3-8B batch 64: 2 against 4 and 8; Qwen3-32B batch
# 32: unsplit against 2; Qwen3-8B batch 16 K = 15: 2 against 4; batch 1, K = 5:
# 16 back to back, 12 alone; batch 2: 12 against 13, 8 and 16; batch 4: 8
# against 12 and 16; batch 1, K = 15 and K = 25 (one 64- or 104-row group per
# KV head on the tcgen05 kernel): 12, the largest split whose clusters are
# all resident at one CTA per SM).
PLAN_CASES = [
    ((1, 6, 32, 8, 128, 4096, 1), (C.ATTN_MMA_SYNC, 16)),   # Qwen3-8B, batch 1, K = 5
    ((1, 6, 32, 8, 128, 4096, 0), (C.ATTN_MMA_SYNC, 12)),   # the same, on an idle GPU
    ((2, 6, 32, 8, 128, 4096, 1), (C.ATTN_MMA_SYNC, 12)),   # batch 2: 16 clusters at once
    ((4, 6, 32, 8, 128, 4096, 1), (C.ATTN_MMA_SYNC, 8)),    # batch 4: 32 clusters at once
    ((16, 8, 32, 8, 128, 8192, 1), (C.ATTN_MMA_SYNC, 4)),   # Qwen3-8B, batch 16, K = 7
    ((1, 16, 32, 8, 128, 4096, 1), (C.ATTN_TCGEN05, 12)),   # batch 1, K = 15: one wave
    ((1, 26, 32, 8, 128, 4096, 1), (C.ATTN_TCGEN05, 12)),   # batch 1, K = 25: 104 rows, one group
    ((16, 16, 32, 8, 128, 8192, 1), (C.ATTN_TCGEN05, 2)),   # batch 16, K = 15
    ((32, 8, 64, 8, 128, 16384, 1), (C.ATTN_TCGEN05, 1)),   # Qwen3-32B, batch 32
    ((64, 8, 32, 8, 128, 32768, 1), (C.ATTN_MMA_SYNC, 2)),  # Llama-3-8B, batch 64
]


@pytest.mark.parametrize("shape,plan", PLAN_CASES, ids=lambda v: str(v))
def test_attention_plan_on_a_gb300_model(lib, shape, plan):
    B, R, Hq, Hkv, D, ctx, stable = shape
    dims = C.AttnDims(B, R, Hq, Hkv, D, 16, (ctx + R + 15) // 16, 1 << 20, 0.0,
                      C.ATTN_KV_STABLE if stable else 0)
    assert C.verify_attn_plan_model(dims, ctx, 152, _gb300_resident) == plan


def test_attention_plan_model_rules(lib):
    # a batch of a few units: the largest even split up to 16 whose clusters
    # are all resident; at most 12 without the stable-cache promise
    st = C.AttnDims(1, 6, 32, 8, 128, 16, 300, 1 << 20, 0.0, C.ATTN_KV_STABLE)
    dims = C.AttnDims(1, 6, 32, 8, 128, 16, 300, 1 << 20, 0.0, 0)
    assert C.verify_attn_plan_model(st, 4096, 152, lambda k, r, kb, s: 304 // s) == (0, 16)
    assert C.verify_attn_plan_model(dims, 4096, 152, lambda k, r, kb, s: 304 // s) == (0, 12)
    assert C.verify_attn_plan_model(st, 4096, 152, lambda k, r, kb, s: 7 if s >= 14 else 304 // s) \
        == (0, 12)
    # no cluster of more than one CTA can be scheduled: no split
    assert C.verify_attn_plan_model(dims, 4096, 152, lambda k, r, kb, s: 152 if s == 1 else 0) \
        == (0, 1)
    # short contexts: at least four 64-key tiles per CTA (256 keys -> 1 split)
    assert C.verify_attn_plan_model(dims, 256, 152, _gb300_resident) == (0, 1)
    assert C.verify_attn_plan_model(dims, 512, 152, _gb300_resident) == (0, 2)
    # more than 32 query rows per KV head with G <= 64: the tcgen05 kernel;
    # a KV head shared by 128 query heads stays on the mma.sync kernel
    big = C.AttnDims(4, 8, 64, 8, 128, 16, 300, 1 << 20, 0.0, 0)
    assert C.verify_attn_plan_model(big, 4096, 152, _gb300_resident)[0] == C.ATTN_TCGEN05
    g128 = C.AttnDims(4, 2, 128, 1, 128, 16, 300, 1 << 20, 0.0, 0)
    assert C.verify_attn_plan_model(g128, 4096, 152, _gb300_resident)[0] == C.ATTN_MMA_SYNC
    # argument checks
    f = lib.cospec_verify_attn_plan_model
    k, sp = ctypes.c_int(), ctypes.c_int()
    cb = C.RESIDENT_FN(lambda *a: 1)
    assert f(ctypes.byref(dims), 4096, 0, cb, None, ctypes.byref(k), ctypes.byref(sp)) == -1
    assert f(ctypes.byref(dims), 4096, 152, C.RESIDENT_FN(), None, ctypes.byref(k),
             ctypes.byref(sp)) == -1
    assert f(ctypes.byref(dims), 300 * 16 + 1, 152, cb, None, ctypes.byref(k), ctypes.byref(sp)) == -1


def test_lmhead_host_validation(lib):
    f = lib.cospec_lmhead_argmax_features
    assert f(0, 4096, 1000, *([None] * 6), 0, None) == 0          # no rows: nothing to do
    assert f(4, 4096, 1000, *([None] * 6), 0, None) == -1         # null pointers
    assert f(-1, 4096, 1000, *([None] * 6), 0, None) == -1
    fake = ctypes.c_void_p(1 << 20)                                # never dereferenced
    assert f(4, 4000, 1000, fake, fake, fake, fake, fake, fake, 1 << 30, None) == -2   # d % 64
    assert f(4, 4096, 1000, ctypes.c_void_p((1 << 20) + 2), fake, fake, fake, fake, fake,
             1 << 30, None) == -1                                  # misaligned hidden
    assert lib.cospec_lmhead_workspace(6, 4096, 151936) > 0


def test_cuda_failure_is_recorded_without_a_device(lib):
    # On a host without a GPU every call that gets past its argument checks
    # fails in its first CUDA call; that error is what cospec_last_cuda_error
    # then names (per host thread: run in a fresh one).
    if torch.cuda.is_available():
        pytest.skip("needs a host without a GPU")
    fake = ctypes.c_void_p(1 << 20)                                # never dereferenced
    got = {}

    def run():
        got["before"] = lib.cospec_last_cuda_error()
        got["status"] = lib.cospec_lmhead_argmax_features_noalloc(6, 4096, 1000, fake, fake, fake,
                                                                  fake, fake, None)
        got["after"] = lib.cospec_last_cuda_error()
        got["ws"] = lib.cospec_lmhead_argmax_features(6, 4096, 1000, fake, fake, fake, fake, fake,
                                                      fake, 1 << 30, None)

    t = threading.Thread(target=run)
    t.start()
    t.join()
    assert got["before"] == b"cudaSuccess"
    assert got["status"] == -4 and got["ws"] == -4
    assert got["after"] not in (b"cudaSuccess", b"cudaErrorUnknown")


def test_arbitrate_host_validation(lib):
    f = lib.cospec_arbitrate
    fake = ctypes.c_void_p(1 << 20)
    assert f(4, 32, fake, fake, fake, 16, fake, fake, fake, 0.0, 0.6, 0, fake, fake, None) == -2
    assert f(4, 5, fake, fake, fake, 16, fake, fake, fake, 0.0, 0.6, 3, fake, fake, None) == -1
    assert f(4, 5, fake, fake, fake, 16, fake, fake, fake, 0.0, float("nan"), 0, fake, fake, None) == -1
    assert f(4, 5, fake, fake, fake, 16, None, fake, fake, 0.0, 0.6, 0, fake, fake, None) == -1
    assert f(4, 5, fake, fake, fake, 2048, fake, fake, fake, 0.0, 0.6, 0, fake, fake, None) == -2
    assert f(0, 5, None, None, None, 16, None, None, None, 0.0, 0.6, 0, None, None, None) == 0


def test_commit_host_validation(lib):
    f = lib.cospec_accept_commit
    fake = ctypes.c_void_p(1 << 20)
    d = _dims(batch=2, rows=6)
    args = [fake] * 7
    # batch in dims must match B, rows must be K + 1
    assert f(3, 5, 36, ctypes.byref(d), *args, 10 ** 9, fake, fake, fake, fake, None) == -1
    assert f(2, 4, 36, ctypes.byref(d), *args, 10 ** 9, fake, fake, fake, fake, None) == -1
    # layer stride smaller than one pool
    assert f(2, 5, 36, ctypes.byref(d), *args, 1024, fake, fake, fake, fake, None) == -1
    # several layers into one shared pool (stride 0) would race for the same cells
    assert f(2, 5, 36, ctypes.byref(d), *args, 0, fake, fake, fake, fake, None) == -1
    assert f(2, 5, 2, ctypes.byref(d), *args, 0, fake, fake, fake, fake, None) == -1
    assert f(2, 5, 36, ctypes.byref(d), *([None] * 7), 10 ** 9, fake, fake, fake, fake, None) == -1


def test_sample_host_validation(lib):
    f = lib.cospec_lmhead_sample_features
    fake = ctypes.c_void_p(1 << 20)
    args = lambda T, seed: (4, 4096, 1000, fake, fake, fake, T, seed, fake, fake, fake, 1 << 30, None)
    assert f(*args(0.0, fake)) == -1                                  # temperature must be > 0
    assert f(*args(-1.0, fake)) == -1
    assert f(*args(float("nan"), fake)) == -1
    assert f(*args(float("inf"), fake)) == -1
    assert f(*args(1e-45, fake)) == -1                                # 1 / T overflows
    assert f(*args(1.0, None)) == -1                                  # seed pointer missing
    assert f(*args(1.0, ctypes.c_void_p((1 << 20) + 4))) == -1        # seed not 8-byte aligned
    assert f(0, 4096, 1000, *([None] * 3), 1.0, None, None, None, None, 0, None) == 0
    assert f(4, 4000, 1000, fake, fake, fake, 1.0, fake, fake, fake, fake, 1 << 30, None) == -2


def test_logits_and_sps_host_validation(lib):
    fake = ctypes.c_void_p(1 << 20)                                   # never dereferenced
    f = lib.cospec_lmhead_logits_features
    args = lambda T, logits: (4, 4096, 1000, fake, fake, fake, T, fake, fake, logits, fake, 1 << 30,
                              None)
    assert f(*args(0.0, fake)) == -1                                  # temperature must be > 0
    assert f(*args(float("inf"), fake)) == -1
    assert f(*args(1.0, None)) == -1                                  # logits pointer missing
    assert f(*args(1.0, ctypes.c_void_p((1 << 20) + 2))) == -1        # logits not 4-byte aligned
    assert f(0, 4096, 1000, *([None] * 3), 1.0, *([None] * 4), 0, None) == 0
    g = lib.cospec_sps_accept
    ws = lib.cospec_sps_workspace(8)
    assert ws >= 8 * 64 * 16 and lib.cospec_sps_workspace(0) == 0
    sargs = lambda B, K, seed, wsb: (B, K, 1000, fake, fake, fake, fake, seed, fake, fake, fake,
                                     fake, wsb, None)
    assert g(*sargs(8, 32, fake, ws)) == -2                           # K <= 31
    assert g(*sargs(8, 5, None, ws)) == -1                            # seed missing
    assert g(*sargs(8, 5, ctypes.c_void_p((1 << 20) + 4), ws)) == -1  # seed not 8-byte aligned
    assert g(*sargs(8, 5, fake, ws - 1)) == -3                        # workspace too small
    assert g(0, 5, 1000, *([None] * 9), 0, None) == 0                 # empty batch
    assert g(8, 5, 1000, fake, fake, fake, None, fake, fake, fake, fake, fake, ws, None) == -1


C_PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "cospec.h"
int main(void) {
  cospec_attn_dims d;
  int kernel = -1, splits = -1;
  memset(&d, 0, sizeof d);
  d.batch = 1; d.rows = 6; d.num_q_heads = 32; d.num_kv_heads = 8; d.head_dim = 96;
  d.page_size = 16; d.max_pages_per_seq = 300; d.num_pages = 300;
  if (strcmp(cospec_status_string(COSPEC_OK), "ok") != 0) return 1;
  if (cospec_verify_attn_plan(&d, 4096, &kernel, &splits) != COSPEC_ERR_UNSUPPORTED) return 2;
  if (cospec_lmhead_argmax_features(0, 4096, 1000, NULL, NULL, NULL, NULL, NULL, NULL, 0,
                                    NULL) != COSPEC_OK) return 3;
  puts("c abi ok");
  return 0;
}
"""


def test_header_is_plain_c_and_links(lib, tmp_path):
    # the header compiles as strict C99 and a C program links and calls the library
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "abi.c"
    src.write_text(C_PROGRAM)
    exe = tmp_path / "abi"
    libdir = os.path.dirname(C.LIB_PATH)
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror",
                        "-I", os.path.join(ROOT, "include"), str(src), "-L", libdir, "-lcospec",
                        f"-Wl,-rpath,{libdir}", "-o", str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert out.returncode == 0 and out.stdout.strip() == "c abi ok", (out.returncode, out.stderr)
