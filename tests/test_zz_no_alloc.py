"""The allocation-free LM-head entry point (for callers that cannot allocate
device memory or pass a workspace) gives the same outputs as the workspace
entry point, on two calls in a row, through the C ABI."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2605_24793_gb300 import build as BLD
from paper_2605_24793_gb300 import cospec as C

from .parity_util import assert_close

pytestmark = pytest.mark.gpu


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    lib = C.load_library(BLD.build())
    torch.cuda.set_device(0)
    rng = np.random.default_rng(2024)
    # different problems back to back: a call must not see an earlier call's
    # scratch contents; M = 512 runs two full 256-row passes that reuse the
    # scratch inside one call
    for M, d, V in ((6, 4096, 151936), (300, 512, 5000), (512, 1024, 40000)):
        hidden = torch.from_numpy(rng.standard_normal((M, d), dtype=np.float32)).to(torch.bfloat16).cuda()
        w = torch.from_numpy(rng.standard_normal((V, d), dtype=np.float32) * 0.05).to(torch.bfloat16).cuda()
        dfr = torch.from_numpy(rng.integers(-1, V, M).astype(np.int32)).cuda()
        am_ws = torch.empty(M, dtype=torch.int32, device="cuda")
        st_ws = torch.empty((M, 5), dtype=torch.float32, device="cuda")
        ws = torch.empty(lib.cospec_lmhead_workspace(M, d, V), dtype=torch.uint8, device="cuda")
        assert lib.cospec_lmhead_argmax_features(M, d, V, _ptr(hidden), _ptr(w), _ptr(dfr), _ptr(am_ws),
                                                 _ptr(st_ws), _ptr(ws), ws.numel(), _stream()) == 0
        am = torch.full((M,), -7, dtype=torch.int32, device="cuda")
        st = torch.full((M, 5), 7.0, dtype=torch.float32, device="cuda")
        assert lib.cospec_lmhead_argmax_features_noalloc(M, d, V, _ptr(hidden), _ptr(w), _ptr(dfr),
                                                         _ptr(am), _ptr(st), _stream()) == 0
        torch.cuda.synchronize()
        assert np.array_equal(am.cpu().numpy(), am_ws.cpu().numpy())
        assert_close(st.cpu().numpy(), st_ws.cpu().numpy(), "no-alloc stats")
    assert C.get_device_error() == 0


def test_noalloc_rejects_requests_beyond_its_scratch():
    lib = C.load_library(BLD.build())
    M, d, V = 513, 128, 256
    hidden = torch.zeros((M, d), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((V, d), dtype=torch.bfloat16, device="cuda")
    dfr = torch.full((M,), -1, dtype=torch.int32, device="cuda")
    am = torch.empty(M, dtype=torch.int32, device="cuda")
    st = torch.empty((M, 5), dtype=torch.float32, device="cuda")
    assert lib.cospec_lmhead_argmax_features_noalloc(M, d, V, _ptr(hidden), _ptr(w), _ptr(dfr),
                                                     _ptr(am), _ptr(st), _stream()) == -2
