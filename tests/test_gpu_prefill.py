"""The arbitrator's attention for one request on the device: its context
prefilled causally in chunks (verify attention + commit), then its
draft/target region attended with the full block mask, against the oracle's
dense attention under the paper's hybrid mask (Sec. 3.3)."""
import numpy as np
import pytest
import torch

from oracle import cospec_oracle as O
from paper_2605_24793_gb300 import build as BLD
from paper_2605_24793_gb300 import cospec as C
from paper_2605_24793_gb300.prefill import BlockPrefill, ChunkedPrefill

from .parity_util import assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    C.load_library(BLD.build())
    torch.cuda.set_device(0)


def _bf16(rng, shape):
    return torch.from_numpy(rng.standard_normal(shape, dtype=np.float32)).to(torch.bfloat16).cuda()


@pytest.mark.parametrize("method", [BlockPrefill, ChunkedPrefill], ids=["block", "chunked"])
@pytest.mark.parametrize("L,B,T,Hq,Hkv,D,region", [
    (2, 2, 200, 8, 2, 64, 9),        # ragged last chunk (200 = 6 x 32 + 8), K = 3 region
    (1, 1, 33, 32, 8, 128, 17),      # one full chunk and one row, K = 7 region
    (1, 3, 96, 16, 8, 128, 53),      # three full chunks, K = 25 region (53 rows)
    (1, 1, 1000, 8, 2, 128, 17),     # 32 chunks, the last of 8 rows
])
def test_prefill_then_region_matches_dense_hybrid_attention(method, L, B, T, Hq, Hkv, D, region):
    rng = np.random.default_rng(T * 7 + region)
    G = Hq // Hkv
    q = _bf16(rng, (L, B, T, Hq, D))
    k = _bf16(rng, (L, B, T, Hkv, D))
    v = _bf16(rng, (L, B, T, Hkv, D))
    pf = method(L, B, T, Hq, Hkv, D, extra_tokens=region)
    out = pf.run(q, k, v)
    torch.cuda.synchronize()
    assert C.get_device_error() == 0
    assert np.array_equal(pf.ctx_len.cpu().numpy(), np.full(B, T))
    # the region: 2K+3 rows over the prefilled context, bidirectional among themselves
    qr = _bf16(rng, (L, B, region, Hq, D))
    kr = _bf16(rng, (L, B, region, Hkv, D))
    vr = _bf16(rng, (L, B, region, Hkv, D))
    outr = torch.empty((L, B, region, Hq, D), dtype=torch.bfloat16, device="cuda")
    for l in range(L):
        C.verify_attn(qr[l], kr[l], vr[l], pf.k_pages[l], pf.v_pages[l], pf.page_table, pf.ctx_len,
                      outr[l], T, block_full=True)
    torch.cuda.synchronize()
    assert C.get_device_error() == 0
    vis = O.hybrid_mask(T, region)
    f = lambda t: t.float().cpu().numpy()
    for l in range(L):
        for b in range(B):
            for h in range(Hq):
                kv = h // G
                qq = np.concatenate([f(q[l, b, :, h]), f(qr[l, b, :, h])])
                kk = np.concatenate([f(k[l, b, :, kv]), f(kr[l, b, :, kv])])
                vv = np.concatenate([f(v[l, b, :, kv]), f(vr[l, b, :, kv])])
                ref = O.dense_masked_attention(qq, kk, vv, vis)
                assert_close(f(out[l, b, :, h]), ref[:T], f"context rows l={l} b={b} h={h}")
                assert_close(f(outr[l, b, :, h]), ref[T:], f"region rows l={l} b={b} h={h}")
    # the cache holds the context's keys and values, position by position
    kp = pf.k_pages.cpu().view(torch.int16).numpy()
    table = pf.page_table.cpu().numpy()
    kb = k.cpu().view(torch.int16).numpy()
    for b in range(B):
        t = np.arange(T)
        np.testing.assert_array_equal(kp[:, table[b, t // 16], :, t % 16].transpose(1, 0, 2, 3), kb[:, b])
