"""Host-side shape checks of the Python binding (no GPU, no library call):
consistent tensors pass, and each tensor that would make a kernel read or
write past its end is rejected before anything is launched."""
import pytest
import torch

from paper_2605_24793_gb300 import cospec as C


def _attn(B=3, R=6, Hq=32, Hkv=8, D=128, pages=40, P=16, maxp=9):
    bf = torch.bfloat16
    return dict(q=torch.empty(B, R, Hq, D, dtype=bf), k_blk=torch.empty(B, R, Hkv, D, dtype=bf),
                v_blk=torch.empty(B, R, Hkv, D, dtype=bf),
                k_pages=torch.empty(pages, Hkv, P, D, dtype=bf),
                v_pages=torch.empty(pages, Hkv, P, D, dtype=bf),
                page_table=torch.empty(B, maxp, dtype=torch.int32),
                ctx_len=torch.empty(B, dtype=torch.int32), out=torch.empty(B, R, Hq, D, dtype=bf))


def test_attention_shapes():
    t = _attn()
    C.check_attn_shapes(**t)
    bad = {
        "q": torch.empty(3, 6, 32 * 128, dtype=torch.bfloat16),            # not 4-D
        "k_blk": torch.empty(3, 5, 8, 128, dtype=torch.bfloat16),          # rows
        "v_blk": torch.empty(2, 6, 8, 128, dtype=torch.bfloat16),          # batch
        "k_pages": torch.empty(40, 8, 16, 64, dtype=torch.bfloat16),       # head_dim
        "v_pages": torch.empty(39, 8, 16, 128, dtype=torch.bfloat16),      # pool size
        "page_table": torch.empty(2, 9, dtype=torch.int32),                # batch
        "ctx_len": torch.empty(4, dtype=torch.int32),                      # batch
        "out": torch.empty(3, 6, 32, 64, dtype=torch.bfloat16),
    }
    for name, wrong in bad.items():
        case = dict(t, **{name: wrong})
        with pytest.raises(ValueError):
            C.check_attn_shapes(**case)


def test_arbitrate_shapes():
    B, K, H = 4, 5, 16
    ok = dict(draft=torch.empty(B, K, dtype=torch.int32),
              argmax=torch.empty(B, K + 1, dtype=torch.int32),
              stats=torch.empty(B, K + 1, 5), w1=torch.empty(H, 8), b1=torch.empty(H),
              w2=torch.empty(H), mode=C.POLICY_MLP, p_out=torch.empty(B, K),
              accept=torch.empty(B, K, dtype=torch.uint8))
    C.check_arbitrate_shapes(**ok)
    # the forced policies read no weights
    C.check_arbitrate_shapes(**dict(ok, w1=None, b1=None, w2=None, mode=C.POLICY_TARGET))
    for name, wrong in {"argmax": torch.empty(B, K, dtype=torch.int32),
                        "stats": torch.empty(B, K + 1, 4), "w1": torch.empty(H, 7),
                        "b1": torch.empty(H - 1), "w2": torch.empty(H + 1),
                        "p_out": torch.empty(B, K + 1),
                        "accept": torch.empty(B - 1, K, dtype=torch.uint8)}.items():
        with pytest.raises(ValueError):
            C.check_arbitrate_shapes(**dict(ok, **{name: wrong}))


def test_commit_shapes():
    B, K, L, Hkv, D, pages, P = 3, 4, 2, 8, 128, 30, 16
    bf = torch.bfloat16
    ok = dict(draft=torch.empty(B, K, dtype=torch.int32),
              argmax=torch.empty(B, K + 1, dtype=torch.int32),
              accept=torch.empty(B, K, dtype=torch.uint8),
              k_blk=torch.empty(L, B, K + 1, Hkv, D, dtype=bf),
              v_blk=torch.empty(L, B, K + 1, Hkv, D, dtype=bf),
              k_pages=torch.empty(L, pages, Hkv, P, D, dtype=bf),
              v_pages=torch.empty(L, pages, Hkv, P, D, dtype=bf),
              page_table=torch.empty(B, 5, dtype=torch.int32),
              ctx_len=torch.empty(B, dtype=torch.int32), accept_len=torch.empty(B, dtype=torch.int32),
              emitted=torch.empty(B, K + 1, dtype=torch.int32))
    C.check_commit_shapes(**ok)
    # one pool shared by every layer
    shared = torch.empty(1, pages, Hkv, P, D, dtype=bf)
    C.check_commit_shapes(**dict(ok, k_pages=shared, v_pages=shared))
    for name, wrong in {"argmax": torch.empty(B, K, dtype=torch.int32),
                        "accept": torch.empty(B, K + 1, dtype=torch.uint8),
                        "k_blk": torch.empty(L, B, K, Hkv, D, dtype=bf),
                        "v_blk": torch.empty(L + 1, B, K + 1, Hkv, D, dtype=bf),
                        "k_pages": torch.empty(L + 1, pages, Hkv, P, D, dtype=bf),
                        "v_pages": torch.empty(L, pages, Hkv, P, 64, dtype=bf),
                        "page_table": torch.empty(B + 1, 5, dtype=torch.int32),
                        "accept_len": torch.empty(B + 1, dtype=torch.int32),
                        "emitted": torch.empty(B, K, dtype=torch.int32)}.items():
        with pytest.raises(ValueError):
            C.check_commit_shapes(**dict(ok, **{name: wrong}))
    # block K/V whose head count or head_dim differs from the pools'
    with pytest.raises(ValueError):
        C.check_commit_shapes(**dict(ok, k_blk=torch.empty(L, B, K + 1, 4, D, dtype=bf),
                                     v_blk=torch.empty(L, B, K + 1, 4, D, dtype=bf)))
