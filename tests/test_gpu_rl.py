"""RL-stage rewards and advantages on the device (Sec. 3.4) against the
oracle, through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import cospec_rl as RL
from paper_2605_24793_gb300 import build as BLD
from paper_2605_24793_gb300 import cospec as C

from .parity_util import assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    C.load_library(BLD.build())
    torch.cuda.set_device(0)
    assert C.get_device_error() == 0


def _batch(rng, groups, K, mode, max_m=6, max_r=8):
    group_off = [0]; correct = []; round_off = [0]
    match, accept, ell = [], [], []
    for x in range(groups):
        for m in range(int(rng.integers(1, max_m + 1))):
            c = {"mixed": rng.random() < 0.5, "pos": True, "neg": False}[mode]
            correct.append(int(c))
            for r in range(int(rng.integers(0, max_r + 1))):      # rollouts with no round too
                d = (rng.random(K) < 0.6).astype(np.uint8)
                a = np.where(d == 1, 1, (rng.random(K) < 0.5)).astype(np.uint8)
                match.append(d); accept.append(a)
                ell.append((-rng.exponential(1.5, K)).astype(np.float32))
            round_off.append(len(match))
        group_off.append(len(correct))
    R = len(match)
    return (np.array(group_off, np.int32), np.array(correct, np.uint8), np.array(round_off, np.int32),
            K, np.array(match, np.uint8).reshape(R, K), np.array(accept, np.uint8).reshape(R, K),
            np.array(ell, np.float32).reshape(R, K))


def _run(batch, obj=None, prm=None):
    go, co, ro, K, ma, ac, el = batch
    cu = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    kw = {}
    if obj is not None:
        kw = dict(ratio=cu(obj[0]), p_new=cu(obj[1]), p_ref=cu(obj[2]))
    out = C.rl_advantages(cu(go), cu(co), cu(ro), cu(ma), cu(ac), cu(el), prm, **kw)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _compare(got, ref):
    assert np.array_equal(got["eff"], ref["eff"])
    assert_close(got["g"], ref["g"], "g")
    assert np.array_equal(np.isnan(got["rho"]), np.isnan(ref["rho"]))
    assert_close(got["rho"][~np.isnan(ref["rho"])], ref["rho"][~np.isnan(ref["rho"])], "rho")
    for k in ("J", "Jbar", "adv", "adv_dec"):
        assert_close(got[k], ref[k], k)


def test_hand_case():
    go, co, ro = np.array([0, 2], np.int32), np.array([1, 0], np.uint8), np.array([0, 2, 4], np.int32)
    ma = np.array([[1, 0, 0], [1, 1, 1], [0, 1, 0], [0, 0, 1]], np.uint8)
    ac = np.array([[1, 1, 0], [1, 1, 1], [1, 1, 1], [0, 1, 1]], np.uint8)
    el = np.array([[0, -1, -3], [0, 0, 0], [-2, 0, -0.5], [-1.5, -0.7, 0]], np.float32)
    got = _run((go, co, ro, 3, ma, ac, el))
    np.testing.assert_allclose(got["J"], [1.0, -2.75], rtol=1e-6)
    np.testing.assert_allclose(got["adv"], [1.0, -1.0], rtol=1e-5)
    np.testing.assert_allclose(got["adv_dec"][2], [-2 / 2.75, 0, -0.5 / 2.75], rtol=1e-5)


@pytest.mark.parametrize("mode", ["mixed", "pos", "neg"])
@pytest.mark.parametrize("K", [6, 25, 64])
def test_matches_oracle(mode, K):
    rng = np.random.default_rng(K * 10 + {"mixed": 1, "pos": 2, "neg": 3}[mode])
    batch = _batch(rng, 60, K, mode)
    R = batch[4].shape[0]
    obj = (rng.uniform(0.5, 1.5, (R, K)).astype(np.float32),
           rng.uniform(0.05, 0.95, (R, K)).astype(np.float32),
           rng.uniform(0.05, 0.95, (R, K)).astype(np.float32))
    got = _run(batch, obj)
    ref = RL.rl_advantages(*batch, RL.RLParams(), ratio=obj[0], p_new=obj[1], p_ref=obj[2])
    _compare(got, ref)
    assert_close(got["loss"], np.array(ref["loss_terms"]), "objective terms")
    assert C.get_device_error() == 0


def test_large_batch_and_many_rounds():
    # 512 prompt groups of 8 rollouts with up to 48 rounds at K = 25
    rng = np.random.default_rng(99)
    batch = _batch(rng, 512, 25, "mixed", max_m=8, max_r=48)
    got = _run(batch)
    ref = RL.rl_advantages(*batch, RL.RLParams())
    _compare(got, ref)


def test_bad_offsets_set_the_error_bit_and_skip_the_group():
    rng = np.random.default_rng(5)
    go, co, ro, K, ma, ac, el = _batch(rng, 4, 5, "mixed")
    go = go.copy()
    go[2] = go[1] - 1                                # group 1 runs backwards
    _run((go, co, ro, K, ma, ac, el))
    assert C.get_device_error() & C.DEVERR_OFFSETS
    assert C.get_device_error() == 0                 # read and cleared


def test_host_validation():
    lib = C.load_library()
    p = C.RLParams()
    fake = C.ctypes.c_void_p(1 << 20)
    args = lambda K, pr, ratio=None: (1, 1, 1, K, fake, fake, fake, fake, fake, fake,
                                      C.ctypes.byref(pr), ratio, None, None, fake, fake, fake, fake,
                                      fake, fake, fake, None, fake, 1 << 20, None)
    assert lib.cospec_rl_advantages(*args(0, p)) == -1              # K outside [1, 64]
    assert lib.cospec_rl_advantages(*args(65, p)) == -1
    assert lib.cospec_rl_advantages(*args(5, p, ratio=fake)) == -1  # objective inputs: all or none
    bad = C.RLParams(eps=0.0)
    assert lib.cospec_rl_advantages(*args(5, bad)) == -1
