"""Least-squares calibration of the batch-time coefficients on the GPU vs the oracle (Sec. 4.1).

The GPU accumulates the normal equations with fp64 atomics and solves them by a
scaled Cholesky factorization; the oracle solves each model's least-squares
problem with an SVD.  Both are accurate to far better than the tolerance below
on these well-conditioned logs, so the coefficients must agree to 1e-7 relative.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu
RTOL = 1e-7


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def R():
    from paper_2607_18253_gb300 import router
    return router


def router_for(M):
    wl = W.small_workload(0, num_instances=M, num_models=M, budget_range=(8, 96), min_gap=8)
    return R().LatencyRouter.from_workload(wl)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def coef_of(M, seed):
    rng = np.random.default_rng(seed)
    a = rng.uniform(3.0, 10.0, M)
    b = rng.uniform(0.05, 0.12, M)
    g = b + rng.uniform(0.1, 0.4, M)
    return W.coefficients(a, b, g).astype(np.float64)


@pytest.mark.parametrize("grouped", [True, False])
@pytest.mark.parametrize("shared", [True, False])
def test_calibration_matches_the_oracle(grouped, shared):
    M = 6
    coef = coef_of(M, 1)
    F, m, t = W.batch_log(300_000 if grouped else 60_000, M, seed=2, coef=coef, noise=0.04, grouped=grouped)
    rt = router_for(M)
    for _ in range(2):  # a second call starts from fresh sums
        got = rt.calibrate(dev(F), dev(m), dev(t), shared_beta1=shared).cpu().numpy()
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        np.testing.assert_allclose(got, oracle.calibrate(F, m, t, M, shared_beta1=shared), rtol=RTOL)


def test_noiseless_log_recovers_the_coefficients():
    M = 3
    coef = coef_of(M, 3)
    F, m, t = W.batch_log(50_000, M, seed=4, coef=coef, noise=0.0)
    got = router_for(M).calibrate(dev(F), dev(m), dev(t), shared_beta1=False).cpu().numpy()
    np.testing.assert_allclose(got, coef, rtol=1e-9)


def test_missing_models_and_bad_rows():
    M = 4
    coef = coef_of(M, 5)
    F, m, t = W.batch_log(20_000, M, seed=6, coef=coef, noise=0.02)
    m = m.copy()
    m[m == 3] = 0        # model 3 absent
    m[:3] = 2            # model 2: just three rows
    m[m == 2] = 1
    m[:3] = 2
    rt = router_for(M)
    got = rt.calibrate(dev(F), dev(m), dev(t), shared_beta1=True).cpu().numpy()
    ref = oracle.calibrate(F, m, t, M, shared_beta1=True)
    assert np.all(np.isnan(got[2:])) and np.all(np.isnan(ref[2:]))
    np.testing.assert_allclose(got[:2], ref[:2], rtol=RTOL)
    assert rt.status() == R().LR_OK
    bad = m.copy()
    bad[10] = 99
    t2 = t.copy()
    t2[11] = np.nan
    got = rt.calibrate(dev(F), dev(bad), dev(t2), shared_beta1=True).cpu().numpy()
    assert rt.status() == R().LR_EINVAL
    keep = np.ones(len(m), bool)
    keep[[10, 11]] = False
    np.testing.assert_allclose(got[:2], oracle.calibrate(F[keep], m[keep], t[keep], M)[:2], rtol=RTOL)


def test_unaligned_inputs_take_the_direct_path():
    # arrays starting one row in are not 16-byte aligned: the kernel reads rows directly
    M = 4
    coef = coef_of(M, 7)
    F, m, t = W.batch_log(100_001, M, seed=8, coef=coef, noise=0.03)
    Fd, md, td = dev(F), dev(m), dev(t)
    rt = router_for(M)
    got = rt.calibrate(Fd[1:], md[1:], td[1:], shared_beta1=False).cpu().numpy()
    assert rt.status() == R().LR_OK
    np.testing.assert_allclose(got, oracle.calibrate(F[1:], m[1:], t[1:], M, shared_beta1=False), rtol=RTOL)
    aligned = rt.calibrate(Fd, md, td, shared_beta1=False).cpu().numpy()
    np.testing.assert_allclose(aligned, oracle.calibrate(F, m, t, M, shared_beta1=False), rtol=RTOL)


def test_large_values_take_the_exact_128_bit_path():
    # features at or above 2^26 (up to just below 2^32) and times at or above 2^8 s skip
    # the 64-bit register sums and add to the 128-bit sums directly; rows of both kinds
    # interleave within warps
    M = 3
    coef = coef_of(M, 9)
    F, m, t = W.batch_log(40_000, M, seed=10, coef=coef, noise=0.03)
    F = F.copy()
    t = t.copy()
    big = np.arange(len(t)) % 3 == 0
    F[big, 3] *= 64      # up to ~6.7e7 > 2^26
    F[big, 4] = np.minimum(F[big, 4] * 64, (1 << 32) - 1)
    slow = np.arange(len(t)) % 7 == 0
    t[slow] += 300.0     # beyond 2^8 s
    assert (F[big] >> 26).any() and (t[slow] >= 256.0).all() and (F < (1 << 32)).all()
    rt = router_for(M)
    for shared in (True, False):
        got = rt.calibrate(dev(F), dev(m), dev(t), shared_beta1=shared).cpu().numpy()
        assert rt.status() == R().LR_OK
        np.testing.assert_allclose(got, oracle.calibrate(F, m, t, M, shared_beta1=shared), rtol=RTOL)


def test_many_models():
    # 128 models, the most the kernel takes: its shared sums leave room for two stages
    M = 128
    coef = coef_of(M, 11)
    F, m, t = W.batch_log(400_000, M, seed=12, coef=coef, noise=0.04, grouped=True)
    got = router_for(M).calibrate(dev(F), dev(m), dev(t), shared_beta1=False).cpu().numpy()
    np.testing.assert_allclose(got, oracle.calibrate(F, m, t, M, shared_beta1=False), rtol=RTOL)


def test_long_slices_flush_within_128_rows():
    # more than 128 rows a consumer lane (10M rows over one CTA per SM): the warps flush
    # their 64-bit sums before they could overflow, mid-model
    M = 2
    coef = coef_of(M, 13)
    F, m, t = W.batch_log(10_000_000, M, seed=14, coef=coef, noise=0.02)
    rt = router_for(M)
    got = rt.calibrate(dev(F), dev(m), dev(t), shared_beta1=True).cpu().numpy()
    assert rt.status() == R().LR_OK
    np.testing.assert_allclose(got, oracle.calibrate(F, m, t, M, shared_beta1=True), rtol=RTOL)
