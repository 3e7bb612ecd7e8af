"""The estimators of include/fp_estimate.h (Eqs. 1-3, Sec. 5.3; the linear
memory model, Sec. 5.2) against the oracle's plain solves.  Host functions
of the library: no GPU."""
import numpy as np
import pytest

from oracle import estimator as E


@pytest.fixture(scope="module")
def fp():
    import __graft_entry__

    __graft_entry__.build()
    import paper_2501_13111_gb300 as fp

    return fp


def test_eq1_eq23_and_prediction_match_the_oracle(fp):
    rng = np.random.default_rng(7)
    for _ in range(50):
        la, lb = sorted(rng.choice(np.arange(1, 500), 2, replace=False))
        lat = rng.uniform(1, 100, 4)
        f1 = fp.fp_solve_eq1(int(la), lat[0], int(lb), lat[1])
        f2 = fp.fp_solve_eq1(int(la), lat[2], int(lb), lat[3])
        r1, r2 = E.solve_eq1(la, lat[0], lb, lat[1]), E.solve_eq1(la, lat[2], lb, lat[3])
        np.testing.assert_allclose([f1.ttft, f1.tpot], r1, rtol=1e-9, atol=1e-9)
        np.testing.assert_allclose([f2.ttft, f2.tpot], r2, rtol=1e-9, atol=1e-9)
        t = fp.fp_solve_eq23(1, f1, 2, f2)
        rt = E.solve_eq23(1, r1[0], r1[1], 2, r2[0], r2[1])
        np.testing.assert_allclose([t.ttft_layer, t.ttft_other, t.tpot_layer, t.tpot_other], rt, rtol=1e-9, atol=1e-9)
        L, N = int(rng.integers(1, 81)), int(rng.integers(1, 2000))
        np.testing.assert_allclose(fp.fp_predict_latency(t, L, N), E.predict_latency(L, N, *rt), rtol=1e-9)


def test_linear_data_is_recovered_exactly(fp):
    # latency(L, n) = L (3 + 0.5 n) + (7 + 0.25 n): every term is recovered
    lat = lambda L, n: L * (3 + 0.5 * n) + (7 + 0.25 * n)
    fits = {L: fp.fp_solve_eq1(16, lat(L, 16), 64, lat(L, 64)) for L in (1, 2)}
    t = fp.fp_solve_eq23(1, fits[1], 2, fits[2])
    assert (t.ttft_layer, t.ttft_other, t.tpot_layer, t.tpot_other) == pytest.approx((3, 7, 0.5, 0.25))
    assert fp.fp_predict_latency(t, 32, 100) == pytest.approx(lat(32, 100))
    assert fp.fp_extrapolate_memory(1, 10.0, 2, 13.0, 80) == pytest.approx(10 + 3 * 79)
    assert fp.fp_extrapolate_memory(2, 13.0, 1, 10.0, 80) == pytest.approx(E.extrapolate_memory(2, 13.0, 1, 10.0, 80))


def test_singular_systems_are_rejected(fp):
    with pytest.raises(fp.FPError):
        fp.fp_solve_eq1(16, 1.0, 16, 2.0)
    f = fp.fp_solve_eq1(16, 1.0, 64, 2.0)
    with pytest.raises(fp.FPError):
        fp.fp_solve_eq23(2, f, 2, f)
    with pytest.raises(fp.FPError):
        fp.fp_extrapolate_memory(1, 1.0, 1, 2.0, 4)
