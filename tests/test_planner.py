"""Host planner of the library (C++ through the C ABI) against the fp64 oracle planner (no GPU).

Widths must match exactly; sigma^2 and weights to 1e-9 relative; scales and basis to fp32
rounding (after the shared sign convention).  Sec. 5 Steps 1-2, Algorithm 1 calibration half.
"""
import numpy as np
import pytest

from oracle import aatc_oracle as O
import workloads as W


def _compare(aatc, cfg, avg_bits, anisotropic, var_only=False, n=W.N_CALIB):
    ck, cv, cq = W.layer_calibration(cfg, 0, anisotropic_queries=anisotropic, n=n)
    dm = aatc.dims(1, cfg.n_kv_heads, cfg.n_q_heads)
    lib = aatc.calibrate(dm, ck[None], cv[None], cq[None], avg_bits, var_only=var_only, n_threads=4)
    g = cfg.group
    for h in range(cfg.n_kv_heads):
        for kind, x in ((0, ck[h]), (1, cv[h])):
            qs = [cq[j].astype(np.float64) for j in range(h * g, (h + 1) * g)] if kind == 0 else None
            ref = O.plan_stream(x.astype(np.float64), avg_bits, queries_by_head=qs,
                                weights="var" if var_only else "aatc")
            got_bits = lib["bits"][0, h, kind].astype(np.int64)
            assert np.array_equal(got_bits, ref["bits"]), (h, kind)
            np.testing.assert_allclose(lib["sigma2"][0, h, kind], ref["sigma2"], rtol=1e-9, atol=1e-14)
            np.testing.assert_allclose(lib["weights"][0, h, kind], ref["weights"], rtol=1e-9)
            np.testing.assert_allclose(lib["scales"][0, h, kind], ref["scales"], rtol=2e-7)
            np.testing.assert_allclose(lib["basis"][0, h, kind], ref["basis"], atol=2e-7)
    return lib


@pytest.mark.parametrize("avg_bits", [1.5, 2.75, 4.0])
def test_planner_matches_oracle_tiny(aatc, avg_bits):
    _compare(aatc, W.CONFIGS["tiny"], avg_bits, anisotropic=False)


def test_planner_matches_oracle_gqa_anisotropic(aatc):
    """Two kv-heads, group 4, anisotropic queries: exercises w^K != const (Eq. waterfilling-keys)."""
    cfg = W.Config(9, "gqa", 1, 2, 8, 1, 256, (2.0,), 1, "planner test")
    lib = _compare(aatc, cfg, 2.0, anisotropic=True, n=2048)
    w = lib["weights"][0, 0, 0]
    assert w.max() / w.min() > 1.5          # the weighting is doing something
    assert np.all(lib["weights"][0, :, 1] == 1.0)


def test_planner_var_only(aatc):
    cfg = W.CONFIGS["tiny"]
    lib = _compare(aatc, cfg, 2.0, anisotropic=True, var_only=True, n=1024)
    assert np.all(lib["weights"] == 1.0)


def test_planner_layout_identity(aatc):
    """Widths non-increasing, budget met exactly, R and W as the paper's 2.75-bit point implies."""
    cfg = W.CONFIGS["tiny"]
    ck, cv, cq = W.layer_calibration(cfg, 0, n=1024)
    lib = aatc.calibrate(aatc.dims(1, 1, 4), ck[None], cv[None], cq[None], 2.75)
    b = lib["bits"].reshape(-1, 128).astype(int)
    assert np.all(np.diff(b, axis=1) <= 0)
    assert np.all(b.sum(axis=1) == 352)
    assert O.record_words(list(b)) == 11


def test_planner_up_to_16_bits_matches_oracle(aatc):
    """b_max = 16 (Sec. 5 allows b in 0..16): at 7 average bits the leading channels take more
    than 8 bits; widths match the oracle exactly and the budget is met."""
    cfg = W.CONFIGS["tiny"]
    ck, cv, cq = W.layer_calibration(cfg, 0, n=1024)
    lib = aatc.calibrate(aatc.dims(1, 1, 4, b_max=16), ck[None], cv[None], cq[None], 7.0)
    for kind, x in ((0, ck[0]), (1, cv[0])):
        qs = [cq[j].astype(np.float64) for j in range(4)] if kind == 0 else None
        ref = O.plan_stream(x.astype(np.float64), 7.0, b_max=16, queries_by_head=qs)
        got = lib["bits"][0, 0, kind].astype(np.int64)
        assert np.array_equal(got, ref["bits"])
        assert got.sum() == 7 * 128 and got.max() > 8 and got.max() <= 16
    with pytest.raises(aatc.AatcError) as e:
        aatc.calibrate(aatc.dims(1, 1, 4, b_max=17), ck[None], cv[None], cq[None], 7.0)
    assert e.value.status == 1
