"""Global cross-layer allocation (Eq. waterfilling-keys summed over layers; Algorithm 1 'Allocate
bits globally'; protected first layers and per-layer 95th-percentile normalisation from the AATC
experimental setup): the oracle pinned by brute force and by its invariants, then the library's
host planner checked against the oracle bit for bit."""
import itertools

import numpy as np
import pytest

from oracle import aatc_oracle as O


def _random_stats(rng, L, H, d, layer_scale=None):
    s2 = rng.lognormal(0.0, 1.5, (L, H, 2, d))
    s2 = -np.sort(-s2, axis=-1)                       # storage order: descending
    w = np.ones((L, H, 2, d))
    w[:, :, 0] = rng.lognormal(0.0, 0.7, (L, H, d))
    if layer_scale is not None:
        s2 *= np.asarray(layer_scale)[:, None, None, None]
    # storage order is by g = w sigma^2 descending within each stream
    for l in range(L):
        for h in range(H):
            for k in range(2):
                o = np.argsort(-(w[l, h, k] * s2[l, h, k]), kind="stable")
                s2[l, h, k] = s2[l, h, k][o]
                w[l, h, k] = w[l, h, k][o]
    return s2, w


def test_oracle_pool_is_optimal_by_brute_force():
    """Two unprotected layers, one head, d = 3, b_max = 3: the pooled greedy allocation reaches
    the minimum of sum g~ 4^-b over every integer allocation with the same total."""
    rng = np.random.default_rng(5)
    L, H, d, b_max = 2, 1, 3, 3
    for trial in range(20):
        s2, w = _random_stats(rng, L, H, d)
        avg = [1.0, 4.0 / 3.0][trial % 2]
        bits = O.global_allocation(s2, w, avg, avg, n_protect=0, b_max=b_max)
        for kind in (0, 1):
            g = []
            for l in range(L):
                ps = O.percentile_linear(s2[l, :, kind].ravel(), 95.0)
                pw = O.percentile_linear(w[l, :, kind].ravel(), 95.0)
                g.append(s2[l, 0, kind] / ps * w[l, 0, kind] / pw)
            g = np.concatenate(g)
            budget = int(round(avg * d)) * L * H
            best = min(np.sum(g * 4.0 ** -np.array(b)) for b in itertools.product(range(b_max + 1), repeat=L * d)
                       if sum(b) == budget)
            got = np.sum(g * 4.0 ** -bits[:, 0, kind].ravel())
            assert got == pytest.approx(best, rel=1e-12)
            assert bits[:, :, kind].sum() == budget


def test_oracle_layer_normalisation_makes_layer_scale_irrelevant():
    """Scaling sigma^2 (or w) of one layer by a constant leaves the allocation unchanged: the
    per-layer 95th-percentile normalisation removes it (the point of that normalisation)."""
    rng = np.random.default_rng(6)
    s2, w = _random_stats(rng, 6, 2, 128)
    base = O.global_allocation(s2, w, 2.75, 2.75, n_protect=3)
    s2b = s2.copy()
    s2b[4] *= 37.0
    wb = w.copy()
    wb[3, :, 0] *= 0.01
    assert np.array_equal(O.global_allocation(s2b, w, 2.75, 2.75, n_protect=3), base)
    assert np.array_equal(O.global_allocation(s2, wb, 2.75, 2.75, n_protect=3), base)
    # a pool without the normalisation would move bits towards the louder layer
    g_raw = np.concatenate([(w[l, :, 1] * s2b[l, :, 1]).ravel() for l in range(3, 6)])
    raw = O.greedy_allocation(g_raw, 352 * 3 * 2, 8).reshape(3, 2, 128)
    assert raw[1].sum() > base[4, :, 1].sum()


def test_oracle_protected_layers_and_budget():
    rng = np.random.default_rng(7)
    L, H, d = 6, 2, 128
    s2, w = _random_stats(rng, L, H, d)
    bits = O.global_allocation(s2, w, 2.75, 2.75, n_protect=3)
    for l in range(3):
        for h in range(H):
            assert bits[l, h, 1].sum() == 352                       # average for values
            assert bits[l, h, 0].sum() == 352 + 128                 # one bit more for keys
            assert np.array_equal(bits[l, h, 0], O.greedy_allocation(w[l, h, 0] * s2[l, h, 0], 480, 8))
    assert bits[:, :, 0].sum() == 352 * L * H and bits[:, :, 1].sum() == 352 * L * H
    assert (np.diff(bits, axis=-1) <= 0).all()                       # non-increasing per stream
    assert bits.max() <= 8


@pytest.mark.parametrize("L,H,n_protect,avg", [(6, 2, 3, 2.75), (5, 8, 3, 2.0), (4, 2, 3, 4.0), (4, 4, 0, 1.5), (1, 8, 0, 2.75)])
def test_library_global_allocation_matches_oracle(aatc, L, H, n_protect, avg):
    rng = np.random.default_rng(100 + L * 10 + H)
    s2, w = _random_stats(rng, L, H, 128, layer_scale=np.exp(rng.normal(0, 2, L)))
    dm = aatc.dims(L, H, 4 * H)
    got = aatc.allocate_global(dm, s2, w, avg, avg, n_protect=n_protect)
    want = O.global_allocation(s2, w, avg, avg, n_protect=n_protect)
    assert np.array_equal(got.astype(np.int64), want)


@pytest.mark.parametrize("L,H,n_protect,avg", [(5, 2, 3, 6.0), (4, 2, 0, 9.0)])
def test_library_global_allocation_up_to_16_bits_matches_oracle(aatc, L, H, n_protect, avg):
    """Widths in {0..16} (the paper's range): the pool gives some channels more than 8 bits and
    the library still matches the oracle bit for bit."""
    rng = np.random.default_rng(200 + L * 10 + H)
    s2, w = _random_stats(rng, L, H, 128, layer_scale=np.exp(rng.normal(0, 2, L)))
    dm = aatc.dims(L, H, 4 * H, b_max=16)
    got = aatc.allocate_global(dm, s2, w, avg, avg, n_protect=n_protect).astype(np.int64)
    want = O.global_allocation(s2, w, avg, avg, n_protect=n_protect, b_max=16)
    assert np.array_equal(got, want)
    assert got.max() > 8 and got.max() <= 16


def test_library_global_allocation_rejects_bad_budgets(aatc):
    rng = np.random.default_rng(3)
    s2, w = _random_stats(rng, 4, 2, 128)
    dm = aatc.dims(4, 2, 8)
    with pytest.raises(RuntimeError):
        aatc.allocate_global(dm, s2, w, 2.7, 2.75)                  # not a multiple of 1/128
    with pytest.raises(RuntimeError):
        aatc.allocate_global(dm, s2, w, 2.0, 2.0, n_protect=3)      # protected keys exceed the total
    with pytest.raises(RuntimeError):
        aatc.allocate_global(aatc.dims(3, 2, 8), s2[:3], w[:3], 4.0, 4.0, n_protect=3)   # keys over budget
    with pytest.raises(ValueError):
        O.global_allocation(s2[:3], w[:3], 4.0, 4.0, n_protect=3)
    bad = s2.copy()
    bad[1, 0, 0, 5] = np.nan
    with pytest.raises(RuntimeError):
        aatc.allocate_global(dm, bad, w, 2.75, 2.75)
