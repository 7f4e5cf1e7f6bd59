"""Plan files (calibration once per model, Algorithm 1's offline half): the host arrays of a plan
survive a save / load bit for bit, and damaged or mismatched files are refused (no GPU)."""
import os

import numpy as np
import pytest

import workloads as W


def _random_plan(rng, dm):
    shape = (dm.n_layers, dm.n_kv_heads, 2, 128)
    basis = rng.standard_normal(shape + (128,)).astype(np.float32)
    basis.reshape(-1)[:7] = [0.0, -0.0, np.inf, -np.inf, np.nan, 1e-45, -3.4e38]   # every bit pattern kept
    bits = np.sort(rng.integers(0, dm.b_max + 1, shape), axis=-1)[..., ::-1].astype(np.uint8)
    scales = rng.uniform(0.1, 9.0, shape).astype(np.float32)
    return basis, bits, scales


@pytest.mark.parametrize("L,H,G,b_max", [(1, 1, 4, 8), (3, 2, 8, 16)])
def test_round_trip_is_bit_exact(aatc, tmp_path, L, H, G, b_max):
    dm = aatc.dims(L, H, G, b_max=b_max)
    basis, bits, scales = _random_plan(np.random.default_rng(L * 10 + H), dm)
    path = str(tmp_path / "plan.aatc")
    aatc.save_plan(path, dm, basis, bits, scales)
    dm2, p = aatc.load_plan(path)
    assert (dm2.d, dm2.n_layers, dm2.n_kv_heads, dm2.n_q_heads, dm2.b_max) == (128, L, H, G, b_max)
    assert np.array_equal(p["basis"].view(np.uint32), basis.view(np.uint32))
    assert np.array_equal(p["bits"], bits)
    assert np.array_equal(p["scales"].view(np.uint32), scales.view(np.uint32))
    # header 48 B + payload + 8 B checksum
    S = L * H * 2
    assert os.path.getsize(path) == 48 + S * 128 * 128 * 4 + S * 128 + S * 128 * 4 + 8


def test_calibrated_plan_round_trip(aatc, tmp_path):
    cfg = W.CONFIGS["tiny"]
    ck, cv, cq = W.layer_calibration(cfg, 0, n=1024)
    dm = aatc.dims(1, 1, 4)
    cal = aatc.calibrate(dm, ck[None], cv[None], cq[None], 2.75)
    path = str(tmp_path / "tiny.aatc")
    aatc.save_plan(path, dm, cal["basis"], cal["bits"], cal["scales"])
    _, p = aatc.load_plan(path)
    for k in ("basis", "bits", "scales"):
        assert np.array_equal(p[k], cal[k].reshape(p[k].shape)), k


def test_damaged_files_are_refused(aatc, tmp_path):
    dm = aatc.dims(1, 2, 4)
    basis, bits, scales = _random_plan(np.random.default_rng(3), dm)
    path = str(tmp_path / "p.aatc")
    aatc.save_plan(path, dm, basis, bits, scales)
    good = open(path, "rb").read()

    def refused(data, status=9):
        bad = str(tmp_path / "bad.aatc")
        with open(bad, "wb") as f:
            f.write(data)
        with pytest.raises(aatc.AatcError) as e:
            aatc.load_plan(bad)
        assert e.value.status == status

    flipped = bytearray(good)
    flipped[48 + 1000] ^= 0x10                               # one payload bit: checksum mismatch
    refused(bytes(flipped))
    refused(good[:-1])                                       # short
    refused(good + b"\0")                                    # trailing bytes
    refused(b"AATCPLAX" + good[8:])                          # magic
    v2 = bytearray(good)
    v2[8] = 2                                                # version
    refused(bytes(v2))
    dims_bad = bytearray(good)
    dims_bad[16] = 64                                        # d = 64
    refused(bytes(dims_bad))
    wide = bytearray(good)
    off_bits = 48 + 2 * 2 * 128 * 128 * 4
    wide[off_bits] = 9                                       # a width above b_max, checksum refreshed below
    import struct
    payload = bytes(wide[48:-8])
    h = 1469598103934665603
    for byte in payload:
        h = ((h ^ byte) * 1099511628211) & 0xFFFFFFFFFFFFFFFF
    refused(bytes(wide[:-8]) + struct.pack("<Q", h))
    with pytest.raises(aatc.AatcError) as e:
        aatc.load_plan(str(tmp_path / "missing.aatc"))
    assert e.value.status == 9


def test_save_and_load_argument_errors(aatc, tmp_path):
    dm = aatc.dims(1, 1, 4)
    basis, bits, scales = _random_plan(np.random.default_rng(4), dm)
    bits[0, 0, 0, 0] = 9                                     # above b_max = 8
    with pytest.raises(aatc.AatcError) as e:
        aatc.save_plan(str(tmp_path / "x.aatc"), dm, basis, bits, scales)
    assert e.value.status == 1
    with pytest.raises(aatc.AatcError) as e:                 # directory that does not exist
        aatc.save_plan(str(tmp_path / "no" / "x.aatc"), dm, basis, np.zeros_like(bits), scales)
    assert e.value.status == 9
    # loading into dims that differ from the file's
    path = str(tmp_path / "ok.aatc")
    aatc.save_plan(path, dm, basis, np.zeros_like(bits), scales)
    lib = aatc.load()
    import ctypes
    other = aatc.dims(1, 1, 8)
    out_b = np.empty_like(basis)
    out_w = np.empty_like(bits)
    out_s = np.empty_like(scales)
    assert lib.aatc_plan_load(os.fsencode(path), ctypes.byref(other), out_b.ctypes.data, out_w.ctypes.data,
                              out_s.ctypes.data) == 1
