"""The C-ABI library loads, exports every symbol include/aatc.h declares, and validates its
arguments on the host before touching the GPU (no GPU needed)."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "aatc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(aatc_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(aatc):
    names = _declared()
    assert "aatc_encode" in names and "aatc_decode_attention" in names and "aatc_plan_create" in names
    lib = ctypes.CDLL(aatc.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(aatc.SIGNATURES), "binding signatures must mirror the header"


def test_status_strings(aatc):
    lib = aatc.load()
    assert lib.aatc_status_string(0) == b"ok"
    assert lib.aatc_status_string(4) == b"workspace too small"
    assert lib.aatc_version() >= 200


def test_calibrate_rejects_bad_arguments(aatc):
    ck = np.zeros((1, 1, 16, 128), np.float32)
    with pytest.raises(aatc.AatcError) as e:
        aatc.calibrate(aatc.dims(1, 1, 4), ck, ck, None, 9.0)          # > b_max bits
    assert e.value.status == 2
    with pytest.raises(aatc.AatcError) as e:
        aatc.calibrate(aatc.dims(1, 1, 4), ck, ck, None, 2.755)        # 352.64 bits: not integral
    assert e.value.status == 2
    bad = aatc.Dims(64, 1, 1, 4, 8)                                    # d != 128
    with pytest.raises((aatc.AatcError, ValueError)):
        aatc.calibrate(bad, ck, ck, None, 2.0)
    with pytest.raises(aatc.AatcError) as e:
        aatc.calibrate(aatc.dims(1, 1, 3, 8), ck, ck, None, 2.0)       # 3 % 1 == 0 ok; b_max fine
        aatc.calibrate(aatc.Dims(128, 1, 2, 3, 8), np.zeros((1, 2, 16, 128), np.float32),
                       np.zeros((1, 2, 16, 128), np.float32), None, 2.0)   # 3 q-heads over 2 kv-heads
    assert e.value.status == 1


def test_plan_create_validates_before_any_cuda_call(aatc):
    lib = aatc.load()
    dm = aatc.dims(1, 1, 4)
    basis = np.tile(np.eye(128, dtype=np.float32), (2, 1, 1))
    scales = np.ones((2, 128), np.float32)
    h = ctypes.c_void_p()
    inc = np.zeros((2, 128), np.uint8)
    inc[0, 5] = 3                                                      # widths must be non-increasing
    assert lib.aatc_plan_create(ctypes.byref(dm), basis.ctypes.data, inc.ctypes.data, scales.ctypes.data, None,
                                ctypes.byref(h)) == 1
    big = np.full((2, 128), 9, np.uint8)                               # > b_max
    assert lib.aatc_plan_create(ctypes.byref(dm), basis.ctypes.data, big.ctypes.data, scales.ctypes.data, None,
                                ctypes.byref(h)) == 1
    ok_bits = np.full((2, 128), 2, np.uint8)
    zero_scale = scales.copy()
    zero_scale[1, 7] = 0.0                                             # scale must be > 0 where bits > 0
    assert lib.aatc_plan_create(ctypes.byref(dm), basis.ctypes.data, ok_bits.ctypes.data, zero_scale.ctypes.data,
                                None, ctypes.byref(h)) == 1
    nan_basis = basis.copy()
    nan_basis[0, 3, 3] = np.nan
    assert lib.aatc_plan_create(ctypes.byref(dm), nan_basis.ctypes.data, ok_bits.ctypes.data, scales.ctypes.data,
                                None, ctypes.byref(h)) == 1
    over = aatc.dims(1, 1, 4, b_max=17)                                # above the paper's 16
    assert lib.aatc_plan_create(ctypes.byref(over), basis.ctypes.data, ok_bits.ctypes.data, scales.ctypes.data,
                                None, ctypes.byref(h)) == 1
    wide = aatc.dims(1, 1, 4, b_max=16)
    many_wide = np.full((2, 128), 2, np.uint8)
    many_wide[1, :33] = 9                                              # 33 channels above 8 bits
    assert lib.aatc_plan_create(ctypes.byref(wide), basis.ctypes.data, many_wide.ctypes.data, scales.ctypes.data,
                                None, ctypes.byref(h)) == 5
    assert lib.aatc_plan_destroy(None) == 0
    # a plan handle without the live magic is rejected (use after destroy / garbage handle)
    junk = (ctypes.c_uint32 * 64)()
    assert lib.aatc_encode(ctypes.addressof(junk), 0, 16, 16, 1, 0, 1, 16, 1, None) == 1
    assert lib.aatc_decode_attention(ctypes.addressof(junk), 0, 16, 16, 1, 1, 1, 16, 16, 1 << 20, None) == 1
