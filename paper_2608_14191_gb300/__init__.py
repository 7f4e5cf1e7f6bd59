"""GB300 (sm_103a) hot path of Attention-Aware Transform Coding (AATC), arxiv 2608.14191.

Thin Python binding over the C ABI in ``include/aatc.h`` (library ``libaatc.so`` built in-tree
by :mod:`paper_2608_14191_gb300.build`).  The binding only marshals arguments: PyTorch
tensors provide device memory and the current CUDA stream; every step of the path runs in
the library.  There is no fallback: if the shared object is missing the import of
:data:`lib` raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HEAD_DIM = 128
_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libaatc.so")

_STATUS = {
    0: "ok", 1: "invalid argument", 2: "bit budget not representable", 3: "token range exceeds cache capacity",
    4: "workspace too small", 5: "unsupported shape", 6: "CUDA error", 7: "out of memory", 8: "device error flag set",
    9: "plan file unreadable or corrupt",
}


class AatcError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = f"{where}: {_STATUS.get(status, 'unknown')} (status {status})"
        if status == 6 and _lib is not None:
            msg += f", cudaError {_lib.aatc_last_cuda_error()}"
        super().__init__(msg)


class Dims(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("n_layers", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("b_max", ctypes.c_int32)]


_lib = None
_P, _I32, _SZ, _F64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t, ctypes.c_double

# name -> (restype, argtypes); mirrors include/aatc.h
SIGNATURES = {
    "aatc_status_string": (ctypes.c_char_p, [_I32]),
    "aatc_last_cuda_error": (_I32, []),
    "aatc_version": (_I32, []),
    "aatc_calibrate": (_I32, [ctypes.POINTER(Dims), _P, _P, _I32, _P, _I32, _F64, _F64, _I32, _P, _P, _P, _P, _P, _I32]),
    "aatc_calibrate_head_group": (_I32, [_I32, _I32, _P, _I32, _P, _I32, _F64, _I32, _I32, _P, _P, _P, _P, _P]),
    "aatc_selftest_bounded_wait": (_I32, [_I32, _P, _P]),
    "aatc_plan_save": (_I32, [ctypes.c_char_p, _P, _P, _P, _P]),
    "aatc_plan_file_dims": (_I32, [ctypes.c_char_p, _P]),
    "aatc_plan_load": (_I32, [ctypes.c_char_p, _P, _P, _P, _P]),
    "aatc_allocate_global": (_I32, [ctypes.POINTER(Dims), _P, _P, _F64, _F64, _I32, _P]),
    "aatc_whitening_transform": (_I32, [_I32, _I32, _P, _P, _P, _P, _P, _P, _P]),
    "aatc_hidden_operand": (_I32, [ctypes.POINTER(Dims), _I32, _P, _P, _P, _P]),
    "aatc_encode_hidden": (_I32, [_P, _I32, _P, _I32, _P, _I32, _I32, _I32, _P, _I32, _P]),
    "aatc_prefill_workspace_bytes": (_I32, [_P, _I32, _I32, ctypes.POINTER(_SZ)]),
    "aatc_prefill_attention": (_I32, [_P, _I32, _P, _I32, _I32, _P, _I32, _I32, _I32, _P, _P, _SZ, _P]),
    "aatc_decode_attention_sw": (_I32, [_P, _I32, _P, _P, _I32, _I32, _I32, _I32, _P, _P, _I32, _I32, _P, _P, _SZ,
                                        _P]),
    "aatc_plan_create": (_I32, [ctypes.POINTER(Dims), _P, _P, _P, _P, ctypes.POINTER(_P)]),
    "aatc_group_plan_create": (_I32, [_P, _I32, _P, _P, _P, _P, _P]),
    "aatc_plan_destroy": (_I32, [_P]),
    "aatc_plan_info": (_I32, [_P, ctypes.POINTER(_I32), _P]),
    "aatc_cache_bytes": (_I32, [_P, _I32, _I32, ctypes.POINTER(_SZ)]),
    "aatc_encode": (_I32, [_P, _I32, _P, _P, _I32, _I32, _I32, _P, _I32, _P]),
    "aatc_decode_workspace_bytes": (_I32, [_P, _I32, _I32, ctypes.POINTER(_SZ)]),
    "aatc_decode_attention": (_I32, [_P, _I32, _P, _P, _I32, _I32, _I32, _P, _P, _SZ, _P]),
    "aatc_decode_attention_noalloc": (_I32, [_P, _I32, _P, _P, _I32, _I32, _I32, _P, _P]),
    "aatc_dequantize": (_I32, [_P, _I32, _P, _I32, _I32, _I32, _I32, _P, _P]),
    "aatc_get_device_error": (_I32, [_P, ctypes.POINTER(_I32), _I32]),
    "aatc_bf16_decode_workspace_bytes": (_I32, [_I32, _I32, _I32, _I32, ctypes.POINTER(_SZ)]),
    "aatc_bf16_decode_attention": (_I32, [_P, _P, _P, _I32, _I32, _I32, _I32, _I32, _P, _P, _SZ, _P]),
}


def load(path: str = LIB_PATH):
    """Load libaatc.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(status: int, where: str):
    if status != 0:
        raise AatcError(status, where)


def _ptr(a) -> int:
    """Address of a torch tensor or numpy array (must be contiguous)."""
    if hasattr(a, "data_ptr"):
        if not a.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return a.data_ptr()
    if not a.flags["C_CONTIGUOUS"]:
        raise ValueError("array must be C-contiguous")
    return a.ctypes.data


def _stream(stream=None) -> int:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


try:                      # the binding's device helpers compare against torch dtypes
    import torch as _torch
    _F32 = _torch.float32
except ImportError:       # host-only use (planner, plan files) works without torch
    _F32 = None


def _arg_error(where: str, what: str):
    raise AatcError(1, f"{where} ({what})")


_DEVICE_TYPE = "cuda"     # where device arguments must live


def _on_device(t) -> bool:
    try:
        return t.is_cuda if _DEVICE_TYPE == "cuda" else t.device.type == _DEVICE_TYPE
    except AttributeError:
        return False


def _dev_tensor(t, where: str, name: str, dtype=None, ndim: int | None = None, shape=None):
    """Checks a device argument before its pointer goes to the library, which cannot see sizes:
    a CUDA tensor, of `dtype`, with `ndim` dimensions and the given sizes (None = any)."""
    if not _on_device(t):
        _arg_error(where, f"{name} must be a {_DEVICE_TYPE} tensor")
    if dtype is not None and t.dtype != dtype:
        _arg_error(where, f"{name} must be {dtype}, not {t.dtype}")
    sh = t.shape
    if ndim is not None and len(sh) != ndim:
        _arg_error(where, f"{name} must have {ndim} dimensions, not {len(sh)}")
    if shape is not None:
        for i, n in enumerate(shape):
            if n is not None and sh[i] != n:
                _arg_error(where, f"{name} size {i} must be {n}, not {sh[i]}")


def _cache_ok(plan, cache, batch: int, max_tokens: int, where: str):
    if not _on_device(cache):
        _arg_error(where, f"cache must be a {_DEVICE_TYPE} tensor")
    need = plan.cache_bytes(batch, max_tokens)
    if cache.nbytes < need:
        _arg_error(where, f"cache holds {cache.nbytes} bytes, {need} needed")


def _out_ok(out, n: int, where: str):
    if not _on_device(out) or out.dtype != _F32:
        _arg_error(where, f"out must be a {_DEVICE_TYPE} tensor of torch.float32")
    if out.numel() < n:
        _arg_error(where, f"out holds {out.numel()} values, {n} needed")


def dims(n_layers: int, n_kv_heads: int, n_q_heads: int, b_max: int = 8) -> Dims:
    return Dims(HEAD_DIM, n_layers, n_kv_heads, n_q_heads, b_max)


def calibrate(dm: Dims, calib_k: np.ndarray, calib_v: np.ndarray, calib_q: np.ndarray | None,
              avg_bits_k: float, avg_bits_v: float | None = None, var_only: bool = False,
              n_threads: int = 0):
    """Host planner (Sec. 5 Steps 1-2).  calib_k/v: fp32 [L][H_kv][N][128]; calib_q: fp32
    [L][H_q][Nq][128] or None.  Returns dict(basis, bits, scales, sigma2, weights)."""
    lib = load()
    ck = np.ascontiguousarray(calib_k, dtype=np.float32)
    cv = np.ascontiguousarray(calib_v, dtype=np.float32)
    cq = None if calib_q is None else np.ascontiguousarray(calib_q, dtype=np.float32)
    L, H = dm.n_layers, dm.n_kv_heads
    if ck.shape[:2] != (L, H) or ck.shape[3] != HEAD_DIM or cv.shape != ck.shape:
        raise ValueError("calibration arrays must be [L][H_kv][N][128]")
    if cq is not None and (cq.shape[:2] != (L, dm.n_q_heads) or cq.shape[3] != HEAD_DIM):
        raise ValueError("calibration queries must be [L][H_q][Nq][128]")
    S = L * H * 2
    basis = np.empty((L, H, 2, HEAD_DIM, HEAD_DIM), np.float32)
    bits = np.empty((L, H, 2, HEAD_DIM), np.uint8)
    scales = np.empty((L, H, 2, HEAD_DIM), np.float32)
    sigma2 = np.empty((L, H, 2, HEAD_DIM), np.float64)
    weights = np.empty((L, H, 2, HEAD_DIM), np.float64)
    st = lib.aatc_calibrate(ctypes.byref(dm), _ptr(ck), _ptr(cv), ck.shape[2], None if cq is None else _ptr(cq),
                            0 if cq is None else cq.shape[2], float(avg_bits_k),
                            float(avg_bits_k if avg_bits_v is None else avg_bits_v), 1 if var_only else 0,
                            _ptr(basis), _ptr(bits), _ptr(scales), _ptr(sigma2), _ptr(weights), int(n_threads))
    _check(st, "aatc_calibrate")
    assert S == basis.shape[0] * H * 2
    return {"basis": basis, "bits": bits, "scales": scales, "sigma2": sigma2, "weights": weights}


def calibrate_head_group(calib: np.ndarray, calib_q: np.ndarray | None, avg_bits: float, group: int = 1,
                         b_max: int = 8, var_only: bool = False):
    """aatc_calibrate_head_group: one transform and one allocation over the concatenated kv-heads
    of a group.  calib: fp32 [g_h][N][128]; calib_q: fp32 [g_h * group][Nq][128] (keys) or None.
    Returns dict(basis [d][d], bits [d], scales [d], sigma2 [d], weights [d]), d = 128 g_h."""
    c = np.ascontiguousarray(calib, dtype=np.float32)
    if c.ndim != 3 or c.shape[2] != HEAD_DIM:
        raise ValueError("calib must be [g_h][N][128]")
    g_h = c.shape[0]
    cq = None if calib_q is None else np.ascontiguousarray(calib_q, dtype=np.float32)
    if cq is not None and (cq.ndim != 3 or cq.shape[0] != g_h * group or cq.shape[2] != HEAD_DIM):
        raise ValueError("calib_q must be [g_h * group][Nq][128]")
    d = HEAD_DIM * g_h
    basis = np.empty((d, d), np.float32)
    bits = np.empty(d, np.uint8)
    scales = np.empty(d, np.float32)
    sigma2 = np.empty(d, np.float64)
    weights = np.empty(d, np.float64)
    _check(load().aatc_calibrate_head_group(g_h, int(group), _ptr(c), c.shape[1], None if cq is None else _ptr(cq),
                                            0 if cq is None else cq.shape[1], float(avg_bits), int(b_max),
                                            1 if var_only else 0, _ptr(basis), _ptr(bits), _ptr(scales),
                                            _ptr(sigma2), _ptr(weights)), "aatc_calibrate_head_group")
    return {"basis": basis, "bits": bits, "scales": scales, "sigma2": sigma2, "weights": weights}


def save_plan(path: str, dm: Dims, basis: np.ndarray, bits: np.ndarray, scales: np.ndarray):
    """aatc_plan_save: write a plan's host arrays (as calibrate returns them) to a plan file."""
    L, H = dm.n_layers, dm.n_kv_heads
    b = np.ascontiguousarray(basis, dtype=np.float32)
    w = np.ascontiguousarray(bits, dtype=np.uint8)
    sc = np.ascontiguousarray(scales, dtype=np.float32)
    if b.size != L * H * 2 * HEAD_DIM * HEAD_DIM or w.size != L * H * 2 * HEAD_DIM or sc.size != w.size:
        raise ValueError("basis / bits / scales do not match the dims")
    _check(load().aatc_plan_save(os.fsencode(path), ctypes.byref(dm), _ptr(b), _ptr(w), _ptr(sc)),
           "aatc_plan_save")


def load_plan(path: str):
    """aatc_plan_file_dims + aatc_plan_load: (dims, dict(basis, bits, scales)) from a plan file, in
    the layouts calibrate returns."""
    lib = load()
    dm = Dims()
    _check(lib.aatc_plan_file_dims(os.fsencode(path), ctypes.byref(dm)), "aatc_plan_file_dims")
    shape = (dm.n_layers, dm.n_kv_heads, 2, HEAD_DIM)
    basis = np.empty(shape + (HEAD_DIM,), np.float32)
    bits = np.empty(shape, np.uint8)
    scales = np.empty(shape, np.float32)
    _check(lib.aatc_plan_load(os.fsencode(path), ctypes.byref(dm), _ptr(basis), _ptr(bits), _ptr(scales)),
           "aatc_plan_load")
    return dm, {"basis": basis, "bits": bits, "scales": scales}


def selftest_bounded_wait(limit_us: int, flags, stream=None):
    """aatc_selftest_bounded_wait: a kernel whose bounded wait runs out (nothing arrives); it sets
    bit 1 of the device int32 `flags` (a torch tensor) and returns."""
    _check(load().aatc_selftest_bounded_wait(int(limit_us), _ptr(flags), _stream(stream)),
           "aatc_selftest_bounded_wait")


def allocate_global(dm: Dims, sigma2: np.ndarray, weights: np.ndarray, avg_bits_k: float,
                    avg_bits_v: float | None = None, n_protect: int = 3) -> np.ndarray:
    """aatc_allocate_global: one water-filling pool per kind over all layers (first n_protect
    layers per stream).  sigma2, weights: fp64 [L][H_kv][2][128] as calibrate returns them.
    Returns bits uint8 [L][H_kv][2][128]."""
    s2 = np.ascontiguousarray(sigma2, dtype=np.float64)
    w = np.ascontiguousarray(weights, dtype=np.float64)
    shape = (dm.n_layers, dm.n_kv_heads, 2, HEAD_DIM)
    if s2.shape != shape or w.shape != shape:
        raise ValueError("sigma2 / weights must be [L][H_kv][2][128]")
    bits = np.empty(shape, np.uint8)
    _check(load().aatc_allocate_global(ctypes.byref(dm), _ptr(s2), _ptr(w), float(avg_bits_k),
                                       float(avg_bits_k if avg_bits_v is None else avg_bits_v), int(n_protect),
                                       _ptr(bits)), "aatc_allocate_global")
    return bits


def whitening_transform(x: np.ndarray, w: np.ndarray) -> dict:
    """aatc_whitening_transform (Sec. 5 Step 1): x fp32 [n][d_model] calibration activations,
    w fp32 [d_model][128] one head's projection.  Returns dict(A, B, S, P, A_hat) with
    W = A B, A_hat = A sqrt(S) = W P."""
    xx = np.ascontiguousarray(x, dtype=np.float32)
    ww = np.ascontiguousarray(w, dtype=np.float32)
    n, dm = xx.shape
    if ww.shape != (dm, HEAD_DIM):
        raise ValueError("w must be [d_model][128]")
    a = np.empty((dm, HEAD_DIM), np.float32)
    b = np.empty((HEAD_DIM, HEAD_DIM), np.float32)
    sv = np.empty(HEAD_DIM, np.float64)
    pm = np.empty((HEAD_DIM, HEAD_DIM), np.float32)
    ah = np.empty((dm, HEAD_DIM), np.float32)
    _check(load().aatc_whitening_transform(dm, n, _ptr(xx), _ptr(ww), _ptr(a), _ptr(b), _ptr(sv), _ptr(pm),
                                           _ptr(ah)), "aatc_whitening_transform")
    return {"A": a, "B": b, "S": sv, "P": pm, "A_hat": ah}


def hidden_operand(dm: Dims, w_k: np.ndarray, w_v: np.ndarray, basis: np.ndarray) -> np.ndarray:
    """aatc_hidden_operand: w_k, w_v fp32 [L][d_model][H_kv*128], basis as calibrate returns it.
    Returns uint16 bf16 bits [L][H_kv][2][128][d_model] (copy it to the device as bfloat16)."""
    wk = np.ascontiguousarray(w_k, dtype=np.float32)
    wv = np.ascontiguousarray(w_v, dtype=np.float32)
    bs = np.ascontiguousarray(basis, dtype=np.float32)
    L, H = dm.n_layers, dm.n_kv_heads
    if wk.ndim != 3 or wk.shape[0] != L or wk.shape[2] != H * HEAD_DIM or wv.shape != wk.shape:
        raise ValueError("w_k / w_v must be [L][d_model][H_kv*128]")
    d_model = wk.shape[1]
    out = np.empty((L, H, 2, HEAD_DIM, d_model), np.uint16)
    _check(load().aatc_hidden_operand(ctypes.byref(dm), d_model, _ptr(wk), _ptr(wv), _ptr(bs), _ptr(out)),
           "aatc_hidden_operand")
    return out


class Plan:
    """Device plan (aatc_plan_t).  Create from the planner outputs; destroyed on close()."""

    def __init__(self, dm: Dims, basis: np.ndarray, bits: np.ndarray, scales: np.ndarray, stream=None):
        lib = load()
        self.dims = dm
        self._basis = np.ascontiguousarray(basis, dtype=np.float32)
        self._bits = np.ascontiguousarray(bits, dtype=np.uint8)
        self._scales = np.ascontiguousarray(scales, dtype=np.float32)
        h = ctypes.c_void_p()
        st = lib.aatc_plan_create(ctypes.byref(dm), _ptr(self._basis), _ptr(self._bits), _ptr(self._scales),
                                  _stream(stream), ctypes.byref(h))
        _check(st, "aatc_plan_create")
        self.handle = h.value
        w = _I32()
        ret = np.empty((dm.n_layers, dm.n_kv_heads, 2), np.int32)
        _check(lib.aatc_plan_info(self.handle, ctypes.byref(w), _ptr(ret)), "aatc_plan_info")
        self.n_words = w.value
        self.retained = ret

    @property
    def group(self) -> int:
        return self.dims.n_q_heads // self.dims.n_kv_heads

    group_heads = 1

    def cache_bytes(self, batch: int, max_tokens: int) -> int:
        key = (int(batch), int(max_tokens))
        memo = self.__dict__.setdefault("_cache_bytes", {})
        if key not in memo:
            n = _SZ()
            _check(load().aatc_cache_bytes(self.handle, batch, max_tokens, ctypes.byref(n)), "aatc_cache_bytes")
            memo[key] = n.value
        return memo[key]

    def new_cache(self, batch: int, max_tokens: int, device="cuda"):
        import torch
        return torch.empty(self.cache_bytes(batch, max_tokens) // 4, dtype=torch.int32, device=device)

    def workspace_bytes(self, batch: int, n_ctx: int) -> int:
        n = _SZ()
        _check(load().aatc_decode_workspace_bytes(self.handle, batch, n_ctx, ctypes.byref(n)),
               "aatc_decode_workspace_bytes")
        return n.value

    def device_error(self, clear: bool = False) -> int:
        f = _I32()
        _check(load().aatc_get_device_error(self.handle, ctypes.byref(f), int(clear)), "aatc_get_device_error")
        return f.value

    def close(self):
        if getattr(self, "handle", None):
            _check(load().aatc_plan_destroy(self.handle), "aatc_plan_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class GroupPlan(Plan):
    """Head-group device plan (aatc_group_plan_create): one transform per group of g_h kv-heads.
    basis fp32 [L][H_kv / g_h][2][n][n], bits uint8 [L][H_kv / g_h][2][n], scales fp32 of the
    same shape, n = 128 g_h (aatc_calibrate_head_group's outputs per group stream)."""

    def __init__(self, dm: Dims, g_h: int, basis: np.ndarray, bits: np.ndarray, scales: np.ndarray, stream=None):
        lib = load()
        self.dims = dm
        self.group_heads = int(g_h)
        n = HEAD_DIM * self.group_heads
        ng = dm.n_kv_heads // max(1, self.group_heads)
        self._basis = np.ascontiguousarray(basis, dtype=np.float32)
        self._bits = np.ascontiguousarray(bits, dtype=np.uint8)
        self._scales = np.ascontiguousarray(scales, dtype=np.float32)
        if (self._basis.shape != (dm.n_layers, ng, 2, n, n) or self._bits.shape != (dm.n_layers, ng, 2, n)
                or self._scales.shape != (dm.n_layers, ng, 2, n)):
            raise ValueError("group plan arrays must be [L][H_kv/g_h][2][n][n], [L][H_kv/g_h][2][n] (n = 128 g_h)")
        h = ctypes.c_void_p()
        st = lib.aatc_group_plan_create(ctypes.byref(dm), self.group_heads, _ptr(self._basis), _ptr(self._bits),
                                        _ptr(self._scales), _stream(stream), ctypes.byref(h))
        _check(st, "aatc_group_plan_create")
        self.handle = h.value
        w = _I32()
        ret = np.empty((dm.n_layers, dm.n_kv_heads, 2), np.int32)
        _check(lib.aatc_plan_info(self.handle, ctypes.byref(w), _ptr(ret)), "aatc_plan_info")
        self.n_words = w.value
        self.retained = ret


def encode(plan: Plan, layer: int, K, V, cache, start: int, max_tokens: int, stream=None):
    """aatc_encode: K, V bf16 [batch][n_tokens][H_kv][128] (device); writes positions
    [start, start + n_tokens) of the packed cache."""
    import torch
    _dev_tensor(K, "aatc_encode", "K", torch.bfloat16, 4, (None, None, plan.dims.n_kv_heads, HEAD_DIM))
    _dev_tensor(V, "aatc_encode", "V", torch.bfloat16, 4, tuple(K.shape))
    batch, n_tokens = K.shape[0], K.shape[1]
    _cache_ok(plan, cache, batch, max_tokens, "aatc_encode")
    _check(load().aatc_encode(plan.handle, layer, _ptr(K), _ptr(V), batch, start, n_tokens, _ptr(cache),
                              max_tokens, _stream(stream)), "aatc_encode")


def encode_hidden(plan: Plan, layer: int, x, a_hat, cache, start: int, max_tokens: int, stream=None):
    """aatc_encode_hidden: x bf16 [batch][n_tokens][d_model] hidden states (device), a_hat bf16
    [L][H_kv][2][128][d_model] from hidden_operand (device); writes positions [start, start +
    n_tokens) of the packed cache with the codes of x W U (keys and values of every kv-head)."""
    import torch
    _dev_tensor(x, "aatc_encode_hidden", "x", torch.bfloat16, 3)
    batch, n_tokens, d_model = x.shape
    _dev_tensor(a_hat, "aatc_encode_hidden", "a_hat", torch.bfloat16)
    if a_hat.numel() != plan.dims.n_layers * plan.dims.n_kv_heads * 2 * HEAD_DIM * d_model:
        _arg_error("aatc_encode_hidden", "a_hat must be [L][H_kv][2][128][d_model] for the d_model of x")
    _cache_ok(plan, cache, batch, max_tokens, "aatc_encode_hidden")
    _check(load().aatc_encode_hidden(plan.handle, layer, _ptr(x), d_model, _ptr(a_hat), batch, start, n_tokens,
                                     _ptr(cache), max_tokens, _stream(stream)), "aatc_encode_hidden")


def prefill_attention(plan: Plan, layer: int, q, q_start: int, cache, n_ctx: int, max_tokens: int, out=None,
                      workspace=None, stream=None):
    """aatc_prefill_attention: q bf16 [batch][n_q][H_q][128] at positions q_start .. q_start + n_q - 1,
    causal over the packed cache tokens [0, n_ctx) -> fp32 [batch][n_q][H_q][128]."""
    import torch
    _dev_tensor(q, "aatc_prefill_attention", "q", torch.bfloat16, 4, (None, None, plan.dims.n_q_heads, HEAD_DIM))
    batch, n_q = q.shape[0], q.shape[1]
    _cache_ok(plan, cache, batch, max_tokens, "aatc_prefill_attention")
    if out is None:
        out = torch.empty((batch, n_q, plan.dims.n_q_heads, HEAD_DIM), dtype=torch.float32, device=q.device)
    _out_ok(out, batch * n_q * plan.dims.n_q_heads * HEAD_DIM, "aatc_prefill_attention")
    nb = _SZ()
    _check(load().aatc_prefill_workspace_bytes(plan.handle, batch, n_ctx, ctypes.byref(nb)),
           "aatc_prefill_workspace_bytes")
    if workspace is None:
        workspace = torch.empty(max(4, (nb.value + 3) // 4), dtype=torch.float32, device=q.device)
    _check(load().aatc_prefill_attention(plan.handle, layer, _ptr(q), q_start, n_q, _ptr(cache), batch, n_ctx,
                                         max_tokens, _ptr(out), _ptr(workspace),
                                         workspace.numel() * workspace.element_size(), _stream(stream)),
           "aatc_prefill_attention")
    return out


def decode_attention(plan: Plan, layer: int, q, cache, n_ctx: int, max_tokens: int, out=None, workspace=None,
                     stream=None):
    """aatc_decode_attention: q bf16 [batch][H_q][128] -> fp32 [batch][H_q][128]."""
    import torch
    _dev_tensor(q, "aatc_decode_attention", "q", torch.bfloat16, 3, (None, plan.dims.n_q_heads, HEAD_DIM))
    batch = q.shape[0]
    _cache_ok(plan, cache, batch, max_tokens, "aatc_decode_attention")
    if out is None:
        out = torch.empty((batch, plan.dims.n_q_heads, HEAD_DIM), dtype=torch.float32, device=q.device)
    _out_ok(out, batch * plan.dims.n_q_heads * HEAD_DIM, "aatc_decode_attention")
    nbytes = plan.workspace_bytes(batch, n_ctx)
    if workspace is None:
        workspace = torch.empty(max(1, nbytes // 4), dtype=torch.float32, device=q.device)
    _check(load().aatc_decode_attention(plan.handle, layer, _ptr(q), _ptr(cache), batch, n_ctx, max_tokens,
                                        _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                        _stream(stream)), "aatc_decode_attention")
    return out


def decode_attention_sw(plan: Plan, layer: int, q, cache, t_first: int, t_end: int, max_tokens: int,
                        k_full=None, v_full=None, n_full: int = 0, out=None, workspace=None, stream=None,
                        full_row0: int = 0):
    """aatc_decode_attention_sw: packed tokens [t_first, t_end) plus the n_full tokens at rows
    [full_row0, full_row0 + n_full) of k_full / v_full (bf16 [batch][cap][H_kv][128]; the row
    stride between sequences stays cap) in one softmax -> fp32 [batch][H_q][128]."""
    import torch
    where = "aatc_decode_attention_sw"
    _dev_tensor(q, where, "q", torch.bfloat16, 3, (None, plan.dims.n_q_heads, HEAD_DIM))
    batch = q.shape[0]
    _cache_ok(plan, cache, batch, max_tokens, where)
    if k_full is not None or v_full is not None:
        _dev_tensor(k_full, where, "k_full", torch.bfloat16, 4, (batch, None, plan.dims.n_kv_heads, HEAD_DIM))
        _dev_tensor(v_full, where, "v_full", torch.bfloat16, 4, tuple(k_full.shape))
    if out is None:
        out = torch.empty((batch, plan.dims.n_q_heads, HEAD_DIM), dtype=torch.float32, device=q.device)
    _out_ok(out, batch * plan.dims.n_q_heads * HEAD_DIM, where)
    cap = 0 if k_full is None else int(k_full.shape[1])
    if full_row0 < 0 or (k_full is not None and (not k_full.is_contiguous() or not v_full.is_contiguous()
                                                 or full_row0 + int(n_full) > cap)):
        _arg_error(where, "k_full / v_full must be contiguous and hold rows [full_row0, full_row0 + n_full)")
    if t_end > t_first and workspace is None:
        workspace = torch.empty(max(1, plan.workspace_bytes(batch, t_end) // 4), dtype=torch.float32,
                                device=q.device)
    ws_ptr = None if workspace is None else _ptr(workspace)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    row_bytes = int(full_row0) * plan.dims.n_kv_heads * HEAD_DIM * 2
    _check(load().aatc_decode_attention_sw(plan.handle, layer, _ptr(q), _ptr(cache), batch, t_first, t_end,
                                           max_tokens, None if k_full is None else _ptr(k_full) + row_bytes,
                                           None if v_full is None else _ptr(v_full) + row_bytes, int(n_full), cap,
                                           _ptr(out),
                                           ws_ptr, ws_bytes, _stream(stream)), "aatc_decode_attention_sw")
    return out


def decode_attention_noalloc(plan: Plan, layer: int, q, out, cache, n_ctx: int, max_tokens: int, stream=None):
    """aatc_decode_attention_noalloc: as decode_attention, but with no workspace and no allocation
    (the caller passes `out`; the library's fixed scratch holds the split partials)."""
    import torch
    where = "aatc_decode_attention_noalloc"
    _dev_tensor(q, where, "q", torch.bfloat16, 3, (None, plan.dims.n_q_heads, HEAD_DIM))
    _cache_ok(plan, cache, q.shape[0], max_tokens, where)
    _out_ok(out, q.shape[0] * plan.dims.n_q_heads * HEAD_DIM, where)
    _check(load().aatc_decode_attention_noalloc(plan.handle, layer, _ptr(q), _ptr(cache), q.shape[0], n_ctx,
                                                max_tokens, _ptr(out), _stream(stream)),
           "aatc_decode_attention_noalloc")
    return out


def dequantize(plan: Plan, layer: int, cache, batch: int, t0: int, n: int, max_tokens: int, stream=None):
    """aatc_dequantize test hook -> fp32 [batch][n][H_kv][2][128]."""
    import torch
    _cache_ok(plan, cache, batch, max_tokens, "aatc_dequantize")
    out = torch.empty((batch, n, plan.dims.n_kv_heads, 2, HEAD_DIM), dtype=torch.float32, device=cache.device)
    _check(load().aatc_dequantize(plan.handle, layer, _ptr(cache), batch, t0, n, max_tokens, _ptr(out),
                                  _stream(stream)), "aatc_dequantize")
    return out


def bf16_workspace_bytes(batch: int, n_kv: int, n_q: int, n_ctx: int) -> int:
    n = _SZ()
    _check(load().aatc_bf16_decode_workspace_bytes(batch, n_kv, n_q, n_ctx, ctypes.byref(n)),
           "aatc_bf16_decode_workspace_bytes")
    return n.value


def bf16_decode_attention(K, V, q, n_ctx: int, out=None, workspace=None, stream=None):
    """Uncompressed reference decode: K, V bf16 [batch][max_tokens][H_kv][128]; q bf16 [batch][H_q][128]."""
    import torch
    where = "aatc_bf16_decode_attention"
    _dev_tensor(K, where, "K", torch.bfloat16, 4, (None, None, None, HEAD_DIM))
    _dev_tensor(V, where, "V", torch.bfloat16, 4, tuple(K.shape))
    batch, max_tokens, n_kv = K.shape[0], K.shape[1], K.shape[2]
    _dev_tensor(q, where, "q", torch.bfloat16, 3, (batch, None, HEAD_DIM))
    n_q = q.shape[1]
    if out is None:
        out = torch.empty((batch, n_q, HEAD_DIM), dtype=torch.float32, device=q.device)
    _out_ok(out, batch * n_q * HEAD_DIM, where)
    if workspace is None:
        workspace = torch.empty(max(1, bf16_workspace_bytes(batch, n_kv, n_q, n_ctx) // 4), dtype=torch.float32,
                                device=q.device)
    _check(load().aatc_bf16_decode_attention(_ptr(K), _ptr(V), _ptr(q), batch, n_ctx, max_tokens, n_kv, n_q,
                                             _ptr(out), _ptr(workspace), workspace.numel() * 4, _stream(stream)),
           "aatc_bf16_decode_attention")
    return out
