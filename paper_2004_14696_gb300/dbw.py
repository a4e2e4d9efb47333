"""Thin ctypes binding of libdbw (include/dbw.h), same entry-point names.

Argument marshalling only: torch tensors are checked for device, dtype and
contiguity, their data pointers and the current CUDA stream are passed to the C
ABI, and a non-zero status raises ``DbwError`` with the library's message.  All
compute runs in libdbw's CUDA kernels; there is no CPU path.  Loading fails
loudly if the library has not been built (``__graft_entry__.build()``).
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdbw.so")

DBW_OK, DBW_EINVAL, DBW_EALIGN, DBW_ECUDA, DBW_EUNSUPPORTED = 0, -1, -2, -3, -4
PREC_FP32, PREC_BF16 = 0, 1
NMAX, DMAX, LMAX = 1024, 64, 8
CHOOSE_BLIND = 1
ALL_ROW_NORMS = 1
NOALLOC_SCRATCH_BYTES = 4 << 20   # DBW_NOALLOC_SCRATCH_BYTES
FLAG_K1, FLAG_L_SKIPPED, FLAG_EMPTY_MASK, FLAG_BAD_STATE = 1, 2, 4, 8
PSW_NOT_CONVERGED, PSW_RANGE, PSW_UNPOLISHED = 1, 2, 4
STAT_K, STAT_SS, STAT_GBAR_SQ, STAT_V, STAT_N, STAT_F, STAT_L, STAT_FLAGS, STAT_VCLOCK = range(9)
STATS_LEN = 9
PARTIALS_MAGIC = 0x44425750415254


class PswHeader(C.Structure):
    """Mirror of ``dbw_psw_header`` (the start of the push-and-wait state buffer)."""
    _fields_ = [
        ("n", C.c_int32), ("h", C.c_int32), ("sweeps", C.c_int32), ("flags", C.c_int32),
        ("vclock", C.c_double), ("unit", C.c_double), ("iterations", C.c_int64),
        ("off_r", C.c_int64), ("off_pend", C.c_int64), ("off_pendv", C.c_int64), ("off_sum", C.c_int64),
        ("off_cnt", C.c_int64), ("off_x", C.c_int64), ("reserved", C.c_int64 * 6),
    ]


class DbwState(C.Structure):
    """Mirror of ``dbw_state`` (plain old data, copied to/from the device as bytes)."""
    _fields_ = [
        ("n", C.c_int32), ("D", C.c_int32), ("t", C.c_int32), ("k_last", C.c_int32),
        ("c", C.c_int32), ("cntV", C.c_int32), ("cntN", C.c_int32), ("cntL", C.c_int32),
        ("flags", C.c_int32), ("has_last", C.c_int32), ("k_next", C.c_int32), ("reserved", C.c_int32),
        ("F_last", C.c_double), ("F_prev", C.c_double), ("N_last", C.c_double), ("V_last", C.c_double),
        ("vclock", C.c_double),
        ("ringV", C.c_double * DMAX), ("ringN", C.c_double * DMAX), ("ringL", C.c_double * DMAX),
        ("S", C.c_double * NMAX),
    ]


STATE_BYTES = C.sizeof(DbwState)


class DbwError(RuntimeError):
    def __init__(self, fn, code, msg):
        super().__init__(f"{fn} failed ({code}): {msg}")
        self.code = code


_lib = None
_vp, _i32, _i64, _sz, _f32, _f64 = C.c_void_p, C.c_int, C.c_int64, C.c_size_t, C.c_float, C.c_double

_SIGS = {
    "dbw_last_error_string": (C.c_char_p, []),
    "dbw_abi_version": (_i32, []),
    "dbw_param_count": (_i64, [_i32, _vp]),
    "dbw_worker_grads_workspace_bytes": (_sz, [_i32, _vp, _i32, _i32, _i32]),
    "dbw_worker_grads_activations": (_i32, [_i32, _vp, _i32, _i32, _i32, _i32, _vp, _vp, _vp]),
    "dbw_worker_grads": (_i32, [_i32, _vp, _i32, _vp, _i64, _vp, _i64, _vp, _vp, _i32, _i32, _vp, _i64, _vp,
                                _vp, _sz, _vp]),
    "dbw_select_fastest": (_i32, [_vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp]),
    "dbw_aggregate_partials_bytes": (_sz, [_i32, _i64]),
    "dbw_aggregate_update": (_i32, [_vp, _i64, _i32, _i64, _vp, _f32, _vp, _vp, _i32, _vp, _sz, _vp]),
    "dbw_aggregate_update_noalloc": (_i32, [_vp, _i64, _i32, _i64, _vp, _f32, _vp, _vp, _i32, _vp, _vp]),
    "dbw_received_grads_workspace_bytes": (_sz, [_i32, _vp, _i32, _i32, _i32]),
    "dbw_received_partials_bytes": (_sz, [_i32]),
    "dbw_received_grads_update": (_i32, [_i32, _vp, _i32, _vp, _i64, _vp, _i64, _vp, _vp, _i32, _i32, _vp, _f32,
                                         _vp, _vp, _vp, _sz, _vp, _sz, _vp]),
    "dbw_psw_bytes": (_sz, [_i32]),
    "dbw_psw_init": (_i32, [_vp, _i32, _vp]),
    "dbw_psw_arrivals": (_i32, [_vp, _i32, _vp, _vp, _vp]),
    "dbw_psw_record": (_i32, [_vp, _i32, _vp, _vp, _vp, _vp]),
    "dbw_psw_estimate": (_i32, [_vp, _i32, _f64, _i32, _vp, _vp]),
    "dbw_choose_b_times": (_i32, [_vp, _vp, _f64, _f64, _i32, _vp, _vp, _vp]),
    "dbw_state_init": (_i32, [_vp, _i32, _i32, _vp]),
    "dbw_grad_stats": (_i32, [_vp, _i32, _vp, _vp, _vp, _f64, _vp, _vp, _vp, _vp]),
    "dbw_choose_b": (_i32, [_vp, _f64, _f64, _i32, _vp, _vp, _vp]),
    "dbw_profile_dw": (_i32, [_i32]),
    "dbw_profile_dw_read": (_i32, [_vp, _vp, _vp]),
    "dbw_profile_gemm": (_i32, [_i32]),
    "dbw_profile_gemm_read": (_i32, [_vp, _vp]),
    "dbw_test_arm_wait_timeout": (_i32, [_i32, _f64]),
}


def lib():
    """The loaded libdbw (raises if it is missing: there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def exported_symbols():
    return list(_SIGS)


def _check(fn, rc):
    if rc != DBW_OK:
        raise DbwError(fn, rc, lib().dbw_last_error_string().decode())


def _ptr(t, dtype=None, name="tensor", nullable=False):
    if t is None:
        if nullable:
            return None
        raise ValueError(f"{name} must not be None")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _widths(widths):
    arr = (C.c_int32 * len(widths))(*[int(x) for x in widths])
    return len(widths) - 1, arr


# ----------------------------------------------------------------- queries
def dbw_param_count(widths):
    L, arr = _widths(widths)
    return int(lib().dbw_param_count(L, arr))


def dbw_worker_grads_workspace_bytes(widths, n, B, prec):
    L, arr = _widths(widths)
    return int(lib().dbw_worker_grads_workspace_bytes(L, arr, n, B, prec))


def dbw_worker_grads_activations(widths, n, B, prec, layer):
    """(byte offset in ws, leading dimension, element bytes) of layer ``layer``'s input activations."""
    L, arr = _widths(widths)
    off, ld, eb = C.c_size_t(), C.c_int64(), C.c_int()
    rc = lib().dbw_worker_grads_activations(L, arr, n, B, prec, layer, C.byref(off), C.byref(ld), C.byref(eb))
    _check("dbw_worker_grads_activations", rc)
    return off.value, ld.value, eb.value


def hidden_activations(ws, widths, n, B, prec, layer):
    """View of the hidden activations [n*B, width] a dbw_worker_grads call left in ws (device tensor)."""
    off, ld, eb = dbw_worker_grads_activations(widths, n, B, prec, layer)
    M = n * B
    raw = ws[off:off + M * ld * eb]
    t = raw.view(torch.bfloat16 if eb == 2 else torch.float32).view(M, ld)
    return t[:, : int(widths[layer])]


def dbw_aggregate_partials_bytes(n, d):
    return int(lib().dbw_aggregate_partials_bytes(n, d))


def dbw_received_grads_workspace_bytes(widths, n, B, prec):
    L, arr = _widths(widths)
    return int(lib().dbw_received_grads_workspace_bytes(L, arr, n, B, prec))


def dbw_received_partials_bytes(n):
    return int(lib().dbw_received_partials_bytes(n))


# ----------------------------------------------------------------- compute
def dbw_worker_grads(widths, prec, w, pool, labels, idx, n, B, G, loss, ws, stream=None):
    L, arr = _widths(widths)
    d = w.numel()
    rc = lib().dbw_worker_grads(
        L, arr, prec, _ptr(w, torch.float32, "w"), d, _ptr(pool, torch.float32, "pool"), pool.shape[0],
        _ptr(labels, torch.int32, "labels"), _ptr(idx, torch.int32, "idx"), n, B, _ptr(G, torch.float32, "G"),
        G.shape[1], _ptr(loss, torch.float32, "loss"), _ptr(ws, torch.uint8, "ws"), ws.numel(), _stream(stream))
    _check("dbw_worker_grads", rc)


def dbw_received_grads_update(widths, prec, w, pool, labels, idx, n, B, mask, lr, loss, partials, ws, gbar=None,
                              stream=None):
    """One iteration for the received workers only (no [n, d] matrix): w updated in
    place, loss [n] (NaN for workers mask leaves out), partials for dbw_grad_stats."""
    L, arr = _widths(widths)
    rc = lib().dbw_received_grads_update(
        L, arr, prec, _ptr(w, torch.float32, "w"), w.numel(), _ptr(pool, torch.float32, "pool"), pool.shape[0],
        _ptr(labels, torch.int32, "labels"), _ptr(idx, torch.int32, "idx"), n, B, _ptr(mask, torch.uint8, "mask"),
        float(lr), _ptr(gbar, torch.float32, "gbar", nullable=True), _ptr(loss, torch.float32, "loss"),
        _ptr(partials, torch.uint8, "partials"), partials.numel(), _ptr(ws, torch.uint8, "ws"), ws.numel(),
        _stream(stream))
    _check("dbw_received_grads_update", rc)


def dbw_psw_bytes(n):
    return int(lib().dbw_psw_bytes(n))


def dbw_psw_init(psw, n, stream=None):
    _check("dbw_psw_init", lib().dbw_psw_init(_ptr(psw, torch.uint8, "psw"), n, _stream(stream)))


def dbw_psw_arrivals(psw, n, omega, arrivals, stream=None):
    rc = lib().dbw_psw_arrivals(_ptr(psw, torch.uint8, "psw"), n, _ptr(omega, torch.float64, "omega"),
                                _ptr(arrivals, torch.float64, "arrivals"), _stream(stream))
    _check("dbw_psw_arrivals", rc)


def dbw_psw_record(psw, n, order, tsorted, k, stream=None):
    rc = lib().dbw_psw_record(_ptr(psw, torch.uint8, "psw"), n, _ptr(order, torch.int32, "order"),
                              _ptr(tsorted, torch.float64, "tsorted"), _ptr(k, torch.int32, "k"), _stream(stream))
    _check("dbw_psw_record", rc)


def dbw_psw_estimate(psw, n, T_hat, tol=1e-6, max_sweeps=100000, stream=None):
    rc = lib().dbw_psw_estimate(_ptr(psw, torch.uint8, "psw"), n, float(tol), int(max_sweeps),
                                _ptr(T_hat, torch.float64, "T_hat"), _stream(stream))
    _check("dbw_psw_estimate", rc)


def dbw_choose_b_times(state, T_hat, lr, beta, b_out, ratio_out=None, flags=0, stream=None):
    rc = lib().dbw_choose_b_times(_ptr(state, torch.uint8, "state"), _ptr(T_hat, torch.float64, "T_hat"), float(lr),
                                  float(beta), int(flags), _ptr(b_out, torch.int32, "b_out"),
                                  _ptr(ratio_out, torch.float64, "ratio_out", nullable=True), _stream(stream))
    _check("dbw_choose_b_times", rc)


def new_psw(n, device="cuda", stream=None):
    """A device push-and-wait state buffer for n workers, initialised."""
    t = torch.empty(dbw_psw_bytes(n), dtype=torch.uint8, device=device)
    dbw_psw_init(t, n, stream)
    return t


def read_psw(psw, n):
    """Host copy of the push-and-wait state: header fields and its arrays (synchronises)."""
    raw = psw.cpu().numpy()
    hdr = PswHeader.from_buffer_copy(raw[:C.sizeof(PswHeader)].tobytes())
    nn = n * n

    def arr(off, dtype, count):
        return np.frombuffer(raw[off:off + count * np.dtype(dtype).itemsize].tobytes(), dtype=dtype)
    pend = arr(hdr.off_pend, np.int32, 2 * n).reshape(n, 2)
    return {"n": hdr.n, "h": hdr.h, "sweeps": hdr.sweeps, "flags": hdr.flags, "vclock": hdr.vclock,
            "iterations": hdr.iterations, "r": arr(hdr.off_r, np.float64, n),
            "pend": pend, "pendv": arr(hdr.off_pendv, np.float64, n),
            "sums": arr(hdr.off_sum, np.uint64, nn).reshape(n, n).astype(np.float64) * hdr.unit,
            "sums_raw": arr(hdr.off_sum, np.uint64, nn).reshape(n, n),
            "cnts": arr(hdr.off_cnt, np.int32, nn).reshape(n, n), "x": arr(hdr.off_x, np.float32, nn).reshape(n, n)}


def dbw_select_fastest(times, b, order, mask, tsorted, k_out=None, stream=None):
    rc = lib().dbw_select_fastest(
        _ptr(times, torch.float64, "times"), times.numel(), _ptr(b, torch.int32, "b"),
        _ptr(order, torch.int32, "order"), _ptr(mask, torch.uint8, "mask"), _ptr(tsorted, torch.float64, "tsorted"),
        _ptr(k_out, torch.int32, "k_out", nullable=True), _stream(stream))
    _check("dbw_select_fastest", rc)


def dbw_aggregate_update(G, n, d, mask, lr, w, partials, gbar=None, stream=None, flags=0):
    rc = lib().dbw_aggregate_update(
        _ptr(G, torch.float32, "G"), G.shape[1], n, d, _ptr(mask, torch.uint8, "mask"), float(lr),
        _ptr(w, torch.float32, "w"), _ptr(gbar, torch.float32, "gbar", nullable=True), int(flags),
        _ptr(partials, torch.uint8, "partials"), partials.numel(), _stream(stream))
    _check("dbw_aggregate_update", rc)


def dbw_aggregate_update_noalloc(G, n, d, mask, lr, w, sums_out, gbar=None, stream=None, flags=0):
    """dbw_aggregate_update without caller scratch (for callers that cannot allocate);
    writes the reduced totals to sums_out [n + 2] fp64."""
    rc = lib().dbw_aggregate_update_noalloc(
        _ptr(G, torch.float32, "G"), G.shape[1], n, d, _ptr(mask, torch.uint8, "mask"), float(lr),
        _ptr(w, torch.float32, "w"), _ptr(gbar, torch.float32, "gbar", nullable=True), int(flags),
        _ptr(sums_out, torch.float64, "sums_out"), _stream(stream))
    _check("dbw_aggregate_update_noalloc", rc)


def dbw_state_init(state, n, D, stream=None):
    rc = lib().dbw_state_init(_ptr(state, torch.uint8, "state"), n, D, _stream(stream))
    _check("dbw_state_init", rc)


def dbw_grad_stats(partials, n, mask, loss, tsorted, lr, state, stats_out=None, row_sqnorm=None, stream=None):
    rc = lib().dbw_grad_stats(
        _ptr(partials, torch.uint8, "partials"), n, _ptr(mask, torch.uint8, "mask"), _ptr(loss, torch.float32, "loss"),
        _ptr(tsorted, torch.float64, "tsorted"), float(lr), _ptr(state, torch.uint8, "state"),
        _ptr(stats_out, torch.float64, "stats_out", nullable=True),
        _ptr(row_sqnorm, torch.float64, "row_sqnorm", nullable=True), _stream(stream))
    _check("dbw_grad_stats", rc)


def dbw_choose_b(state, lr, beta, b_out, ratio_out=None, flags=0, stream=None):
    rc = lib().dbw_choose_b(
        _ptr(state, torch.uint8, "state"), float(lr), float(beta), int(flags), _ptr(b_out, torch.int32, "b_out"),
        _ptr(ratio_out, torch.float64, "ratio_out", nullable=True), _stream(stream))
    _check("dbw_choose_b", rc)


def dbw_test_arm_wait_timeout(stage, wait_ms):
    """Arms the next weight-gradient launch to lose the load of one pipeline stage
    (tests of the bounded-wait path); stage < 0 disarms."""
    _check("dbw_test_arm_wait_timeout", lib().dbw_test_arm_wait_timeout(int(stage), float(wait_ms)))


def dbw_profile_dw(enable):
    _check("dbw_profile_dw", lib().dbw_profile_dw(1 if enable else 0))


def dbw_profile_dw_read():
    """(summed ms, launches, summed algorithmic bytes) of the timed weight-gradient launches."""
    ms, n, b = C.c_double(), C.c_int64(), C.c_double()
    _check("dbw_profile_dw_read", lib().dbw_profile_dw_read(C.byref(ms), C.byref(n), C.byref(b)))
    return ms.value, n.value, b.value


def dbw_profile_gemm(enable):
    _check("dbw_profile_gemm", lib().dbw_profile_gemm(1 if enable else 0))


def dbw_profile_gemm_read():
    """(summed ms, launches) of the timed persistent tensor-core GEMM launches."""
    ms, n = C.c_double(), C.c_int64()
    _check("dbw_profile_gemm_read", lib().dbw_profile_gemm_read(C.byref(ms), C.byref(n)))
    return ms.value, n.value


# ----------------------------------------------------------------- helpers
def new_state(n, D, device="cuda", stream=None):
    """Device buffer holding a dbw_state initialised for n workers and window D."""
    st = torch.empty(STATE_BYTES, dtype=torch.uint8, device=device)
    dbw_state_init(st, n, D, stream)
    return st


def read_state(state_tensor):
    """Copy a device dbw_state to the host as a ``DbwState`` (synchronises)."""
    raw = state_tensor.detach().cpu().numpy().tobytes()
    return DbwState.from_buffer_copy(raw)


def write_state(state_tensor, st: DbwState):
    """Overwrite a device dbw_state from a host ``DbwState``."""
    buf = torch.frombuffer(bytearray(bytes(st)), dtype=torch.uint8)
    state_tensor.copy_(buf)
