"""ctypes binding of the BMLP C-ABI (include/bmlp.h).

Argument marshalling only: every step of training and evaluation runs in the
CUDA kernels of ``libbmlp.so``.  There is no fallback: if the library or a GB300
is missing, the calls raise.

Buffers may be torch tensors (CUDA or CPU) or numpy arrays; CPU/numpy buffers
are host pointers, which the library stages through its own device buffers.
``stream`` is a ``torch.cuda.Stream``, a raw ``cudaStream_t`` integer, or None
(torch's current stream when torch CUDA is initialised, else the legacy
default stream).
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

from . import _build

BMLP_OK = 0
BMLP_EINVAL = -1
BMLP_ENOMEM = -2
BMLP_ECUDA = -3
BMLP_ETIMEOUT = -4
BMLP_ESTATE = -5
BMLP_ENODEV = -6
BMLP_EPOCH_END = 1
BMLP_FWD_AUTO, BMLP_FWD_POPC, BMLP_FWD_TCGEN05, BMLP_FWD_B1MMA, BMLP_FWD_S8MMA = 0, 1, 2, 3, 4
BMLP_GROUPS_CONTIGUOUS, BMLP_GROUPS_FIXED, BMLP_GROUPS_RESHUFFLED = 0, 1, 2
PROFILE_KINDS = ("train_forward", "cls_select", "update", "eval_forward", "eval_out", "copy",
                 "r_events")

_ERRNAMES = {-1: "EINVAL", -2: "ENOMEM", -3: "ECUDA", -4: "ETIMEOUT", -5: "ESTATE", -6: "ENODEV"}


class BmlpError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("bmlp error %s (%d): %s" % (_ERRNAMES.get(code, "?"), code, msg))
        self.code = code


class bmlp_hparams(C.Structure):
    _fields_ = [("bs", C.c_int32), ("r_num", C.c_int32), ("r_den", C.c_int32),
                ("p_r0", C.c_double), ("gamma", C.POINTER(C.c_int32)), ("fwd_impl", C.c_int32),
                ("group_mode", C.c_int32)]


_lib = None
_lock = threading.Lock()
_vp = C.c_void_p
_i32p = C.POINTER(C.c_int32)
_i64p = C.POINTER(C.c_int64)
_f64p = C.POINTER(C.c_double)

# (name, restype, argtypes) of every entry point of include/bmlp.h
SIGNATURES = [
    ("bmlp_create", C.c_int, [_i32p, C.c_int32, C.c_int32, C.c_int16, C.c_uint64,
                              C.POINTER(bmlp_hparams), C.POINTER(_vp)]),
    ("bmlp_destroy", None, [_vp]),
    ("bmlp_train", C.c_int, [_vp, _vp, _vp, C.c_int64, C.c_uint32, _vp, _i64p]),
    ("bmlp_predict", C.c_int, [_vp, _vp, C.c_int64, _vp, _vp]),
    ("bmlp_get_state", C.c_int, [_vp, C.c_int32, _vp, _vp, _vp, _f64p, _i64p]),
    ("bmlp_set_state", C.c_int, [_vp, C.c_int32, _vp, C.c_double, C.c_int64]),
    ("bmlp_get_info", C.c_int, [_vp, _i32p, _i32p, _i32p, _i32p, _i32p, _i32p]),
    ("bmlp_last_error", C.c_char_p, [_vp]),
    ("bmlp_gamma_rule", C.c_int32, [C.c_int32]),
    ("bmlp_reinforce_tables", C.c_int, [C.c_double, C.c_int32, C.c_int32, _vp, _vp, _vp]),
    ("bmlp_debug_last_step", C.c_int, [_vp, C.c_int32, _vp, _vp, _vp, _vp]),
    ("bmlp_set_profiling", C.c_int, [_vp, C.c_int32]),
    ("bmlp_get_profile", C.c_int, [_vp, C.c_int32, _i64p, _f64p]),
    ("bmlp_reset_profile", C.c_int, [_vp]),
    ("bmlp_launch_count", C.c_int64, [_vp]),
    ("bmlp_predict_noalloc", C.c_int, [_vp, _vp, C.c_int64, _vp, _vp]),
    ("bmlp_layer_forward", C.c_int, [_vp, C.c_int32, _vp, C.c_int64, _vp, _vp]),
    ("bmlp_update_stats", C.c_int, [_vp, _vp, _vp, _vp, C.c_int32]),
    ("bmlp_predict_layers", C.c_int, [_vp, _vp, C.c_int64, _vp, _vp]),
    ("bmlp_layer_errors", C.c_int, [_vp, _i64p, C.c_int32]),
    ("bmlp_binarize_median", C.c_int, [_vp, C.c_int64, C.c_int32, _vp, _vp]),
    ("bmlp_expand_weights", C.c_int, [C.c_uint64, C.c_int32, C.c_int32, _vp, _vp]),
    ("bmlp_expand_sign", C.c_int, [_vp, C.c_int64, C.c_int32, _vp, C.c_int32, _vp, _vp]),
    ("bmlp_debug_wait_probe", C.c_int, [_vp, C.c_int32, C.c_double]),
    ("bmlp_engine_peak", C.c_int, [C.c_int32, C.c_int64, _f64p, _f64p]),
    ("bmlp_debug_fail_alloc", C.c_int, [C.c_int64]),
    ("bmlp_debug_alloc_stats", C.c_int, [_i64p, _i64p]),
    ("bmlp_layer_forward_engine", C.c_int, [_vp, C.c_int32, C.c_int32, _vp, C.c_int64, _vp, _vp]),
]


def library_path() -> str:
    return _build.LIB


def lib(build_if_missing: bool = True):
    """Load libbmlp.so (building it with nvcc first if it is missing)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.LIB
            if not os.path.exists(path):
                if not build_if_missing:
                    raise OSError("libbmlp.so is not built: run __graft_entry__.build()")
                _build.build()
            L = C.CDLL(path)
            for name, res, args in SIGNATURES:
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
    return _lib


def _check(rc, h=None):
    if rc != BMLP_OK:
        msg = lib().bmlp_last_error(h)
        raise BmlpError(rc, msg.decode() if msg else "")


def _ptr(buf):
    """Raw pointer of a torch tensor or numpy array (must be contiguous)."""
    if buf is None:
        return None
    if isinstance(buf, np.ndarray):
        assert buf.flags["C_CONTIGUOUS"], "numpy buffer must be C-contiguous"
        return buf.ctypes.data
    if hasattr(buf, "data_ptr"):
        assert buf.is_contiguous(), "tensor must be contiguous"
        return buf.data_ptr()
    raise TypeError("expected a torch tensor or a numpy array, got %r" % type(buf))


def _stream(stream):
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available() and torch.cuda.is_initialized():
                return torch.cuda.current_stream().cuda_stream
        except ImportError:
            pass
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# -- the C-ABI, one Python function per entry point ------------------------------

def bmlp_create(widths, classes, h_max=255, seed=0, bs=100, r=(1, 4), p_r0=0.5, gamma=None,
                fwd_impl=BMLP_FWD_AUTO, group_mode=BMLP_GROUPS_CONTIGUOUS):
    w = (C.c_int32 * len(widths))(*[int(v) for v in widths])
    hp = bmlp_hparams()
    hp.bs = bs
    hp.r_num, hp.r_den = int(r[0]), int(r[1])
    hp.p_r0 = float(p_r0)
    g = None
    if gamma is not None:
        g = (C.c_int32 * len(gamma))(*[int(v) for v in gamma])
        hp.gamma = C.cast(g, _i32p)
    hp.fwd_impl = fwd_impl
    hp.group_mode = group_mode
    h = _vp()
    rc = lib().bmlp_create(w, len(widths), classes, h_max, seed & (2 ** 64 - 1), C.byref(hp), C.byref(h))
    _check(rc, None)
    return h.value


def bmlp_destroy(h):
    lib().bmlp_destroy(h)


def bmlp_train(h, x_packed, labels, n=None, flags=0, stream=None, count_errors=False):
    n = labels.shape[0] if n is None else n
    err = C.c_int64(-1)
    rc = lib().bmlp_train(h, _ptr(x_packed), _ptr(labels), n, flags, _stream(stream),
                          C.byref(err) if count_errors else None)
    _check(rc, h)
    return int(err.value) if count_errors else None


def bmlp_predict(h, x_packed, labels_out, n=None, stream=None):
    n = labels_out.shape[0] if n is None else n
    _check(lib().bmlp_predict(h, _ptr(x_packed), n, _ptr(labels_out), _stream(stream)), h)


def bmlp_predict_noalloc(h, x_packed, labels_out, n=None, stream=None):
    """Allocation-free bmlp_predict for callers that cannot allocate device
    memory (device buffers only; n * ceil(max K_l / 64) <= 2^20)."""
    n = labels_out.shape[0] if n is None else n
    _check(lib().bmlp_predict_noalloc(h, _ptr(x_packed), n, _ptr(labels_out), _stream(stream)), h)


def bmlp_predict_layers(h, x_packed, labels_out, n=None, stream=None):
    """Early-exit predictions of every layer into labels_out (L x n, layer-major)."""
    n = labels_out.shape[-1] if n is None else n
    _check(lib().bmlp_predict_layers(h, _ptr(x_packed), n, _ptr(labels_out), _stream(stream)), h)


def bmlp_layer_errors(h, reset=False):
    """Local 01-loss counts of layers 1..L since creation or the last reset."""
    L = C.c_int32()
    lib().bmlp_get_info(h, C.byref(L), None, None, None, None, None)
    out = (C.c_int64 * L.value)()
    _check(lib().bmlp_layer_errors(h, out, 1 if reset else 0), h)
    return [int(v) for v in out]


def bmlp_binarize_median(x, out, stream=None):
    """Median binarisation of n x K fp32 patterns (device) into packed bits."""
    n, K = x.shape
    _check(lib().bmlp_binarize_median(_ptr(x), n, K, _ptr(out), _stream(stream)), None)


def bmlp_expand_weights(seed, K, D, E_out, stream=None):
    """The packed K x D +-1 expansion matrix (device, K x ceil(D/64) int64)."""
    _check(lib().bmlp_expand_weights(seed, K, D, _ptr(E_out), _stream(stream)), None)


def bmlp_expand_sign(x, E, K, out, stream=None):
    """Expansion layer: n x D uint8 patterns (device) -> packed sign(x E^T)."""
    n, D = x.shape
    _check(lib().bmlp_expand_sign(_ptr(x), n, D, _ptr(E), K, _ptr(out), _stream(stream)), None)


def bmlp_debug_wait_probe(h, arrive, seconds=0.05, leave_pending=False):
    """Run the bounded-wait probe; raises BmlpError(BMLP_ETIMEOUT) if it expired.
    leave_pending: nothing arrives and the expiry is left for the next
    synchronising call to report."""
    a = -1 if leave_pending else (1 if arrive else 0)
    _check(lib().bmlp_debug_wait_probe(h, a, float(seconds)), h)


def bmlp_layer_forward(h, layer, a_in, a_out, n=None, stream=None):
    """a_out = sign(a_in W_layer), packed rows on the device."""
    n = a_out.shape[0] if n is None else n
    _check(lib().bmlp_layer_forward(h, layer, _ptr(a_in), n, _ptr(a_out), _stream(stream)), h)


def bmlp_layer_forward_engine(h, layer, engine, a_in, a_out, n=None, stream=None):
    """bmlp_layer_forward on the given engine (BMLP_FWD_POPC / TCGEN05 / B1MMA)."""
    n = a_out.shape[0] if n is None else n
    _check(lib().bmlp_layer_forward_engine(h, layer, engine, _ptr(a_in), n, _ptr(a_out),
                                           _stream(stream)), h)


def bmlp_debug_fail_alloc(nth):
    """Arm (nth >= 1) or disarm (0) the one-shot failure of the nth allocation."""
    _check(lib().bmlp_debug_fail_alloc(int(nth)), None)


def bmlp_debug_alloc_stats():
    """(allocations the library holds, their bytes), over all live handles."""
    n, b = C.c_int64(), C.c_int64()
    _check(lib().bmlp_debug_alloc_stats(C.byref(n), C.byref(b)), None)
    return n.value, b.value


def bmlp_engine_peak(engine, iters):
    """(bit-pairs per second over the device, ms of the timed launch) of one
    contraction unit's peak kernel."""
    bp, ms = C.c_double(), C.c_double()
    _check(lib().bmlp_engine_peak(engine, iters, C.byref(bp), C.byref(ms)), None)
    return bp.value, ms.value


def bmlp_update_stats(h, reset=False):
    """(rows visited, rows streamed, algorithmic bytes) of the update kernel."""
    r, st, by = C.c_int64(), C.c_int64(), C.c_int64()
    _check(lib().bmlp_update_stats(h, C.byref(r), C.byref(st), C.byref(by), 1 if reset else 0), h)
    return r.value, st.value, by.value


def bmlp_get_info(h):
    L = C.c_int32()
    lib().bmlp_get_info(h, C.byref(L), None, None, None, None, None)
    widths = (C.c_int32 * (L.value + 1))()
    gam = (C.c_int32 * L.value)()
    cls, bs, fwd = C.c_int32(), C.c_int32(), C.c_int32()
    _check(lib().bmlp_get_info(h, C.byref(L), widths, C.byref(cls), gam, C.byref(bs), C.byref(fwd)), h)
    return dict(L=L.value, widths=list(widths), classes=cls.value, gamma=list(gam), bs=bs.value,
                fwd_impl=fwd.value)


def bmlp_get_state(h, layer):
    """Returns (H int16 K_l x K_{l-1}, W uint64 K_l x nw, P int8 K_l x c, p_r, step)."""
    info = bmlp_get_info(h)
    Kin, Kout, c = info["widths"][layer - 1], info["widths"][layer], info["classes"]
    H = np.empty((Kout, Kin), np.int16)
    W = np.empty((Kout, (Kin + 63) // 64), np.uint64)
    P = np.empty((Kout, c), np.int8)
    pr = C.c_double()
    step = C.c_int64()
    _check(lib().bmlp_get_state(h, layer, H.ctypes.data, W.ctypes.data, P.ctypes.data,
                                C.byref(pr), C.byref(step)), h)
    return H, W, P, pr.value, step.value


def bmlp_set_state(h, layer, H=None, p_r=0.0, step=-1):
    Hc = None if H is None else np.ascontiguousarray(H, dtype=np.int16)
    _check(lib().bmlp_set_state(h, layer, None if Hc is None else Hc.ctypes.data, p_r, step), h)


def bmlp_debug_last_step(h, layer):
    info = bmlp_get_info(h)
    K, bs = info["widths"][layer], info["bs"]
    G = K // info["gamma"][layer - 1]
    Z = np.empty((bs, K), np.int16)
    A = np.empty((bs, (K + 63) // 64), np.uint64)
    mark = np.empty(bs, np.uint8)
    sel = np.empty((bs, G), np.int16)
    _check(lib().bmlp_debug_last_step(h, layer, Z.ctypes.data, A.ctypes.data, mark.ctypes.data,
                                      sel.ctypes.data), h)
    return Z, A, mark, sel


def bmlp_gamma_rule(K):
    return lib().bmlp_gamma_rule(K)


def bmlp_reinforce_tables(p_r, K, n):
    """Sampler thresholds of a block of n inputs: (any, first[n], gap[n-1])."""
    any_ = np.zeros(1, np.uint64)
    first = np.zeros(64, np.uint64)
    gap = np.zeros(64, np.uint64)
    _check(lib().bmlp_reinforce_tables(p_r, K, n, any_.ctypes.data, first.ctypes.data,
                                       gap.ctypes.data), None)
    return int(any_[0]), first[:n].copy(), gap[:max(n - 1, 0)].copy()


def bmlp_last_error(h=None):
    m = lib().bmlp_last_error(h)
    return m.decode() if m else ""


def bmlp_set_profiling(h, every=1):
    """every: 0 off, 1 every mini-batch, S every S-th mini-batch (True = 1)."""
    _check(lib().bmlp_set_profiling(h, int(every)), h)


def bmlp_get_profile(h):
    out = {}
    for i, name in enumerate(PROFILE_KINDS):
        n, ms = C.c_int64(), C.c_double()
        _check(lib().bmlp_get_profile(h, i, C.byref(n), C.byref(ms)), h)
        out[name] = (n.value, ms.value)
    return out


def bmlp_reset_profile(h):
    _check(lib().bmlp_reset_profile(h), h)


def bmlp_launch_count(h):
    return int(lib().bmlp_launch_count(h))


# -- convenience object -----------------------------------------------------------

class BMLP:
    """Owning wrapper of a bmlp_t handle."""

    def __init__(self, widths, classes, h_max=255, seed=0, bs=100, r=(1, 4), p_r0=0.5,
                 gamma=None, fwd_impl=BMLP_FWD_AUTO, group_mode=BMLP_GROUPS_CONTIGUOUS):
        self.h = bmlp_create(widths, classes, h_max, seed, bs, r, p_r0, gamma, fwd_impl,
                             group_mode)
        self.info = bmlp_get_info(self.h)

    def close(self):
        if getattr(self, "h", None):
            bmlp_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def train(self, x_packed, labels, epoch_end=False, stream=None, count_errors=False, n=None):
        return bmlp_train(self.h, x_packed, labels, n, BMLP_EPOCH_END if epoch_end else 0, stream,
                          count_errors)

    def predict(self, x_packed, labels_out, stream=None, n=None):
        bmlp_predict(self.h, x_packed, labels_out, n, stream)

    def predict_layers(self, x_packed, labels_out, stream=None, n=None):
        bmlp_predict_layers(self.h, x_packed, labels_out, n, stream)

    def layer_errors(self, reset=False):
        return bmlp_layer_errors(self.h, reset)

    def state(self, layer):
        return bmlp_get_state(self.h, layer)

    def set_state(self, layer, H=None, p_r=0.0, step=-1):
        bmlp_set_state(self.h, layer, H, p_r, step)
