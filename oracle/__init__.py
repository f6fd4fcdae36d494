"""CPU oracle of the fully binary BMLP training rule -- TEST INFRASTRUCTURE.

Loads ``bmlp_oracle.c`` (plain C, compiled here with gcc) through ctypes and
wraps it for numpy.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline / reference legs of ``bench.py`` may import this package; the GPU
library and its Python binding never do.

What each function follows (arXiv 2412.00119):
  ``philox4x32_10``            -- Salmon et al., SC'11 (the random stream)
  ``gamma_rule``               -- Sec. 4.3, choice of the group size
  ``reinforce_prob``           -- Alg. 3 l.8, q = p_r sqrt(2/(pi K_l))
  ``r_block_tables``/``r_events`` -- Alg. 3 l.5-12, which weights are reinforced
  ``layer_forward``            -- Alg. 1 l.8-9
  ``local_output``/``local_loss`` -- Alg. 1 l.10-17 and Eq. 1
  ``select``                   -- Alg. 2
  ``perceptron_update``        -- Alg. 3
  ``OracleModel.train``        -- Alg. 1 as a whole (NetworkUpdate)
  ``OracleModel.predict``      -- forward-only evaluation through P_L (Sec. 3.1)
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bmlp_oracle.c")
_LIB = os.path.join(_HERE, "libbmlp_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP, no FP contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-std=gnu11", "-Wall",
               "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
        subprocess.check_call(cmd)
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = C.CDLL(build())
            _declare(_lib)
    return _lib


class use_library:
    """Context manager: run the wrappers below against another build of the
    oracle source (the pin tests use it to check that planted mistakes in the
    oracle are caught)."""

    def __init__(self, path):
        self.path = path
        self.prev = None

    def __enter__(self):
        global _lib
        other = C.CDLL(self.path)
        _declare(other)
        with _lock:
            self.prev = _lib
            _lib = other
        return other

    def __exit__(self, *exc):
        global _lib
        with _lock:
            _lib = self.prev
        return False


def compile_variant(src_text: str, out_path: str) -> str:
    """Compile an edited copy of the oracle source to ``out_path``."""
    src = out_path + ".c"
    with open(src, "w") as f:
        f.write(src_text)
    subprocess.check_call(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-std=gnu11",
                           "-shared", "-fPIC", "-o", out_path, src, "-lm"])
    return out_path


def source() -> str:
    with open(_SRC) as f:
        return f.read()


_i32p = C.POINTER(C.c_int32)
_i8p = C.POINTER(C.c_int8)
_u8p = C.POINTER(C.c_uint8)
_u32p = C.POINTER(C.c_uint32)
_u64p = C.POINTER(C.c_uint64)
_i64p = C.POINTER(C.c_int64)


def _declare(L):
    L.or_philox4x32_10.argtypes = [_u32p, _u32p, _u32p]
    L.or_philox4x32_10.restype = None
    L.or_init_h.argtypes = [C.c_uint64, C.c_int32, C.c_int32, C.c_int32]
    L.or_init_h.restype = C.c_int32
    L.or_init_rho.argtypes = [C.c_uint64, C.c_int32, C.c_int32, C.c_int32]
    L.or_init_rho.restype = C.c_int32
    L.or_reinforce_prob.argtypes = [C.c_double, C.c_int32]
    L.or_reinforce_prob.restype = C.c_double
    L.or_r_block_tables.argtypes = [C.c_double, C.c_int32, _u64p, _u64p, _u64p]
    L.or_r_block_tables.restype = None
    L.or_r_events.argtypes = [C.c_uint64, C.c_int32, C.c_int32, C.c_uint32, C.c_int32, C.c_double,
                              _u8p]
    L.or_r_events.restype = None
    L.or_gamma_rule.argtypes = [C.c_int32]
    L.or_gamma_rule.restype = C.c_int32
    L.or_layer_forward.argtypes = [_i8p, C.c_int32, C.c_int32, _i32p, C.c_int32, _i32p, _i8p]
    L.or_layer_forward.restype = None
    L.or_local_output.argtypes = [_i8p, C.c_int32, C.c_int32, _i8p, C.c_int32, _i32p]
    L.or_local_output.restype = None
    L.or_local_loss.argtypes = [_i32p, C.c_int32, C.c_int32, _i32p, C.c_int32, C.c_int32,
                                C.c_int32, _i32p, _u8p, _i32p, _u8p]
    L.or_local_loss.restype = None
    L.or_select.argtypes = [_i32p, C.c_int32, C.c_int32, _i8p, C.c_int32, _i32p, _u8p,
                            C.c_int32, _i32p, _i32p]
    L.or_group_members.argtypes = [C.c_uint64, C.c_int32, C.c_int32, C.c_int32, C.c_uint32, _i32p]
    L.or_group_members.restype = C.c_int
    L.or_set_group_mode.argtypes = [C.c_void_p, C.c_int32]
    L.or_set_group_mode.restype = C.c_int
    L.or_select.restype = None
    L.or_perceptron_update.argtypes = [_i32p, C.c_int32, C.c_int32, _i8p, _i32p, _i8p,
                                       C.c_int32, _i32p, C.c_int32, C.c_int32, C.c_int32,
                                       C.c_double, C.c_uint64, C.c_int32, C.c_uint32]
    L.or_perceptron_update.restype = None
    L.or_perceptron_update_at.argtypes = [_i32p, C.c_int32, C.c_int32, C.c_int32, _i8p, _i32p, _i8p,
                                          C.c_int32, _i32p, C.c_int32, C.c_int32, C.c_int32,
                                          C.c_double, C.c_uint64, C.c_int32, C.c_uint32]
    L.or_perceptron_update_at.restype = None
    L.or_create.argtypes = [_i32p, C.c_int32, C.c_int32, C.c_int32, C.c_uint64, C.c_int32,
                            C.c_int32, C.c_int32, C.c_double, _i32p, C.POINTER(C.c_void_p)]
    L.or_create.restype = C.c_int
    L.or_destroy.argtypes = [C.c_void_p]
    L.or_destroy.restype = None
    L.or_train.argtypes = [C.c_void_p, _i8p, _i32p, C.c_int64, C.c_int32, _i64p]
    L.or_train.restype = C.c_int
    L.or_predict.argtypes = [C.c_void_p, _i8p, C.c_int64, _i32p]
    L.or_predict.restype = C.c_int
    L.or_predict_layers.argtypes = [C.c_void_p, _i8p, C.c_int64, _i32p]
    L.or_predict_layers.restype = C.c_int
    L.or_layer_errors.argtypes = [C.c_void_p, _i64p, C.c_int32]
    L.or_layer_errors.restype = C.c_int
    L.or_binarize_median.argtypes = [C.POINTER(C.c_float), C.c_int64, C.c_int32, _i8p]
    L.or_binarize_median.restype = C.c_int
    L.or_expand_weight.argtypes = [C.c_uint64, C.c_int32, C.c_int32]
    L.or_expand_weight.restype = C.c_int32
    L.or_expand_weights.argtypes = [C.c_uint64, C.c_int32, C.c_int32, _i8p]
    L.or_expand_weights.restype = C.c_int
    L.or_expand_sign.argtypes = [_u8p, C.c_int64, C.c_int32, _i8p, C.c_int32, _i8p]
    L.or_expand_sign.restype = C.c_int
    L.or_num_layers.argtypes = [C.c_void_p]
    L.or_num_layers.restype = C.c_int32
    L.or_width.argtypes = [C.c_void_p, C.c_int32]
    L.or_width.restype = C.c_int32
    L.or_gamma.argtypes = [C.c_void_p, C.c_int32]
    L.or_gamma.restype = C.c_int32
    L.or_get_pr.argtypes = [C.c_void_p]
    L.or_get_pr.restype = C.c_double
    L.or_get_step.argtypes = [C.c_void_p]
    L.or_get_step.restype = C.c_int64
    L.or_get_layer.argtypes = [C.c_void_p, C.c_int32, _i32p, _i8p]
    L.or_get_layer.restype = C.c_int
    L.or_set_layer.argtypes = [C.c_void_p, C.c_int32, _i32p]
    L.or_set_layer.restype = C.c_int
    L.or_set_scalars.argtypes = [C.c_void_p, C.c_double, C.c_int64]
    L.or_set_scalars.restype = C.c_int
    L.or_set_threads.argtypes = [C.c_int32]
    L.or_set_threads.restype = C.c_int


def _p(a, t):
    return a.ctypes.data_as(t)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def set_threads(n: int) -> int:
    """OpenMP threads the oracle uses (0 = keep); returns the current count."""
    return lib().or_set_threads(int(n))


# -- element definitions ------------------------------------------------------

def philox4x32_10(ctr, key):
    c = _c(ctr, np.uint32)
    k = _c(key, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().or_philox4x32_10(_p(c, _u32p), _p(k, _u32p), _p(out, _u32p))
    return out


def init_h(seed, l, k, i):
    return lib().or_init_h(seed, l, k, i)


def init_rho(seed, l, k, j):
    return lib().or_init_rho(seed, l, k, j)


def reinforce_prob(p_r, K):
    return lib().or_reinforce_prob(p_r, K)


def r_block_tables(q, n):
    """Thresholds of a block of n inputs: (any, first[n], gap[n-1])."""
    any_ = np.zeros(1, np.uint64)
    first = np.zeros(64, np.uint64)
    gap = np.zeros(64, np.uint64)
    lib().or_r_block_tables(q, n, _p(any_, _u64p), _p(first, _u64p), _p(gap, _u64p))
    return int(any_[0]), first[:n].copy(), gap[:max(n - 1, 0)].copy()


def r_events(seed, l, k, t, K_prev, q):
    """Reinforcement events of neuron k (uint8 per input, 1 = reinforced)."""
    fire = np.zeros(max(K_prev, 1), np.uint8)
    lib().or_r_events(seed, l, k, t & 0xFFFFFFFF, K_prev, q, _p(fire, _u8p))
    return fire[:K_prev]


def gamma_rule(K):
    return lib().or_gamma_rule(K)


# -- the algorithm's steps, one call each -------------------------------------

def layer_forward(a_prev, H):
    """Alg. 1 l.8-9.  a_prev: b x K_prev (+-1); H: K_prev x K.  Returns (z, a)."""
    a_prev = _c(a_prev, np.int8)
    H = _c(H, np.int32)
    b, Kp = a_prev.shape
    assert H.shape[0] == Kp
    K = H.shape[1]
    z = np.zeros((b, K), np.int32)
    a = np.zeros((b, K), np.int8)
    lib().or_layer_forward(_p(a_prev, _i8p), b, Kp, _p(H, _i32p), K, _p(z, _i32p), _p(a, _i8p))
    return z, a


def local_output(a, P):
    """Alg. 1 l.10.  a: b x K; P: K x c.  Returns yhat: b x c."""
    a = _c(a, np.int8)
    P = _c(P, np.int8)
    b, K = a.shape
    c = P.shape[1]
    yhat = np.zeros((b, c), np.int32)
    lib().or_local_output(_p(a, _i8p), b, K, _p(P, _i8p), c, _p(yhat, _i32p))
    return yhat


def local_loss(yhat, y, K, r_num=1, r_den=4):
    """Eq. 1 and Alg. 1 l.11-17.  Returns (pred, ell, tau, mark)."""
    yhat = _c(yhat, np.int32)
    y = _c(y, np.int32)
    b, c = yhat.shape
    pred = np.zeros(b, np.int32)
    ell = np.zeros(b, np.uint8)
    tau = np.zeros(b, np.int32)
    mark = np.zeros(b, np.uint8)
    lib().or_local_loss(_p(yhat, _i32p), b, c, _p(y, _i32p), K, r_num, r_den, _p(pred, _i32p),
                        _p(ell, _u8p), _p(tau, _i32p), _p(mark, _u8p))
    return pred, ell, tau, mark


def select(z, P, y, mark, gamma, member=None):
    """Alg. 2 l.4-10.  Returns sel: b x G (selected neuron per group, -1 = none).
    member (O19): group g = member[g*gamma:(g+1)*gamma]; None = contiguous."""
    z = _c(z, np.int32)
    P = _c(P, np.int8)
    y = _c(y, np.int32)
    mark = _c(mark, np.uint8)
    b, K = z.shape
    c = P.shape[1]
    G = K // gamma
    sel = np.zeros((b, G), np.int32)
    mem = None if member is None else _c(member, np.int32)
    lib().or_select(_p(z, _i32p), b, K, _p(P, _i8p), c, _p(y, _i32p), _p(mark, _u8p), gamma,
                    None if mem is None else _p(mem, _i32p), _p(sel, _i32p))
    return sel


def group_members(seed, l, K, mode, t=0):
    """Group order of layer l (O19): member[j] = neuron at position j."""
    out = np.zeros(K, np.int32)
    rc = lib().or_group_members(seed & (2**64 - 1), l, K, mode, t & 0xFFFFFFFF, _p(out, _i32p))
    if rc != 0:
        raise ValueError("or_group_members failed: %d" % rc)
    return out


def perceptron_update(H, a_prev, y, P, sel, h_max, q, seed, l, t, k0=0):
    """Alg. 3 on a copy of H (K_prev x K), reinforcement probability q.
    k0: H and P hold neurons k0 .. k0 + K - 1 of the layer, sel holds neuron
    indices of the layer (or -1), and the reinforcement stream is keyed by
    those indices.  Returns the updated H."""
    H = np.array(H, dtype=np.int32, order="C", copy=True)
    a_prev = _c(a_prev, np.int8)
    y = _c(y, np.int32)
    P = _c(P, np.int8)
    sel = _c(sel, np.int32)
    Kp, K = H.shape
    b, G = sel.shape
    lib().or_perceptron_update_at(_p(H, _i32p), Kp, K, k0, _p(a_prev, _i8p), _p(y, _i32p),
                                  _p(P, _i8p), P.shape[1], _p(sel, _i32p), b, G, h_max, float(q),
                                  seed, l, t & 0xFFFFFFFF)
    return H


def binarize_median(x):
    """MedianBinarization (Alg. 1 l.5, O16): n x K fp32 -> n x K +-1 int8."""
    x = _c(x, np.float32)
    n, K = x.shape
    a = np.zeros((n, K), np.int8)
    rc = lib().or_binarize_median(x.ctypes.data_as(C.POINTER(C.c_float)), n, K, _p(a, _i8p))
    if rc != 0:
        raise ValueError("or_binarize_median failed: %d" % rc)
    return a


def expand_weight(seed, k, i):
    """Expansion weight e_{k,i} in {+-1} (O20)."""
    return int(lib().or_expand_weight(seed, k, i))


def expand_weights(seed, K, D):
    """The K x D +-1 int8 expansion matrix of O20."""
    e = np.zeros((K, D), np.int8)
    rc = lib().or_expand_weights(seed, K, D, _p(e, _i8p))
    if rc != 0:
        raise ValueError("or_expand_weights failed: %d" % rc)
    return e


def expand_sign(x, e):
    """Expansion layer (O20): n x D uint8, K x D +-1 -> n x K +-1 int8."""
    x = _c(x, np.uint8)
    e = _c(e, np.int8)
    n, D = x.shape
    K, De = e.shape
    if De != D:
        raise ValueError("x has %d inputs, e has %d" % (D, De))
    a = np.zeros((n, K), np.int8)
    rc = lib().or_expand_sign(_p(x, _u8p), n, D, _p(e, _i8p), K, _p(a, _i8p))
    if rc != 0:
        raise ValueError("or_expand_sign failed: %d" % rc)
    return a


# -- the whole rule -------------------------------------------------------------

class OracleModel:
    """A BMLP trained by Alg. 1-3 on the CPU (plain, slow, for checking)."""

    def __init__(self, widths, classes, h_max=255, seed=0, bs=100, r=(1, 4), p_r0=0.5,
                 gamma=None):
        w = _c(widths, np.int32)
        g = None if gamma is None else _c(gamma, np.int32)
        h = C.c_void_p()
        rc = lib().or_create(_p(w, _i32p), len(w), classes, h_max, seed & (2**64 - 1), bs,
                             r[0], r[1], p_r0, None if g is None else _p(g, _i32p), C.byref(h))
        if rc != 0:
            raise ValueError("or_create failed: %d" % rc)
        self._h = h
        self.widths = [int(v) for v in w]
        self.L = len(w) - 1
        self.classes = classes

    def close(self):
        if self._h:
            lib().or_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def train(self, x, y, epoch_end=False):
        """x: n x K_0 (+-1 int8), y: n labels.  Returns the last-layer error count."""
        x = _c(x, np.int8)
        y = _c(y, np.int32)
        n = y.shape[0]
        assert x.shape == (n, self.widths[0])
        err = C.c_int64(0)
        rc = lib().or_train(self._h, _p(x, _i8p), _p(y, _i32p), n, 1 if epoch_end else 0,
                            C.byref(err))
        if rc != 0:
            raise ValueError("or_train failed: %d" % rc)
        return int(err.value)

    def predict(self, x):
        x = _c(x, np.int8)
        n = x.shape[0]
        out = np.zeros(n, np.int32)
        rc = lib().or_predict(self._h, _p(x, _i8p), n, _p(out, _i32p))
        if rc != 0:
            raise ValueError("or_predict failed: %d" % rc)
        return out

    def predict_layers(self, x):
        """Early-exit predictions (O17): (L, n), row l-1 = argmax of a_l P_l."""
        x = _c(x, np.int8)
        n = x.shape[0]
        out = np.zeros((self.L, n), np.int32)
        rc = lib().or_predict_layers(self._h, _p(x, _i8p), n, _p(out, _i32p))
        if rc != 0:
            raise ValueError("or_predict_layers failed: %d" % rc)
        return out

    def layer_errors(self, reset=False):
        """Local 01-loss counts of layers 1..L since creation or the last reset."""
        out = np.zeros(self.L, np.int64)
        lib().or_layer_errors(self._h, _p(out, _i64p), 1 if reset else 0)
        return [int(v) for v in out]

    def set_group_mode(self, mode):
        """Group membership of every layer (O19): 0 contiguous, 1 fixed random,
        2 redrawn at every mini-batch step."""
        if lib().or_set_group_mode(self._h, mode) != 0:
            raise ValueError("or_set_group_mode failed")

    def gamma(self, l):
        return lib().or_gamma(self._h, l)

    def H(self, l):
        """Hidden weights of layer l (1-based), K_{l-1} x K_l, paper orientation."""
        H = np.zeros((self.widths[l - 1], self.widths[l]), np.int32)
        lib().or_get_layer(self._h, l, _p(H, _i32p), None)
        return H

    def P(self, l):
        P = np.zeros((self.widths[l], self.classes), np.int8)
        lib().or_get_layer(self._h, l, None, _p(P, _i8p))
        return P

    def set_H(self, l, H):
        H = _c(H, np.int32)
        assert H.shape == (self.widths[l - 1], self.widths[l])
        if lib().or_set_layer(self._h, l, _p(H, _i32p)) != 0:
            raise ValueError("or_set_layer failed")

    @property
    def p_r(self):
        return lib().or_get_pr(self._h)

    @property
    def step(self):
        return int(lib().or_get_step(self._h))

    def set_scalars(self, p_r, step):
        if lib().or_set_scalars(self._h, p_r, step) != 0:
            raise ValueError("or_set_scalars failed")
