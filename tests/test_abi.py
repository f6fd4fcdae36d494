"""The C-ABI library without a GPU: it loads, exports every entry point that
include/bmlp.h declares, validates arguments before touching CUDA, and its
host-side arithmetic agrees with the oracle's independent version."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from conftest import ROOT

import paper_2412_00119_gb300 as pkg
from paper_2412_00119_gb300 import bmlp as B


def declared_functions():
    with open(os.path.join(ROOT, "include", "bmlp.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bmlp_[a-z_0-9]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    lib = pkg.lib()
    names = declared_functions()
    assert len(names) >= 15
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(n for n, _, _ in B.SIGNATURES) == names


def test_gamma_rule_matches_oracle(oracle_mod):
    for K in list(range(1, 400)) + [525, 784, 1024, 1035, 2025, 2048, 4096, 8192, 10000]:
        assert B.bmlp_gamma_rule(K) == oracle_mod.gamma_rule(K), K
    assert B.bmlp_gamma_rule(0) == -1


def test_sampler_tables_match_oracle(oracle_mod):
    """The library's reinforcement-sampler thresholds (host code) equal the
    oracle's, entry for entry, for every block length."""
    for p_r in (0.0, 1e-9, 0.01, 0.1234567, 0.25, 0.5, 0.9, 1.0, 3.0):
        for K in (1, 2, 3, 10, 64, 100, 256, 784, 1024, 4096, 8192, 65536):
            q = oracle_mod.reinforce_prob(p_r, K)
            for n in (1, 2, 5, 17, 63, 64):
                a, f, g = B.bmlp_reinforce_tables(p_r, K, n)
                ao, fo, go = oracle_mod.r_block_tables(q, n)
                assert a == ao and np.array_equal(f, fo) and np.array_equal(g, go), (p_r, K, n)
    with pytest.raises(B.BmlpError):
        B.bmlp_reinforce_tables(0.5, 10, 65)
    with pytest.raises(B.BmlpError):
        B.bmlp_reinforce_tables(0.5, 0, 8)


@pytest.mark.parametrize("kw,msg", [
    (dict(widths=[10], classes=2), "n_widths"),
    (dict(widths=[10, 0], classes=2), "width"),
    (dict(widths=[10, 8], classes=1), "classes"),
    (dict(widths=[10, 8], classes=2, h_max=4), "h_max"),
    (dict(widths=[10, 8], classes=2, h_max=16385), "h_max"),
    (dict(widths=[10, 8], classes=2, bs=2000), "bs"),
    (dict(widths=[10, 8], classes=2, gamma=[3]), "gamma"),
    (dict(widths=[10, 8], classes=2, r=(-1, 4)), "r must"),
    (dict(widths=[10, 8], classes=2, fwd_impl=7), "fwd_impl"),
    (dict(widths=[10, 8], classes=2, group_mode=3), "group_mode"),
    (dict(widths=[10, 20000], classes=2, gamma=[100], group_mode=1), "16384"),
])
def test_create_rejects_bad_arguments(kw, msg):
    with pytest.raises(B.BmlpError) as ei:
        B.bmlp_create(**kw)
    assert ei.value.code == B.BMLP_EINVAL
    assert msg in str(ei.value)


def test_create_without_gpu_reports_no_device():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(B.BmlpError) as ei:
        B.bmlp_create([16, 8], 2)
    assert ei.value.code == B.BMLP_ENODEV


def test_binarize_rejects_bad_arguments():
    lib = pkg.lib()
    assert lib.bmlp_binarize_median(None, -1, 8, None, None) == B.BMLP_EINVAL
    assert b"n < 0" in lib.bmlp_last_error(None)
    assert lib.bmlp_binarize_median(None, 4, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_binarize_median(None, 0, 8, None, None) == B.BMLP_OK
    x = np.zeros((4, 8), np.float32)
    out = np.zeros((4, 1), np.uint64)
    assert lib.bmlp_binarize_median(x.ctypes.data, 4, 8, out.ctypes.data, None) == B.BMLP_EINVAL
    assert b"device pointers" in lib.bmlp_last_error(None)


def test_expansion_rejects_bad_arguments():
    lib = pkg.lib()
    assert lib.bmlp_expand_weights(1, 0, 8, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_expand_weights(1, 8, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_expand_weights(1, 8, (1 << 23) + 1, None, None) == B.BMLP_EINVAL
    assert b"2^23" in lib.bmlp_last_error(None)
    E = np.zeros((8, 1), np.uint64)
    assert lib.bmlp_expand_weights(1, 8, 8, E.ctypes.data, None) == B.BMLP_EINVAL
    assert b"device pointer" in lib.bmlp_last_error(None)
    assert lib.bmlp_expand_sign(None, -1, 8, None, 8, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_expand_sign(None, 4, 8, None, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_expand_sign(None, 4, 0, None, 8, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_expand_sign(None, 0, 8, None, 8, None, None) == B.BMLP_OK
    x = np.zeros((4, 8), np.uint8)
    out = np.zeros((4, 1), np.uint64)
    assert lib.bmlp_expand_sign(x.ctypes.data, 4, 8, E.ctypes.data, 8, out.ctypes.data,
                                None) == B.BMLP_EINVAL
    assert b"device pointers" in lib.bmlp_last_error(None)


def test_null_handle_calls_fail_cleanly():
    lib = pkg.lib()
    assert lib.bmlp_predict_layers(None, None, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_layer_errors(None, None, 0) == B.BMLP_EINVAL
    assert lib.bmlp_debug_wait_probe(None, 0, 0.05) == B.BMLP_EINVAL
    assert lib.bmlp_train(None, None, None, 0, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_predict(None, None, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_get_state(None, 1, None, None, None, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_launch_count(None) == -1
    lib.bmlp_destroy(None)
    assert lib.bmlp_layer_forward_engine(None, 1, 1, None, 0, None, None) == B.BMLP_EINVAL
    assert lib.bmlp_predict_noalloc(None, None, 0, None, None) == B.BMLP_EINVAL


def test_engine_peak_rejects_bad_arguments():
    lib = pkg.lib()
    with pytest.raises(B.BmlpError) as ei:
        B.bmlp_engine_peak(99, 10)
    assert ei.value.code == B.BMLP_EINVAL and "engine" in str(ei.value)
    with pytest.raises(B.BmlpError):
        B.bmlp_engine_peak(B.BMLP_FWD_POPC, 0)
    assert lib.bmlp_engine_peak(B.BMLP_FWD_POPC, 10, None, None) == B.BMLP_EINVAL


def test_alloc_injection_host_side():
    """Arming and disarming the injected allocation failure and reading the
    live-allocation counters need no device; no handle exists here."""
    assert B.bmlp_debug_alloc_stats() == (0, 0)
    with pytest.raises(B.BmlpError):
        B.bmlp_debug_fail_alloc(-1)
    B.bmlp_debug_fail_alloc(3)
    B.bmlp_debug_fail_alloc(0)
