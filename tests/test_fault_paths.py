"""Failure paths of the library, forced on the host -- no GPU fault, trap or
hang is involved:

  * an allocation that fails (injected: bmlp_debug_fail_alloc) at every
    allocation point of bmlp_create, and in the host-buffer staging of
    bmlp_train: BMLP_ENOMEM, nothing leaked (bmlp_debug_alloc_stats), the
    handle (when there is one) still trains bit for bit like the oracle;
  * an expired bounded device wait left pending across a training step (the
    wait probe with nothing arriving): that step changes neither H nor W, the
    error is reported by the next synchronising call, and training then
    continues exactly like the oracle with that step skipped."""
import os

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2412_00119_gb300 import bmlp as B
from test_gpu_parity import assert_same_state, dev_x, dev_y

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(DEV)
    O.set_threads(os.cpu_count() or 1)
    B.lib()
    yield
    B.bmlp_debug_fail_alloc(0)


def _allocations_of_create(widths, classes, **kw):
    base = B.bmlp_debug_alloc_stats()
    h = B.bmlp_create(widths, classes, **kw)
    n = B.bmlp_debug_alloc_stats()[0] - base[0]
    B.bmlp_destroy(h)
    assert B.bmlp_debug_alloc_stats() == base
    return n


@pytest.mark.parametrize("fwd", [B.BMLP_FWD_TCGEN05, B.BMLP_FWD_POPC])
def test_create_frees_everything_after_each_failed_allocation(fwd):
    widths, c = (200, 130, 70), 10
    kw = dict(seed=3, bs=50, gamma=[13, 7], fwd_impl=fwd)
    n_alloc = _allocations_of_create(widths, c, **kw)
    assert n_alloc >= 10 * 2 + 4
    base = B.bmlp_debug_alloc_stats()
    for nth in range(1, n_alloc + 1):
        B.bmlp_debug_fail_alloc(nth)
        with pytest.raises(B.BmlpError) as ei:
            B.bmlp_create(widths, c, **kw)
        assert ei.value.code == B.BMLP_ENOMEM, nth
        assert "injected" in str(ei.value), nth
        assert B.bmlp_debug_alloc_stats() == base, nth
    # past the last allocation point the injection never fires
    B.bmlp_debug_fail_alloc(n_alloc + 1)
    h = B.bmlp_create(widths, c, **kw)
    B.bmlp_destroy(h)
    B.bmlp_debug_fail_alloc(0)
    assert B.bmlp_debug_alloc_stats() == base


def test_staging_allocation_failure_leaves_handle_usable():
    widths, c = (130, 96), 5
    cfg = W.small_config(widths, c, 300, 0, teacher_hidden=16)
    tr = W.make_split(cfg, "train")
    gpu = B.BMLP(widths, c, seed=5, bs=100)
    ref = O.OracleModel(list(widths), c, seed=5, bs=100)
    held = B.bmlp_debug_alloc_stats()
    B.bmlp_debug_fail_alloc(1)   # the first staging buffer of a host-buffer call
    with pytest.raises(B.BmlpError) as ei:
        gpu.train(tr.xp, tr.y)
    assert ei.value.code == B.BMLP_ENOMEM
    assert B.bmlp_debug_alloc_stats() == held
    assert_same_state(gpu, ref, "after the failed call")
    eg = gpu.train(tr.xp, tr.y, epoch_end=True, count_errors=True)
    er = ref.train(tr.pm1(), tr.y, epoch_end=True)
    assert eg == er
    assert_same_state(gpu, ref, "after the retried call")
    gpu.close()


def test_pending_timeout_skips_the_update():
    widths, c, bs = (200, 130, 70), 10, 50
    cfg = W.small_config(widths, c, 400, 0, teacher_hidden=16)
    tr = W.make_split(cfg, "train")
    gpu = B.BMLP(widths, c, seed=8, bs=bs, gamma=[13, 7], fwd_impl=B.BMLP_FWD_TCGEN05)
    ref = O.OracleModel(list(widths), c, seed=8, bs=bs, gamma=[13, 7])
    x, y, xo = dev_x(tr.xp), dev_y(tr.y), tr.pm1()
    gpu.train(x[:200], y[:200])
    ref.train(xo[:200], tr.y[:200])
    assert_same_state(gpu, ref, "before the expiry")
    B.bmlp_debug_wait_probe(gpu.h, arrive=False, seconds=0.05, leave_pending=True)
    with pytest.raises(B.BmlpError) as ei:   # one mini-batch while the expiry is pending
        gpu.train(x[200:250], y[200:250], count_errors=True)
    assert ei.value.code == B.BMLP_ETIMEOUT
    # the skipped mini-batch changed no weight; only the step counter moved
    ref.set_scalars(ref.p_r, ref.step + 1)
    assert_same_state(gpu, ref, "after the skipped mini-batch")
    gpu.train(x[250:], y[250:])
    ref.train(xo[250:], tr.y[250:])
    assert_same_state(gpu, ref, "after training on")
    gpu.close()
