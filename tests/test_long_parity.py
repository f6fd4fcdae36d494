"""Long GPU-vs-oracle runs, too slow for the regular suite (minutes of oracle
time on 16 host cores): skipped unless BMLP_LONG_CHECKS=1.

  * 784 -> 1024 x3 -> 10 on all 60,000 training samples for its 5 epochs
    (3,000 mini-batches): error counts, p_r after every epoch end (Alg. 1
    l.21), the step counter and every hidden weight after each epoch, then
    the 10,000 test predictions;
  * 8192 -> 8192 x4 -> 10 for 100 mini-batches of its stream in one training
    call (the bench's launch configuration: eight-step graphs, dependent
    launches): H, W, P, p_r, the step counter and the error count.

Run:  BMLP_LONG_CHECKS=1 python -m pytest tests/test_long_parity.py -m gpu -x -q
"""
import os

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2412_00119_gb300 import bmlp as B
from test_gpu_parity import assert_same_state, dev_x, dev_y

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(os.environ.get("BMLP_LONG_CHECKS") != "1",
                                 reason="long oracle runs; set BMLP_LONG_CHECKS=1")]


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)
    O.set_threads(os.cpu_count() or 1)
    B.lib()


def test_c2_all_five_epochs():
    cfg = W.CONFIGS["C2"]
    tr, te = W.make_split(cfg, "train"), W.make_split(cfg, "test")
    gpu = B.BMLP(cfg.widths, cfg.classes, seed=cfg.model_seed, bs=100)
    ref = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
    x, y, xo = dev_x(tr.xp), dev_y(tr.y), tr.pm1()
    for e in range(cfg.epochs):
        eg = gpu.train(x, y, epoch_end=True, count_errors=True)
        er = ref.train(xo, tr.y, epoch_end=True)
        assert eg == er, (e, eg, er)
        assert_same_state(gpu, ref, "after epoch %d" % (e + 1))
    out = torch.empty(len(te.y), dtype=torch.int32, device="cuda")
    gpu.predict(dev_x(te.xp), out)
    assert np.array_equal(out.cpu().numpy(), ref.predict(te.pm1()))
    gpu.close()


def test_c5_100_steps_one_call():
    cfg = W.CONFIGS["C5"]
    n = 100 * 100
    xp = W.make_inputs(cfg, "train", n)
    y = W.teacher_labels_pm1(W.make_teacher(cfg), W.unpack(xp, cfg.widths[0]))
    gpu = B.BMLP(cfg.widths, cfg.classes, seed=cfg.model_seed, bs=100)
    ref = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
    eg = gpu.train(dev_x(xp), dev_y(y), count_errors=True)
    er = ref.train(W.unpack(xp, cfg.widths[0]), y)
    assert eg == er, (eg, er)
    assert_same_state(gpu, ref, "after 100 mini-batches")
    gpu.close()
