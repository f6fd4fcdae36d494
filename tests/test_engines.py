"""The forward contraction (Alg. 1 l.8-9) on every unit that runs it: the
CUDA-core XOR/popcount kernel, the e4m3 tcgen05 kernel and the b1 mma.sync
kernel give the oracle's packed sign(a W) bit for bit, at the training shape
(100 patterns on an 8192 x 8192 layer), on ragged shapes, and on sampled rows
of the 65,536-pattern sweep; and each unit's peak kernel runs."""
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2412_00119_gb300 import bmlp as B
from test_gpu_parity import dev_x

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
ENGINES = {"popc": B.BMLP_FWD_POPC, "tcgen05": B.BMLP_FWD_TCGEN05, "b1mma": B.BMLP_FWD_B1MMA}


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(DEV)
    O.set_threads(os.cpu_count() or 1)
    B.lib()


# (widths, n): single bit; one 16 x 8 tile; ragged K / neurons / patterns;
# the training shape; odd word counts (8-byte rows)
CASES = [((1, 8), 5), ((64, 16), 8), ((130, 257, 129), 129), ((1100, 700, 300), 1000),
         ((8192, 8192), 100), ((960, 1000), 33), ((3072, 4096), 104), ((8192, 8192), 300)]


@pytest.mark.parametrize("engine", sorted(ENGINES))
@pytest.mark.parametrize("widths,n", CASES)
def test_layer_forward_engine_matches_oracle(widths, n, engine):
    gpu = B.BMLP(widths, 4, seed=9, bs=64)
    ref = O.OracleModel(list(widths), 4, seed=9, bs=64)
    for l in range(1, len(widths)):
        xp = W.random_packed(100 * l + n, n, widths[l - 1])
        out = torch.full((n, W.words(widths[l])), -1, dtype=torch.int64, device=DEV)
        B.bmlp_layer_forward_engine(gpu.h, l, ENGINES[engine], dev_x(xp), out)
        _, a = O.layer_forward(W.unpack(xp, widths[l - 1]), ref.H(l))
        assert np.array_equal(out.cpu().numpy().view(np.uint64), W.pack(a)), (engine, widths, l)
    gpu.close()


@pytest.mark.parametrize("engine", sorted(ENGINES))
def test_sweep_shape_sampled(engine):
    """65,536 patterns through one 8192 x 8192 layer (the evaluation sweep's
    launch): 400 sampled rows, both ends among them, equal the oracle's."""
    widths, n = (8192, 8192), 65536
    gpu = B.BMLP(widths, 4, seed=12, bs=64)
    ref = O.OracleModel(list(widths), 4, seed=12, bs=64)
    xp = W.random_packed(4242, n, widths[0])
    out = torch.full((n, W.words(widths[1])), -1, dtype=torch.int64, device=DEV)
    B.bmlp_layer_forward_engine(gpu.h, 1, ENGINES[engine], dev_x(xp), out)
    rng = np.random.default_rng(5)
    rows = np.unique(np.concatenate([np.arange(130), np.arange(n - 130, n),
                                     rng.integers(0, n, 140)]))
    _, a = O.layer_forward(W.unpack(xp[rows], widths[0]), ref.H(1))
    assert np.array_equal(out.cpu().numpy().view(np.uint64)[rows], W.pack(a))
    gpu.close()


def test_b1_unaligned_rows():
    """Input rows at an 8-byte (not 16-byte) offset take the word-by-word
    staging path of the b1 kernel; same bits."""
    widths, n = (1100, 700), 150
    gpu = B.BMLP(widths, 4, seed=9, bs=64)
    ref = O.OracleModel(list(widths), 4, seed=9, bs=64)
    nw = W.words(widths[0])
    xp = W.random_packed(31, n, widths[0])
    flat = torch.zeros(n * nw + 1, dtype=torch.int64, device=DEV)
    flat[1:] = dev_x(xp).reshape(-1)
    x = flat[1:].view(n, nw)
    assert x.data_ptr() % 16 == 8
    out = torch.full((n, W.words(widths[1])), -1, dtype=torch.int64, device=DEV)
    B.bmlp_layer_forward_engine(gpu.h, 1, B.BMLP_FWD_B1MMA, x, out)
    _, a = O.layer_forward(W.unpack(xp, widths[0]), ref.H(1))
    assert np.array_equal(out.cpu().numpy().view(np.uint64), W.pack(a))
    gpu.close()


@pytest.mark.parametrize("engine", [B.BMLP_FWD_POPC, B.BMLP_FWD_TCGEN05, B.BMLP_FWD_B1MMA,
                                    B.BMLP_FWD_S8MMA])
def test_engine_peak_kernel_runs(engine):
    rate, ms = B.bmlp_engine_peak(engine, 2000)
    assert math.isfinite(rate) and rate > 0 and ms > 0
