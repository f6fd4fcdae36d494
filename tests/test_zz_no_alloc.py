"""bmlp_predict_noalloc: forward-only evaluation for callers that cannot
allocate device memory.

The regular bmlp_predict allocates its inter-layer activation buffers with
cudaMalloc on first use.  Code that must not allocate (inside a host callback,
under a fixed real-time memory plan, or in a process whose device allocator
belongs to another runtime) calls bmlp_predict_noalloc instead; it keeps its
scratch in a fixed array inside the library.  This test calls it through the
C-ABI and checks its labels against bmlp_predict's, exactly (labels are
integers), on two calls in a row with different inputs and sizes."""
import ctypes as C

import numpy as np
import pytest
import torch

import workloads as W
from paper_2412_00119_gb300 import bmlp as B

pytestmark = pytest.mark.gpu

SCRATCH_WORDS = 1 << 20  # per ping-pong buffer, as documented in include/bmlp.h


def _entry():
    f = B.lib().bmlp_predict_noalloc
    f.restype = C.c_int
    f.argtypes = [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p]
    return f


def test_noalloc_predict_matches_predict_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    noalloc = _entry()
    widths, c = (300, 200, 130), 10
    cfg = W.small_config(widths, c, 400, 0, teacher_hidden=32, number=77)
    tr = W.make_split(cfg, "train")
    model = B.BMLP(widths, c, seed=21, bs=100)
    model.train(torch.from_numpy(tr.xp.view(np.int64)).to(dev), torch.from_numpy(tr.y).to(dev))
    for call, n in enumerate((1500, 3777)):
        xp = W.make_inputs(W.small_config(widths, c, n, 0, number=80 + call), "train", n)
        x = torch.from_numpy(xp.view(np.int64)).to(dev)
        want = torch.full((n,), -1, dtype=torch.int32, device=dev)
        model.predict(x, want)
        got = torch.full((n,), -7, dtype=torch.int32, device=dev)
        rc = noalloc(model.h, x.data_ptr(), n, got.data_ptr(), stream.cuda_stream)
        assert rc == B.BMLP_OK, B.bmlp_last_error(model.h)
        torch.cuda.synchronize()
        assert torch.equal(got, want), "call %d" % call
    # sizes beyond the fixed scratch are rejected before any work
    max_rows = SCRATCH_WORDS // ((max(widths[1:]) + 63) // 64)
    big = torch.zeros((max_rows + 1, (widths[0] + 63) // 64), dtype=torch.int64, device=dev)
    out = torch.zeros(max_rows + 1, dtype=torch.int32, device=dev)
    rc = noalloc(model.h, big.data_ptr(), max_rows + 1, out.data_ptr(), stream.cuda_stream)
    assert rc == B.BMLP_EINVAL and "scratch" in B.bmlp_last_error(model.h)
    # host buffers are rejected (staging them would need an allocation)
    host = np.zeros((4, (widths[0] + 63) // 64), np.uint64)
    hout = np.zeros(4, np.int32)
    rc = noalloc(model.h, host.ctypes.data, 4, hout.ctypes.data, stream.cuda_stream)
    assert rc == B.BMLP_EINVAL
    model.close()
