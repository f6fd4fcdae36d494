"""The GPU library against the CPU oracle after every epoch of the five seeded
workloads, bit for bit (tolerance 0: every quantity of the rule is an integer
or a bit).  The oracle's side is stored as SHA-256 digests in
tests/golden/epochs_<config>.json, written by tests/golden/make_epoch_hashes.py,
which calls only the oracle and the input generators (the full runs take the
oracle about an hour on 8 host cores; the GPU side takes seconds).

Per checkpoint -- the end of every epoch (Alg. 1 l.21), and for the 8192-wide
stress workload the ends of its first 20 and 100 mini-batches -- the test
compares every layer's hidden weights H, visible weights W and local
classifier P, the epoch's last-layer error count, p_r and the step counter,
and the test predictions.  It first checks that this machine generates the
same inputs and labels the digests were made from."""
import hashlib
import json
import os

import numpy as np
import pytest
import torch

import workloads as W
from conftest import golden_path
from paper_2412_00119_gb300 import bmlp as B

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(DEV)
    B.lib()


def sha(a, dtype):
    return hashlib.sha256(np.ascontiguousarray(a, dtype=dtype).tobytes()).hexdigest()


def load(key):
    with open(golden_path("epochs_%s.json" % key)) as f:
        return json.load(f)


def dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).to(DEV)


def check_state(gpu, g, cp, where):
    for l in range(1, len(g["widths"])):
        H, Wp, P, p_r, step = gpu.state(l)
        want = cp["layers"][l - 1]
        assert sha(H, "<i2") == want["H"], "H of layer %d differs %s" % (l, where)
        assert sha(Wp, "<u8") == want["W"], "W of layer %d differs %s" % (l, where)
        assert sha(P, "i1") == want["P"], "P of layer %d differs %s" % (l, where)
    assert p_r == float.fromhex(cp["p_r"]), (p_r, cp["p_r"], where)
    assert step == cp["step"], (step, cp["step"], where)


def model(g):
    return B.BMLP(g["widths"], g["classes"], h_max=g["h_max"], seed=g["model_seed"], bs=g["bs"],
                  r=tuple(g["r"]), p_r0=g["p_r0"])


@pytest.mark.parametrize("key", ["C1", "C2", "C3", "C4"])
def test_every_epoch_matches_oracle(key):
    g = load(key)
    cfg = W.CONFIGS[key]
    tr, te = W.make_split(cfg, "train"), W.make_split(cfg, "test")
    assert sha(tr.xp, "<u8") == g["inputs"]["train_x"], "training inputs differ on this machine"
    assert sha(tr.y, "<i4") == g["inputs"]["train_y"], "training labels differ on this machine"
    assert sha(te.xp, "<u8") == g["inputs"]["test_x"], "test inputs differ on this machine"
    gpu = model(g)
    x, y, xt = dev(tr.xp, np.int64), dev(tr.y, np.int32), dev(te.xp, np.int64)
    assert len(g["checkpoints"]) == cfg.epochs
    for cp in g["checkpoints"]:
        where = "after epoch %d of %s" % (cp["epoch"], key)
        err = gpu.train(x, y, epoch_end=True, count_errors=True)
        assert err == cp["errors"], (err, cp["errors"], where)
        check_state(gpu, g, cp, where)
        out = torch.full((len(te.y),), -1, dtype=torch.int32, device=DEV)
        gpu.predict(xt, out)
        assert sha(out.cpu().numpy(), "<i4") == cp["test_pred"], "test predictions differ " + where
    gpu.close()


def test_stress_prefix_matches_oracle():
    """8192 -> 8192 x4 -> 10 in the bench's launch configuration (tensor-core
    forward, eight-step graphs): 20 mini-batches, then 80 more, in two calls."""
    g = load("C5")
    cfg = W.CONFIGS["C5"]
    n = g["inputs"]["n_train"]
    xp = W.make_inputs(cfg, "train", n)
    y = W.teacher_labels_pm1(W.make_teacher(cfg), W.unpack(xp, cfg.widths[0]))
    xt = W.make_inputs(cfg, "test", g["inputs"]["n_test"])
    assert sha(xp, "<u8") == g["inputs"]["train_x"], "training inputs differ on this machine"
    assert sha(y, "<i4") == g["inputs"]["train_y"], "training labels differ on this machine"
    assert sha(xt, "<u8") == g["inputs"]["test_x"], "test inputs differ on this machine"
    gpu = model(g)
    assert gpu.info["fwd_impl"] == B.BMLP_FWD_TCGEN05
    x, yd = dev(xp, np.int64), dev(y, np.int32)
    done = 0
    for cp in g["checkpoints"]:
        a, b = 100 * done, 100 * cp["minibatches"]
        err = gpu.train(x[a:b], yd[a:b], count_errors=True)
        done = cp["minibatches"]
        where = "after %d mini-batches" % done
        assert err == cp["errors"], (err, cp["errors"], where)
        check_state(gpu, g, cp, where)
        if "test_pred" in cp:
            out = torch.full((len(xt),), -1, dtype=torch.int32, device=DEV)
            gpu.predict(dev(xt, np.int64), out)
            assert sha(out.cpu().numpy(), "<i4") == cp["test_pred"], "predictions differ " + where
    gpu.close()
