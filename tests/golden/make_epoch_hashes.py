"""Write tests/golden/epochs_<config>.json: SHA-256 digests of the CPU oracle's
model state after every epoch of the five seeded workloads, for the GPU test
that checks the library against them (tests/test_epoch_golden.py).

Only the oracle (oracle/, Alg. 1-3 step by step) and the input generators
(workloads.py) are called here; nothing comes from the GPU library.

What is recorded per checkpoint (the end of every epoch; for the 8192-wide
stress workload, whose single epoch is 10,000 mini-batches, the ends of its
first 20 and 100 mini-batches):
  * every layer's hidden weights H (int16, K_l rows of K_{l-1}: neuron-major,
    the export format of bmlp_get_state), visible weights W = pack(sign(H))
    (uint64, K_l rows of ceil(K_{l-1}/64) words) and local classifier P
    (int8, K_l x c), as SHA-256 of their little-endian bytes;
  * the last-layer 01-loss count of the epoch's training passes (Alg. 1
    l.11-17), p_r after the epoch end (Alg. 1 l.21) as a float hex string, and
    the step counter;
  * the SHA-256 of the test predictions (int32, argmax of a_L P_L, Sec. 3.1)
    and their accuracy against the teacher labels (information only).
Inputs and labels are hashed too, so that a test run on another machine
first proves it trains on the same data.

Run (minutes to about an hour on 8 host cores; each config is written as
soon as it finishes):
    python tests/golden/make_epoch_hashes.py [C1 C2 ...]
"""
from __future__ import annotations

import hashlib
import json
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import oracle as O  # noqa: E402
import workloads as W  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))

# the stress workload: checkpoints (mini-batches trained so far) and the test
# patterns predicted at the last one
C5_CHECKPOINTS = (20, 100)
C5_TEST = 1024


def sha(a, dtype) -> str:
    return hashlib.sha256(np.ascontiguousarray(a, dtype=dtype).tobytes()).hexdigest()


def state_digest(ref) -> list:
    out = []
    for l in range(1, ref.L + 1):
        H = ref.H(l).T  # K_l x K_{l-1}, neuron-major
        out.append({"H": sha(H, "<i2"),
                    "W": sha(W.pack(np.where(H > 0, 1, -1)), "<u8"),
                    "P": sha(ref.P(l), "i1")})
    return out


def golden_path(key: str) -> str:
    return os.path.join(HERE, "epochs_%s.json" % key)


def epochs_golden(key: str) -> dict:
    cfg = W.CONFIGS[key]
    t0 = time.time()
    tr, te = W.make_split(cfg, "train"), W.make_split(cfg, "test")
    ref = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
    xo, xt = tr.pm1(), te.pm1()
    rec = {"config": key, "widths": list(cfg.widths), "classes": cfg.classes,
           "model_seed": cfg.model_seed, "bs": 100, "h_max": 255, "r": [1, 4], "p_r0": 0.5,
           "inputs": {"train_x": sha(tr.xp, "<u8"), "train_y": sha(tr.y, "<i4"),
                      "test_x": sha(te.xp, "<u8"), "test_y": sha(te.y, "<i4"),
                      "n_train": int(len(tr.y)), "n_test": int(len(te.y))},
           "checkpoints": []}
    for e in range(cfg.epochs):
        err = ref.train(xo, tr.y, epoch_end=True)
        pred = ref.predict(xt)
        rec["checkpoints"].append({
            "epoch": e + 1, "minibatches": int(ref.step), "errors": int(err),
            "p_r": float(ref.p_r).hex(), "step": int(ref.step), "layers": state_digest(ref),
            "test_pred": sha(pred, "<i4"), "test_acc": float(np.mean(pred == te.y))})
        print("%s epoch %d: errors %d, p_r %r, test acc %.4f (%.0f s)"
              % (key, e + 1, err, ref.p_r, np.mean(pred == te.y), time.time() - t0), flush=True)
    ref.close()
    rec["oracle_seconds"] = time.time() - t0
    return rec


def stress_golden() -> dict:
    cfg = W.CONFIGS["C5"]
    t0 = time.time()
    n = 100 * max(C5_CHECKPOINTS)
    xp = W.make_inputs(cfg, "train", n)
    xo = W.unpack(xp, cfg.widths[0])
    y = W.teacher_labels_pm1(W.make_teacher(cfg), xo)
    xt = W.make_inputs(cfg, "test", C5_TEST)
    ref = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
    rec = {"config": "C5", "widths": list(cfg.widths), "classes": cfg.classes,
           "model_seed": cfg.model_seed, "bs": 100, "h_max": 255, "r": [1, 4], "p_r0": 0.5,
           "inputs": {"train_x": sha(xp, "<u8"), "train_y": sha(y, "<i4"),
                      "test_x": sha(xt, "<u8"), "n_train": n, "n_test": C5_TEST},
           "checkpoints": []}
    done = 0
    for cp in C5_CHECKPOINTS:
        a, b = 100 * done, 100 * cp
        err = ref.train(xo[a:b], y[a:b])
        done = cp
        c = {"minibatches": cp, "errors": int(err), "p_r": float(ref.p_r).hex(),
             "step": int(ref.step), "layers": state_digest(ref)}
        if cp == C5_CHECKPOINTS[-1]:
            pred = ref.predict(W.unpack(xt, cfg.widths[0]))
            c["test_pred"] = sha(pred, "<i4")
        rec["checkpoints"].append(c)
        print("C5 after %d mini-batches: errors %d (%.0f s)" % (cp, err, time.time() - t0),
              flush=True)
    ref.close()
    rec["oracle_seconds"] = time.time() - t0
    return rec


def main(argv) -> int:
    keys = argv or ["C1", "C2", "C3", "C5", "C4"]
    cores = O.set_threads(os.cpu_count() or 1)
    for key in keys:
        rec = stress_golden() if key == "C5" else epochs_golden(key)
        rec["oracle_threads"] = cores
        rec["written_by"] = "tests/golden/make_epoch_hashes.py (CPU oracle only)"
        with open(golden_path(key), "w") as f:
            json.dump(rec, f, indent=1)
            f.write("\n")
        print("wrote", golden_path(key), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main(sys.argv[1:]))
