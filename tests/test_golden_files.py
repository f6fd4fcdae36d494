"""CPU checks of the per-epoch digest fixtures (tests/golden/epochs_*.json):
each was written by the oracle-only script, names its workload's exact shape
and seeds, and covers every epoch of that workload (the stress workload: its
20- and 100-mini-batch prefix)."""
import json
import math

import pytest

import workloads as W
from conftest import golden_path

KEYS = ("C1", "C2", "C3", "C4", "C5")


@pytest.mark.parametrize("key", KEYS)
def test_digest_file_covers_its_workload(key):
    with open(golden_path("epochs_%s.json" % key)) as f:
        g = json.load(f)
    cfg = W.CONFIGS[key]
    assert g["written_by"].startswith("tests/golden/make_epoch_hashes.py")
    assert g["config"] == key and g["widths"] == list(cfg.widths) and g["classes"] == cfg.classes
    assert g["model_seed"] == cfg.model_seed and g["bs"] == 100 and g["h_max"] == 255
    assert g["r"] == [1, 4] and g["p_r0"] == 0.5
    L = len(cfg.widths) - 1
    for cp in g["checkpoints"]:
        assert len(cp["layers"]) == L
        for lay in cp["layers"]:
            assert all(len(lay[k]) == 64 for k in ("H", "W", "P"))
        float.fromhex(cp["p_r"])
    if key == "C5":
        assert [c["minibatches"] for c in g["checkpoints"]] == [20, 100]
        assert "test_pred" in g["checkpoints"][-1]
    else:
        assert [c["epoch"] for c in g["checkpoints"]] == list(range(1, cfg.epochs + 1))
        steps = cfg.n_train // 100
        assert [c["step"] for c in g["checkpoints"]] == [steps * (e + 1) for e in range(cfg.epochs)]
        # p_r after each epoch end is p_r times sqrt(E) of that epoch (Alg. 1 l.21)
        # (IEEE double, correctly rounded sqrt: the same value, bit for bit)
        p = 0.5
        for c in g["checkpoints"]:
            p = p * math.sqrt(float(c["errors"]) / float(cfg.n_train))
            assert float.fromhex(c["p_r"]) == p
