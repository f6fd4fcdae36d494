"""The Random Prototypes workload (Sec. 4.1.1) and the paper's Table C1.

CPU: the generator has the properties Sec. 4.1.1 states.  GPU: training on it
is bit-exact with the oracle, and the test accuracies of the 2-hidden-layer
BMLPs of Table C1 (widths 35 ... 525, bs 100, 50 epochs, p_r 0.5, r 0.25, 10
realizations of the initial conditions) are reproduced within the stated
tolerance of the printed means."""
import os

import numpy as np
import pytest

import oracle as O
import workloads as W


def test_generator_properties():
    """K_0 = 1000, 10 balanced classes, 10,000 + 2,000 distinct samples, each
    entry flipped from its class prototype with probability 0.44 (binomial 5
    sigma bound on the flip count)."""
    tr, te = W.random_prototypes(5)
    assert tr.xp.shape == (10000, 16) and te.xp.shape == (2000, 16)
    assert np.array_equal(np.bincount(tr.y), np.full(10, 1000))
    assert np.array_equal(np.bincount(te.y), np.full(10, 200))
    allx = np.concatenate([tr.xp, te.xp])
    assert len({r.tobytes() for r in allx}) == 12000
    x = np.concatenate([tr.pm1(), te.pm1()]).astype(np.int32)
    y = np.concatenate([tr.y, te.y])
    # the prototype of a class is the per-entry majority of its 1,200 samples
    # (an entry's sum is 144 +- 35 in the prototype's direction)
    proto = np.stack([np.where(x[y == j].sum(axis=0) >= 0, 1, -1) for j in range(10)])
    flips = (x != proto[y]).sum()
    n = x.size
    assert abs(flips - 0.44 * n) < 5 * np.sqrt(n * 0.44 * 0.56), flips / n


# Table C1, rows "Ours": hidden width -> (mean, std) test accuracy in %.
TABLE_C1 = {35: (79.10, 1.27), 75: (87.65, 0.56), 135: (92.25, 0.45), 255: (93.60, 0.67),
            525: (94.83, 0.56)}


@pytest.mark.gpu
def test_parity_on_prototypes():
    """1000 -> 75 -> 75 -> 10 on 2,000 prototype samples for two epochs: H, W,
    p_r, step and test predictions equal the oracle's."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    O.set_threads(os.cpu_count() or 1)
    tr, te = W.random_prototypes(11, 2000, 500)
    gpu = B.BMLP([1000, 75, 75], 10, seed=3, bs=100)
    ref = O.OracleModel([1000, 75, 75], 10, seed=3, bs=100)
    x = torch.from_numpy(tr.xp.view(np.int64)).cuda()
    y = torch.from_numpy(tr.y).cuda()
    for _ in range(2):
        assert gpu.train(x, y, epoch_end=True, count_errors=True) == ref.train(tr.pm1(), tr.y,
                                                                               epoch_end=True)
    for l in (1, 2):
        H, _, _, p_r, step = gpu.state(l)
        assert np.array_equal(H.astype(np.int32), ref.H(l).T), l
        assert p_r == ref.p_r and step == ref.step
    out = torch.empty(500, dtype=torch.int32, device="cuda")
    gpu.predict(torch.from_numpy(te.xp.view(np.int64)).cuda(), out)
    assert np.array_equal(out.cpu().numpy(), ref.predict(te.pm1()))
    gpu.close()


@pytest.mark.gpu
def test_table_c1_reproduction():
    """Mean test accuracy over 10 model seeds after 50 epochs, per hidden
    width, within 3 printed standard deviations + 1 point of Table C1 (the
    dataset is a fresh draw of the Sec. 4.1.1 generator; the GPU path is
    bit-exact with the oracle, so the numbers are deterministic)."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tr, te = W.random_prototypes(2024)
    x = torch.from_numpy(tr.xp.view(np.int64)).cuda()
    y = torch.from_numpy(tr.y).cuda()
    xt = torch.from_numpy(te.xp.view(np.int64)).cuda()
    out = torch.empty(len(te.y), dtype=torch.int32, device="cuda")
    rows = []
    for width, (mean_p, std_p) in TABLE_C1.items():
        acc = []
        for seed in range(10):
            m = B.BMLP([1000, width, width], 10, seed=seed, bs=100)
            for _ in range(50):
                m.train(x, y, epoch_end=True)
            m.predict(xt, out)
            acc.append(100.0 * float((out.cpu().numpy() == te.y).mean()))
            m.close()
        mean = float(np.mean(acc))
        rows.append((width, mean, float(np.std(acc, ddof=1)), mean_p, std_p))
    print("\nwidth  ours (mean +- std)  Table C1")
    for r in rows:
        print("%5d  %6.2f +- %.2f      %6.2f +- %.2f" % r)
    for width, mean, _, mean_p, std_p in rows:
        assert abs(mean - mean_p) <= 3 * std_p + 1.0, (width, mean, mean_p)


@pytest.mark.gpu
def test_group_membership_does_not_matter():
    """Sec. 4.3: a fixed random partition, or one redrawn at every step, trains
    as well as contiguous groups.  1000 -> 255 -> 255 -> 10 (gamma 85, three
    groups per layer), 20 epochs, 10 model seeds: the three mean test
    accuracies lie within 1.5 points of each other."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tr, te = W.random_prototypes(2024)
    x = torch.from_numpy(tr.xp.view(np.int64)).cuda()
    y = torch.from_numpy(tr.y).cuda()
    xt = torch.from_numpy(te.xp.view(np.int64)).cuda()
    out = torch.empty(len(te.y), dtype=torch.int32, device="cuda")
    means = []
    for mode in (B.BMLP_GROUPS_CONTIGUOUS, B.BMLP_GROUPS_FIXED, B.BMLP_GROUPS_RESHUFFLED):
        acc = []
        for seed in range(10):
            m = B.BMLP([1000, 255, 255], 10, seed=seed, bs=100, group_mode=mode)
            for _ in range(20):
                m.train(x, y, epoch_end=True)
            m.predict(xt, out)
            acc.append(100.0 * float((out.cpu().numpy() == te.y).mean()))
            m.close()
        means.append(float(np.mean(acc)))
    print("\ncontiguous / fixed random / reshuffled: %.2f / %.2f / %.2f" % tuple(means))
    assert max(means) - min(means) <= 1.5, means


@pytest.mark.gpu
def test_hidden_bits_sweep():
    """App. A.5: fewer bits for the hidden weights (h_max = 2^b - 1) bring
    catastrophic forgetting; with one bit only the visible weights remain.
    1000 -> 135 -> 135 -> 10, 50 epochs, 3 model seeds: accuracy rises with b,
    one bit stays near chance (< 20 %) and eight bits reach > 85 %."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tr, te = W.random_prototypes(2024)
    x = torch.from_numpy(tr.xp.view(np.int64)).cuda()
    y = torch.from_numpy(tr.y).cuda()
    xt = torch.from_numpy(te.xp.view(np.int64)).cuda()
    out = torch.empty(len(te.y), dtype=torch.int32, device="cuda")
    means = []
    for bits in (1, 4, 8):
        acc = []
        for seed in range(3):
            m = B.BMLP([1000, 135, 135], 10, h_max=2 ** bits - 1, seed=seed, bs=100)
            for _ in range(50):
                m.train(x, y, epoch_end=True)
            m.predict(xt, out)
            acc.append(100.0 * float((out.cpu().numpy() == te.y).mean()))
            m.close()
        means.append(float(np.mean(acc)))
    print("\nbits 1 / 4 / 8: %.2f / %.2f / %.2f" % tuple(means))
    assert means[0] < 20.0 < means[1] < means[2] and means[2] > 85.0, means
