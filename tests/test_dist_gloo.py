"""Multi-rank host logic of bench.py on CPU (gloo, world_size 2).

With N GPUs every rank trains an independent replica (model seed + rank) with
no collective on the data path; the only collectives are the timing reductions
(max of the elapsed time, sum of the samples) and barriers."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import numpy as np
    import torch.distributed as dist

    import bench
    import oracle as O

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, lr = bench.dist_env()
    elapsed = 1.5 + rank                      # rank 1 is the slow one
    mx = bench.max_over_ranks(elapsed)
    total = bench.sum_over_ranks(1000.0 * (rank + 1))
    bench.barrier()
    seed = bench.replica_seed(5, rank)
    m = O.OracleModel([16, 8], 2, seed=seed, bs=4)
    H = m.H(1)
    m.close()
    out.put((rank, r, w, lr, mx, total, seed, H.tobytes()))
    dist.destroy_process_group()


def test_two_rank_reductions_and_independent_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, rr0, w0, l0, mx0, tot0, s0, H0), (r1, rr1, w1, l1, mx1, tot1, s1, H1) = res
    assert (rr0, rr1, w0, w1, l0, l1) == (0, 1, 2, 2, 0, 1)
    assert mx0 == mx1 == 2.5                      # time = max over ranks
    assert tot0 == tot1 == 3000.0                 # samples = sum over ranks
    assert s0 != s1 and H0 != H1                  # independent replicas


def test_single_process_helpers_are_identity():
    import bench
    assert bench.max_over_ranks(3.0) == 3.0
    assert bench.sum_over_ranks(7.0) == 7.0
    bench.barrier()
    assert bench.dist_env()[1] >= 1


def test_bench_arithmetic():
    import bench
    w = (8192, 8192, 8192, 8192, 8192)
    assert bench.bitpairs_per_sample(w, 10) == 4 * 8192 * (8192 + 10)
    # bit-sliced H (8 planes of 32 weights: one byte per weight) read + write
    # (8192 x 8192 x 1 x 2 bytes) + packed W (8192 x 128 x 8) per layer
    assert bench.update_bytes_per_launch(w) == 4 * (8192 * 8192 * 2 + 8192 * 128 * 8)
    # 25 groups x 8 planes = 200 words per row; one plane (h_max = 1): 25 words
    # padded to 28; 16 planes (h_max = 257): 400 words
    assert bench.update_bytes_per_launch((784, 256)) == 256 * (2 * 4 * 200 + 13 * 8)
    assert bench.update_bytes_per_launch((784, 256), h_max=1) == 256 * (2 * 4 * 28 + 13 * 8)
    assert bench.update_bytes_per_launch((784, 256), h_max=257) == 256 * (2 * 4 * 400 + 13 * 8)
    assert [bench.hidden_planes(h) for h in (1, 3, 5, 7, 15, 17, 255, 257, 16383)] == \
        [1, 2, 4, 4, 4, 8, 8, 16, 16]


def test_step_roofline_arithmetic():
    """The whole-step roofline of the bench line: t_roof = max(HBM bytes at the
    copy peak, the forward's bit-pairs at the engine's peak), frac = t_roof /
    measured; the popcount-peak figure is reported beside it."""
    import bench
    w = (8192, 8192, 8192, 8192, 8192)
    bp = 100 * bench.bitpairs_per_sample(w, 10)
    fwd_bytes = bench.forward_weight_bytes(w)
    assert fwd_bytes == 4 * 8192 * 128 * 8
    upd = 433_000_000
    r = bench.step_roofline(0.184, upd, w, 10, 6784.8, 3397.6e12, 161e12, "tensor (e4m3)")
    t_hbm = (upd + fwd_bytes) / 6784.8e9
    assert r["bound"] == "hbm" and abs(r["us_roof"] - t_hbm * 1e6) < 1e-9
    assert abs(r["frac"] - t_hbm / 184e-6) < 1e-12
    assert abs(r["vs_popcount_peak"]["us_popc"] - bp / 161e12 * 1e6) < 1e-9
    assert abs(r["vs_popcount_peak"]["frac"] - max(t_hbm, bp / 161e12) / 184e-6) < 1e-12
    # a compute-bound case names the engine
    r2 = bench.step_roofline(0.184, 0, w, 10, 6784.8, 1e12, 161e12, "alu (popcount)")
    assert r2["bound"] == "alu (popcount)" and abs(r2["us_compute"] - bp / 1e12 * 1e6) < 1e-6


# -- neuron sharding (paper_2412_00119_gb300.sharding) ------------------------------

def _sharded_worker(rank, world, port, out, *args):
    try:
        _sharded_run(rank, world, port, out, *args)
    except Exception as e:   # reported to the test instead of a silent timeout
        out.put(("error", rank, repr(e)))
        raise


def _sharded_run(rank, world, port, out, widths, classes, gammas, n, bs, epochs, seed):
    """One rank of a neuron-sharded training run, every step of the rule taken
    from the oracle on this rank's slice of every layer; the only exchange is
    the all-gather of the slices' activations (Sec. 3.1)."""
    import numpy as np
    import torch
    import torch.distributed as dist

    import oracle as O
    import workloads as W
    from paper_2412_00119_gb300 import sharding as S

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    O.set_threads(1)
    L = len(widths) - 1
    plan = S.neuron_slices(widths, gammas, world)
    mine = plan[rank]
    cfg = W.small_config(widths, classes, n, 0, teacher_hidden=16, number=61)
    tr = W.make_split(cfg, "train")
    x, y = tr.pm1(), tr.y
    full = O.OracleModel(list(widths), classes, seed=seed, bs=bs, gamma=list(gammas))
    H = [full.H(l)[:, mine[l - 1][0]:mine[l - 1][1]].copy() for l in range(1, L + 1)]
    P = [full.P(l) for l in range(1, L + 1)]
    full.close()
    p_r, t, gathered = 0.5, 0, 0
    errs = []
    for _ in range(epochs):
        err = 0
        for s0 in range(0, n, bs):
            xb, yb = x[s0:s0 + bs], y[s0:s0 + bs]
            a_prev, ins, zs, marks = xb, [], [], []
            for l in range(1, L + 1):
                k0, k1 = mine[l - 1]
                z, a = O.layer_forward(a_prev, H[l - 1])
                # all-gather of the slices' activations (padded to the widest slice)
                wmax = max(p[l - 1][1] - p[l - 1][0] for p in plan)
                buf = torch.zeros((len(yb), wmax), dtype=torch.int8)
                buf[:, :k1 - k0] = torch.from_numpy(a)
                parts = [torch.zeros_like(buf) for _ in range(world)]
                dist.all_gather(parts, buf)
                gathered += 1
                a_full = np.concatenate([parts[r][:, :plan[r][l - 1][1] - plan[r][l - 1][0]].numpy()
                                         for r in range(world)], axis=1)
                yhat = O.local_output(a_full, P[l - 1])
                _, ell, _, mark = O.local_loss(yhat, yb, widths[l])
                if l == L:
                    err += int(ell.sum())
                ins.append(a_prev)
                zs.append(z)
                marks.append(mark)
                a_prev = a_full
            for l in range(1, L + 1):
                if not marks[l - 1].any():
                    continue   # O6: no update of a layer with an empty M_l
                k0, k1 = mine[l - 1]
                if k1 == k0:
                    continue
                Ps = P[l - 1][k0:k1]
                sel = O.select(zs[l - 1], Ps, yb, marks[l - 1], gammas[l - 1])
                sel = np.where(sel >= 0, sel + k0, -1)
                H[l - 1] = O.perceptron_update(H[l - 1], ins[l - 1], yb, Ps, sel, 255,
                                               O.reinforce_prob(p_r, widths[l]), seed, l, t, k0=k0)
            t += 1
        errs.append(err)
        p_r = p_r * np.sqrt(err / n)   # Alg. 1 l.21: the same error count on every rank
    got = [None] * world
    dist.all_gather_object(got, [h.tobytes() for h in H])
    if rank == 0:
        out.put((errs, p_r, t, gathered, got, plan))
    dist.destroy_process_group()


@pytest.mark.parametrize("world,widths,gammas", [
    (2, (130, 256, 192), (64, 32)),      # unequal slices of layer 2 (3 units of 64)
    (2, (70, 64, 128), (64, 64)),        # one layer with a single unit: one rank idle there
    (3, (96, 384, 200), (64, 8)),        # three ranks; 200 = 3 units of 64 + a remainder of 8
])
def test_neuron_sharded_training_equals_one_rank(world, widths, gammas):
    """Neuron-sharded training on gloo ranks -- each rank the oracle's steps on
    its slices, one all-gather of activations per layer and mini-batch -- gives
    the single-rank oracle's hidden weights, error counts and p_r bit for bit
    over two epochs (the reinforcement stream is keyed by the neuron's index in
    its layer, so the slices draw what one model draws)."""
    import numpy as np

    import oracle as O
    import workloads as W

    classes, n, bs, epochs, seed = 10, 240, 40, 2, 17
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    args = (world, port, q, widths, classes, gammas, n, bs, epochs, seed)
    procs = [ctx.Process(target=_sharded_worker, args=(r,) + args) for r in range(world)]
    for p in procs:
        p.start()
    res = q.get(timeout=300)
    assert res[0] != "error", res
    errs, p_r, t, gathered, got, plan = res
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    L = len(widths) - 1
    assert gathered == L * epochs * (n // bs)   # one exchange per layer and mini-batch
    cfg = W.small_config(widths, classes, n, 0, teacher_hidden=16, number=61)
    tr = W.make_split(cfg, "train")
    ref = O.OracleModel(list(widths), classes, seed=seed, bs=bs, gamma=list(gammas))
    ref_errs = [ref.train(tr.pm1(), tr.y, epoch_end=True) for _ in range(epochs)]
    assert errs == ref_errs
    assert p_r == ref.p_r and t == ref.step
    for l in range(1, L + 1):
        k = widths[l - 1]
        parts = [np.frombuffer(got[r][l - 1], np.int32).reshape(k, -1) for r in range(world)]
        assert np.array_equal(np.concatenate(parts, axis=1), ref.H(l)), "layer %d" % l
    ref.close()


def test_neuron_slices_plan():
    from paper_2412_00119_gb300 import sharding as S
    widths, gammas = (784, 8192, 8192, 4096, 100), (64, 64, 128, 100)
    for world in (1, 2, 3, 4, 8):
        plan = S.neuron_slices(widths, gammas, world)
        assert len(plan) == world
        for l in range(1, len(widths)):
            K, unit = widths[l], S.slice_unit(gammas[l - 1])
            edges = [plan[r][l - 1] for r in range(world)]
            assert edges[0][0] == 0 and edges[-1][1] == K
            for r in range(world - 1):
                assert edges[r][1] == edges[r + 1][0]              # contiguous cover
            for a, b in edges:
                assert a % unit == 0                                # whole groups and words
                assert (b - a) % gammas[l - 1] == 0
            sizes = [b - a for a, b in edges]
            assert max(sizes) - min(sizes) <= unit + K % unit       # balanced to one unit
    assert S.slice_unit(64) == 64 and S.slice_unit(100) == 1600 and S.slice_unit(96) == 192
    assert S.gather_words_per_step((8192,) * 5, 100) == 4 * 100 * 128
    with pytest.raises(ValueError):
        S.neuron_slices((10, 9), (2,), 2)
