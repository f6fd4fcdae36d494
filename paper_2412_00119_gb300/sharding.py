"""Neuron sharding of a BMLP across ranks (one process per GPU): the plan.

Every layer trains on its own input and its own local error signal (Sec. 3.1),
and the group selection of Alg. 2 looks only inside a group, so a layer can be
split across ranks by neurons along group boundaries.  Rank r owns a contiguous
slice [k0, k1) of the neurons of every layer l -- its rows of H_l and W_l and
its rows of P_l -- with k0 and k1 multiples of lcm(gamma_l, 64): whole groups,
and whole 64-bit words of the packed activations.

Per mini-batch and layer the ranks exchange one thing: the packed activations
a_l of their slices, an all-gather of bs x ceil(K_l / 64) words.  Each rank
needs the whole a_l for the next layer's forward pass (Alg. 1 l.8), for the
local classifier yhat_l = a_l P_l with its 01-loss and margin (Eq. 1,
Alg. 1 l.10-17), which every rank then computes identically, and for the
update of layer l + 1 (Alg. 3 reads a_l).  Everything else is local: the
pre-activations and selections of the slice's groups (Alg. 2), the clipped
perceptron and the reinforcement events (Alg. 3; the random stream is keyed by
the neuron's index in its layer, so a slice draws exactly what one GPU would),
and the repack of W.  The last layer's error count -- hence E and the p_r
rescale of Alg. 1 l.21 -- is the same on every rank.  So N ranks train the
same model as one GPU, bit for bit, with one collective per layer.

This module holds the host-side plan; tests/test_dist_gloo.py runs the
decomposition on CPU ranks with the oracle's per-layer steps.
"""
from __future__ import annotations

import math


def slice_unit(gamma: int) -> int:
    """Neuron granularity of a slice: whole groups and whole packed words."""
    return gamma * 64 // math.gcd(gamma, 64)


def neuron_slices(widths, gammas, world: int):
    """For each rank, the (k0, k1) slice of every layer l = 1..L.

    widths: K_0..K_L; gammas: the L group sizes.  A layer of u units of
    slice_unit(gamma_l) neurons gives the first u % world ranks one unit more
    than the others (a rank may get an empty slice when u < world).  A layer
    whose width is not a multiple of its unit puts the remainder (a whole
    number of groups) on the last rank that holds neurons."""
    if world < 1:
        raise ValueError("world must be >= 1")
    L = len(widths) - 1
    if len(gammas) != L:
        raise ValueError("one group size per layer")
    plan = [[None] * L for _ in range(world)]
    for l in range(L):
        K, g = widths[l + 1], gammas[l]
        if g < 1 or K % g:
            raise ValueError("gamma of layer %d must divide K_l" % (l + 1))
        unit = slice_unit(g)
        units = K // unit
        edges = [0]
        for r in range(world):
            edges.append(edges[-1] + unit * (units // world + (1 if r < units % world else 0)))
        # the remainder (K % unit, whole groups) joins the last non-empty slice
        last = max([r for r in range(world) if edges[r + 1] > edges[r]] or [world - 1])
        for r in range(last + 1, world + 1):
            edges[r] += K - units * unit
        for r in range(world):
            plan[r][l] = (edges[r], edges[r + 1])
    return plan


def gather_words_per_step(widths, bs: int) -> int:
    """64-bit words every rank receives per mini-batch: the packed
    activations of all layers (its own slice included)."""
    return sum(bs * ((K + 63) // 64) for K in widths[1:])
