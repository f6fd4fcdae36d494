"""Pins of the CPU oracle: checks against what the paper and the mathematics fix.

Each ``check_*`` raises AssertionError on failure.  ``test_oracle_pins.py`` runs
them against the oracle as built, and against copies of the oracle source with
a planted mistake (each mutant must fail at least one check).

Sources of the expected values:
  * Philox4x32-10 known-answer vectors (Salmon et al., SC'11 / Random123);
  * the two worked examples of the group-size rule (Sec. 4.3);
  * hand-worked cases of Eq. 1 / Alg. 1 l.13-15, Alg. 2 and Alg. 3
    (``tests/golden/*.txt``, each derived in its comment header);
  * exhaustive brute force of the +-1 dot product, N - 2 popcount(a XOR w);
  * exact rational arithmetic for the reinforcement probability and the
    sampler's thresholds, the law of independent Bernoulli(q) events (marginal
    rate, pair independence, per-block binomial counts; and, for small blocks,
    the exact probability of every event set against the product law), a
    binomial bound on the reinforcement rate, and the closed form of Alg. 1
    l.21;
  * invariants of Alg. 3 (odd h, |h| <= h_max, one lattice unit per event,
    reinforcement moves away from 0) and the learnability of a separable task;
  * the rank form of the lower median (brute force), the truncated network
    for early-exit predictions, and the evaluation path for the local error
    counts;
  * for the expansion front end: the Philox stream recomputed from the
    KAT-pinned primitive, and special cases (zero pattern, one or two lit
    inputs, 0/1 patterns as counts).
"""
from __future__ import annotations

import math
from decimal import Decimal, getcontext
from fractions import Fraction

import numpy as np

import oracle as O
from conftest import read_golden


# -- random stream ---------------------------------------------------------------

def check_philox_kat():
    for line in read_golden("philox4x32_10_kat.txt"):
        v = [int(t, 16) for t in line.split()]
        out = O.philox4x32_10(v[0:4], v[4:6])
        assert [int(o) for o in out] == v[6:10], (line, [hex(int(o)) for o in out])


# -- expansion front end (O20) ----------------------------------------------------

def check_expand_weights_stream(seed=0x1234_5678_9ABC):
    """Expansion weights (O20): e_{k,i} = +1 iff bit 31 of word i%4 of the
    KAT-pinned Philox at counter (i/4, k, 33*2^16, 0), recomputed here from
    the primitive over a ragged D; balanced (P(+1) = 1/2 within 5 sigma over
    200,000 weights); a stream of its own, not that of the initial weights."""
    K, D = 7, 13
    e = O.expand_weights(seed, K, D)
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for k in range(K):
        for i in range(D):
            w = O.philox4x32_10([i // 4, k, 33 << 16, 0], key)
            assert e[k, i] == (1 if (int(w[i % 4]) >> 31) else -1), (k, i)
            assert O.expand_weight(seed, k, i) == e[k, i], (k, i)
    h1 = np.array([[O.init_h(seed, 1, k, i) for i in range(D)] for k in range(K)])
    assert not np.array_equal(e, h1)
    big = O.expand_weights(seed, 200, 1000)
    assert set(np.unique(big)) == {-1, 1}
    assert abs((big == 1).mean() - 0.5) < 5 * math.sqrt(0.25 / big.size)


def check_expand_sign(seed=11):
    """Expansion layer (O20), a_k = +1 iff sum_i x_i e_{k,i} >= 0, against
    what fixes it without the sum as written: a zero pattern gives all +1
    (sign(0) = +1); a pattern with one lit input i gives a_k = e_{k,i}; two
    lit inputs u > v on weights +1 / -1 give +1 and on -1 / +1 give -1 (for
    u >= 128 too: the inputs are unsigned); on 0/1 patterns a_k = +1 iff at
    least half of the lit inputs carry weight +1 (a count); and, as a cross-
    check, the exact int64 matrix product for pixel-like inputs with K != D."""
    rng = np.random.default_rng(seed)
    K, D = 9, 23
    e = O.expand_weights(seed, K, D)
    assert np.all(O.expand_sign(np.zeros((2, D), np.uint8), e) == 1)
    for i in range(D):
        for v in (1, 7, 128, 255):
            x = np.zeros((1, D), np.uint8)
            x[0, i] = v
            assert np.array_equal(O.expand_sign(x, e)[0], e[:, i]), (i, v)
    for k in range(K):
        pos = np.flatnonzero(e[k] == 1)
        neg = np.flatnonzero(e[k] == -1)
        if len(pos) == 0 or len(neg) == 0:
            continue
        for u, v in ((255, 254), (200, 100), (128, 1), (2, 1)):
            x = np.zeros((2, D), np.uint8)
            x[0, pos[0]], x[0, neg[0]] = u, v
            x[1, pos[0]], x[1, neg[0]] = v, u
            a = O.expand_sign(x, e)
            assert a[0, k] == 1 and a[1, k] == -1, (k, u, v)
    xb = (rng.random((300, D)) < 0.4).astype(np.uint8)
    a = O.expand_sign(xb, e)
    for mu in range(len(xb)):
        lit = xb[mu] == 1
        for k in range(K):
            plus = int((e[k][lit] == 1).sum())
            assert a[mu, k] == (1 if 2 * plus >= int(lit.sum()) else -1), (mu, k)
    Kp, Dp = 37, 61
    ep = O.expand_weights(seed + 1, Kp, Dp)
    xp = np.where(rng.random((50, Dp)) < 0.5, 0, rng.integers(1, 256, (50, Dp))).astype(np.uint8)
    want = np.where(xp.astype(np.int64) @ ep.astype(np.int64).T >= 0, 1, -1)
    assert np.array_equal(O.expand_sign(xp, ep), want)


# -- group size ----------------------------------------------------------------

def check_gamma_golden():
    for line in read_golden("gamma_rule.txt"):
        K, g = (int(t) for t in line.split())
        assert O.gamma_rule(K) == g, (K, O.gamma_rule(K), g)


# -- forward ---------------------------------------------------------------------

def _all_pm1(N):
    codes = np.arange(2 ** N)
    bits = (codes[:, None] >> np.arange(N)[None, :]) & 1
    return codes, np.where(bits == 1, 1, -1).astype(np.int8)


def check_dot_bruteforce(Nmax=8):
    """z = N - 2 popcount(a XOR w) over every pair of +-1 vectors, N <= Nmax."""
    for N in range(1, Nmax + 1):
        codes, V = _all_pm1(N)
        # hidden weights: odd integers whose sign is V, magnitudes 1..7
        mag = 1 + 2 * (np.arange(V.size).reshape(V.shape) % 4)
        H = (V.astype(np.int32) * mag).T.copy()        # N x 2^N, column w = vector w
        z, a = O.layer_forward(V, H)
        pc = np.array([bin(int(c)).count("1") for c in range(2 ** N)])
        expect = N - 2 * pc[codes[:, None] ^ codes[None, :]]
        assert np.array_equal(z, expect), N
        assert np.array_equal(a, np.where(expect >= 0, 1, -1)), N


def check_sign_zero():
    """sign(0) = +1 for activations (reading O1): z = 0 gives a = +1."""
    a_prev = np.array([[1, -1], [1, 1], [-1, -1]], np.int8)
    H = np.array([[1], [1]], np.int32)
    z, a = O.layer_forward(a_prev, H)
    assert z[:, 0].tolist() == [0, 2, -2]
    assert a[:, 0].tolist() == [1, 1, -1]


def check_local_output_popcount(seed=0):
    rng = np.random.default_rng(seed)
    for (b, K, c) in [(5, 1, 2), (7, 63, 3), (9, 130, 10), (3, 257, 100)]:
        a = np.where(rng.random((b, K)) < 0.5, 1, -1).astype(np.int8)
        P = np.where(rng.random((K, c)) < 0.5, 1, -1).astype(np.int8)
        yhat = O.local_output(a, P)
        dis = (a[:, :, None] != P[None, :, :]).sum(axis=1)
        assert np.array_equal(yhat, K - 2 * dis)


# -- local loss and marking ------------------------------------------------------

def check_local_loss_golden():
    for line in read_golden("local_loss_cases.txt"):
        head, yh, exp = (s.split() for s in line.split("|"))
        K, y = int(head[0]), int(head[1])
        yhat = np.array([[int(v) for v in yh]], np.int32)
        pred, ell, tau, mark = O.local_loss(yhat, np.array([y]), K, 1, 4)
        got = [int(pred[0]), int(ell[0]), int(tau[0]), int(mark[0])]
        assert got == [int(v) for v in exp], (line, got)


def check_local_loss_special(seed=1):
    """r = 0 marks exactly the errors; a huge r marks every pattern."""
    rng = np.random.default_rng(seed)
    yhat = rng.integers(-20, 21, size=(200, 7)).astype(np.int32)
    y = rng.integers(0, 7, size=200).astype(np.int32)
    pred, ell, tau, mark = O.local_loss(yhat, y, 64, 0, 1)
    assert np.array_equal(mark, ell)
    pred, ell, tau, mark = O.local_loss(yhat, y, 64, 10 ** 6, 1)
    assert mark.all()
    srt = np.sort(yhat, axis=1)
    assert np.array_equal(tau, srt[:, -1] - srt[:, -2])


# -- selection -------------------------------------------------------------------

def _parse_select():
    z, rho, sels, marks = [], [], [], []
    y = gamma = None
    for line in read_golden("select_case.txt"):
        t = line.split()
        if t[0] == "z":
            z.append([int(v) for v in t[1:]])
        elif t[0] == "rho":
            rho.append([int(v) for v in t[1:]])
        elif t[0] == "y":
            y = [int(v) for v in t[1:]]
        elif t[0] == "gamma":
            gamma = int(t[1])
        elif t[0] == "mark":
            marks.append([int(v) for v in t[1:]])
            sels.append([])
        elif t[0] == "sel":
            sels[-1].append([int(v) for v in t[1:]])
    return (np.array(z, np.int32), np.array(rho, np.int8), np.array(y, np.int32), gamma,
            marks, sels)


def check_select_golden():
    z, rho, y, gamma, marks, sels = _parse_select()
    for mark, sel in zip(marks, sels):
        got = O.select(z, rho, y, np.array(mark, np.uint8), gamma)
        assert got.tolist() == sel, (mark, got.tolist(), sel)


def check_select_special(seed=2):
    """gamma = 1: every neuron with negative stability is selected (Alg. 2 with
    G = K_l); gamma = K_l: one selection per pattern, the largest negative delta."""
    rng = np.random.default_rng(seed)
    b, K, c = 20, 24, 5
    z = rng.integers(-9, 10, size=(b, K)).astype(np.int32)
    P = np.where(rng.random((K, c)) < 0.5, 1, -1).astype(np.int8)
    y = rng.integers(0, c, size=b).astype(np.int32)
    mark = np.ones(b, np.uint8)
    delta = z * P[:, y].T
    sel1 = O.select(z, P, y, mark, 1)
    assert np.array_equal(sel1, np.where(delta < 0, np.arange(K)[None, :], -1))
    selK = O.select(z, P, y, mark, K)
    for mu in range(b):
        neg = [k for k in range(K) if delta[mu, k] < 0]
        if not neg:
            assert selK[mu, 0] == -1
        else:
            best = max(delta[mu, k] for k in neg)
            assert selK[mu, 0] == min(k for k in neg if delta[mu, k] == best)


# -- perceptron level --------------------------------------------------------------

def _parse_perceptron():
    d = {}
    for line in read_golden("perceptron_case.txt"):
        t = line.split()
        d.setdefault(t[0], []).append([int(v) for v in t[1:]])
    return d


def check_perceptron_golden():
    d = _parse_perceptron()
    H = np.array(d["H"], np.int32)
    a = np.array(d["a"], np.int8)
    y = np.array(d["y"][0], np.int32)
    rho = np.array(d["rho"], np.int8)
    sel = np.array(d["sel"], np.int32)
    cp = O.perceptron_update(H, a, y, rho, sel, 3, 0.0, 7, 1, 0)
    assert cp.tolist() == d["cp"], cp.tolist()
    cpr = O.perceptron_update(H, a, y, rho, sel, 3, 1.0, 7, 1, 0)
    assert cpr.tolist() == d["cpr"], cpr.tolist()


def check_cp_monotone(seed=12):
    """Alg. 3 l.2-4 with one CP tuple (mu, k) and no reinforcement: every
    hidden weight of neuron k moves by 2 a^mu_i rho_{k,y} unless that would
    cross the bound h_max (then it stays), no other weight moves, and the
    pattern's stability delta_k = z_k rho_{k,y} does not decrease: each sign
    flip of a visible weight of k raises it by exactly 2."""
    rng = np.random.default_rng(seed)
    for trial in range(300):
        Kp, K, c = int(rng.integers(3, 40)), int(rng.integers(2, 12)), int(rng.integers(2, 5))
        h_max = 7 if trial % 3 == 0 else 255
        H = (2 * rng.integers(-(h_max + 1) // 2, (h_max + 1) // 2, (Kp, K)) + 1).astype(np.int32)
        a = rng.choice([-1, 1], (1, Kp)).astype(np.int8)
        P = rng.choice([-1, 1], (K, c)).astype(np.int8)
        y = np.array([rng.integers(0, c)], np.int32)
        k = int(rng.integers(0, K))
        H2 = O.perceptron_update(H, a, y, P, np.array([[k]], np.int32), h_max, 0.0, seed, 1, 0)
        rho = int(P[k, y[0]])
        step = 2 * a[0].astype(np.int32) * rho
        want = H.copy()
        want[:, k] = np.where(np.abs(H[:, k] + step) <= h_max, H[:, k] + step, H[:, k])
        assert np.array_equal(H2, want), trial
        s_old, s_new = np.where(H[:, k] > 0, 1, -1), np.where(H2[:, k] > 0, 1, -1)
        d_old = int((a[0] * s_old).sum()) * rho
        d_new = int((a[0] * s_new).sum()) * rho
        assert d_new - d_old == 2 * int((s_old != s_new).sum()) >= 0, trial


def _ceil_frac(x: Fraction) -> int:
    return -((-x.numerator) // x.denominator)


def check_threshold_exact():
    """q is p_r sqrt(2 / (pi K)) to within 2 ulp (40-digit decimal evaluation);
    every threshold of the block sampler is ceil(x 2^32) of its double x (exact
    rational check), and x is within 1e-12 of the exact (1-q)^m expression."""
    getcontext().prec = 40
    pi = Decimal("3.141592653589793238462643383279502884197")
    for p_r in (0.5, 0.25, 0.1234567, 1e-3, 0.9):
        for K in (1, 2, 10, 64, 256, 784, 1024, 4096, 8192):
            q = O.reinforce_prob(p_r, K)
            qd = Decimal(p_r) * (Decimal(2) / (pi * K)).sqrt()
            assert abs(Decimal(q) - qd) <= 2 * Decimal(math.ulp(q)), (p_r, K)
    two32 = 1 << 32
    for q in (0.0044077, 0.0285, 0.05, 0.3, 0.77):
        qf = Fraction(q)
        for n in (1, 2, 7, 64):
            any_, first, gap = O.r_block_tables(q, n)
            s = 1.0 - q
            pw = [1.0]
            for _ in range(n):
                pw.append(pw[-1] * s)
            p_any = 1.0 - pw[n]
            exact_any = 1 - (1 - qf) ** n
            assert abs(Fraction(p_any) - exact_any) < Fraction(1, 10 ** 12), (q, n)
            assert any_ == _ceil_frac(Fraction(p_any) * two32), (q, n, any_)
            for j in range(n):
                x = (1.0 - pw[j + 1]) / p_any
                ex = (1 - (1 - qf) ** (j + 1)) / exact_any
                assert abs(Fraction(x) - ex) < Fraction(1, 10 ** 12), (q, n, j)
                want = two32 if x >= 1.0 else _ceil_frac(Fraction(x) * two32)
                assert int(first[j]) == want, (q, n, j, int(first[j]), want)
            assert int(first[n - 1]) == two32
            for g in range(n - 1):
                x = 1.0 - pw[g + 1]
                assert abs(Fraction(x) - (1 - (1 - qf) ** (g + 1))) < Fraction(1, 10 ** 12)
                assert int(gap[g]) == _ceil_frac(Fraction(x) * two32), (q, n, g)
            assert np.all(np.diff(first.astype(np.float64)) >= 0)
            assert np.all(np.diff(gap.astype(np.float64)) >= 0)
    any0, first0, gap0 = O.r_block_tables(0.0, 64)
    assert any0 == 0 and np.all(gap0 == 0)
    for q in (1.0, 3.5):
        a1, f1, g1 = O.r_block_tables(q, 64)
        assert a1 == two32 and np.all(f1 == two32) and np.all(g1 == two32)


def check_reinforce_rate():
    """Reinforcement alone (no tuples): each weight moves with probability q, by
    exactly 2 sign(h); the count obeys a binomial bound; draws repeat for the
    same step and differ between steps."""
    Kp, K = 512, 512
    rng = np.random.default_rng(3)
    H = (np.where(rng.random((Kp, K)) < 0.5, 1, -1) * (1 + 2 * rng.integers(0, 3, (Kp, K))))
    H = H.astype(np.int32)
    a = np.ones((1, Kp), np.int8)
    sel = -np.ones((1, K), np.int32)
    rho = np.ones((K, 2), np.int8)
    y = np.zeros(1, np.int32)
    q = 0.02
    H1 = O.perceptron_update(H, a, y, rho, sel, 255, q, 11, 2, 5)
    d = H1 - H
    moved = d != 0
    n = moved.sum()
    mean, sd = q * H.size, math.sqrt(q * (1 - q) * H.size)
    assert abs(n - mean) < 5 * sd, (n, mean, sd)
    assert np.array_equal(d[moved], 2 * np.sign(H[moved]))
    H1b = O.perceptron_update(H, a, y, rho, sel, 255, q, 11, 2, 5)
    assert np.array_equal(H1, H1b)
    H2 = O.perceptron_update(H, a, y, rho, sel, 255, q, 11, 2, 6)
    overlap = ((H2 - H) != 0) & moved
    assert overlap.sum() < 5 * q * n + 10


def _events(q, K_prev, rows, seed=5, l=1, t=3):
    return np.array([O.r_events(seed, l, k, t, K_prev, q) for k in range(rows)], np.float64)


def check_event_law():
    """The reinforcement events of a row are independent Bernoulli(q): every
    input fires with frequency q (whole blocks and a ragged last block), pairs
    inside a block and across a block boundary fire together with frequency
    q^2, and the number of events of a 64-input block follows Binomial(64, q)
    (chi-square).  q = 0 and q >= 1 give no event / every input."""
    for q, rows in ((0.01, 4000), (0.05, 3000), (0.3, 1500)):
        K_prev = 200                                   # blocks of 64, 64, 64, 8
        ev = _events(q, K_prev, rows)
        n = ev.shape[0]
        # marginal rate per input position (pooled over rows)
        f = ev.mean(axis=0)
        sd = math.sqrt(q * (1 - q) / n)
        assert np.all(np.abs(f - q) < 5.5 * sd), (q, float(np.abs(f - q).max() / sd))
        assert abs(ev.mean() - q) < 5 * math.sqrt(q * (1 - q) / ev.size), (q, ev.mean())
        # pairs: neighbours, a block boundary, the ragged block, far apart
        for i, j in ((0, 1), (30, 31), (62, 63), (63, 64), (127, 128), (191, 192), (195, 199),
                     (5, 70)):
            both = (ev[:, i] * ev[:, j]).mean()
            sd2 = math.sqrt(q * q * (1 - q * q) / n)
            assert abs(both - q * q) < 5.5 * sd2 + 1e-12, (q, i, j, both)
        # events per full block: Binomial(64, q)
        counts = ev[:, :192].reshape(n * 3, 64).sum(axis=1).astype(np.int64)
        lam = 64 * q
        kmax = int(lam + 4 * math.sqrt(lam) + 2)
        pmf = [math.comb(64, c) * q ** c * (1 - q) ** (64 - c) for c in range(kmax)]
        obs = np.bincount(np.minimum(counts, kmax), minlength=kmax + 1)
        exp = np.array(pmf + [1 - sum(pmf)]) * counts.size
        keep = exp >= 5
        chi2 = float((((obs - exp) ** 2 / np.maximum(exp, 1e-300))[keep]).sum())
        dof = int(keep.sum()) - 1
        assert chi2 < dof + 6 * math.sqrt(2 * dof) + 10, (q, chi2, dof)
    assert _events(0.0, 130, 50).sum() == 0
    for q in (1.0, 2.0):
        assert np.all(_events(q, 130, 20) == 1)


def _least_with(V, tab, hi):
    """The least j <= hi with V < tab[j], or hi + 1 when there is none (a
    linear scan: the definition, not the oracle's search)."""
    for j in range(hi + 1):
        if V < int(tab[j]):
            return j
    return hi + 1


def _block_law(any_, first, gap, n):
    """Exact probability of every event set of an n-input block under the
    block sampler of reading O9 with these thresholds, as Fractions: the
    block draw U fires the block with measure any / 2^32; the first event is
    at j with measure (first[j] - first[j-1]) / 2^32; after an event at p the
    next comes g + 1 inputs later with measure (gap[g] - gap[g-1]) / 2^32 for
    g <= n - 2 - p, and none with the rest.  Keys: tuples of positions."""
    two32 = 1 << 32
    law = {(): Fraction(two32 - any_, two32)}

    def walk(events, prob):
        p = events[-1]
        if p == n - 1:
            law[tuple(events)] = law.get(tuple(events), 0) + prob
            return
        gmax = n - 2 - p
        stop = Fraction(two32 - int(gap[gmax]), two32)
        law[tuple(events)] = law.get(tuple(events), 0) + prob * stop
        prev = 0
        for g in range(gmax + 1):
            m = Fraction(int(gap[g]) - prev, two32)
            prev = int(gap[g])
            if m:
                walk(events + [p + 1 + g], prob * m)

    prev = 0
    for j in range(n):
        m = Fraction(int(first[j]) - prev, two32)
        prev = int(first[j])
        if m:
            walk([j], Fraction(any_, two32) * m)
    return law


class _EventDraws:
    """V_0, V_1, ... of one block: the words of Philox((b, k, (4 + r) 2^16 + l,
    t)) for r = 0, 1, ..., in order."""

    def __init__(self, b, k, l, t, key):
        self.b, self.k, self.l, self.t, self.key = b, k, l, t, key
        self.i = 0
        self.words = []

    def __call__(self):
        if self.i % 4 == 0:
            ctr = (self.b, self.k, ((4 + self.i // 4) << 16) + self.l, self.t)
            self.words = [int(w) for w in O.philox4x32_10(ctr, self.key)]
        v = self.words[self.i % 4]
        self.i += 1
        return v


def check_sampler_exact_law():
    """Reading O9 realises independent Bernoulli(q) events exactly up to the
    2^-32 rounding of its thresholds: for small blocks, the exact probability
    of every event set under the sampler (from the oracle's tables) sums to 1
    and lies within (n + 2) 2^-31 of q^|S| (1-q)^(n-|S|).  And the oracle's
    events are those the sampler's definition gives on its documented stream:
    block draw U = word b % 4 of Philox((b/4, k, 3 * 2^16 + l, t)), event
    draws V = the words of Philox((b, k, (4 + r) 2^16 + l, t)), r = 0, 1, ...,
    key = (seed mod 2^32, seed div 2^32); the first event at the least j with
    V < first[j]; after an event at p, the next at p + 1 + g for the least
    g <= n - 2 - p with V < gap[g], else none."""
    for q in (0.0044077, 0.05, 0.3, 0.77):
        for n in (1, 2, 3, 5, 8):
            any_, first, gap = O.r_block_tables(q, n)
            law = _block_law(any_, first, gap, n)
            assert sum(law.values()) == 1, (q, n)
            tol = Fraction(n + 2, 1 << 31)
            qf = Fraction(q)
            for mask in range(1 << n):
                S = tuple(i for i in range(n) if mask >> i & 1)
                want = qf ** len(S) * (1 - qf) ** (n - len(S))
                assert abs(law.get(S, Fraction(0)) - want) <= tol, (q, n, S)
    seed, l, t = 0x1234_5678_9ABC_DEF1, 2, 77
    key = (seed & 0xFFFFFFFF, seed >> 32)
    for q, K_prev in ((0.05, 200), (0.3, 130), (0.0044077, 64)):
        tabs = {n: O.r_block_tables(q, n) for n in {64, K_prev % 64 or 64}}
        for k in range(40 if q > 0.01 else 160):
            want = np.zeros(K_prev, np.uint8)
            for b in range((K_prev + 63) // 64):
                n = min(64, K_prev - 64 * b)
                any_, first, gap = tabs[n]
                U = int(O.philox4x32_10((b // 4, k, (3 << 16) + l, t), key)[b % 4])
                if not U < any_:
                    continue
                V = _EventDraws(b, k, l, t, key)
                p = _least_with(V(), first, n - 1)
                want[64 * b + p] = 1
                while p < n - 1:
                    gmax = n - 2 - p
                    g = _least_with(V(), gap, gmax)
                    if g > gmax:
                        break
                    p += 1 + g
                    want[64 * b + p] = 1
            got = O.r_events(seed, l, k, t, K_prev, q)
            assert np.array_equal(got, want), (q, K_prev, k)


def check_update_invariants(seed=4):
    """One CP tuple changes each h of its neuron by exactly one lattice unit (2)
    unless clipped; reinforcement never flips a sign; h stays odd and bounded."""
    rng = np.random.default_rng(seed)
    Kp, K, c, h_max = 40, 12, 3, 5
    H = (np.where(rng.random((Kp, K)) < 0.5, 1, -1) *
         (1 + 2 * rng.integers(0, 3, (Kp, K)))).astype(np.int32)
    a = np.where(rng.random((3, Kp)) < 0.5, 1, -1).astype(np.int8)
    y = rng.integers(0, c, 3).astype(np.int32)
    rho = np.where(rng.random((K, c)) < 0.5, 1, -1).astype(np.int8)
    sel = -np.ones((3, 1), np.int32)
    sel[1, 0] = 7                       # one tuple: (mu=1, k=7), gamma = K
    H1 = O.perceptron_update(H, a, y, rho, sel, h_max, 0.0, 1, 1, 0)
    d = H1 - H
    assert np.all(d[:, [k for k in range(K) if k != 7]] == 0)
    step = 2 * a[1] * rho[7, y[1]]
    want = np.clip(H[:, 7] + step, -h_max, h_max)
    assert np.array_equal(H1[:, 7], want)
    assert np.all(np.abs(d[:, 7]) <= 2)
    assert np.all((d[:, 7] == 0) == (np.abs(H[:, 7] + step) > h_max))
    # reinforcement only, probability 1
    H2 = O.perceptron_update(H, a, y, rho, -np.ones((3, 1), np.int32), h_max, 1.0, 1, 1, 0)
    assert np.array_equal(np.sign(H2), np.sign(H))
    assert np.array_equal(H2, np.clip(H + 2 * np.sign(H), -h_max, h_max))
    for M in (H1, H2):
        assert np.all(M % 2 != 0) and np.all(np.abs(M) <= h_max)


# -- the whole rule ------------------------------------------------------------

def _bias_data(rng, n, K, c):
    x = np.where(rng.random((n, K)) < 0.5, 1, -1).astype(np.int8)
    y = rng.integers(0, c, n).astype(np.int32)
    return x, y


def check_training_invariants(seed=5):
    """Over whole training runs with a small h_max (lots of clipping): h odd,
    |h| <= h_max, every h changes by at most 2 (n_k + 1) per step."""
    rng = np.random.default_rng(seed)
    widths, c, h_max = [50, 24, 16], 3, 7
    m = O.OracleModel(widths, c, h_max=h_max, seed=9, bs=10, p_r0=0.9, gamma=[4, 4])
    x, y = _bias_data(rng, 60, widths[0], c)
    prev = [m.H(l) for l in (1, 2)]
    for s in range(6):
        m.train(x[10 * s:10 * s + 10], y[10 * s:10 * s + 10])
        for l in (1, 2):
            H = m.H(l)
            assert np.all(H % 2 != 0) and np.all(np.abs(H) <= h_max)
            # at most bs tuples per neuron per step, plus one reinforcement event
            assert np.all(np.abs(H - prev[l - 1]) <= 2 * (10 + 1))
            prev[l - 1] = H
    assert m.step == 6


def check_no_mark_no_update(seed=6):
    """When no pattern of a layer is marked, the layer is not updated at all --
    not even reinforced (reading O6).  Labels = the model's own predictions with
    r = 0 leave M_L empty."""
    rng = np.random.default_rng(seed)
    m = O.OracleModel([30, 40], 2, seed=12, bs=25, r=(0, 1), p_r0=1.0)
    x, _ = _bias_data(rng, 100, 30, 2)
    y = m.predict(x)
    H0 = m.H(1)
    err = m.train(x, y)
    assert err == 0
    assert np.array_equal(m.H(1), H0)
    assert m.step == 4


def check_epoch_end_pr(seed=7):
    """Alg. 1 l.21: p_r <- p_r sqrt(E^e), E^e the epoch's error fraction."""
    getcontext().prec = 40
    rng = np.random.default_rng(seed)
    m = O.OracleModel([20, 32, 32], 4, seed=2, bs=10, p_r0=0.5)
    x, y = _bias_data(rng, 50, 20, 4)
    e1 = m.train(x[:30], y[:30])
    e2 = m.train(x[30:], y[30:], epoch_end=True)
    want = Decimal(0.5) * (Decimal(e1 + e2) / Decimal(50)).sqrt()
    assert abs(Decimal(m.p_r) - want) <= 2 * Decimal(math.ulp(float(want))), (m.p_r, want)
    pr1 = m.p_r
    e3 = m.train(x, y, epoch_end=True)
    want2 = Decimal(pr1) * (Decimal(e3) / Decimal(50)).sqrt()
    assert abs(Decimal(m.p_r) - want2) <= 2 * Decimal(math.ulp(float(want2)) + 1e-300)


def margin_teacher_task(seed, n, K0=64, c=4, margin=8):
    """A linearly separable +-1 task with a margin: labels = argmax of a random
    +-1 teacher x V, keeping only samples whose top-1 minus top-2 score >= margin."""
    rng = np.random.default_rng(seed)
    V = np.where(rng.random((K0, c)) < 0.5, 1, -1)
    xs, ys, have = [], [], 0
    while have < n:
        x = np.where(rng.random((4096, K0)) < 0.5, 1, -1)
        s = x @ V
        o = np.sort(s, axis=1)
        keep = (o[:, -1] - o[:, -2]) >= margin
        xs.append(x[keep])
        ys.append(np.argmax(s[keep], axis=1))
        have += int(keep.sum())
    x = np.concatenate(xs)[:n].astype(np.int8)
    y = np.concatenate(ys)[:n].astype(np.int32)
    return x, y


LEARN_MIN_TRAIN_ACC = 0.95   # observed: 0.994 after 5 epochs (seed 3 model, seed 1 data)


def check_learnable():
    """The rule learns a separable teacher task: 64 -> 256 -> 4, 1000 samples,
    bs = 100, 5 epochs; train accuracy >= 0.95."""
    x, y = margin_teacher_task(1, 1500)
    xtr, ytr, xte, yte = x[:1000], y[:1000], x[1000:], y[1000:]
    m = O.OracleModel([64, 256], 4, seed=3, bs=100)
    for _ in range(5):
        m.train(xtr, ytr, epoch_end=True)
    acc = (m.predict(xtr) == ytr).mean()
    assert acc >= LEARN_MIN_TRAIN_ACC, acc
    return acc, (m.predict(xte) == yte).mean()


def check_resume_equivalence(seed=8):
    """Training in one call equals training in two calls split at a batch
    boundary, and a model rebuilt from the saved state continues identically."""
    rng = np.random.default_rng(seed)
    x, y = _bias_data(rng, 120, 33, 3)
    a = O.OracleModel([33, 20, 16], 3, seed=4, bs=20, gamma=[5, 4])
    a.train(x, y)
    b = O.OracleModel([33, 20, 16], 3, seed=4, bs=20, gamma=[5, 4])
    b.train(x[:60], y[:60])
    c = O.OracleModel([33, 20, 16], 3, seed=4, bs=20, gamma=[5, 4])
    for l in (1, 2):
        c.set_H(l, b.H(l))
    c.set_scalars(b.p_r, b.step)
    b.train(x[60:], y[60:])
    c.train(x[60:], y[60:])
    for l in (1, 2):
        assert np.array_equal(a.H(l), b.H(l))
        assert np.array_equal(a.H(l), c.H(l))
    assert a.step == b.step == c.step == 6


# -- front end and early exit (O16, O17) -----------------------------------------

def check_binarize_median_rank(seed=9):
    """MedianBinarization (O16) against its rank form: x_i > m, m the
    ceil(K/2)-th smallest value, holds iff at least ceil(K/2) values of the
    pattern are strictly below x_i.  Exhaustive over small K with many ties,
    negative values and signed zeros; distinct values give floor(K/2) ones; a
    constant pattern gives none."""
    rng = np.random.default_rng(seed)
    for K in range(1, 12):
        pool = np.array([-2.0, -1.0, -0.0, 0.0, 0.5, 1.0, 3.0], np.float32)
        x = pool[rng.integers(0, len(pool), (200, K))]
        a = O.binarize_median(x)
        below = (x[:, None, :] < x[:, :, None]).sum(axis=2)   # below[mu, i] = #{j: x_j < x_i}
        want = np.where(below >= (K + 1) // 2, 1, -1)
        assert np.array_equal(a, want), K
        d = np.stack([rng.permutation(K) for _ in range(20)]).astype(np.float32) - K / 3.0
        assert np.all((O.binarize_median(d) == 1).sum(axis=1) == K // 2), K
        assert np.all(O.binarize_median(np.full((3, K), 1.5, np.float32)) == -1)


def check_early_exit_truncation(seed=10):
    """The early-exit prediction of layer l (O17) is the prediction of the same
    network cut after layer l: H_1..H_l and P_l depend only on (seed, l), so
    the truncated model is that network."""
    rng = np.random.default_rng(seed)
    widths, c = [40, 24, 16, 12], 5
    x, y = _bias_data(rng, 90, widths[0], c)
    full = O.OracleModel(widths, c, seed=3, bs=30, gamma=[4, 4, 4])
    full.train(x[:60], y[:60])
    pl = full.predict_layers(x)
    assert pl.shape == (3, 90)
    assert np.array_equal(pl[-1], full.predict(x))
    for l in (1, 2):
        cut = O.OracleModel(widths[:l + 1], c, seed=3, bs=30, gamma=[4] * l)
        for j in range(1, l + 1):
            cut.set_H(j, full.H(j))
        assert np.array_equal(cut.predict(x), pl[l - 1]), l


def check_layer_errors_match_eval(seed=11):
    """The local 01-loss count of layer l (O17) adds up, mini-batch by
    mini-batch, the patterns whose layer-l early-exit prediction with that
    mini-batch's pre-update weights differs from the label; the last layer's
    count is the train call's error count."""
    rng = np.random.default_rng(seed)
    widths, c, bs = [36, 20, 16], 4, 25
    x, y = _bias_data(rng, 100, widths[0], c)
    m = O.OracleModel(widths, c, seed=6, bs=bs, gamma=[4, 4])
    want = np.zeros(2, np.int64)
    last = 0
    for s0 in range(0, 100, bs):
        pl = m.predict_layers(x[s0:s0 + bs])
        want += (pl != y[s0:s0 + bs][None, :]).sum(axis=1)
        last += m.train(x[s0:s0 + bs], y[s0:s0 + bs])
    got = m.layer_errors(reset=True)
    assert got == [int(v) for v in want], (got, want)
    assert got[-1] == last
    assert m.layer_errors() == [0, 0]


# -- group membership (O19) -------------------------------------------------------

def check_group_members(seed=12):
    """Modes 1 and 2 order the neurons by the Philox key of O19 (recomputed here
    from the KAT-pinned Philox with numpy's stable lexsort); mode 0 is the
    identity; mode 1 does not depend on the step, mode 2 does, and equals
    mode 1 at t = 0.  Over many layers the partition is uniform: neurons 0 and
    1 share a group with probability (gamma-1)/(K-1), and neuron 0's position
    is uniform (chi-square)."""
    for K in (1, 5, 24, 130):
        assert np.array_equal(O.group_members(seed, 1, K, 0), np.arange(K))
        for l in (1, 3):
            for t in (0, 7):
                u = np.array([O.philox4x32_10([k // 4, 0, (32 << 16) + l, t],
                                              [seed & 0xFFFFFFFF, seed >> 32])[k % 4]
                              for k in range(K)], np.uint64)
                want = np.lexsort((np.arange(K), u))
                assert np.array_equal(O.group_members(seed, l, K, 2, t), want), (K, l, t)
                assert np.array_equal(O.group_members(seed, l, K, 1, t),
                                      O.group_members(seed, l, K, 2, 0))
    assert not np.array_equal(O.group_members(seed, 1, 130, 2, 1), O.group_members(seed, 1, 130, 2, 2))
    K, gamma, trials = 24, 6, 3000
    same, pos0 = 0, np.zeros(K, np.int64)
    for s in range(trials):
        m = O.group_members(1000 + s, 1 + s % 7, K, 1)
        where = np.argsort(m)
        same += int(where[0] // gamma == where[1] // gamma)
        pos0[where[0]] += 1
    p = (gamma - 1) / (K - 1)
    assert abs(same - p * trials) < 5 * np.sqrt(trials * p * (1 - p)), same
    chi2 = ((pos0 - trials / K) ** 2 / (trials / K)).sum()
    assert chi2 < 60, chi2   # 23 degrees of freedom: P(chi2 > 60) < 1e-4


def check_select_with_members(seed=13):
    """Alg. 2 over an arbitrary partition: the selected neuron lies in its
    group, has delta < 0, and no member of the group has a larger negative
    delta or the same delta with a smaller index; a group without a negative
    delta gives -1; the identity order reproduces contiguous groups."""
    rng = np.random.default_rng(seed)
    b, K, c, gamma = 30, 24, 4, 6
    for _ in range(20):
        z = rng.integers(-3, 4, size=(b, K)).astype(np.int32)    # many ties
        P = np.where(rng.random((K, c)) < 0.5, 1, -1).astype(np.int8)
        y = rng.integers(0, c, size=b).astype(np.int32)
        mark = (rng.random(b) < 0.8).astype(np.uint8)
        member = rng.permutation(K).astype(np.int32)
        sel = O.select(z, P, y, mark, gamma, member)
        assert np.array_equal(O.select(z, P, y, mark, gamma, np.arange(K)),
                              O.select(z, P, y, mark, gamma))
        delta = z * P[:, y].T
        for mu in range(b):
            for g in range(K // gamma):
                grp = member[g * gamma:(g + 1) * gamma]
                neg = [k for k in grp if delta[mu, k] < 0]
                if not mark[mu] or not neg:
                    assert sel[mu, g] == -1
                    continue
                best = max(delta[mu, k] for k in neg)
                assert sel[mu, g] == min(k for k in neg if delta[mu, k] == best), (mu, g)


def check_group_mode_single_group(seed=14):
    """With gamma = K_l the only group is the whole layer whatever the order,
    so training in modes 1 and 2 equals mode 0 exactly."""
    rng = np.random.default_rng(seed)
    x, y = _bias_data(rng, 120, 30, 3)
    ref = O.OracleModel([30, 12, 8], 3, seed=2, bs=20, gamma=[12, 8])
    ref.train(x, y)
    for mode in (1, 2):
        m = O.OracleModel([30, 12, 8], 3, seed=2, bs=20, gamma=[12, 8])
        m.set_group_mode(mode)
        m.train(x, y)
        for l in (1, 2):
            assert np.array_equal(m.H(l), ref.H(l)), (mode, l)
    a = O.OracleModel([30, 12, 8], 3, seed=2, bs=20, gamma=[4, 4])
    a.set_group_mode(2)
    a.train(x, y)
    assert not np.array_equal(a.H(1), ref.H(1))


ALL_CHECKS = [
    check_philox_kat,
    check_expand_weights_stream,
    check_expand_sign,
    check_gamma_golden,
    check_dot_bruteforce,
    check_sign_zero,
    check_local_output_popcount,
    check_local_loss_golden,
    check_local_loss_special,
    check_select_golden,
    check_select_special,
    check_perceptron_golden,
    check_cp_monotone,
    check_threshold_exact,
    check_reinforce_rate,
    check_event_law,
    check_sampler_exact_law,
    check_update_invariants,
    check_training_invariants,
    check_no_mark_no_update,
    check_epoch_end_pr,
    check_learnable,
    check_resume_equivalence,
    check_binarize_median_rank,
    check_early_exit_truncation,
    check_layer_errors_match_eval,
    check_group_members,
    check_select_with_members,
    check_group_mode_single_group,
]
