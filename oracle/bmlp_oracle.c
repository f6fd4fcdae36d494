/*
 * bmlp_oracle.c -- TEST INFRASTRUCTURE, NOT THE PRODUCT.
 *
 * A plain, slow CPU implementation of the fully binary training rule for binary
 * multi-layer perceptrons (BMLPs) of "Training multi-layer binary neural
 * networks with random local binary error signals" (arXiv 2412.00119):
 *   - Sec. 3.1            architecture (H_l, W_l = sign(H_l), fixed random P_l)
 *   - Algorithm 1, Eq. 1  network level: forward pass, local 01-loss, robustness
 *   - Algorithm 2         layer level: groups of gamma, easiest perceptron
 *   - Algorithm 3         perceptron level: clipped perceptron + reinforcement
 *   - Sec. 4.3            the rule that picks gamma from the layer width
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference
 * leg may load this library.  The GPU library never links, includes or calls it,
 * and the two share no code.
 *
 * Style on purpose: unpacked +-1 values in int8, int32 arithmetic, H_l stored in
 * the paper's own K_{l-1} x K_l orientation (element h_{ik} at [i*K_l + k]),
 * loops in the order the algorithms state them.  No bit packing, no tiling, no
 * fusion.  The only concession to speed is an OpenMP parallel-for over
 * independent outputs (neurons k), which changes no arithmetic.
 *
 * Readings of places where the paper is silent (each one is listed, with its
 * reason, in the design notes of the repository):
 *   O1  sign(0) = +1 for activations (Alg. 1 l.9).  Hidden weights are odd, so
 *       sign(h) is never 0 (see O3).
 *   O2  argmax ties resolve to the lowest class index (Eq. 1).
 *   O3  h starts at +-1 and moves in steps of +-2, so it stays odd; it is
 *       clipped to [-h_max, h_max] after every single update event, h_max odd
 *       (8-bit hidden weights, Table 4, give h_max = 255).
 *   O4  tau = (largest local output) - (second largest, counted with
 *       multiplicity), so a tie for the maximum gives tau = 0 (Alg. 1 l.13).
 *   O5  r is rational, r = r_num / r_den; "tau < r K_l" is tested exactly as
 *       tau * r_den < r_num * K_l (Alg. 1 l.14).
 *   O6  LayerUpdate (selection, CP and R) runs only when M_l is non-empty
 *       (Sec. 3.3 first sentence; Alg. 1 l.18 calls it unconditionally).
 *   O7  Groups are contiguous: neuron k is in group floor(k / gamma) (Alg. 2
 *       l.2).  A group whose neurons all have delta >= 0 contributes no tuple;
 *       among equal largest negative deltas the lowest k wins (Alg. 2 l.7).
 *   O8  Tuples of U_l are applied in (mu ascending, g ascending) order, the
 *       order in which Alg. 2 builds U_l (Alg. 3 l.2-4).
 *   O9  Alg. 3 l.7-8 reinforces each hidden weight independently with
 *       probability q = p_r sqrt(2 / (pi K_l)) (q in IEEE double, taken as 1
 *       when larger).  The events of one neuron row are sampled block by
 *       block (blocks of 64 consecutive inputs, the last one shorter) with
 *       32-bit Philox draws compared against integer thresholds thr(x) =
 *       ceil(x 2^32) (0 for x <= 0, 2^32 for x >= 1), where (1-q)^m is the
 *       left-to-right IEEE product of m factors (1-q):
 *         - a block of n inputs holds at least one event iff its draw
 *           U < thr(1 - (1-q)^n);
 *         - then its first event is at the least j with
 *           V < thr((1 - (1-q)^(j+1)) / (1 - (1-q)^n)), and after an event at p
 *           the next one is at p + 1 + g for the least g <= n - 2 - p with
 *           V < thr(1 - (1-q)^(g+1)); there is none when no such g exists.
 *       This is the law of n independent Bernoulli(q) events (first success
 *       given at least one, then geometric gaps), up to the 2^-32 rounding of
 *       the thresholds.
 *   O10 K in sqrt(2 / (pi K_l)) is the layer width K_l, as printed (Alg. 3 l.8).
 *   O11 E^e = (# training patterns of the epoch whose last-layer 01-loss was 1 in
 *       the training forward pass) / (# patterns of the epoch); p_r <- p_r *
 *       sqrt(E^e) compounds over epochs (Alg. 1 l.21).
 *   O12 The training and evaluation entry points take inputs that are already
 *       +-1, so MedianBinarization (Alg. 1 l.5) is the identity there; the
 *       front end for real-valued patterns is a separate step (O16).
 *   O13 A last mini-batch shorter than bs is processed as a batch of its own
 *       size; the step counter t counts mini-batches since creation.
 *   O14 gamma rule of Sec. 4.3: among the divisors of K_l, the one whose distance
 *       to the interval [75, 105] is smallest; among equally distant divisors the
 *       largest (the paper's examples: 525 -> 105, 2025 -> 81).
 *   O16 MedianBinarization of a real-valued pattern x in R^K (Alg. 1 l.5,
 *       Sec. 3.2: the median value is the threshold): the median of the
 *       pattern's own K values, taken as the lower median m = the
 *       ceil(K/2)-th smallest; a_i = +1 iff x_i > m (strict, compared in
 *       fp32), else -1.  With distinct values exactly floor(K/2) inputs are
 *       +1; a constant pattern is all -1.
 *   O19 Group membership (Sec. 4.3: by permutation symmetry the groups may
 *       be a random partition fixed once, or redrawn at every step).  Mode 0:
 *       contiguous groups (O7).  Modes 1 and 2: order the neurons k of layer l
 *       by the key u_k = word k%4 of Philox (k/4, 0, 32*2^16 + l, t'), ties to
 *       the smaller k; group g is the neurons at positions g*gamma ..
 *       (g+1)*gamma - 1 of that order; t' = 0 (mode 1, fixed) or the step t
 *       (mode 2, redrawn every mini-batch).  Inside a group the easiest
 *       neuron is chosen as in O7, ties to the lowest neuron index k.
 *   O17 Early exit (Sec. 3.1: the intermediate P_l may serve early-exit
 *       strategies): the prediction of layer l is argmax_j of
 *       yhat_l = a_l P_l, ties to the lowest class (O2); the local error
 *       count of layer l is the number of training patterns whose 01-loss
 *       l_l of Eq. 1 was 1 in their training forward pass.
 *   O20 Expansion layer for integer-valued inputs (Sec. 3.2, footnote to the
 *       binarisation step: a fixed random input layer with weights in {+-1}
 *       and sign activation lets the BMLP take non-binary inputs directly).
 *       Inputs are unsigned 8-bit integers (pixel intensities); expansion
 *       weight e_{k,i} (k < K expansion neurons, i < D inputs) is uniform on
 *       {+-1}, drawn like the initial weights from its own Philox stream
 *       (below); a_k = +1 iff sum_i x_i e_{k,i} >= 0 (O1), the sum taken
 *       exactly in integers.
 *
 * Philox stream layout (counter-based; Salmon, Moraes, Dror, Shaw, "Parallel
 * random numbers: as easy as 1, 2, 3", SC'11).  key = (seed mod 2^32,
 * seed div 2^32); counter words (c0, c1, c2, c3):
 *   initial h_{ik} of layer l : (i/4, k, 1*2^16 + l, 0); word i%4; h = +1 iff bit 31 set
 *   rho_{kj} of P_l           : (j/4, k, 2*2^16 + l, 0); word j%4; rho = +1 iff bit 31 set
 *   block draw U of block b (inputs 64b .. 64b+63) of neuron k, step t:
 *                               (b/4, k, 3*2^16 + l, t); word b%4
 *   event draws V_0, V_1, ... of that block, in this order:
 *                               words 0..3 of (b, k, (4 + r)*2^16 + l, t), r = 0, 1, ...
 *                               (at most 16 calls per block: r <= 15)
 *   group-order key u_k of neuron k (O19): (k/4, 0, 32*2^16 + l, t'); word k%4
 *   expansion weight e_{k,i} (O20)         : (i/4, k, 33*2^16, 0); word i%4;
 *                               e = +1 iff bit 31 set
 *   Layers are numbered l = 1..L as in the paper.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_EINVAL -1
#define OR_ENOMEM -2

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon et al., SC'11): 10 rounds of the 4x32 S-box with the */
/* published multipliers and Weyl key increments.                             */
/* ------------------------------------------------------------------------ */
void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; round++) {
    if (round > 0) {
      k0 += W0;
      k1 += W1;
    }
    uint64_t p0 = (uint64_t)M0 * (uint64_t)x0;
    uint64_t p1 = (uint64_t)M1 * (uint64_t)x2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t y0 = hi1 ^ x1 ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x3 ^ k1;
    uint32_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

static void philox_at(uint64_t seed, uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                      uint32_t out[4]) {
  uint32_t ctr[4] = {c0, c1, c2, c3};
  uint32_t key[2] = {(uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32)};
  or_philox4x32_10(ctr, key, out);
}

/* Initial hidden weight h_{ik} of layer l (Alg. 1 l.2: uniform on {+-1}). */
int32_t or_init_h(uint64_t seed, int32_t l, int32_t k, int32_t i) {
  uint32_t w[4];
  philox_at(seed, (uint32_t)(i / 4), (uint32_t)k, (1u << 16) + (uint32_t)l, 0u, w);
  return (w[i % 4] >> 31) ? +1 : -1;
}

/* Fixed random classifier weight rho_{kj} of P_l (Sec. 3.1: uniform on {+-1}). */
int32_t or_init_rho(uint64_t seed, int32_t l, int32_t k, int32_t j) {
  uint32_t w[4];
  philox_at(seed, (uint32_t)(j / 4), (uint32_t)k, (2u << 16) + (uint32_t)l, 0u, w);
  return (w[j % 4] >> 31) ? +1 : -1;
}

/* Reinforcement probability of Alg. 3 l.8: q = p_r sqrt(2 / (pi K_l)). */
double or_reinforce_prob(double p_r, int32_t K_l) {
  return p_r * sqrt(2.0 / (M_PI * (double)K_l));
}

/* thr(x) of reading O9: the integer T with (V < T) <=> (V / 2^32 < x) for
 * every 32-bit V. */
static uint64_t thr(double x) {
  if (!(x > 0.0)) return 0;
  if (x >= 1.0) return (uint64_t)1 << 32;
  return (uint64_t)ceil(x * 4294967296.0);
}

/* The thresholds of reading O9 for a block of n inputs (1 <= n <= 64):
 * any = thr(1 - (1-q)^n); first[j] = thr((1 - (1-q)^(j+1)) / (1 - (1-q)^n)),
 * j < n; gap[g] = thr(1 - (1-q)^(g+1)), g < n - 1. */
void or_r_block_tables(double q, int32_t n, uint64_t* any, uint64_t* first, uint64_t* gap) {
  if (q > 1.0) q = 1.0;
  const double s = 1.0 - q;
  double pw[65];  /* pw[m] = (1-q)^m */
  pw[0] = 1.0;
  for (int32_t m = 1; m <= n; m++) pw[m] = pw[m - 1] * s;
  const double p_any = 1.0 - pw[n];
  *any = thr(p_any);
  for (int32_t j = 0; j < n; j++) first[j] = thr((1.0 - pw[j + 1]) / p_any);
  for (int32_t g = 0; g + 1 < n; g++) gap[g] = thr(1.0 - pw[g + 1]);
}

/* The sequence of event draws V_0, V_1, ... of one block (stream layout). */
typedef struct {
  uint64_t seed;
  uint32_t b, k, l, t;
  uint32_t w[4];
  int32_t used;  /* draws taken so far */
} ev_stream;

static uint32_t next_draw(ev_stream* e) {
  if (e->used % 4 == 0)
    philox_at(e->seed, e->b, e->k, ((4u + (uint32_t)(e->used / 4)) << 16) + e->l, e->t, e->w);
  return e->w[e->used++ % 4];
}

/* Reinforcement events of neuron k of layer l at step t (Alg. 3 l.5-12,
 * reading O9): fire[i] = 1 iff h_{ik} is reinforced, i < K_prev. */
void or_r_events(uint64_t seed, int32_t l, int32_t k, uint32_t t, int32_t K_prev, double q,
                 uint8_t* fire) {
  uint64_t any[2], first[2][64], gap[2][64];
  const int32_t tail = K_prev % 64;
  or_r_block_tables(q, 64, &any[0], first[0], gap[0]);
  if (tail) or_r_block_tables(q, tail, &any[1], first[1], gap[1]);
  memset(fire, 0, (size_t)K_prev);
  for (int32_t b = 0; 64 * b < K_prev; b++) {
    const int32_t n = (K_prev - 64 * b < 64) ? K_prev - 64 * b : 64;
    const int32_t x = (n == 64) ? 0 : 1;
    uint32_t w[4];
    philox_at(seed, (uint32_t)(b / 4), (uint32_t)k, (3u << 16) + (uint32_t)l, t, w);
    if (!((uint64_t)w[b % 4] < any[x])) continue;  /* no event in this block */
    ev_stream e = {seed, (uint32_t)b, (uint32_t)k, (uint32_t)l, t, {0, 0, 0, 0}, 0};
    /* first event: the least j with V < first[j] (first[n-1] = 2^32, so the
     * scan stops inside the block) */
    uint32_t V = next_draw(&e);
    int32_t p = 0;
    while (p < n - 1 && !((uint64_t)V < first[x][p])) p++;
    fire[64 * b + p] = 1;
    /* later events: geometric gaps, cut at the end of the block */
    while (p < n - 1) {
      V = next_draw(&e);
      int32_t g = 0;
      while (g <= n - 2 - p && !((uint64_t)V < gap[x][g])) g++;
      if (g > n - 2 - p) break;
      p = p + 1 + g;
      fire[64 * b + p] = 1;
    }
  }
}

/* Sec. 4.3: gamma* = the divisor of K_l closest to the range [75, 105]
 * (reading O14 for ties). */
int32_t or_gamma_rule(int32_t K_l) {
  const int32_t lo = 75, hi = 105;
  int32_t best = -1, best_dist = 0;
  if (K_l <= 0) return -1;
  for (int32_t g = 1; g <= K_l; g++) {
    if (K_l % g != 0) continue;
    int32_t dist = (g < lo) ? (lo - g) : (g > hi) ? (g - hi) : 0;
    if (best < 0 || dist < best_dist || (dist == best_dist && g > best)) {
      best = g;
      best_dist = dist;
    }
  }
  return best;
}

static int32_t clip(int32_t h, int32_t h_max) {
  return h > h_max ? h_max : (h < -h_max ? -h_max : h);
}

static int32_t sign_of(int32_t v) { return v >= 0 ? +1 : -1; } /* O1 */

/* Group membership of layer l (O19): member[j] = the neuron at position j of
 * the group order (group g = member[g*gamma .. (g+1)*gamma - 1]). */
typedef struct {
  uint32_t u;
  int32_t k;
} or_keyed;

static int or_cmp_keyed(const void* pa, const void* pb) {
  const or_keyed* a = (const or_keyed*)pa;
  const or_keyed* b = (const or_keyed*)pb;
  if (a->u != b->u) return a->u < b->u ? -1 : 1;
  return (a->k > b->k) - (a->k < b->k);
}

int or_group_members(uint64_t seed, int32_t l, int32_t K, int32_t mode, uint32_t t,
                     int32_t* member) {
  if (K < 1 || !member || mode < 0 || mode > 2) return OR_EINVAL;
  if (mode == 0) {
    for (int32_t k = 0; k < K; k++) member[k] = k;
    return OR_OK;
  }
  or_keyed* v = (or_keyed*)malloc(sizeof(or_keyed) * (size_t)K);
  if (!v) return OR_ENOMEM;
  const uint32_t tt = (mode == 2) ? t : 0u;
  for (int32_t k = 0; k < K; k++) {
    uint32_t w[4];
    philox_at(seed, (uint32_t)k / 4u, 0u, (32u << 16) + (uint32_t)l, tt, w);
    v[k].u = w[k % 4];
    v[k].k = k;
  }
  qsort(v, (size_t)K, sizeof(or_keyed), or_cmp_keyed);
  for (int32_t j = 0; j < K; j++) member[j] = v[j].k;
  free(v);
  return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Network level, Algorithm 1                                                 */
/* ------------------------------------------------------------------------ */

/* Alg. 1 l.8-9 for one layer and b patterns:
 *   z^mu_k = sum_i a^mu_i sign(h_{ik}),   a^mu_k = sign(z^mu_k).
 * a_prev: b x K_prev (+-1), H: K_prev x K (paper orientation), z: b x K, a: b x K. */
void or_layer_forward(const int8_t* a_prev, int32_t b, int32_t K_prev, const int32_t* H, int32_t K,
                      int32_t* z, int8_t* a) {
#pragma omp parallel for schedule(static)
  for (int32_t mu = 0; mu < b; mu++) {
    int32_t* zr = z + (int64_t)mu * K;
    for (int32_t k = 0; k < K; k++) zr[k] = 0;
    for (int32_t i = 0; i < K_prev; i++) {
      const int32_t ai = a_prev[(int64_t)mu * K_prev + i];
      const int32_t* hrow = H + (int64_t)i * K;
      for (int32_t k = 0; k < K; k++) zr[k] += ai * (hrow[k] > 0 ? 1 : -1);
    }
    if (a)
      for (int32_t k = 0; k < K; k++) a[(int64_t)mu * K + k] = (int8_t)sign_of(zr[k]);
  }
}

/* Alg. 1 l.10: yhat^mu_j = sum_k a^mu_k rho_{kj}.  P: K x c. */
void or_local_output(const int8_t* a, int32_t b, int32_t K, const int8_t* P, int32_t c,
                     int32_t* yhat) {
  for (int32_t mu = 0; mu < b; mu++)
    for (int32_t j = 0; j < c; j++) {
      int32_t s = 0;
      for (int32_t k = 0; k < K; k++) s += a[(int64_t)mu * K + k] * P[(int64_t)k * c + j];
      yhat[(int64_t)mu * c + j] = s;
    }
}

/* Eq. 1 and Alg. 1 l.11-17 for b patterns.  Outputs (each may be NULL):
 * pred (argmax, O2), ell (01-loss), tau (O4), mark (mu in M_l, O5). */
void or_local_loss(const int32_t* yhat, int32_t b, int32_t c, const int32_t* y, int32_t K,
                   int32_t r_num, int32_t r_den, int32_t* pred, uint8_t* ell, int32_t* tau,
                   uint8_t* mark) {
  for (int32_t mu = 0; mu < b; mu++) {
    const int32_t* v = yhat + (int64_t)mu * c;
    int32_t jmax = 0;
    for (int32_t j = 1; j < c; j++)
      if (v[j] > v[jmax]) jmax = j;
    int32_t second = INT32_MIN;
    for (int32_t j = 0; j < c; j++)
      if (j != jmax && v[j] > second) second = v[j];
    int32_t t = (c > 1) ? v[jmax] - second : 0;
    uint8_t l01 = (jmax != y[mu]) ? 1 : 0;
    uint8_t m = (l01 == 1) || ((int64_t)t * r_den < (int64_t)r_num * K);
    if (pred) pred[mu] = jmax;
    if (ell) ell[mu] = l01;
    if (tau) tau[mu] = t;
    if (mark) mark[mu] = m;
  }
}

/* ------------------------------------------------------------------------ */
/* Layer level, Algorithm 2                                                   */
/* ------------------------------------------------------------------------ */

/* For every mu in M_l (mark[mu] != 0) and every group g of gamma neurons
 * (member == NULL: contiguous, neuron g*gamma + j; else neuron member[g*gamma + j],
 * O19): delta_k = z^mu_k rho_{k, y^mu}; k* = argmax_{k in g} {delta_k : delta_k < 0},
 * ties to the lowest k.  sel[mu * G + g] = k*, or -1 when mu is not marked or
 * no delta in g is negative. */
void or_select(const int32_t* z, int32_t b, int32_t K, const int8_t* P, int32_t c,
               const int32_t* y, const uint8_t* mark, int32_t gamma, const int32_t* member,
               int32_t* sel) {
  const int32_t G = K / gamma;
  int32_t* delta = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
  for (int32_t mu = 0; mu < b; mu++) {
    for (int32_t g = 0; g < G; g++) sel[(int64_t)mu * G + g] = -1;
    if (!mark[mu]) continue;
    for (int32_t k = 0; k < K; k++)
      delta[k] = z[(int64_t)mu * K + k] * P[(int64_t)k * c + y[mu]];
    for (int32_t g = 0; g < G; g++) {
      int32_t best = -1;
      for (int32_t j = g * gamma; j < (g + 1) * gamma; j++) {
        const int32_t k = member ? member[j] : j;
        if (delta[k] < 0 &&
            (best < 0 || delta[k] > delta[best] || (delta[k] == delta[best] && k < best)))
          best = k;
      }
      sel[(int64_t)mu * G + g] = best;
    }
  }
  free(delta);
}

/* ------------------------------------------------------------------------ */
/* Perceptron level, Algorithm 3                                              */
/* ------------------------------------------------------------------------ */

/* Clipped perceptron over U_l, in (mu, g) order (O8), then reinforcement of
 * every h of the layer with probability q at step t (O9, O10), for the
 * neurons k0 .. k0 + K - 1 of layer l (the whole layer: k0 = 0).  H: K_prev x K
 * (column j = neuron k0 + j); P: K x c (row j = neuron k0 + j); sel holds
 * neuron indices of the layer (k0 <= k < k0 + K) or -1.  The reinforcement
 * stream of a neuron is keyed by its index in the layer (Alg. 3 l.5-12, O9). */
void or_perceptron_update_at(int32_t* H, int32_t K_prev, int32_t K, int32_t k0, const int8_t* a_prev,
                             const int32_t* y, const int8_t* P, int32_t c, const int32_t* sel,
                             int32_t b, int32_t G, int32_t h_max, double q, uint64_t seed,
                             int32_t l, uint32_t t) {
  /* Clipped Perceptron, Alg. 3 l.2-4 */
  for (int32_t mu = 0; mu < b; mu++)
    for (int32_t g = 0; g < G; g++) {
      int32_t k = sel[(int64_t)mu * G + g];
      if (k < 0) continue;
      k -= k0;
      int32_t rho = P[(int64_t)k * c + y[mu]];
      for (int32_t i = 0; i < K_prev; i++) {
        int32_t* h = &H[(int64_t)i * K + k];
        *h = clip(*h + 2 * a_prev[(int64_t)mu * K_prev + i] * rho, h_max);
      }
    }
  /* Reinforcement, Alg. 3 l.5-12 */
#pragma omp parallel
  {
    uint8_t* fire = (uint8_t*)malloc((size_t)(K_prev > 0 ? K_prev : 1));
#pragma omp for schedule(static)
    for (int32_t k = 0; k < K; k++) {
      or_r_events(seed, l, k0 + k, t, K_prev, q, fire);
      for (int32_t i = 0; i < K_prev; i++)
        if (fire[i]) {
          int32_t* h = &H[(int64_t)i * K + k];
          *h = clip(*h + 2 * (*h > 0 ? 1 : -1), h_max);
        }
    }
    free(fire);
  }
}

void or_perceptron_update(int32_t* H, int32_t K_prev, int32_t K, const int8_t* a_prev,
                          const int32_t* y, const int8_t* P, int32_t c, const int32_t* sel,
                          int32_t b, int32_t G, int32_t h_max, double q, uint64_t seed,
                          int32_t l, uint32_t t) {
  or_perceptron_update_at(H, K_prev, K, 0, a_prev, y, P, c, sel, b, G, h_max, q, seed, l, t);
}

/* ------------------------------------------------------------------------ */
/* The whole rule: a model and NetworkUpdate (Alg. 1)                         */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t L;        /* number of layers */
  int32_t* K;       /* K[0..L] */
  int32_t c;        /* classes */
  int32_t h_max;    /* odd bound of |h| */
  uint64_t seed;
  int32_t bs, r_num, r_den;
  double p_r;       /* current reinforcement probability */
  int32_t* gamma;   /* gamma[1..L] */
  int64_t t;        /* mini-batches processed since creation */
  int64_t epoch_err, epoch_n;
  int64_t* layer_err; /* layer_err[l]: local 01-loss count of layer l (O17) */
  int32_t group_mode; /* O19: 0 contiguous, 1 fixed random, 2 redrawn every step */
  int32_t** H;      /* H[l]: K[l-1] x K[l] */
  int8_t** P;       /* P[l]: K[l] x c */
} or_model;

void or_destroy(or_model* m) {
  if (!m) return;
  if (m->H)
    for (int32_t l = 1; l <= m->L; l++) free(m->H[l]);
  if (m->P)
    for (int32_t l = 1; l <= m->L; l++) free(m->P[l]);
  free(m->H);
  free(m->P);
  free(m->K);
  free(m->gamma);
  free(m->layer_err);
  free(m);
}

/* widths = K_0..K_L (n_widths = L+1).  gamma may be NULL (Sec. 4.3 rule). */
int or_create(const int32_t* widths, int32_t n_widths, int32_t classes, int32_t h_max,
              uint64_t seed, int32_t bs, int32_t r_num, int32_t r_den, double p_r0,
              const int32_t* gamma, or_model** out) {
  if (!out || !widths || n_widths < 2 || classes < 2 || h_max < 1 || (h_max % 2) == 0 ||
      bs < 1 || r_num < 0 || r_den < 1 || !(p_r0 >= 0.0))
    return OR_EINVAL;
  for (int32_t l = 0; l < n_widths; l++)
    if (widths[l] < 1) return OR_EINVAL;
  or_model* m = (or_model*)calloc(1, sizeof(or_model));
  if (!m) return OR_ENOMEM;
  m->L = n_widths - 1;
  m->c = classes;
  m->h_max = h_max;
  m->seed = seed;
  m->bs = bs;
  m->r_num = r_num;
  m->r_den = r_den;
  m->p_r = p_r0;
  m->K = (int32_t*)calloc((size_t)n_widths, sizeof(int32_t));
  m->gamma = (int32_t*)calloc((size_t)n_widths, sizeof(int32_t));
  m->H = (int32_t**)calloc((size_t)n_widths, sizeof(int32_t*));
  m->P = (int8_t**)calloc((size_t)n_widths, sizeof(int8_t*));
  m->layer_err = (int64_t*)calloc((size_t)n_widths, sizeof(int64_t));
  if (!m->K || !m->gamma || !m->H || !m->P || !m->layer_err) {
    or_destroy(m);
    return OR_ENOMEM;
  }
  memcpy(m->K, widths, sizeof(int32_t) * (size_t)n_widths);
  for (int32_t l = 1; l <= m->L; l++) {
    int32_t g = gamma ? gamma[l - 1] : or_gamma_rule(m->K[l]);
    if (g < 1 || m->K[l] % g != 0) {
      or_destroy(m);
      return OR_EINVAL;
    }
    m->gamma[l] = g;
  }
  /* Alg. 1 l.2: initialise H_l and P_l uniformly on {+-1}. */
  for (int32_t l = 1; l <= m->L; l++) {
    int32_t Kp = m->K[l - 1], K = m->K[l];
    m->H[l] = (int32_t*)malloc(sizeof(int32_t) * (size_t)Kp * (size_t)K);
    m->P[l] = (int8_t*)malloc((size_t)K * (size_t)classes);
    if (!m->H[l] || !m->P[l]) {
      or_destroy(m);
      return OR_ENOMEM;
    }
#pragma omp parallel for schedule(static)
    for (int32_t i = 0; i < Kp; i++)
      for (int32_t k = 0; k < K; k++) m->H[l][(int64_t)i * K + k] = or_init_h(seed, l, k, i);
    for (int32_t k = 0; k < K; k++)
      for (int32_t j = 0; j < classes; j++)
        m->P[l][(int64_t)k * classes + j] = (int8_t)or_init_rho(seed, l, k, j);
  }
  *out = m;
  return OR_OK;
}

/* NetworkUpdate over n patterns in dataset order (Alg. 1 l.4-20); with
 * epoch_end != 0 the epoch is closed afterwards (l.21).  x: n x K_0 (+-1),
 * y: n labels in 0..c-1.  *n_err_out (may be NULL) = last-layer 01-loss count. */
int or_train(or_model* m, const int8_t* x, const int32_t* y, int64_t n, int32_t epoch_end,
             int64_t* n_err_out) {
  if (!m || n < 0 || (n > 0 && (!x || !y))) return OR_EINVAL;
  for (int64_t mu = 0; mu < n; mu++)
    if (y[mu] < 0 || y[mu] >= m->c) return OR_EINVAL;
  const int32_t L = m->L, c = m->c;
  int8_t** a = (int8_t**)calloc((size_t)L + 1, sizeof(int8_t*));
  int32_t** z = (int32_t**)calloc((size_t)L + 1, sizeof(int32_t*));
  uint8_t** mark = (uint8_t**)calloc((size_t)L + 1, sizeof(uint8_t*));
  int32_t* yhat = (int32_t*)malloc(sizeof(int32_t) * (size_t)m->bs * (size_t)c);
  uint8_t* ell = (uint8_t*)malloc((size_t)m->bs);
  int32_t* sel = NULL;
  int32_t* member = NULL;
  int64_t n_err = 0;
  int rc = OR_OK;
  if (!a || !z || !mark || !yhat || !ell) rc = OR_ENOMEM;
  for (int32_t l = 1; rc == OR_OK && l <= L; l++) {
    a[l] = (int8_t*)malloc((size_t)m->bs * (size_t)m->K[l]);
    z[l] = (int32_t*)malloc(sizeof(int32_t) * (size_t)m->bs * (size_t)m->K[l]);
    mark[l] = (uint8_t*)malloc((size_t)m->bs);
    if (!a[l] || !z[l] || !mark[l]) rc = OR_ENOMEM;
  }
  int32_t Kmax = 0;
  for (int32_t l = 1; l <= L; l++)
    if (m->K[l] > Kmax) Kmax = m->K[l];
  if (rc == OR_OK) {
    sel = (int32_t*)malloc(sizeof(int32_t) * (size_t)m->bs * (size_t)Kmax);
    member = (int32_t*)malloc(sizeof(int32_t) * (size_t)Kmax);
    if (!sel || !member) rc = OR_ENOMEM;
  }
  for (int64_t start = 0; rc == OR_OK && start < n; start += m->bs) {
    const int32_t b = (int32_t)((n - start) < m->bs ? (n - start) : m->bs); /* O13 */
    const int32_t* yb = y + start;
    a[0] = (int8_t*)(x + start * m->K[0]); /* O12: already +-1 */
    /* forward pass and local losses, Alg. 1 l.6-17 */
    for (int32_t l = 1; l <= L; l++) {
      or_layer_forward(a[l - 1], b, m->K[l - 1], m->H[l], m->K[l], z[l], a[l]);
      or_local_output(a[l], b, m->K[l], m->P[l], c, yhat);
      or_local_loss(yhat, b, c, yb, m->K[l], m->r_num, m->r_den, NULL, ell, NULL, mark[l]);
      for (int32_t mu = 0; mu < b; mu++) m->layer_err[l] += ell[mu]; /* O17 */
      if (l == L)
        for (int32_t mu = 0; mu < b; mu++) n_err += ell[mu];
    }
    /* LayerUpdate of every layer with this mini-batch's activations, Alg. 1 l.18 */
    for (int32_t l = 1; l <= L; l++) {
      int any = 0;
      for (int32_t mu = 0; mu < b; mu++) any |= mark[l][mu];
      if (!any) continue; /* O6 */
      const int32_t G = m->K[l] / m->gamma[l];
      if (m->group_mode != 0)
        or_group_members(m->seed, l, m->K[l], m->group_mode, (uint32_t)m->t, member);
      or_select(z[l], b, m->K[l], m->P[l], c, yb, mark[l], m->gamma[l],
                m->group_mode != 0 ? member : NULL, sel);
      or_perceptron_update(m->H[l], m->K[l - 1], m->K[l], a[l - 1], yb, m->P[l], c, sel, b, G,
                           m->h_max, or_reinforce_prob(m->p_r, m->K[l]), m->seed, l,
                           (uint32_t)m->t);
    }
    m->t += 1;
  }
  if (rc == OR_OK) {
    m->epoch_err += n_err;
    m->epoch_n += n;
    if (epoch_end) { /* Alg. 1 l.21, O11 */
      double E = m->epoch_n > 0 ? (double)m->epoch_err / (double)m->epoch_n : 0.0;
      m->p_r = m->p_r * sqrt(E);
      m->epoch_err = 0;
      m->epoch_n = 0;
    }
    if (n_err_out) *n_err_out = n_err;
  }
  for (int32_t l = 1; l <= L; l++) {
    if (a) free(a[l]);
    if (z) free(z[l]);
    if (mark) free(mark[l]);
  }
  free(a);
  free(z);
  free(mark);
  free(yhat);
  free(ell);
  free(sel);
  free(member);
  return rc;
}

/* Forward-only evaluation (Sec. 3.1: P_L is the output layer).  pred: n labels. */
int or_predict(const or_model* m, const int8_t* x, int64_t n, int32_t* pred) {
  if (!m || n < 0 || (n > 0 && (!x || !pred))) return OR_EINVAL;
  const int32_t L = m->L, c = m->c;
  int32_t Kmax = 0;
  for (int32_t l = 0; l <= L; l++)
    if (m->K[l] > Kmax) Kmax = m->K[l];
  const int32_t chunk = 256;
  int8_t* a0 = (int8_t*)malloc((size_t)chunk * (size_t)Kmax);
  int8_t* a1 = (int8_t*)malloc((size_t)chunk * (size_t)Kmax);
  int32_t* z = (int32_t*)malloc(sizeof(int32_t) * (size_t)chunk * (size_t)Kmax);
  int32_t* yhat = (int32_t*)malloc(sizeof(int32_t) * (size_t)chunk * (size_t)c);
  int rc = (a0 && a1 && z && yhat) ? OR_OK : OR_ENOMEM;
  for (int64_t start = 0; rc == OR_OK && start < n; start += chunk) {
    const int32_t b = (int32_t)((n - start) < chunk ? (n - start) : chunk);
    const int8_t* in = x + start * m->K[0];
    int8_t* cur = a0;
    for (int32_t l = 1; l <= L; l++) {
      or_layer_forward(in, b, m->K[l - 1], m->H[l], m->K[l], z, cur);
      in = cur;
      cur = (cur == a0) ? a1 : a0;
    }
    or_local_output(in, b, m->K[L], m->P[L], c, yhat);
    /* O2: argmax with ties to the lowest class; labels are irrelevant here */
    for (int32_t mu = 0; mu < b; mu++) {
      int32_t jmax = 0;
      for (int32_t j = 1; j < c; j++)
        if (yhat[(int64_t)mu * c + j] > yhat[(int64_t)mu * c + jmax]) jmax = j;
      pred[start + mu] = jmax;
    }
  }
  free(a0);
  free(a1);
  free(z);
  free(yhat);
  return rc;
}

/* Early-exit evaluation (Sec. 3.1, O17): pred[(l-1) n + mu] = argmax_j of
 * a_l P_l for pattern mu, every layer l = 1..L. */
int or_predict_layers(const or_model* m, const int8_t* x, int64_t n, int32_t* pred) {
  if (!m || n < 0 || (n > 0 && (!x || !pred))) return OR_EINVAL;
  const int32_t L = m->L, c = m->c;
  int32_t Kmax = 0;
  for (int32_t l = 0; l <= L; l++)
    if (m->K[l] > Kmax) Kmax = m->K[l];
  const int32_t chunk = 256;
  int8_t* a0 = (int8_t*)malloc((size_t)chunk * (size_t)Kmax);
  int8_t* a1 = (int8_t*)malloc((size_t)chunk * (size_t)Kmax);
  int32_t* z = (int32_t*)malloc(sizeof(int32_t) * (size_t)chunk * (size_t)Kmax);
  int32_t* yhat = (int32_t*)malloc(sizeof(int32_t) * (size_t)chunk * (size_t)c);
  int rc = (a0 && a1 && z && yhat) ? OR_OK : OR_ENOMEM;
  for (int64_t start = 0; rc == OR_OK && start < n; start += chunk) {
    const int32_t b = (int32_t)((n - start) < chunk ? (n - start) : chunk);
    const int8_t* in = x + start * m->K[0];
    int8_t* cur = a0;
    for (int32_t l = 1; l <= L; l++) {
      or_layer_forward(in, b, m->K[l - 1], m->H[l], m->K[l], z, cur);
      or_local_output(cur, b, m->K[l], m->P[l], c, yhat);
      for (int32_t mu = 0; mu < b; mu++) {
        int32_t jmax = 0;
        for (int32_t j = 1; j < c; j++)
          if (yhat[(int64_t)mu * c + j] > yhat[(int64_t)mu * c + jmax]) jmax = j;
        pred[(int64_t)(l - 1) * n + start + mu] = jmax;
      }
      in = cur;
      cur = (cur == a0) ? a1 : a0;
    }
  }
  free(a0);
  free(a1);
  free(z);
  free(yhat);
  return rc;
}

/* Local 01-loss counts of every layer since creation or the last reset (O17):
 * out[l-1] for l = 1..L. */
int or_layer_errors(or_model* m, int64_t* out, int32_t reset) {
  if (!m || !out) return OR_EINVAL;
  for (int32_t l = 1; l <= m->L; l++) {
    out[l - 1] = m->layer_err[l];
    if (reset) m->layer_err[l] = 0;
  }
  return OR_OK;
}

static int or_cmp_float(const void* pa, const void* pb) {
  const float a = *(const float*)pa, b = *(const float*)pb;
  return (a < b) ? -1 : (a > b) ? 1 : 0;
}

/* MedianBinarization (Alg. 1 l.5, O16): x is n x K fp32 (finite), a is n x K
 * +-1.  Each pattern is sorted (library sort) to find its lower median. */
int or_binarize_median(const float* x, int64_t n, int32_t K, int8_t* a) {
  if (n < 0 || K < 1 || (n > 0 && (!x || !a))) return OR_EINVAL;
  int rc = OR_OK;
#pragma omp parallel for schedule(static)
  for (int64_t mu = 0; mu < n; mu++) {
    float* s = (float*)malloc(sizeof(float) * (size_t)K);
    if (!s) {
#pragma omp atomic write
      rc = OR_ENOMEM;
      continue;
    }
    const float* row = x + mu * K;
    memcpy(s, row, sizeof(float) * (size_t)K);
    qsort(s, (size_t)K, sizeof(float), or_cmp_float);
    const float med = s[(K + 1) / 2 - 1];
    for (int32_t i = 0; i < K; i++) a[mu * K + i] = (int8_t)(row[i] > med ? 1 : -1);
    free(s);
  }
  return rc;
}

/* Fixed random expansion weight e_{k,i} (O20): uniform on {+-1}. */
int32_t or_expand_weight(uint64_t seed, int32_t k, int32_t i) {
  uint32_t w[4];
  philox_at(seed, (uint32_t)(i / 4), (uint32_t)k, 33u << 16, 0u, w);
  return (w[i % 4] >> 31) ? +1 : -1;
}

/* The K x D expansion matrix, e[k*D + i] = e_{k,i}. */
int or_expand_weights(uint64_t seed, int32_t K, int32_t D, int8_t* e) {
  if (K < 1 || D < 1 || !e) return OR_EINVAL;
#pragma omp parallel for schedule(static)
  for (int32_t k = 0; k < K; k++)
    for (int32_t i = 0; i < D; i++) e[(int64_t)k * D + i] = (int8_t)or_expand_weight(seed, k, i);
  return OR_OK;
}

/* Expansion layer (O20): x is n x D uint8, e is K x D +-1, a is n x K +-1;
 * a[mu][k] = sign(sum_i x[mu][i] e[k][i]) with sign(0) = +1 (O1). */
int or_expand_sign(const uint8_t* x, int64_t n, int32_t D, const int8_t* e, int32_t K, int8_t* a) {
  if (n < 0 || D < 1 || K < 1 || (n > 0 && (!x || !e || !a))) return OR_EINVAL;
#pragma omp parallel for schedule(static)
  for (int64_t mu = 0; mu < n; mu++) {
    for (int32_t k = 0; k < K; k++) {
      int64_t z = 0;
      for (int32_t i = 0; i < D; i++) z += (int64_t)x[mu * D + i] * (int64_t)e[(int64_t)k * D + i];
      a[mu * K + k] = (int8_t)(z >= 0 ? 1 : -1);
    }
  }
  return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* State access                                                               */
/* ------------------------------------------------------------------------ */
int32_t or_num_layers(const or_model* m) { return m->L; }
int32_t or_width(const or_model* m, int32_t l) { return m->K[l]; }
int32_t or_gamma(const or_model* m, int32_t l) { return m->gamma[l]; }
double or_get_pr(const or_model* m) { return m->p_r; }
int64_t or_get_step(const or_model* m) { return m->t; }

/* H: K[l-1] x K[l] (paper orientation), P: K[l] x c.  Either may be NULL. */
int or_get_layer(const or_model* m, int32_t l, int32_t* H, int8_t* P) {
  if (!m || l < 1 || l > m->L) return OR_EINVAL;
  if (H) memcpy(H, m->H[l], sizeof(int32_t) * (size_t)m->K[l - 1] * (size_t)m->K[l]);
  if (P) memcpy(P, m->P[l], (size_t)m->K[l] * (size_t)m->c);
  return OR_OK;
}

int or_set_layer(or_model* m, int32_t l, const int32_t* H) {
  if (!m || l < 1 || l > m->L || !H) return OR_EINVAL;
  memcpy(m->H[l], H, sizeof(int32_t) * (size_t)m->K[l - 1] * (size_t)m->K[l]);
  return OR_OK;
}

/* Group membership mode of every layer (O19). */
int or_set_group_mode(or_model* m, int32_t mode) {
  if (!m || mode < 0 || mode > 2) return OR_EINVAL;
  m->group_mode = mode;
  return OR_OK;
}

int or_set_scalars(or_model* m, double p_r, int64_t t) {
  if (!m || !(p_r >= 0.0) || t < 0) return OR_EINVAL;
  m->p_r = p_r;
  m->t = t;
  return OR_OK;
}

int or_set_threads(int32_t n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
  return omp_get_max_threads();
#else
  (void)n;
  return 1;
#endif
}
