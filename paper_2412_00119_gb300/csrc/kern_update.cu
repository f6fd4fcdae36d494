// kern_update.cu -- local classifiers, selection and the hidden-weight update of
// the BMLP training rule (arXiv 2412.00119, Alg. 1 l.10-18, Alg. 2, Alg. 3), plus
// initialisation and the evaluation output.
#include <climits>

#include "update_common.cuh"

namespace bk {
namespace {

__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ int64_t batch_start(const StepParams* P) {
  return (int64_t)P->ctrl->s * P->bs;
}

__device__ __forceinline__ int64_t batch_size(const StepParams* P, int64_t start) {
  const int64_t rem = P->n - start;
  return rem < P->bs ? rem : P->bs;
}

}  // namespace

// ---------------------------------------------------------------------------
// Local classifier, 01-loss, robustness margin and group selection.
// Grid (bs, L): CTA (mu, l) handles pattern mu of layer l.
//   yhat_j = K_l - 2 popc(A_l[mu] XOR P_l^T[j])                      (Alg. 1 l.10)
//   pred = argmax (lowest j), loss = [pred != y], tau = top1 - top2   (Eq. 1, l.12-13)
//   mark = loss or tau * r_den < r_num * K_l                         (l.14-15)
//   for marked mu, group g: sel = argmax_{k in g} {delta_k < 0},
//   delta_k = z_k rho_{k,y}, ties to the lowest k; -1 if none        (Alg. 2 l.4-8)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kClsThreads) k_cls_select(const StepParams* __restrict__ P) {
  const int li = blockIdx.y;
  const int mu = blockIdx.x;
  const DevLayer& Ly = P->layer[li];
  Ctrl* ctrl = P->ctrl;
  pdl_wait();
  pdl_trigger();
  const int64_t start = batch_start(P);
  const int64_t bsz = batch_size(P, start);
  if (mu >= bsz) return;
  if (ctrl->timeouts != 0u) {
    // a bounded wait of this step's forward pass expired (or an earlier one
    // is not yet reported): Z and A are not valid, so the pattern is marked
    // for nothing; with every mark 0 the update leaves H and W as they are
    // and only advances the step counters
    if (threadIdx.x == 0) Ly.mark[mu] = 0;
    return;
  }
  const int c = P->c;
  __shared__ int yh[BMLP_MAX_CLASSES];
  __shared__ int s_mark, s_y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;

  const uint64_t* a = Ly.A + (int64_t)mu * Ly.nw_out;
  for (int j = warp; j < c; j += nwarps) {
    const uint64_t* pt = Ly.PT + (int64_t)j * Ly.nw_out;
    int cnt = 0;
    for (int w = lane; w < Ly.nw_out; w += 32) cnt += __popcll(a[w] ^ pt[w]);
    cnt = warp_sum(cnt);
    if (lane == 0) yh[j] = Ly.Kout - 2 * cnt;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int yv = P->y[start + mu];
    if (yv < 0 || yv >= c) {
      if (li == 0) atomicAdd(&ctrl->bad_labels, 1ull);
      yv = 0;  // memory-safe stand-in; the host reports BMLP_EINVAL
    }
    int jmax = 0;
    for (int j = 1; j < c; ++j)
      if (yh[j] > yh[jmax]) jmax = j;
    int second = INT_MIN;
    for (int j = 0; j < c; ++j)
      if (j != jmax && yh[j] > second) second = yh[j];
    const int tau = yh[jmax] - second;
    const int loss = (jmax != yv) ? 1 : 0;
    const int mark = loss || ((long long)tau * P->r_den < (long long)P->r_num * Ly.Kout);
    Ly.mark[mu] = (uint8_t)mark;
    if (mark) atomicOr(&ctrl->any_mark[li], 1u);
    if (loss) atomicAdd(&ctrl->layer_err[li], 1ull);
    if (li == P->L - 1 && loss) atomicAdd(&ctrl->err, 1ull);
    s_mark = mark;
    s_y = yv;
  }
  __syncthreads();

  // selections are stored group-major (sel[g][mu]): the update kernel reads a
  // group's bs selections as one contiguous run
  int16_t* sel = Ly.sel + mu;
  const int64_t sstride = P->bs;
  if (!s_mark) {
    for (int g = threadIdx.x; g < Ly.G; g += blockDim.x) sel[g * sstride] = -1;
    return;
  }
  const int y = s_y;
  const int16_t* z = Ly.Z + (int64_t)mu * Ly.Kout;
  const int gamma = Ly.gamma;
  const int per = gamma >> 3;  // 8-neuron chunks per group
  if (Ly.member == nullptr && (gamma & 7) == 0 && per <= 32 && (per & (per - 1)) == 0) {
    // one thread per 8 neurons: 16-byte z loads, 8 bytes of rho^T, then the
    // group's per lanes (consecutive, aligned) reduce with shuffles
    const int8_t* rt = Ly.rhoT + (int64_t)y * Ly.Kout;
    const int nchunk = Ly.Kout >> 3;
    for (int base = 0; base < nchunk; base += blockDim.x) {
      const int ci = base + threadIdx.x;
      int bestd = INT_MIN, bestk = INT_MAX;
      if (ci < nchunk) {
        const uint4 zv = *reinterpret_cast<const uint4*>(z + 8 * ci);
        const uint2 rv = *reinterpret_cast<const uint2*>(rt + 8 * ci);
        const uint32_t zw[4] = {zv.x, zv.y, zv.z, zv.w};
        const uint32_t rw[2] = {rv.x, rv.y};
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int zj = (int)(int16_t)(zw[j >> 1] >> (16 * (j & 1)));
          const int rj = (int)(int8_t)(rw[j >> 2] >> (8 * (j & 3)));
          const int d = zj * rj;
          if (d < 0 && d > bestd) {  // ascending k: strict '>' keeps the lowest
            bestd = d;
            bestk = 8 * ci + j;
          }
        }
      }
      for (int off = per >> 1; off > 0; off >>= 1) {
        const int od = __shfl_xor_sync(0xffffffffu, bestd, off);
        const int ok = __shfl_xor_sync(0xffffffffu, bestk, off);
        if (od > bestd || (od == bestd && ok < bestk)) {
          bestd = od;
          bestk = ok;
        }
      }
      if (ci < nchunk && (ci & (per - 1)) == 0)
        sel[(ci / per) * sstride] = (bestd == INT_MIN) ? (int16_t)-1 : (int16_t)bestk;
    }
    return;
  }
  // warp per group; the group's neurons are contiguous or listed by the group
  // order (random partition), so ties compare neuron indices explicitly
  const int16_t* member = Ly.member;
  for (int g = warp; g < Ly.G; g += nwarps) {
    int bestd = INT_MIN, bestk = INT_MAX;
    for (int kk = lane; kk < gamma; kk += 32) {
      const int k = member ? (int)member[g * gamma + kk] : g * gamma + kk;
      const int d = (int)z[k] * (int)Ly.rho[(int64_t)k * c + y];
      if (d < 0 && (d > bestd || (d == bestd && k < bestk))) {
        bestd = d;
        bestk = k;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const int od = __shfl_xor_sync(0xffffffffu, bestd, off);
      const int ok = __shfl_xor_sync(0xffffffffu, bestk, off);
      if (od > bestd || (od == bestd && ok < bestk)) {
        bestd = od;
        bestk = ok;
      }
    }
    if (lane == 0) sel[g * sstride] = (bestd == INT_MIN) ? (int16_t)-1 : (int16_t)bestk;
  }
}

// ---------------------------------------------------------------------------
// Hidden-weight update, fused with the visible-weight repack (Alg. 3, Sec. 3.1).
// The grid is persistent (as many CTAs as fit on the device); every warp takes
// rows -- all layers' neuron rows in one numbering -- from the step's row
// counter, kRowChunk at a time, and owns one neuron row k at a time:
//   1. it collects, in ascending mu, the patterns whose selection in group g
//      is k (the CP tuples of k);
//   2. it copies the row's reinforcement-event bitmap (one 64-bit word per
//      block of 64 inputs, drawn by k_r_events) into shared memory with
//      cp.async, overlapping step 1;
//   (a row without CP tuple is not streamed: its H changes only at its
//   reinforcement events, applied as single-weight read-modify-writes, and
//   its W is unchanged because reinforcement never flips a sign)
//   3. it streams the row in chunks of 8 hidden weights, two chunks per lane
//      per iteration, with a rotating queue of four 16-byte vectors in flight
//      per lane: the CP tuples, then the chunk's reinforcement events (its byte
//      of the bitmap; lanes with an event step away from 0, as Alg. 3 orders
//      CP before R), then H and the W byte are written.
// H holds each weight as its lattice index v = (h + h_max)/2 + 2^hb (see
// DevLayer): a CP or R event is a step of +-1 in v, and v stays in
// [2^hb, 2^hb + h_max] subset of (0, 2^15).  A 32-bit word holds two lanes, so a
// packed pair of +-1 steps is one 32-bit add with no carry between lanes.
// After a step a lane can only have left the range by one, to 2^hb - 1 (bit hb
// clear) or to 2^hb + h_max + 1 (= 2^(hb+1) when h_max + 1 = 2^hb, kPow2); the
// clip moves it back.  h > 0 is the lane's bit hb - 1 (kPow2) or v >= 2^hb +
// (h_max + 1)/2.  The CP step per tuple adds the packed +-1 steps
// 2 a^mu_i rho_{k,y^mu}/2 from a 256-entry shared byte table, then clips.
// The partly padded last chunk of a row runs per weight.  Layers with an
// empty M_l are skipped (no CP, no R).  The last warp to finish advances the
// step counters and clears the per-step flags.
// ---------------------------------------------------------------------------
namespace {

using namespace upd;
constexpr int kPre = 4;  // tuples per row whose activation bytes are prefetched
// the prefetched activation bytes of one chunk, one byte per tuple
using TupleBytes = uint32_t;
static_assert(kPre <= (int)sizeof(TupleBytes), "one byte per prefetched tuple");
constexpr int kRowChunk = 1;  // rows a warp takes from the row counter at a time

// shared memory of one update warp: s_list [bs] int32, s_ev [nblk_max] uint64
__host__ __device__ __forceinline__ size_t update_warp_smem(int bs, int nblk_max) {
  return ((sizeof(int32_t) * (size_t)bs + 7) & ~(size_t)7) + sizeof(uint64_t) * (size_t)nblk_max;
}

__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;"
               ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))), "l"(gmem) : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Least j in [0, hi] with V < tab[j], or hi when there is none (tab
// nondecreasing).
__device__ __forceinline__ int least_below(uint32_t V, const unsigned long long* tab, int hi) {
  int lo = 0;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if ((unsigned long long)V < tab[mid]) hi = mid;
    else lo = mid + 1;
  }
  return lo;
}

// The events of block b (n inputs, tables index x) of neuron k at step t,
// given that the block holds at least one: the first from the first-event
// table, the next ones by geometric gaps cut at the block's end; the draws
// are the words of Philox((b, k, (4 + r) 2^16 + l, t)), r = 0, 1, ... in order.
__device__ __forceinline__ uint64_t block_events(const RTables& R, int x, int n, uint32_t b,
                                                 uint32_t k, uint32_t l, uint32_t t, uint32_t key0,
                                                 uint32_t key1) {
  uint32_t r = 0;
  uint4 v = philox4x32_10(make_uint4(b, k, (4u << 16) + l, t), key0, key1);
  int used = 1;
  int p = least_below(v.x, R.first[x], n - 1);
  uint64_t mask = 1ull << p;
#pragma unroll 1
  while (p < n - 1) {
    if (used == 4) {
      ++r;
      v = philox4x32_10(make_uint4(b, k, ((4u + r) << 16) + l, t), key0, key1);
      used = 0;
    }
    const uint32_t V = word_of(v, used++);
    const int gmax = n - 2 - p;
    if (!((unsigned long long)V < R.gap[gmax])) break;  // no further event in the block
    p += 1 + least_below(V, R.gap, gmax);
    mask |= 1ull << p;
  }
  return mask;
}

}  // namespace

size_t update_smem_bytes(int bs, int nblk_max) {
  return (size_t)(kUpdThreads / 32) * update_warp_smem(bs, nblk_max);
}

template <int kHb>
__global__ void __launch_bounds__(kUpdThreads, 4) k_update(const StepParams* __restrict__ P,
                                                           uint32_t key0, uint32_t key1) {
  extern __shared__ int32_t dyn[];
  __shared__ uint4 s_db[256];
  __shared__ uint2 s_fire[16];
  __shared__ unsigned long long s_stats[3];
  Ctrl* ctrl = P->ctrl;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
  // dynamic shared memory, per warp: s_list [bs] int32 | (8-byte aligned)
  // s_ev [nblk_max] uint64
  const size_t wbytes = update_warp_smem(P->bs, P->nblk_max);
  uint8_t* wbase = reinterpret_cast<uint8_t*>(dyn) + (size_t)warp * wbytes;
  int32_t* s_list = reinterpret_cast<int32_t*>(wbase);
  uint64_t* s_ev = reinterpret_cast<uint64_t*>(wbase + ((sizeof(int32_t) * P->bs + 7) & ~(size_t)7));

  if (threadIdx.x == 0) s_stats[0] = s_stats[1] = s_stats[2] = 0ull;
  // s_db[b]: the +-1 lattice steps of the 8 weights of a chunk whose
  // activation byte is b, for rho = +1 (rho = -1 indexes with ~b): d = +1 for
  // a set bit, two lanes per word (d_lo + 2^16 d_hi)
  {
    const int b = threadIdx.x & 255;
    uint32_t wv[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int d0 = ((b >> (2 * j)) & 1) ? 1 : -1, d1 = ((b >> (2 * j + 1)) & 1) ? 1 : -1;
      wv[j] = (uint32_t)(d0 + 65536 * d1);
    }
    if (threadIdx.x < 256) s_db[b] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
  if (threadIdx.x < 32) {
    const int r = threadIdx.x >> 4, n = threadIdx.x & 15;
    // s_fire[n]: 1 in each lane of nibble n whose bit is set, two lanes per word
    if (r == 0)
      s_fire[n] = make_uint2((uint32_t)((n & 1) | ((n >> 1) & 1) << 16),
                             (uint32_t)(((n >> 2) & 1) | ((n >> 3) & 1) << 16));
  }
  // the tables above depend on no earlier kernel; everything below does
  pdl_wait();
  pdl_trigger();
  const unsigned long long t = ctrl->t;
  const uint32_t s = ctrl->s;
  const int64_t start = (int64_t)s * P->bs;
  const int bsz = (int)batch_size(P, start);
  // an expired bounded wait in this step's forward pass: no CP, no R (the
  // selection kernel marked nothing either); the counters still advance
  const bool step_failed = ctrl->timeouts != 0u;
  __syncthreads();

  const int c = P->c;
  Enc E;
  E.h_max = P->h_max;
  E.hb = P->hb;
  E.base = 1 << P->hb;
  Lanes<kHb> LN;
  LN.hb_rt = P->hb;
  LN.over_pair = (uint32_t)(E.base + E.h_max + 1) * kLaneOne;
  LN.pos_pair = (uint32_t)(E.base + (E.h_max + 1) / 2) * kLaneOne;
  const uint32_t pos_from = (uint32_t)(E.base + (E.h_max + 1) / 2);  // lattice index of h = +1
  const uint32_t v_top = (uint32_t)(E.base + E.h_max);
  const int rows_total = P->rows_total;

  // every warp takes chunks of kRowChunk rows (all layers, in order) from the
  // step's row counter until the rows run out
  uint32_t st_rows = 0, st_streamed = 0, st_bytes = 0;  // statistics (per warp)
#pragma unroll 1
  while (true) {
    int base = 0;
    if (lane == 0) base = (int)atomicAdd(&ctrl->upd_next, (unsigned)kRowChunk);
    base = __shfl_sync(kFull, base, 0);
    if (base >= rows_total) break;
#pragma unroll 1
    for (int gr = base; gr < min(base + kRowChunk, rows_total); ++gr) {
      int li = 0;
      while (li + 1 < P->L && gr >= P->layer[li + 1].row_base) ++li;
      if (step_failed || ctrl->any_mark[li] == 0u) continue;   // M_l empty: no CP, no R
      const DevLayer& Ly = P->layer[li];
      const int k = gr - Ly.row_base;
      const int gamma = Ly.gamma;
      const int g = Ly.group_of ? (int)Ly.group_of[k] : k / gamma;
      const int Kin = Ly.Kin;
      const int nch = (Kin + 7) >> 3;             // chunks holding at least one input
      const int full = Kin >> 3;                  // chunks of 8 real inputs
      const int nblk = Ly.nblk;
      const uint32_t arow_bytes = (uint32_t)Ly.nw_in * 8u;
      const uint8_t* aprev = (li == 0) ? reinterpret_cast<const uint8_t*>(P->x + start * P->nw0)
                                       : reinterpret_cast<const uint8_t*>(P->layer[li - 1].A);
      {
        // the row's event bitmap -> shared memory, overlapping the tuple scan
        const uint64_t* evrow = Ly.EV + (int64_t)k * Ly.ev_stride;
        for (int b = lane; b < nblk; b += 32) cp_async8(s_ev + b, evrow + b);
        cp_async_commit();
      }
      // ---- 1. CP tuples of neuron k, ascending mu ----
      int n_t = 0;
      for (int mb = 0; mb < bsz; mb += 32) {
        const int m = mb + lane;
        const bool hit = (m < bsz) && (Ly.sel[(int64_t)g * P->bs + m] == k);
        const unsigned bal = __ballot_sync(kFull, hit);
        if (hit) {
          int yv = P->y[start + m];
          if (yv < 0 || yv >= c) yv = 0;
          const int rho = Ly.rho[(int64_t)k * c + yv];
          s_list[n_t + __popc(bal & ((1u << lane) - 1u))] = m | ((rho > 0) ? 0 : 0x10000);
        }
        n_t += __popc(bal);
      }
      // ---- 2. the row's reinforcement events (drawn by k_r_events) ----
      cp_async_wait<0>();
      __syncwarp();

        int16_t* hrow = Ly.H + (int64_t)k * Ly.ldh;
        if (n_t == 0) {
          // no tuple: H changes only at the reinforcement events, which never
          // flip a sign, so W stays; single-weight read-modify-writes
          int nev = 0;
  #pragma unroll 1
          for (int b = lane; b < nblk; b += 32) {
            uint64_t mask = s_ev[b];
            nev += __popcll(mask);
  #pragma unroll 1
            while (mask != 0ull) {
              const int bit = __ffsll((long long)mask) - 1;
              mask &= mask - 1ull;
              int16_t* hp = hrow + 64 * b + bit;
              const uint32_t v = (uint16_t)*hp;
              *hp = (int16_t)((v >= pos_from) ? min(v + 1u, v_top) : max(v - 1u, (uint32_t)E.base));
            }
          }
          nev = warp_sum(nev);
          st_rows += 1u;
          st_bytes += 4u * (uint32_t)nev;
          __syncwarp();   // s_ev and s_list are reused by the next row
          continue;
        }
        st_rows += 1u;
        st_streamed += 1u;
        st_bytes += 4u * (uint32_t)Ly.ldh + 8u * (uint32_t)Ly.nw_in;

        // ---- 3. CP and W over the row ----
        uint8_t* wrow = reinterpret_cast<uint8_t*>(Ly.W + (int64_t)k * Ly.nw_in);
        // Each iteration handles two chunks per lane, ch and ch + 32 (64 chunks
        // per warp), so the tuple loop and the loop control are shared.  A
        // rotating queue keeps the H vectors of the next iteration in flight (4
        // per lane); the activation bytes of the first kPre tuples are fetched at
        // the top of each iteration.  Every lane runs the same number of
        // iterations.
        uint4 q0 = make_uint4(0, 0, 0, 0), q1 = q0, q2 = q0, q3 = q0;
        if (lane < nch) q0 = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * lane));
        if (lane + 32 < nch) q1 = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * (lane + 32)));
        if (lane + 64 < nch) q2 = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * (lane + 64)));
        if (lane + 96 < nch) q3 = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * (lane + 96)));
        const int iters2 = (nch + 63) >> 6;
        // activation bytes of tuples 0..kPre-1 (one per byte) for the next
        // iteration's two chunks, loaded one iteration ahead
        auto tuple_bytes = [&](int it_next, TupleBytes (&pbo)[2]) {
          pbo[0] = 0u;
          pbo[1] = 0u;
  #pragma unroll
          for (int q = 0; q < kPre; ++q) {
            if (q < n_t) {
              const uint8_t* arow = aprev + (size_t)(s_list[q] & 0xFFFF) * arow_bytes;
  #pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int ch = 64 * it_next + 32 * u + lane;
                if (ch < nch) pbo[u] |= (TupleBytes)__ldg(arow + ch) << (8 * q);
              }
            }
          }
        };
        TupleBytes pbn[2];
        tuple_bytes(0, pbn);
  #pragma unroll 1
        for (int it = 0; it < iters2; ++it) {
          int chv[2];
          bool live[2];
          uint4 w[2];
          TupleBytes pb[2] = {pbn[0], pbn[1]};  // this iteration's tuple bytes
          chv[0] = 64 * it + lane;
          chv[1] = chv[0] + 32;
          live[0] = chv[0] < nch;
          live[1] = chv[1] < nch;
          if (it + 1 < iters2) tuple_bytes(it + 1, pbn);
          w[0] = q0;
          w[1] = q1;
          q0 = q2;
          q1 = q3;
          if (chv[0] + 128 < nch) q2 = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * (chv[0] + 128)));
          if (chv[1] + 128 < nch) q3 = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * (chv[1] + 128)));
  #pragma unroll
          for (int q = 0; q < kPre; ++q) {
            if (q < n_t) {
              const uint32_t xm = (s_list[q] & 0x10000) ? 0xFFu : 0u;  // rho = -1: ~byte
  #pragma unroll
              for (int u = 0; u < 2; ++u) {
                const uint4 d = s_db[((uint32_t)(pb[u] >> (8 * q)) ^ xm) & 0xFFu];
                w[u].x = LN.clip(w[u].x + d.x);
                w[u].y = LN.clip(w[u].y + d.y);
                w[u].z = LN.clip(w[u].z + d.z);
                w[u].w = LN.clip(w[u].w + d.w);
              }
            }
          }
  #pragma unroll 1
          for (int q = kPre; q < n_t; ++q) {
            const int e = s_list[q];
            const uint32_t xm = (e & 0x10000) ? 0xFFu : 0u;
            const uint8_t* arow = aprev + (size_t)(e & 0xFFFF) * arow_bytes;
  #pragma unroll
            for (int u = 0; u < 2; ++u) {
              const uint32_t byte = live[u] ? arow[chv[u]] : 0u;
              const uint4 d = s_db[(byte ^ xm) & 0xFFu];
              w[u].x = LN.clip(w[u].x + d.x);
              w[u].y = LN.clip(w[u].y + d.y);
              w[u].z = LN.clip(w[u].z + d.z);
              w[u].w = LN.clip(w[u].w + d.w);
            }
          }
          // ---- R: the chunks' bytes of the row's event bitmap ----
          uint32_t fb[2];
  #pragma unroll
          for (int u = 0; u < 2; ++u)
            fb[u] = live[u] ? (uint32_t)reinterpret_cast<const uint8_t*>(s_ev)[chv[u]] : 0u;
          if (__any_sync(kFull, (fb[0] | fb[1]) != 0u)) {
  #pragma unroll
            for (int u = 0; u < 2; ++u) {
              if (fb[u] != 0u) {
                const uint2 fl = s_fire[fb[u] & 15u], fh = s_fire[fb[u] >> 4];
                w[u].x = LN.reinforce(w[u].x, fl.x);
                w[u].y = LN.reinforce(w[u].y, fl.y);
                w[u].z = LN.reinforce(w[u].z, fh.x);
                w[u].w = LN.reinforce(w[u].w, fh.y);
              }
            }
          }
  #pragma unroll
          for (int u = 0; u < 2; ++u) {
            uint32_t wbyte = LN.w_byte(w[u]);
            if (live[u] && chv[u] >= full) {
              // the partly padded last chunk: per weight, from the row as
              // loaded (H is written back only below)
              const uint4 w0 = *reinterpret_cast<const uint4*>(hrow + 8 * chv[u]);
              const ChunkOut o = chunk_scalar(w0, chv[u], Kin - 8 * chv[u], s_list, n_t, aprev,
                                              arow_bytes, E, fb[u]);
              w[u] = o.w;
              wbyte = o.wbyte;
            }
            if (live[u]) {
              __stcs(reinterpret_cast<uint4*>(hrow + 8 * chv[u]), w[u]);
              wrow[chv[u]] = (uint8_t)wbyte;
            }
          }
        }
      __syncwarp();   // s_ev and s_list are reused by the next row
    }
  }
  // statistics: per CTA, one atomic per counter
  if (lane == 0) {
    atomicAdd(&s_stats[0], (unsigned long long)st_rows);
    atomicAdd(&s_stats[1], (unsigned long long)st_streamed);
    atomicAdd(&s_stats[2], (unsigned long long)st_bytes);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    atomicAdd(&ctrl->upd_rows, s_stats[0]);
    atomicAdd(&ctrl->upd_streamed, s_stats[1]);
    atomicAdd(&ctrl->upd_bytes, s_stats[2]);
  }

  // step completion: the last warp to finish advances the counters
  __syncwarp();
  if (lane == 0) {
    __threadfence();
    const unsigned prev = atomicAdd(&ctrl->done, 1u);
    if (prev == gridDim.x * nwarps - 1) {
      ctrl->t = t + 1;
      ctrl->s = s + 1;
      for (int i = 0; i < P->L; ++i) ctrl->any_mark[i] = 0u;
      ctrl->upd_next = 0u;
      ctrl->done = 0u;
      __threadfence();
    }
  }
}

// Reinforcement events of the current step (Alg. 3 l.5-12): warp per neuron
// row; lane j draws the block draws of blocks 4j .. 4j+3 (one Philox call), the
// blocks that hold an event are compacted into a per-warp list, and the lanes
// share that list for the event draws (binary searches in the layer's
// threshold tables, staged in shared memory); the row's bitmap goes to
// DevLayer::EV.  It depends only on (seed, layer, neuron, step, p_r), so it
// runs beside the forward passes.
__global__ void __launch_bounds__(kEvThreads) k_r_events(const StepParams* __restrict__ P,
                                                         uint32_t key0, uint32_t key1) {
  __shared__ RTables s_rt;
  __shared__ uint16_t s_cand[kEvRowsPerCta][128];  // blocks with an event, per warp
  const int bid = blockIdx.x;
  int li = 0;
  while (li + 1 < P->L && bid >= P->layer[li + 1].ev_cta_base) ++li;
  const DevLayer& Ly = P->layer[li];
  {
    const unsigned long long* src = reinterpret_cast<const unsigned long long*>(P->rt + li);
    unsigned long long* dst = reinterpret_cast<unsigned long long*>(&s_rt);
    for (int i = threadIdx.x; i < (int)(sizeof(RTables) / 8); i += blockDim.x) dst[i] = src[i];
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = (bid - Ly.ev_cta_base) * kEvRowsPerCta + warp;
  if (k >= Ly.Kout) return;
  const uint32_t l = (uint32_t)li + 1u;
  const uint32_t tt = (uint32_t)P->ctrl->t;
  const int Kin = Ly.Kin, nblk = Ly.nblk;
  uint64_t* ev = Ly.EV + (int64_t)k * Ly.ev_stride;
  uint16_t* cand = s_cand[warp];
  // rounds of 32 block groups (128 blocks): the block draws, one Philox call per
  // lane; the blocks that hold an event are compacted into a list that the
  // lanes then share, one block each, for the event draws
#pragma unroll 1
  for (int g0 = 0; 4 * g0 < nblk; g0 += 32) {
    const int gq = g0 + lane;
    uint32_t cmask = 0;
    if (4 * gq < nblk) {
      const uint4 u = philox4x32_10(make_uint4((uint32_t)gq, (uint32_t)k, (3u << 16) + l, tt), key0,
                                    key1);
#pragma unroll
      for (int wq = 0; wq < 4; ++wq) {
        const int b = 4 * gq + wq;
        if (b < nblk) {
          const int x = (Kin - 64 * b >= 64) ? 0 : 1;
          if ((unsigned long long)word_of(u, wq) < s_rt.any[x]) cmask |= 1u << wq;
          else ev[b] = 0ull;
        }
      }
    }
    // exclusive prefix of the candidate counts over the lanes
    const int cnt = __popc(cmask);
    int incl = cnt;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int v = __shfl_up_sync(kFull, incl, off);
      if (lane >= off) incl += v;
    }
    const int total = __shfl_sync(kFull, incl, 31);
    int pos = incl - cnt;
#pragma unroll
    for (int wq = 0; wq < 4; ++wq)
      if ((cmask >> wq) & 1u) cand[pos++] = (uint16_t)(4 * gq + wq);
    __syncwarp();
#pragma unroll 1
    for (int i = lane; i < total; i += 32) {
      const int b = cand[i];
      const int n = min(64, Kin - 64 * b);
      ev[b] = block_events(s_rt, (n == 64) ? 0 : 1, n, (uint32_t)b, (uint32_t)k, l, tt, key0, key1);
    }
    __syncwarp();
  }
}

// ---------------------------------------------------------------------------
// Group order of a layer with a random partition (Sec. 4.3): CTA l sorts the
// 64-bit keys (u_k << 32 | k), u_k = word k%4 of Philox (k/4, 0, 32*2^16 + l,
// t'), ascending with a bitonic network in shared memory (keys are distinct,
// so ties in u_k go to the smaller k), then member[j] = the k of the j-th key
// and group_of[k] = j / gamma.  t' = the step counter when redrawn every
// step, else 0.
// ---------------------------------------------------------------------------
constexpr int kGroupThreads = 1024;

__global__ void __launch_bounds__(kGroupThreads) k_group_order(const StepParams* __restrict__ P,
                                                               int redraw) {
  extern __shared__ unsigned long long keys[];
  const DevLayer& Ly = P->layer[blockIdx.x];
  if (Ly.member == nullptr) return;
  const int K = Ly.Kout;
  int n = 1;
  while (n < K) n <<= 1;
  const uint32_t t = redraw ? (uint32_t)P->ctrl->t : 0u;
  const uint32_t c2 = (32u << 16) + (uint32_t)(blockIdx.x + 1);
  for (int k = threadIdx.x; k < n; k += kGroupThreads) {
    unsigned long long v = ~0ull;
    if (k < K) {
      const uint4 w = philox4x32_10(make_uint4((uint32_t)k >> 2, 0u, c2, t), P->key0, P->key1);
      const uint32_t u = (k & 3) == 0 ? w.x : (k & 3) == 1 ? w.y : (k & 3) == 2 ? w.z : w.w;
      v = ((unsigned long long)u << 32) | (uint32_t)k;
    }
    keys[k] = v;
  }
  __syncthreads();
  for (int size = 2; size <= n; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (n >> 1); i += kGroupThreads) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool up = (lo & size) == 0;
        const unsigned long long a = keys[lo], b = keys[hi];
        if ((a > b) == up) {
          keys[lo] = b;
          keys[hi] = a;
        }
      }
      __syncthreads();
    }
  }
  for (int j = threadIdx.x; j < K; j += kGroupThreads) {
    const int k = (int)(uint32_t)keys[j];
    Ly.member[j] = (int16_t)k;
    Ly.group_of[k] = (int16_t)(j / Ly.gamma);
  }
}

static size_t group_order_smem(int max_K) {
  int n = 1;
  while (n < max_K) n <<= 1;
  return sizeof(unsigned long long) * (size_t)n;
}

cudaError_t prepare_group_order(int max_K) {
  return cudaFuncSetAttribute(k_group_order, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)group_order_smem(max_K));
}

cudaError_t launch_group_order(int L, int max_K, bool redraw, cudaStream_t st, const StepParams* P) {
  k_group_order<<<(unsigned)L, kGroupThreads, group_order_smem(max_K), st>>>(P, redraw ? 1 : 0);
  return cudaGetLastError();
}

void launch_r_events(unsigned grid, cudaStream_t st, const StepParams* P, uint32_t key0,
                     uint32_t key1) {
  k_r_events<<<grid, kEvThreads, 0, st>>>(P, key0, key1);
}

cudaError_t launch_update(int hb_mode, unsigned grid, size_t smem, cudaStream_t st, bool pdl,
                          const StepParams* P, uint32_t key0, uint32_t key1) {
  if (hb_mode == 8)
    return launch_kernel(k_update<8>, dim3(grid), dim3(kUpdThreads), smem, st, pdl, P, key0, key1);
  if (hb_mode != 0)
    return launch_kernel(k_update<-1>, dim3(grid), dim3(kUpdThreads), smem, st, pdl, P, key0, key1);
  return launch_kernel(k_update<0>, dim3(grid), dim3(kUpdThreads), smem, st, pdl, P, key0, key1);
}

cudaError_t update_kernel_occupancy(int hb_mode, size_t smem, int* per_sm) {
  if (hb_mode == 8)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, k_update<8>, kUpdThreads, smem);
  if (hb_mode != 0)
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, k_update<-1>, kUpdThreads, smem);
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, k_update<0>, kUpdThreads, smem);
}

cudaError_t update_kernel_attributes(cudaFuncAttributes* fa, size_t smem) {
  cudaError_t e = cudaFuncGetAttributes(fa, k_update<8>);
  if (e != cudaSuccess || smem == 0) return e;
  if ((e = cudaFuncSetAttribute(k_update<8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(k_update<-1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(k_update<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

// ---------------------------------------------------------------------------
// Evaluation output: pred = argmax_j (K_L - 2 popc(A_L[mu] XOR P_L^T[j])),
// lowest j on ties.  One warp per pattern.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_predict_out(const uint64_t* __restrict__ A, int64_t M,
                                                     int nw, const uint64_t* __restrict__ PT,
                                                     int c, int K, int32_t* __restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t mu = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (mu >= M) return;
  const uint64_t* a = A + mu * nw;
  int best = INT_MIN, bestj = 0;
  for (int j = 0; j < c; ++j) {
    const uint64_t* pt = PT + (int64_t)j * nw;
    int cnt = 0;
    for (int w = lane; w < nw; w += 32) cnt += __popcll(a[w] ^ pt[w]);
    cnt = warp_sum(cnt);
    const int v = K - 2 * cnt;
    if (v > best) {
      best = v;
      bestj = j;
    }
  }
  if (lane == 0) out[mu] = bestj;
}

// ---------------------------------------------------------------------------
// Initialisation (Alg. 1 l.2): h_ik = +-1 from Philox purpose 1, stored as the
// lattice index v = (h + h_max)/2 + 2^hb; pad entries get 2^hb (never used;
// their W bits stay 0); W = packed sign(H).  One thread per
// chunk of 8 inputs of one neuron row.
// ---------------------------------------------------------------------------
__global__ void k_init_hw(int16_t* H, uint64_t* W, int Kin, int Kout, int ldh, int nw_in, int l,
                          uint32_t key0, uint32_t key1, int h_max, int hb) {
  const int nch = ldh >> 3;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * nch) return;
  const int k = (int)(idx / nch);
  const int ch = (int)(idx % nch);
  const uint4 r0 = philox4x32_10(make_uint4(2u * ch, (uint32_t)k, (1u << 16) + (uint32_t)l, 0u), key0, key1);
  const uint4 r1 = philox4x32_10(make_uint4(2u * ch + 1u, (uint32_t)k, (1u << 16) + (uint32_t)l, 0u), key0, key1);
  const uint32_t w8[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
  int16_t h[8];
  uint32_t wbyte = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int i = 8 * ch + j;
    const int hv = (w8[j] >> 31) ? 1 : -1;
    h[j] = (int16_t)((i < Kin ? (hv + h_max) / 2 : 0) + (1 << hb));  // lattice index v
    if (i < Kin && hv > 0) wbyte |= 1u << j;
  }
  int4 hv;
  hv.x = (int)(((uint32_t)(uint16_t)h[0]) | ((uint32_t)(uint16_t)h[1] << 16));
  hv.y = (int)(((uint32_t)(uint16_t)h[2]) | ((uint32_t)(uint16_t)h[3] << 16));
  hv.z = (int)(((uint32_t)(uint16_t)h[4]) | ((uint32_t)(uint16_t)h[5] << 16));
  hv.w = (int)(((uint32_t)(uint16_t)h[6]) | ((uint32_t)(uint16_t)h[7] << 16));
  *reinterpret_cast<int4*>(H + (int64_t)k * ldh + 8 * ch) = hv;
  reinterpret_cast<uint8_t*>(W + (int64_t)k * nw_in)[ch] = (uint8_t)wbyte;
}

// rho_kj = +-1 from Philox purpose 2 (Sec. 3.1).
__global__ void k_init_rho(int8_t* rho, int Kout, int c, int l, uint32_t key0, uint32_t key1) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * c) return;
  const int k = (int)(idx / c);
  const int j = (int)(idx % c);
  const uint4 r = philox4x32_10(make_uint4((uint32_t)(j >> 2), (uint32_t)k, (2u << 16) + (uint32_t)l, 0u), key0, key1);
  const uint32_t w = (j & 3) == 0 ? r.x : (j & 3) == 1 ? r.y : (j & 3) == 2 ? r.z : r.w;
  rho[idx] = (w >> 31) ? (int8_t)1 : (int8_t)-1;
}

// PT[j] = packed column j of P_l (bit k%64 of word k/64 = rho_kj > 0).
__global__ void k_pack_pt(const int8_t* rho, uint64_t* PT, int Kout, int c, int nw_out) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)c * nw_out) return;
  const int j = (int)(idx / nw_out);
  const int w = (int)(idx % nw_out);
  uint64_t bits = 0;
  for (int b = 0; b < 64; ++b) {
    const int k = 64 * w + b;
    if (k < Kout && rho[(int64_t)k * c + j] > 0) bits |= 1ull << b;
  }
  PT[idx] = bits;
}

// rhoT[j][k] = rho[k][j].
__global__ void k_transpose_rho(const int8_t* rho, int8_t* rhoT, int Kout, int c) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * c) return;
  const int j = (int)(idx / Kout);
  const int k = (int)(idx % Kout);
  rhoT[idx] = rho[(int64_t)k * c + j];
}

// W = packed sign(H) for one layer (H as lattice indices), pad bits 0.
__global__ void k_repack_w(const int16_t* H, uint64_t* W, int Kin, int Kout, int ldh, int nw_in,
                           int h_max, int hb) {
  const int pos_from = (1 << hb) + (h_max + 1) / 2;  // lattice index of h = +1
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * nw_in) return;
  const int k = (int)(idx / nw_in);
  const int w = (int)(idx % nw_in);
  uint64_t bits = 0;
  for (int b = 0; b < 64; ++b) {
    const int i = 64 * w + b;
    if (i < Kin && H[(int64_t)k * ldh + i] >= pos_from) bits |= 1ull << b;
  }
  W[idx] = bits;
}

}  // namespace bk
