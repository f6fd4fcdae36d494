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
// Launched as a programmatic dependent of the last layer's forward pass: the
// CTAs of layers l < L read only what kernels two or more launches back wrote
// (their layer's Z and A, the batch index), so they do all their work before
// waiting, overlapping that forward pass; the CTAs of layer L wait first.
// Every CTA waits before it lets the next kernel start, so a kernel two
// launches back has always completed.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cls_select_body(const StepParams* __restrict__ P, int li, int mu);

__global__ void __launch_bounds__(kClsThreads) k_cls_select(const StepParams* __restrict__ P) {
  const int li = blockIdx.y;
  const int mu = blockIdx.x;
  const bool early = li < P->L - 1;
  if (!early) pdl_wait();
  cls_select_body(P, li, mu);
  if (early) pdl_wait();
  pdl_trigger();
}

__device__ __forceinline__ void cls_select_body(const StepParams* __restrict__ P, int li, int mu) {
  const DevLayer& Ly = P->layer[li];
  Ctrl* ctrl = P->ctrl;
  const int64_t start = batch_start(P);
  const int64_t bsz = batch_size(P, start);
  if (mu >= bsz) return;
  __shared__ int yh[BMLP_MAX_CLASSES];
  __shared__ int s_mark, s_y, s_timeout;
  // one read of the counter for the whole CTA (the last forward pass may be
  // running beside an early CTA and could raise it meanwhile)
  if (threadIdx.x == 0) s_timeout = ctrl->timeouts != 0u;
  __syncthreads();
  if (s_timeout) {
    // a bounded wait of this step's forward pass expired (or an earlier one
    // is not yet reported): Z and A are not valid, so the pattern is marked
    // for nothing; with every mark 0 the update leaves H and W as they are
    // and only advances the step counters (the update kernel also skips the
    // step on its own reading of the counter)
    if (threadIdx.x == 0) Ly.mark[mu] = 0;
    return;
  }
  const int c = P->c;
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

namespace {

using namespace upd;

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
// Initialisation (Alg. 1 l.2): h_ik = +-1 from Philox purpose 1, stored
// bit-sliced (DevLayer::H) as the lattice index u = (h + h_max)/2, i.e.
// (h_max + 1)/2 for +1 and (h_max - 1)/2 for -1; inputs i >= K_in keep u = 0
// and W bit 0; W = packed sign(H).  One thread per group of 32 inputs of one
// neuron row; H and W are zeroed beforehand (row padding).
// ---------------------------------------------------------------------------
__global__ void k_init_hw(uint32_t* H, uint64_t* W, int Kin, int Kout, int ldh, int ngrp, int nplanes,
                          int l, uint32_t key0, uint32_t key1, int h_max) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * ngrp) return;
  const int k = (int)(idx / ngrp);
  const int g = (int)(idx % ngrp);
  uint32_t pos = 0u;   // bit j: h of input 32 g + j is +1
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const uint4 r = philox4x32_10(make_uint4(8u * g + q, (uint32_t)k, (1u << 16) + (uint32_t)l, 0u), key0, key1);
    pos |= ((r.x >> 31) << (4 * q)) | ((r.y >> 31) << (4 * q + 1)) | ((r.z >> 31) << (4 * q + 2)) |
           ((r.w >> 31) << (4 * q + 3));
  }
  const uint32_t valid = upd::group_mask(g, Kin);
  pos &= valid;
  const int up = (h_max + 1) / 2, dn = up - 1;   // u of h = +1, h = -1
  uint32_t* hg = H + (int64_t)k * ldh + (int64_t)g * nplanes;
  for (int p = 0; p < nplanes; ++p) {
    const uint32_t m1 = ((up >> p) & 1) ? upd::kFull : 0u, m0 = ((dn >> p) & 1) ? upd::kFull : 0u;
    hg[p] = ((pos & m1) | (~pos & m0)) & valid;
  }
  reinterpret_cast<uint32_t*>(W + (int64_t)k * ((ngrp + 1) / 2))[g] = pos;
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

// W = packed sign(H) for one layer (H bit-sliced), pad bits 0: per group of
// 32 inputs, the lanes with u >= (h_max + 1)/2.  One thread per group.
__global__ void k_repack_w(const uint32_t* H, uint64_t* W, int Kin, int Kout, int ldh, int ngrp,
                           int nplanes, int h_max) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * ngrp) return;
  const int k = (int)(idx / ngrp);
  const int g = (int)(idx % ngrp);
  const int m = (h_max + 1) / 2;
  const uint32_t* hg = H + (int64_t)k * ldh + (int64_t)g * nplanes;
  uint32_t gt = 0u, eq = upd::kFull;
  for (int p = nplanes - 1; p >= 0; --p) {
    const uint32_t mp = ((m >> p) & 1) ? upd::kFull : 0u;
    gt |= eq & hg[p] & ~mp;
    eq &= ~(hg[p] ^ mp);
  }
  reinterpret_cast<uint32_t*>(W + (int64_t)k * ((ngrp + 1) / 2))[g] = (gt | eq) & upd::group_mask(g, Kin);
}

}  // namespace bk
