// kern_update.cu -- local classifiers, selection and the hidden-weight update of
// the BMLP training rule (arXiv 2412.00119, Alg. 1 l.10-18, Alg. 2, Alg. 3), plus
// initialisation and the evaluation output.
#include <climits>

#include "bmlp_internal.cuh"

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
  const int64_t start = batch_start(P);
  const int64_t bsz = batch_size(P, start);
  if (mu >= bsz) return;
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
    if (li == P->L - 1 && loss) atomicAdd(&ctrl->err, 1ull);
    s_mark = mark;
    s_y = yv;
  }
  __syncthreads();

  int16_t* sel = Ly.sel + (int64_t)mu * Ly.G;
  if (!s_mark) {
    for (int g = threadIdx.x; g < Ly.G; g += blockDim.x) sel[g] = -1;
    return;
  }
  const int y = s_y;
  const int16_t* z = Ly.Z + (int64_t)mu * Ly.Kout;
  const int gamma = Ly.gamma;
  for (int g = warp; g < Ly.G; g += nwarps) {
    int bestd = INT_MIN, bestk = INT_MAX;
    for (int kk = lane; kk < gamma; kk += 32) {
      const int k = g * gamma + kk;
      const int d = (int)z[k] * (int)Ly.rho[(int64_t)k * c + y];
      if (d < 0 && d > bestd) {  // ascending k per lane: strict '>' keeps the lowest
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
    if (lane == 0) sel[g] = (bestd == INT_MIN) ? (int16_t)-1 : (int16_t)bestk;
  }
}

// ---------------------------------------------------------------------------
// Hidden-weight update, fused with the visible-weight repack (Alg. 3, Sec. 3.1).
// CTA = (layer, group g, slice of kUpdRowsPerCta neurons).  A warp owns one
// neuron row k at a time: it collects, in ascending mu, the patterns whose
// selection in group g is k (the CP tuples of k), then streams the row in
// chunks of 8 hidden weights (one 16-byte vector per lane, kUpdUnroll vectors
// in flight per lane):
//   CP: h_i <- clip(h_i + 2 a^mu_i rho_{k,y^mu}) per tuple, in mu order.  The
//       8 weights stay packed as int16 pairs; a shared table turns the
//       activation byte into four packed +-2 delta words and the DPX
//       add-min / max3 instructions clip two weights per instruction.
//   R : U = Philox draw (hi16 lane from purpose 3, lo16 from purpose 4);
//       U < T  ->  h_i <- clip(h_i + 2 sign h_i).  The 16-bit lanes of the
//       Philox output line up with the int16 pairs; a SIMD-within-a-register
//       test against T's high half finds the chunks with an event or a tie
//       (about 4% of chunks at the paper's p_r), and only those take the
//       per-weight path; the low half is drawn only on a tie.
//   W : bit i = (h_i > 0) = NOT sign bit; one byte per chunk, in place.
// Chunks that hold only padding (i >= K_{l-1}) are never touched; a chunk that
// is partly padding takes the per-weight path with the padding masked.
// Layers with an empty M_l are skipped (no CP, no R).  The last CTA to finish
// advances the step counters and clears the per-step flags.
// ---------------------------------------------------------------------------
namespace {

struct UpdCtx {
  const uint8_t* aprev;  // previous layer's packed activations, bytes
  size_t arow_bytes;
  const int32_t* list;   // CP tuples of the row: mu | (rho < 0) << 16
  int n_t;
  int h_max;
  uint32_t Thi, Tlo, Tpair;
  bool fast_r;           // Thi < 2^15: the SIMD test is exact
  uint32_t key0, key1;
  uint32_t k, c2_hi, c2_lo, t;
  const uint4* delta;    // [2][256] packed +-2 deltas per activation byte and rho sign
};

__device__ __forceinline__ int lane_h(const uint32_t (&w)[4], int j) {
  return (int)(int16_t)(uint16_t)(w[j >> 1] >> (16 * (j & 1)));
}

__device__ __forceinline__ void set_lane_h(uint32_t (&w)[4], int j, int h) {
  const int sh = 16 * (j & 1);
  w[j >> 1] = (w[j >> 1] & ~(0xFFFFu << sh)) | (((uint32_t)h & 0xFFFFu) << sh);
}

// Per-weight path: CP (already applied by the caller when `cp_done`), R and W
// for the first `nvalid` weights of the chunk.
__device__ __noinline__ uint32_t chunk_scalar(uint32_t (&w)[4], int ch, int nvalid, bool cp_done,
                                              const UpdCtx& C, uint4 rh) {
  if (!cp_done) {
    for (int q = 0; q < C.n_t; ++q) {
      const int e = C.list[q];
      const int m = e & 0xFFFF;
      const int rho = (e & 0x10000) ? -1 : 1;
      const uint32_t byte = C.aprev[(size_t)m * C.arow_bytes + ch];
      for (int j = 0; j < nvalid; ++j) {
        const int step = ((byte >> j) & 1u) ? rho : -rho;
        set_lane_h(w, j, clip_h(lane_h(w, j) + 2 * step, C.h_max));
      }
    }
  }
  uint32_t ties = 0;
  for (int j = 0; j < 8; ++j) ties |= (lane16(rh, j) == C.Thi ? 1u : 0u) << j;
  uint4 rl = make_uint4(0, 0, 0, 0);
  if (ties)
    rl = philox4x32_10(make_uint4((uint32_t)ch, C.k, C.c2_lo, C.t), C.key0, C.key1);
  uint32_t wbyte = 0;
  for (int j = 0; j < nvalid; ++j) {
    const uint32_t u = lane16(rh, j);
    const bool fire = (u < C.Thi) || (((ties >> j) & 1u) && lane16(rl, j) < C.Tlo);
    int h = lane_h(w, j);
    if (fire) {
      h = clip_h(h + (h > 0 ? 2 : -2), C.h_max);
      set_lane_h(w, j, h);
    }
    wbyte |= (h > 0 ? 1u : 0u) << j;
  }
  return wbyte;
}

// Sign bits of the 8 packed weights -> W byte (bit j = h_j > 0, h never 0).
__device__ __forceinline__ uint32_t w_byte(const uint32_t (&w)[4]) {
  const uint32_t p0 = __byte_perm(w[0], w[1], 0x7531) & 0x80808080u;
  const uint32_t p1 = __byte_perm(w[2], w[3], 0x7531) & 0x80808080u;
  const uint32_t neg = ((p0 * 0x00204081u) >> 28) | (((p1 * 0x00204081u) >> 28) << 4);
  return ~neg & 0xFFu;
}

__device__ __forceinline__ uint32_t chunk_packed(uint32_t (&w)[4], int ch, const UpdCtx& C,
                                                 uint32_t neg_pair, uint32_t pos_pair) {
  // Clipped Perceptron, two weights per DPX instruction
  for (int q = 0; q < C.n_t; ++q) {
    const int e = C.list[q];
    const int m = e & 0xFFFF;
    const uint32_t byte = C.aprev[(size_t)m * C.arow_bytes + ch];
    const uint4 d = C.delta[((e >> 16) & 1) * 256 + byte];
    w[0] = __vimax3_s16x2(__viaddmin_s16x2(w[0], d.x, pos_pair), neg_pair, neg_pair);
    w[1] = __vimax3_s16x2(__viaddmin_s16x2(w[1], d.y, pos_pair), neg_pair, neg_pair);
    w[2] = __vimax3_s16x2(__viaddmin_s16x2(w[2], d.z, pos_pair), neg_pair, neg_pair);
    w[3] = __vimax3_s16x2(__viaddmin_s16x2(w[3], d.w, pos_pair), neg_pair, neg_pair);
  }
  // Reinforcement draws for the 8 weights
  const uint4 rh = philox4x32_10(make_uint4((uint32_t)ch, C.k, C.c2_hi, C.t), C.key0, C.key1);
  uint32_t any = 1;
  if (C.fast_r) {
    // lane fires iff its 16-bit draw u < Thi (< 2^15): top bit clear and low 15
    // bits below Thi; lane ties iff u == Thi (zero lane of u ^ Tpair)
    const uint32_t H = 0x80008000u;
    const uint32_t u[4] = {rh.x, rh.y, rh.z, rh.w};
    any = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t d = ((u[i] & 0x7FFF7FFFu) | H) - C.Tpair;
      const uint32_t x = u[i] ^ C.Tpair;
      any |= (~(d | u[i]) & H) | ((x - 0x00010001u) & ~x & H);
    }
  }
  if (any) return chunk_scalar(w, ch, 8, true, C, rh);
  return w_byte(w);
}

}  // namespace

__global__ void __launch_bounds__(kUpdThreads, 3) k_update(const StepParams* __restrict__ P) {
  extern __shared__ int32_t dyn[];
  __shared__ uint4 s_delta[2 * 256];
  const int bid = blockIdx.x;
  int li = 0;
  while (li + 1 < P->L && bid >= P->layer[li + 1].upd_cta_base) ++li;
  const DevLayer& Ly = P->layer[li];
  Ctrl* ctrl = P->ctrl;
  const unsigned long long t = ctrl->t;
  const uint32_t s = ctrl->s;
  const bool active = ctrl->any_mark[li] != 0u;

  if (active) {
    const int gamma = Ly.gamma;
    const int slices = (gamma + kUpdRowsPerCta - 1) / kUpdRowsPerCta;
    const int local = bid - Ly.upd_cta_base;
    const int g = local / slices;
    const int r0 = (local % slices) * kUpdRowsPerCta;
    const int r1 = min(r0 + kUpdRowsPerCta, gamma);
    const int64_t start = (int64_t)s * P->bs;
    const int bsz = (int)batch_size(P, start);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    int16_t* s_sel = reinterpret_cast<int16_t*>(dyn);               // [bs]
    int32_t* s_list = dyn + (P->bs + 1) / 2 + warp * P->bs;         // [nwarps][bs]

    for (int m = threadIdx.x; m < bsz; m += blockDim.x) s_sel[m] = Ly.sel[(int64_t)m * Ly.G + g];
    // s_delta[r][b]: packed int16 pair p of entry = (+-2 for bit 2p, +-2 for
    // bit 2p+1 of b), sign flipped for r = 1 (rho = -1)
    for (int i = threadIdx.x; i < 512; i += blockDim.x) {
      const int r = i >> 8, b = i & 255;
      uint32_t v[4];
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        int lo = ((b >> (2 * p)) & 1) ? 2 : -2;
        int hi = ((b >> (2 * p + 1)) & 1) ? 2 : -2;
        if (r) { lo = -lo; hi = -hi; }
        v[p] = ((uint32_t)lo & 0xFFFFu) | ((uint32_t)hi << 16);
      }
      s_delta[i] = make_uint4(v[0], v[1], v[2], v[3]);
    }
    __syncthreads();

    const int l = li + 1;
    const int c = P->c;
    UpdCtx C;
    C.h_max = P->h_max;
    const unsigned long long T = P->T[li];
    C.Thi = (uint32_t)(T >> 16);   // 0..65536
    C.Tlo = (uint32_t)(T & 0xFFFFu);
    C.fast_r = C.Thi < 0x8000u;
    C.Tpair = C.Thi * 0x00010001u;
    C.key0 = P->key0;
    C.key1 = P->key1;
    C.c2_hi = (3u << 16) + (uint32_t)l;
    C.c2_lo = (4u << 16) + (uint32_t)l;
    C.t = (uint32_t)t;
    C.delta = s_delta;
    const int Kin = Ly.Kin;
    const int nch = (Kin + 7) >> 3;             // chunks holding at least one input
    const int full = Kin >> 3;                  // chunks of 8 real inputs
    C.arow_bytes = (size_t)Ly.nw_in * 8;
    C.aprev = (li == 0) ? reinterpret_cast<const uint8_t*>(P->x + start * P->nw0)
                        : reinterpret_cast<const uint8_t*>(P->layer[li - 1].A);
    const uint32_t neg_pair = (uint32_t)(-C.h_max & 0xFFFF) * 0x00010001u;
    const uint32_t pos_pair = (uint32_t)C.h_max * 0x00010001u;

    for (int rr = r0 + warp; rr < r1; rr += nwarps) {
      const int k = g * gamma + rr;
      // CP tuples of neuron k, ascending mu
      int n_t = 0;
      for (int base = 0; base < bsz; base += 32) {
        const int m = base + lane;
        const bool hit = (m < bsz) && (s_sel[m] == k);
        const unsigned bal = __ballot_sync(0xffffffffu, hit);
        if (hit) {
          int yv = P->y[start + m];
          if (yv < 0 || yv >= c) yv = 0;
          const int rho = Ly.rho[(int64_t)k * c + yv];
          s_list[n_t + __popc(bal & ((1u << lane) - 1u))] = m | ((rho > 0) ? 0 : 0x10000);
        }
        n_t += __popc(bal);
      }
      __syncwarp();
      C.list = s_list;
      C.n_t = n_t;
      C.k = (uint32_t)k;

      int16_t* hrow = Ly.H + (int64_t)k * Ly.ldh;
      uint8_t* wrow = reinterpret_cast<uint8_t*>(Ly.W + (int64_t)k * Ly.nw_in);
      // kUpdUnroll 16-byte loads in flight per lane before any is processed;
      // H is streamed (read once, written once per step)
      for (int base = lane; base < nch; base += 32 * kUpdUnroll) {
        uint4 hbuf[kUpdUnroll];
#pragma unroll
        for (int u = 0; u < kUpdUnroll; ++u) {
          const int ch = base + 32 * u;
          if (ch < nch) hbuf[u] = __ldcs(reinterpret_cast<const uint4*>(hrow + 8 * ch));
        }
#pragma unroll
        for (int u = 0; u < kUpdUnroll; ++u) {
          const int ch = base + 32 * u;
          if (ch >= nch) break;
          uint32_t w[4] = {hbuf[u].x, hbuf[u].y, hbuf[u].z, hbuf[u].w};
          uint32_t wbyte;
          if (ch < full) {
            wbyte = chunk_packed(w, ch, C, neg_pair, pos_pair);
          } else {
            const uint4 rh = philox4x32_10(make_uint4((uint32_t)ch, C.k, C.c2_hi, C.t), C.key0, C.key1);
            wbyte = chunk_scalar(w, ch, Kin - 8 * ch, false, C, rh);
          }
          __stcs(reinterpret_cast<uint4*>(hrow + 8 * ch), make_uint4(w[0], w[1], w[2], w[3]));
          wrow[ch] = (uint8_t)wbyte;
        }
      }
      __syncwarp();
    }
  }

  // step completion: the last CTA advances the counters
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned prev = atomicAdd(&ctrl->done, 1u);
    if (prev == gridDim.x - 1) {
      ctrl->t = t + 1;
      ctrl->s = s + 1;
      for (int i = 0; i < P->L; ++i) ctrl->any_mark[i] = 0u;
      ctrl->done = 0u;
      __threadfence();
    }
  }
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
// Initialisation (Alg. 1 l.2): h_ik = +-1 from Philox purpose 1, pad entries
// -1 (never used; their W bits stay 0); W = packed sign(H).  One thread per
// chunk of 8 inputs of one neuron row.
// ---------------------------------------------------------------------------
__global__ void k_init_hw(int16_t* H, uint64_t* W, int Kin, int Kout, int ldh, int nw_in, int l,
                          uint32_t key0, uint32_t key1) {
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
    h[j] = (i < Kin) ? ((w8[j] >> 31) ? (int16_t)1 : (int16_t)-1) : (int16_t)-1;
    if (i < Kin && h[j] > 0) wbyte |= 1u << j;
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

// W = packed sign(H) for one layer, pad bits 0.
__global__ void k_repack_w(const int16_t* H, uint64_t* W, int Kin, int Kout, int ldh, int nw_in) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)Kout * nw_in) return;
  const int k = (int)(idx / nw_in);
  const int w = (int)(idx % nw_in);
  uint64_t bits = 0;
  for (int b = 0; b < 64; ++b) {
    const int i = 64 * w + b;
    if (i < Kin && H[(int64_t)k * ldh + i] > 0) bits |= 1ull << b;
  }
  W[idx] = bits;
}

}  // namespace bk
