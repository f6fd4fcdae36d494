// kern_binarize.cu -- MedianBinarization of real-valued input patterns
// (Alg. 1 l.5; Sec. 3.2: the median value is the threshold).
//
//   a_i = +1  iff  x_i > m,   m = the ceil(K/2)-th smallest of the pattern's K
//                              values (lower median), compared in fp32
//
// packed as bits (bit i % 64 of word i / 64 = 1 <-> +1, pad bits 0), the input
// format of bmlp_train / bmlp_predict.
//
// One CTA per pattern.  The median is found exactly by a radix select over the
// order-preserving 32-bit image of the floats (key = bits ^ 0x80000000 for a
// clear sign bit, ~bits for a set one): four passes of 8-bit digits, most
// significant first, each a shared-memory histogram of the keys that share the
// digits chosen so far, then one warp scans the 256 counts and picks the
// bucket holding the target rank.  The comparison x_i > m is made on the
// floats, so -0 and +0 compare equal as they do in fp32.  The pattern's row is
// read five times (four passes and the packing); it stays in L1 between them.
#include "bmlp_internal.cuh"

namespace bk {
namespace {

constexpr int kBinThreads = 256;

__device__ __forceinline__ uint32_t float_key(float v) {
  const uint32_t u = __float_as_uint(v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float key_float(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

__global__ void __launch_bounds__(kBinThreads)
    k_binarize_median(const float* __restrict__ x, int64_t n, int K, int nw, uint64_t* __restrict__ out) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t s_prefix, s_rank;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int64_t mu = blockIdx.x; mu < n; mu += gridDim.x) {
    const float* row = x + mu * (int64_t)K;
    uint32_t prefix = 0, mask = 0;
    uint32_t rank = (uint32_t)((K + 1) / 2 - 1);  // 0-based rank of the lower median
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += kBinThreads) hist[i] = 0;
      __syncthreads();
      for (int i = threadIdx.x; i < K; i += kBinThreads) {
        const uint32_t key = float_key(row[i]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 0xFFu], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        // lane j owns buckets 8j .. 8j + 7; an inclusive scan of the lane sums
        // finds the lane whose buckets hold the rank, then that lane walks them
        uint32_t c[8], sum = 0;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
          c[b] = hist[8 * lane + b];
          sum += c[b];
        }
        uint32_t incl = sum;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
          const uint32_t v = __shfl_up_sync(0xffffffffu, incl, d);
          if (lane >= d) incl += v;
        }
        const uint32_t excl = incl - sum;
        if (excl <= rank && rank < incl) {
          uint32_t below = excl;
          int b = 0;
          while (below + c[b] <= rank) below += c[b++];
          s_prefix = prefix | ((uint32_t)(8 * lane + b) << shift);
          s_rank = rank - below;
        }
      }
      __syncthreads();
      prefix = s_prefix;
      rank = s_rank;
      mask |= 0xFFu << shift;
    }
    const float m = key_float(prefix);
    uint32_t* o = reinterpret_cast<uint32_t*>(out + mu * (int64_t)nw);
    for (int w = warp; w < 2 * nw; w += kBinThreads / 32) {
      const int i = 32 * w + lane;
      const unsigned bits = __ballot_sync(0xffffffffu, i < K && row[i] > m);
      if (lane == 0) o[w] = bits;
    }
    __syncthreads();  // hist, s_prefix and s_rank are reused by the next pattern
  }
}

}  // namespace

void launch_binarize_median(const float* x, int64_t n, int K, int nw, uint64_t* out,
                            cudaStream_t st) {
  const int64_t grid = n < (int64_t)1 << 20 ? n : (int64_t)1 << 20;
  k_binarize_median<<<(unsigned)grid, kBinThreads, 0, st>>>(x, n, K, nw, out);
}

}  // namespace bk
