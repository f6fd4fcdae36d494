// kern_expand.cu -- fixed random expansion layer for integer-valued inputs
// (Sec. 3.2, footnote to the binarisation step: a fixed random input layer
// with weights in {+-1} and sign activation lets the BMLP take non-binary
// inputs directly).
//
//   a_mu,k = +1  iff  z = sum_i x[mu][i] e_k,i >= 0    (sign(0) = +1)
//
// x: unsigned 8-bit inputs (pixel intensities); e_k,i: bit i of row k of the
// packed expansion matrix E (1 <-> +1).  z is summed exactly in int32
// (|z| <= 255 D < 2^31).  The output is packed like every activation (bit
// k % 64 of word k / 64, pad bits 0), i.e. bmlp_train / bmlp_predict input
// for K_0 = K.
//
// k_expand_sign: a 128-pattern x 128-neuron tile per CTA of 256 threads, the
// inputs in chunks of 64 (one word of E per neuron): the chunk's bytes of x
// and the chunk's E bits, expanded to +-1 bytes, are staged in shared memory
// (rows padded to 17 words: conflict-free reads; the next chunk's raw words
// are already in flight in registers), then thread (tx, ty) runs
// dp4a.u32.s32 for patterns ty + 16 i and neurons tx + 16 j, i, j < 8 (64
// int32 sums).  Each warp ballots the signs of 2 patterns x 16 neurons and
// writes 16-bit pieces of the packed rows.  Neuron tiles vary fastest in the
// grid, so the CTAs of one pattern tile run together and read x from L2.
// Why CUDA cores and not tcgen05: e4m3 holds no byte exactly, the int8 tensor
// rate of this part is far below its fp8 rate, and the transform runs once per
// data set, not once per training step.
//
// k_expand_weights: E from the Philox stream of the expansion weights,
// e_k,i = +1 iff bit 31 of word i%4 of Philox (i/4, k, 33*2^16, 0) (the
// library's stream layout is listed in bmlp_internal.cuh); pad bits 0.
#include "bmlp_internal.cuh"

namespace bk {
namespace {

constexpr int kXThreads = 256;
constexpr int kXM = 128;         // patterns per CTA
constexpr int kXN = 128;         // neurons per CTA
constexpr int kXLd = 64 / 4 + 1; // 32-bit words per staged row (64 inputs + pad)
constexpr int kXMaxRowTiles = 65535;

__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
  int d;
  asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

__global__ void __launch_bounds__(kXThreads, 2)
    k_expand_sign(const uint8_t* __restrict__ x, int64_t n, int D, bool vec,
                  const uint64_t* __restrict__ E, int K, int nwD, uint64_t* __restrict__ out,
                  int nwK) {
  __shared__ uint32_t xs[kXM][kXLd];
  __shared__ uint32_t es[kXN][kXLd];
  const int n0 = blockIdx.x * kXN;
  const int64_t m0 = (int64_t)blockIdx.y * kXM;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  int acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0;

  // thread t stages words q = t + 256 v (v < 8) of the x tile -- staged row
  // q / 16, word q % 16 = inputs 4 (q % 16) .. + 3 of the chunk, byte b = input
  // 4 (q % 16) + b, 0 past D and past n -- and half t & 1 of the E word of
  // neuron n0 + t / 2.  The raw words of chunk kc + 1 are loaded into
  // registers before chunk kc is computed, so the loads overlap the dp4a work.
  uint32_t xr[8], er;
  auto load_chunk = [&](int kc) {
    const int i0 = 64 * kc;
#pragma unroll
    for (int v = 0; v < 8; ++v) {
      const int q = threadIdx.x + kXThreads * v;
      const int r = q >> 4, c4 = q & 15;
      const int64_t m = m0 + r;
      const int i = i0 + 4 * c4;
      uint32_t w = 0;
      if (m < n) {
        const uint8_t* row = x + m * (int64_t)D;
        if (vec && i + 4 <= D) {
          w = __ldg(reinterpret_cast<const uint32_t*>(row + i));
        } else {
#pragma unroll
          for (int b = 0; b < 4; ++b)
            if (i + b < D) w |= (uint32_t)__ldg(row + i + b) << (8 * b);
        }
      }
      xr[v] = w;
    }
    const int k = n0 + (threadIdx.x >> 1);
    er = k < K ? (uint32_t)(E[(int64_t)k * nwD + kc] >> (32 * (threadIdx.x & 1))) : 0u;
  };
  load_chunk(0);

#pragma unroll 1
  for (int kc = 0; kc < nwD; ++kc) {
#pragma unroll
    for (int v = 0; v < 8; ++v) {
      const int q = threadIdx.x + kXThreads * v;
      xs[q >> 4][q & 15] = xr[v];
    }
    {
      // E half -> eight words of +-1 bytes (0x01 / 0xFF); neurons past K
      // stage zeros
      const int r = threadIdx.x >> 1, h = threadIdx.x & 1;
      const bool live = n0 + r < K;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        // nibble -> one bit per byte (the shifted copies do not overlap)
        const uint32_t p = (((er >> (4 * q)) & 0xFu) * 0x00204081u) & 0x01010101u;
        es[r][8 * h + q] = live ? ~(p * 0xFEu) : 0u;
      }
    }
    __syncthreads();
    if (kc + 1 < nwD) load_chunk(kc + 1);
#pragma unroll 4
    for (int c4 = 0; c4 < 16; ++c4) {
      uint32_t a[8], b[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) a[i] = xs[ty + 16 * i][c4];
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = es[tx + 16 * j][c4];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = dp4a_us(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }

  // lanes 0..15 hold pattern ty = 2 warp, lanes 16..31 pattern ty = 2 warp + 1,
  // lane tx neuron n0 + tx + 16 j: each half of the ballot is 16 consecutive
  // neurons of one pattern
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t m = m0 + ty + 16 * i;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int nn = n0 + tx + 16 * j;
      const unsigned bits = __ballot_sync(0xffffffffu, nn < K && acc[i][j] >= 0);
      const int piece = (n0 + 16 * j) >> 4;   // 16-bit piece of the packed row
      if ((lane & 15) == 0 && m < n && piece < 4 * nwK)
        reinterpret_cast<uint16_t*>(out + m * (int64_t)nwK)[piece] = (uint16_t)(bits >> (lane & 16));
    }
  }
}

__global__ void k_expand_weights(uint32_t key0, uint32_t key1, int K, int D, int nwD,
                                 uint64_t* __restrict__ E) {
  const int64_t total = (int64_t)K * nwD;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int k = (int)(idx / nwD), w = (int)(idx % nwD);
    uint64_t word = 0;
#pragma unroll 1
    for (int g = 0; g < 16; ++g) {  // inputs 64 w + 4 g .. + 3: one Philox call
      const int i = 64 * w + 4 * g;
      if (i >= D) break;
      const uint4 u = philox4x32_10(make_uint4((uint32_t)(i / 4), (uint32_t)k, 33u << 16, 0u), key0, key1);
      const uint64_t s = (u.x >> 31) | ((u.y >> 31) << 1) | ((u.z >> 31) << 2) | ((u.w >> 31) << 3);
      word |= s << (4 * g);
    }
    const int valid = D - 64 * w;
    if (valid < 64) word &= (1ull << valid) - 1ull;
    E[idx] = word;
  }
}

}  // namespace

void launch_expand_weights(uint64_t seed, int K, int D, uint64_t* E, cudaStream_t st) {
  const int nwD = (D + 63) / 64;
  const int64_t total = (int64_t)K * nwD;
  const int64_t blocks = (total + 255) / 256;
  k_expand_weights<<<(unsigned)(blocks < 4096 ? blocks : 4096), 256, 0, st>>>(
      (uint32_t)(seed & 0xFFFFFFFFu), (uint32_t)(seed >> 32), K, D, nwD, E);
}

void launch_expand_sign(const uint8_t* x, int64_t n, int D, const uint64_t* E, int K, uint64_t* out,
                        cudaStream_t st) {
  const int nwD = (D + 63) / 64, nwK = (K + 63) / 64;
  const unsigned ntiles = (unsigned)((K + kXN - 1) / kXN);
  // patterns in launches of at most 65,535 tiles of 128 (the grid's y limit)
  const int64_t per = (int64_t)kXMaxRowTiles * kXM;
  for (int64_t off = 0; off < n; off += per) {
    const int64_t cnt = (n - off < per) ? n - off : per;
    const uint8_t* xo = x + off * (int64_t)D;
    const bool vec = (D % 4 == 0) && (reinterpret_cast<uintptr_t>(xo) % 4 == 0);
    const dim3 grid(ntiles, (unsigned)((cnt + kXM - 1) / kXM));
    k_expand_sign<<<grid, kXThreads, 0, st>>>(xo, cnt, D, vec, E, K, nwD, out + off * (int64_t)nwK, nwK);
  }
}

}  // namespace bk
