// kern_forward_b1.cu -- the forward contraction of one layer (Alg. 1 l.8-9)
// on the legacy binary tensor-core path, mma.sync.m16n8k256 .b1 xor.popc:
//
//   z^mu_k = K_in - 2 popc(a^mu XOR w_k),   a^mu_k = (z^mu_k >= 0)
//
// computed straight from the packed bits (pad bits are 0 in both operands, so
// their XOR adds nothing).  Kept for the engine comparison (bmlp_engine_peak,
// bmlp_layer_forward_engine): no expansion of bits to bytes is needed, unlike
// the e4m3 tcgen05 path.
//
// Roles: the MMA's 16-row A operand is 16 neurons (rows of W, K-contiguous
// bits, "row" layout) and its 8-column B operand 8 patterns (rows of the
// activation matrix, K-contiguous bits = "col" layout); D[neuron][pattern] is
// the popcount of the XOR.
//
// Tiling: a CTA of 4 warps owns 64 neurons (one packed output word per
// pattern) and 8 NT patterns; a warp owns 16 neurons x NT n-tiles of 8
// patterns.  K advances in supersteps of 512 bits (two MMAs).  Because the
// contraction sums over k, the same permutation of k on both operands leaves
// z unchanged, so thread (g, t) of a warp (g = lane / 4, t = lane % 4) loads
// 16 contiguous bytes -- 32-bit words 4t .. 4t+3 of the superstep -- of its
// neuron rows g and g + 8 straight from global memory into registers, and
// 16 bytes of its pattern row g of each n-tile from shared memory, and feeds
// words (4t, 4t+1) to the first MMA and (4t+2, 4t+3) to the second in the
// register slots the fragment layout assigns to k = 32t.. and 128 + 32t..
// The weights are read once; the activation rows of the CTA are staged in
// shared memory in K chunks of 1024 bits (3-stage cp.async ring), each
// 128-byte row with its 16-byte pieces XOR-swizzled by 4 (row & 1) so that the
// 16-byte fragment reads of two neighbouring rows hit disjoint banks.
#include "bmlp_internal.cuh"

namespace bk {
namespace {

constexpr int kB1Warps = 4;
constexpr int kB1Threads = 32 * kB1Warps;
constexpr int kB1Stages = 3;
constexpr int kB1RowBytes = 128;  // one K chunk of a pattern row (1024 bits)

__device__ __forceinline__ void cp16(void* smem, const void* gmem, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;"
               ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))), "l"(gmem),
               "r"(src_bytes) : "memory");
}

__device__ __forceinline__ void cp8(void* smem, const void* gmem, int src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;"
               ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))), "l"(gmem),
               "r"(src_bytes) : "memory");
}

__device__ __forceinline__ void mma_b1(int (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                       uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.xor.popc {%0,%1,%2,%3}, "
      "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <int NT>
__global__ void __launch_bounds__(kB1Threads) k_forward_b1(const uint64_t* __restrict__ A, int64_t M,
                                                           int nw_in, const uint64_t* __restrict__ W,
                                                           int N, int Kin, uint64_t* __restrict__ Aout,
                                                           int nw_out) {
  constexpr int PT = 8 * NT;
  extern __shared__ __align__(16) uint8_t sb[];   // [kB1Stages][PT][128] then [PT][4] uint16
  uint16_t* s_out = reinterpret_cast<uint16_t*>(sb + kB1Stages * PT * kB1RowBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int nblk = blockIdx.x;                  // 64 neurons: output word nblk
  const int n0 = 64 * nblk + 16 * warp;         // this warp's 16 neurons
  const int64_t m0 = (int64_t)blockIdx.y * PT;  // first pattern of the CTA
  const int nss = (nw_in + 7) >> 3;             // supersteps of 512 bits
  const int nch = (nss + 1) >> 1;               // K chunks of 1024 bits
  const bool avec = (nw_in % 2 == 0) && (reinterpret_cast<uintptr_t>(A) % 16 == 0);
  const bool wvec = (nw_in % 2 == 0) && (reinterpret_cast<uintptr_t>(W) % 16 == 0);

  // ---- activation chunks -> shared memory (zero past M and past nw_in) ----
  auto stage_chunk = [&](int c) {
    uint8_t* dst0 = sb + (c % kB1Stages) * PT * kB1RowBytes;
    for (int i = threadIdx.x; i < PT * 8; i += kB1Threads) {
      const int r = i >> 3, p = i & 7;            // row, 16-byte piece (two words)
      const int w = 16 * c + 2 * p;               // first 64-bit word of the piece
      uint8_t* dst = dst0 + r * kB1RowBytes + 16 * (p ^ (4 * (r & 1)));
      const bool rv = m0 + r < M;
      const uint64_t* src = A + (rv ? (m0 + r) * (int64_t)nw_in : 0) + (w < nw_in ? w : 0);
      const int nwv = rv ? max(0, min(2, nw_in - w)) : 0;  // valid words of the piece
      if (avec) {
        cp16(dst, src, 8 * nwv);
      } else {
        cp8(dst, src, nwv >= 1 ? 8 : 0);
        cp8(dst + 8, nwv >= 2 ? src + 1 : src, nwv >= 2 ? 8 : 0);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  // ---- weight rows g and g + 8 of the warp's 16 neurons ----
  const uint32_t* wr0 = (n0 + g < N) ? reinterpret_cast<const uint32_t*>(W + (int64_t)(n0 + g) * nw_in)
                                     : nullptr;
  const uint32_t* wr1 = (n0 + g + 8 < N)
                            ? reinterpret_cast<const uint32_t*>(W + (int64_t)(n0 + g + 8) * nw_in)
                            : nullptr;
  const int nw32 = 2 * nw_in;
  auto load_w = [&](const uint32_t* r, int ss) -> uint4 {
    const int w = 16 * ss + 4 * t;
    if (r == nullptr || w >= nw32) return make_uint4(0, 0, 0, 0);
    if (wvec) return __ldg(reinterpret_cast<const uint4*>(r + w));
    uint4 v;
    v.x = __ldg(r + w);
    v.y = w + 1 < nw32 ? __ldg(r + w + 1) : 0u;
    v.z = w + 2 < nw32 ? __ldg(r + w + 2) : 0u;
    v.w = w + 3 < nw32 ? __ldg(r + w + 3) : 0u;
    return v;
  };

  int acc[NT][4];
#pragma unroll
  for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0;

#pragma unroll
  for (int c = 0; c < kB1Stages - 1; ++c)
    if (c < nch) stage_chunk(c);
    else asm volatile("cp.async.commit_group;" ::: "memory");
  uint4 wa = load_w(wr0, 0), wb = load_w(wr1, 0);

#pragma unroll 1
  for (int c = 0; c < nch; ++c) {
    asm volatile("cp.async.wait_group %0;" ::"n"(kB1Stages - 2) : "memory");
    __syncthreads();   // chunk c visible to all; chunk c - 1's slot is free
    if (c + kB1Stages - 1 < nch) stage_chunk(c + kB1Stages - 1);
    else asm volatile("cp.async.commit_group;" ::: "memory");
    const uint8_t* sc = sb + (c % kB1Stages) * PT * kB1RowBytes;
#pragma unroll
    for (int sub = 0; sub < 2; ++sub) {
      const int ss = 2 * c + sub;
      if (ss >= nss) break;
      const uint4 a_lo = wa, a_hi = wb;
      wa = load_w(wr0, ss + 1);   // next superstep's weights, one ahead
      wb = load_w(wr1, ss + 1);
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        const int r = 8 * j + g;
        const uint4 b = *reinterpret_cast<const uint4*>(sc + r * kB1RowBytes +
                                                        16 * ((4 * sub + t) ^ (4 * (r & 1))));
        mma_b1(acc[j], a_lo.x, a_hi.x, a_lo.y, a_hi.y, b.x, b.y);
        mma_b1(acc[j], a_lo.z, a_hi.z, a_lo.w, a_hi.w, b.z, b.w);
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");

  // ---- epilogue: sign bits, OR-reduced over the 8 groups of the warp ----
  const bool ok0 = n0 + g < N, ok1 = n0 + g + 8 < N;
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    uint32_t v0 = 0, v1 = 0;   // patterns 8j + 2t and 8j + 2t + 1
    if (ok0 && Kin - 2 * acc[j][0] >= 0) v0 |= 1u << g;
    if (ok0 && Kin - 2 * acc[j][1] >= 0) v1 |= 1u << g;
    if (ok1 && Kin - 2 * acc[j][2] >= 0) v0 |= 1u << (g + 8);
    if (ok1 && Kin - 2 * acc[j][3] >= 0) v1 |= 1u << (g + 8);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      v0 |= __shfl_xor_sync(0xffffffffu, v0, off);
      v1 |= __shfl_xor_sync(0xffffffffu, v1, off);
    }
    if (g == 0) {
      s_out[(8 * j + 2 * t) * kB1Warps + warp] = (uint16_t)v0;
      s_out[(8 * j + 2 * t + 1) * kB1Warps + warp] = (uint16_t)v1;
    }
  }
  __syncthreads();
  for (int p = threadIdx.x; p < PT; p += kB1Threads)
    if (m0 + p < M)
      Aout[(m0 + p) * nw_out + nblk] = reinterpret_cast<const uint64_t*>(s_out)[p];
}

template <int NT>
cudaError_t launch_nt(const uint64_t* A, int64_t M, int nw_in, const uint64_t* W, int N, int Kin,
                      uint64_t* Aout, int nw_out, cudaStream_t st) {
  constexpr int PT = 8 * NT;
  const size_t smem = (size_t)kB1Stages * PT * kB1RowBytes + (size_t)PT * kB1Warps * 2;
  cudaError_t e = cudaFuncSetAttribute(k_forward_b1<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((unsigned)((N + 63) / 64), (unsigned)((M + PT - 1) / PT));
  k_forward_b1<NT><<<grid, kB1Threads, smem, st>>>(A, M, nw_in, W, N, Kin, Aout, nw_out);
  return cudaGetLastError();
}

}  // namespace

// One layer on the b1 mma.sync path: Aout (M x nw_out) = packed sign(A W^T),
// M <= 65535 * 128 patterns per launch.
cudaError_t launch_forward_b1(const uint64_t* A, int64_t M, int nw_in, const uint64_t* W, int N,
                              int Kin, uint64_t* Aout, int nw_out, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  if (M <= 32) return launch_nt<4>(A, M, nw_in, W, N, Kin, Aout, nw_out, st);
  if (M <= 64) return launch_nt<8>(A, M, nw_in, W, N, Kin, Aout, nw_out, st);
  if (M <= 104) return launch_nt<13>(A, M, nw_in, W, N, Kin, Aout, nw_out, st);
  return launch_nt<16>(A, M, nw_in, W, N, Kin, Aout, nw_out, st);
}

}  // namespace bk
