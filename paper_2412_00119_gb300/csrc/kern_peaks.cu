// kern_peaks.cu -- measured peak rates of the units that can run the forward
// contraction of the BMLP (Alg. 1 l.8: z = K_{l-1} - 2 popc(a XOR w), the
// XNOR/popcount term that Table 3 counts) on this device.  Each kernel keeps
// its operands in registers (or shared memory / TMEM for tcgen05) and issues
// one kind of instruction back to back, so that the timed rate is the unit's,
// not the memory system's:
//   POPC    : CUDA-core 32-bit XOR + popcount, 32 bit-pairs per popcount;
//   TCGEN05 : tcgen05.mma.kind::f8f6f4, e4m3 x e4m3 -> fp32, M128 N256 K32
//             (+-1 is exact in e4m3), 128 x 256 x 32 MACs per instruction;
//   B1MMA   : mma.sync.m16n8k256 .b1 xor.popc, 16 x 8 x 256 bit-pairs;
//   S8MMA   : mma.sync.m16n8k32 .s8 (+-1 as int8), 16 x 8 x 32 MACs.
// (tcgen05.mma.kind::i8 is not available on sm_103a: ptxas rejects it, so
// +-1 as int8 on tensor cores is the legacy mma.sync path.)
// Every loop has a fixed trip count; the tcgen05 kernel's completion wait is
// bounded like every other mbarrier wait of the library.
#include "tc_common.cuh"

namespace bk {
namespace {

using namespace tc;

constexpr int kPeakChains = 8;  // independent accumulators per thread / warp

__global__ void __launch_bounds__(256) k_peak_popc(int64_t iters, uint32_t seed, int* sink) {
  uint32_t x[kPeakChains], acc[kPeakChains];
#pragma unroll
  for (int j = 0; j < kPeakChains; ++j) {
    x[j] = seed ^ (threadIdx.x * 0x9E3779B9u + (uint32_t)j * 0x85EBCA6Bu);
    acc[j] = 0;
  }
  const uint32_t y = seed * 0x27D4EB2Fu + blockIdx.x;
#pragma unroll 1
  for (int64_t it = 0; it < iters; ++it) {
#pragma unroll
    for (int j = 0; j < kPeakChains; ++j) {
      x[j] = __funnelshift_l(x[j], x[j], 1) ^ y;
      acc[j] += __popc(x[j]);
    }
  }
  uint32_t s = 0;
#pragma unroll
  for (int j = 0; j < kPeakChains; ++j) s += acc[j];
  if (s == 0xFFFFFFFFu) sink[blockIdx.x] = (int)s;  // keeps the loop alive
}

__global__ void __launch_bounds__(128) k_peak_b1(int64_t iters, uint32_t seed, int* sink) {
  const uint32_t a0 = seed ^ threadIdx.x, a1 = a0 * 3u, a2 = a0 * 5u, a3 = a0 * 7u;
  const uint32_t b0 = seed + threadIdx.x, b1 = b0 * 11u;
  int d[kPeakChains][4];
#pragma unroll
  for (int j = 0; j < kPeakChains; ++j) d[j][0] = d[j][1] = d[j][2] = d[j][3] = j;
#pragma unroll 1
  for (int64_t it = 0; it < iters; ++it) {
#pragma unroll
    for (int j = 0; j < kPeakChains; ++j)
      asm volatile(
          "mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.xor.popc {%0,%1,%2,%3}, "
          "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
          : "+r"(d[j][0]), "+r"(d[j][1]), "+r"(d[j][2]), "+r"(d[j][3])
          : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
  int s = 0;
#pragma unroll
  for (int j = 0; j < kPeakChains; ++j) s += d[j][0] + d[j][1] + d[j][2] + d[j][3];
  if (s == 0x7FFFFFFF) sink[blockIdx.x] = s;
}

__global__ void __launch_bounds__(128) k_peak_s8(int64_t iters, uint32_t seed, int* sink) {
  const uint32_t a0 = 0x01FF01FFu ^ (seed & 0x00FE0000u), a1 = a0, a2 = a0, a3 = a0;
  const uint32_t b0 = 0xFF0101FFu, b1 = b0;
  int d[kPeakChains][4];
#pragma unroll
  for (int j = 0; j < kPeakChains; ++j) d[j][0] = d[j][1] = d[j][2] = d[j][3] = j;
#pragma unroll 1
  for (int64_t it = 0; it < iters; ++it) {
#pragma unroll
    for (int j = 0; j < kPeakChains; ++j)
      asm volatile(
          "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, "
          "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
          : "+r"(d[j][0]), "+r"(d[j][1]), "+r"(d[j][2]), "+r"(d[j][3])
          : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
  int s = 0;
#pragma unroll
  for (int j = 0; j < kPeakChains; ++j) s += d[j][0] + d[j][1] + d[j][2] + d[j][3];
  if (s == 0x7FFFFFFF) sink[blockIdx.x] = s;
}

// tcgen05: one CTA per SM (the shared-memory request keeps a second CTA off
// the SM); thread 0 issues `iters` rounds of four M128 N256 K32 e4m3 MMAs over
// one zeroed 48 KB stage into 256 TMEM columns, then commits; all threads
// wait (bounded) for completion.
constexpr int kPeakTM = 128, kPeakTN = 256;
constexpr int kPeakStage = kPeakTM * KB + kPeakTN * KB;       // 48 KB
constexpr size_t kPeakSmem = 1024 + 120 * 1024;                // one CTA per SM
constexpr uint32_t kPeakIdesc = idesc_f8(kPeakTM, kPeakTN);

__global__ void __launch_bounds__(128, 1) k_peak_tc(int64_t iters, unsigned int* timeouts) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ unsigned long long done;
  __shared__ uint32_t tmem_base;
  __shared__ int failed;
  for (int i = threadIdx.x; i < kPeakStage / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(base)[i] = make_uint4(0, 0, 0, 0);
  if (threadIdx.x == 0) {
    mbar_init(&done, 1);
    failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (threadIdx.x < 32) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&tmem_base)), "r"(kPeakTN) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tmem_base;
  if (threadIdx.x == 0) {
    const uint64_t ad = smem_desc(smem_u32(base));
    const uint64_t bd = smem_desc(smem_u32(base + kPeakTM * KB));
#pragma unroll 1
    for (int64_t it = 0; it < iters; ++it) {
#pragma unroll
      for (int j = 0; j < KB / 32; ++j)
        mma_f8<kPeakIdesc>(tmem, ad + 2 * j, bd + 2 * j, (it > 0 || j > 0) ? 1u : 0u);
    }
    mma_commit(&done);
  }
  __syncwarp();
  const bool ok = mbar_wait(&done, 0, &failed);
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  __syncthreads();
  if (threadIdx.x == 0 && !ok) atomicAdd(timeouts, 1u);
  if (threadIdx.x < 32)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPeakTN)
                 : "memory");
}

}  // namespace

// Bit-pairs (MACs) of one launch of the peak kernel of `engine` with `iters`
// iterations, and the launch itself.
cudaError_t launch_engine_peak(int engine, int64_t iters, int sms, int* sink, unsigned int* timeouts,
                               cudaStream_t st, double* bitpairs) {
  switch (engine) {
    case BMLP_FWD_POPC: {
      const int blocks = 8 * sms;
      *bitpairs = (double)blocks * 256 * kPeakChains * 32.0 * (double)iters;
      k_peak_popc<<<blocks, 256, 0, st>>>(iters, 0x1234567u, sink);
      break;
    }
    case BMLP_FWD_B1MMA: {
      const int blocks = 4 * sms;  // 16 warps per SM
      *bitpairs = (double)blocks * 4 * kPeakChains * (16.0 * 8 * 256) * (double)iters;
      k_peak_b1<<<blocks, 128, 0, st>>>(iters, 0x1234567u, sink);
      break;
    }
    case BMLP_FWD_S8MMA: {
      const int blocks = 4 * sms;
      *bitpairs = (double)blocks * 4 * kPeakChains * (16.0 * 8 * 32) * (double)iters;
      k_peak_s8<<<blocks, 128, 0, st>>>(iters, 0x1234567u, sink);
      break;
    }
    case BMLP_FWD_TCGEN05: {
      cudaError_t e = cudaFuncSetAttribute(k_peak_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)kPeakSmem);
      if (e != cudaSuccess) return e;
      *bitpairs = (double)sms * 4 * ((double)kPeakTM * kPeakTN * 32) * (double)iters;
      k_peak_tc<<<sms, 128, kPeakSmem, st>>>(iters, timeouts);
      break;
    }
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace bk
