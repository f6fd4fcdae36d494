// kern_eval_tc.cu -- tensor-core forward for forward-only evaluation
// (Sec. 3.1; Alg. 1 l.8-9 without the training side outputs).
//
// Same exact e4m3 formulation as the training forward (+-1 -> 0x38 / 0xB8,
// pads 0, fp32 sums exact), tiled for large batches: a CTA computes 128
// patterns x 256 neurons over the whole K range.
//   - 12 producer warps, one thread per stage row (128 activation rows, then
//     256 weight rows): per 128-element k-block the thread loads the row's
//     two bit words (one 16-byte load when the rows are 16-byte aligned),
//     kPrefetch blocks ahead, and expands them into the row's eight 16-byte
//     chunks of the 128B-swizzled K-major stage (48 KB, 4-stage ring);
//   - 1 MMA warp issues tcgen05.mma.kind::f8f6f4 M128 N256 K32 (four per stage)
//     into a 128 x 256 fp32 accumulator in TMEM (256 columns) and commits to
//     the stage's "empty" mbarrier;
//   - the epilogue: the producer warps read TMEM (warp w: lanes 32 (w % 4) ..,
//     column blocks w / 4, w / 4 + 3, ..) and write the sign bits of each
//     pattern as 32-bit pieces of its packed row (pad bits 0).
// Every mbarrier wait is bounded; the first expiry stops every other wait and
// the kernel counts it in *timeouts, releases TMEM and returns.
#include "tc_common.cuh"

namespace bk {
namespace {

using namespace tc;

constexpr int TM = 128;
constexpr int TN = 256;
constexpr int kStages = 4;
constexpr int kPrefetch = 4;  // == kStages: the stage of k-block kb0 + d is d
constexpr int kProducers = TM + TN;  // one stage row per producer thread
constexpr int kProdWarps = kProducers / 32;
constexpr int THREADS = kProducers + 32;
constexpr int A_BYTES = TM * KB;   // 16 KB
constexpr int B_BYTES = TN * KB;   // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 256;
constexpr uint32_t kIdesc = idesc_f8(TM, TN);
static_assert(kPrefetch == kStages, "stage index is the unrolled prefetch slot");

struct __align__(8) EvShared {
  unsigned long long full[kStages];
  unsigned long long empty[kStages];
  unsigned long long done;
  uint32_t tmem_base;
  int failed;
};

constexpr size_t kSmemBytes = 1024 + kStages * STAGE_BYTES + sizeof(EvShared);

// Four K-elements, bits P .. P + 3 of x (P = 0 or 4), as four e4m3 bytes
// (bit 1 -> 0x38 = +1, bit 0 -> 0xB8 = -1): the product places bit P + j at
// bit 8 j + 7; its four shifted copies of the masked nibble do not overlap,
// so it carries nothing.
template <int P>
__device__ __forceinline__ uint32_t e4m3_quad(uint32_t x) {
  static_assert(P == 0 || P == 4, "nibble position");
  constexpr uint32_t kMul = P == 0 ? 0x10204080u : 0x01020408u;
  return ((x & (0xFu << P)) * kMul & 0x80808080u) ^ 0xB8B8B8B8u;
}

// The row's 128 K-elements of one k-block (four 32-bit words, element e =
// bit e % 32 of word e / 32) -> its eight chunks; chunk c (elements 16 c ..
// 16 c + 15) goes to physical chunk c ^ swz.  Elements at index >= valid are
// written 0 (valid < 128 only in the last k-block of a ragged K).
__device__ __forceinline__ void expand_row(uint8_t* row, int swz, uint4 w, int valid) {
  const uint32_t x[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const uint32_t h = x[c >> 1] >> (16 * (c & 1));
    uint4 v = make_uint4(e4m3_quad<0>(h), e4m3_quad<4>(h), e4m3_quad<0>(h >> 8),
                         e4m3_quad<4>(h >> 8));
    if (valid < KB) {
      const int n = valid - 16 * c;
      v.x &= keep_mask(n);
      v.y &= keep_mask(n - 4);
      v.z &= keep_mask(n - 8);
      v.w &= keep_mask(n - 12);
    }
    *reinterpret_cast<uint4*>(row + 16 * (c ^ swz)) = v;
  }
}

// Bits of k-block kb of a row (words 2 kb, 2 kb + 1; 0 past the nw words).
template <bool kVec>
__device__ __forceinline__ uint4 load_block(const uint64_t* src, int kb, int nkb, int nw) {
  if (src == nullptr || kb >= nkb) return make_uint4(0, 0, 0, 0);
  if (kVec) return __ldg(reinterpret_cast<const uint4*>(src) + kb);
  const uint64_t lo = __ldg(src + 2 * kb);
  const uint64_t hi = 2 * kb + 1 < nw ? __ldg(src + 2 * kb + 1) : 0ull;
  return make_uint4((uint32_t)lo, (uint32_t)(lo >> 32), (uint32_t)hi, (uint32_t)(hi >> 32));
}

// kVec: nw even and both operands 16-byte aligned (every row then is)
template <bool kVec>
__global__ void __launch_bounds__(THREADS, 1)
    k_forward_eval_tc(const uint64_t* __restrict__ A, int64_t M, int nw, const uint64_t* __restrict__ W,
                      int N, int Kin, uint64_t* __restrict__ Aout, int nw_out,
                      unsigned int* __restrict__ timeouts) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  EvShared* sh = reinterpret_cast<EvShared*>(base + kStages * STAGE_BYTES);
  const int64_t m0 = (int64_t)blockIdx.y * TM;
  const int MR = (int)min((int64_t)TM, M - m0);   // pattern rows of this CTA
  const int n0 = blockIdx.x * TN;
  const int NB = min(TN, N - n0);                 // neuron rows of this CTA
  const int nkb = (Kin + KB - 1) / KB;
  const int tail = Kin - KB * (nkb - 1);          // valid elements of the last k-block
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* failed = &sh->failed;

  for (int s = 0; s < kStages; ++s) {
    uint4* a4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES);
    for (int i = MR * (KB / 16) + threadIdx.x; i < TM * (KB / 16); i += THREADS)
      a4[i] = make_uint4(0, 0, 0, 0);
    uint4* b4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES + A_BYTES);
    for (int i = NB * (KB / 16) + threadIdx.x; i < TN * (KB / 16); i += THREADS)
      b4[i] = make_uint4(0, 0, 0, 0);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh->full[s], kProdWarps);  // one arrival per producer warp
      mbar_init(&sh->empty[s], 1);
    }
    mbar_init(&sh->done, 1);
    sh->failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&sh->tmem_base)), "r"(TMEM_COLS) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = sh->tmem_base;

  if (threadIdx.x < kProducers) {
    // this thread's stage row: activation row p (p < TM) or weight row p - TM
    const int p = threadIdx.x;
    const bool isA = p < TM;
    const int r = isA ? p : p - TM;
    const uint64_t* src = nullptr;
    if (isA && r < MR) src = A + (m0 + r) * nw;
    if (!isA && r < NB) src = W + (int64_t)(n0 + r) * nw;
    const uint32_t row_off = (isA ? 0u : (uint32_t)A_BYTES) + (uint32_t)(r * KB);
    const int swz = r & 7;

    uint4 pre[kPrefetch];
#pragma unroll
    for (int d = 0; d < kPrefetch; ++d) pre[d] = load_block<kVec>(src, d, nkb, nw);

    for (int kb0 = 0; kb0 < nkb; kb0 += kPrefetch) {
#pragma unroll
      for (int d = 0; d < kPrefetch; ++d) {
        const int kb = kb0 + d;
        if (kb >= nkb) break;
        if (kb0 > 0 &&
            !__all_sync(kFull, mbar_wait(&sh->empty[d], (uint32_t)((kb0 / kStages - 1) & 1), failed)))
          break;
        if (src != nullptr)
          expand_row(base + d * STAGE_BYTES + row_off, swz, pre[d], kb == nkb - 1 ? tail : KB);
        pre[d] = load_block<kVec>(src, kb + kPrefetch, nkb, nw);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->full[d]);
      }
      if (__any_sync(kFull, *failed != 0)) break;
    }
  } else if (threadIdx.x == kProducers) {
    // MMA issuer: lane 0 of the last warp
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % kStages;
      if (!mbar_wait(&sh->full[s], (uint32_t)((kb / kStages) & 1), failed)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint8_t* sa = base + s * STAGE_BYTES;
      const uint64_t ad = smem_desc(smem_u32(sa));
      const uint64_t bd = smem_desc(smem_u32(sa + A_BYTES));
#pragma unroll
      for (int j = 0; j < KB / 32; ++j)
        mma_f8<kIdesc>(tmem, ad + 2 * j, bd + 2 * j, (kb > 0 || j > 0) ? 1u : 0u);
      mma_commit(&sh->empty[s]);
    }
    if (!*failed) mma_commit(&sh->done);
  }

  // epilogue: tcgen05.ld is warp-collective, so the decision is per warp
  bool go = false;
  if (threadIdx.x < kProducers) {
    go = !*failed && mbar_wait(&sh->done, 0, failed);
    go = __all_sync(0xffffffffu, go);
  }
  if (go) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int sub = warp & 3;
    const int m = 32 * sub + lane;
    for (int cb = warp >> 2; cb < TN / 32; cb += kProdWarps / 4) {
      const int col0 = 32 * cb;
      uint32_t v[32];
      asm volatile(
          "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
          "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
          : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
            "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
            "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
            "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
            "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
          : "r"(tmem + ((uint32_t)(32 * sub) << 16) + (uint32_t)col0));
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      // words wholly past N (inside the row's last 64-bit word) are written 0
      if (m < MR && ((n0 + col0) >> 5) < 2 * nw_out) {
        uint32_t bits = 0;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int z = __float2int_rn(__uint_as_float(v[j]));
          if (n0 + col0 + j < N && z >= 0) bits |= 1u << j;
        }
        reinterpret_cast<uint32_t*>(Aout + (m0 + m) * nw_out)[(n0 + col0) >> 5] = bits;
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (threadIdx.x == 0 && *failed) atomicAdd(timeouts, 1u);
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
}

}  // namespace

cudaError_t prepare_forward_eval_tc() {
  cudaError_t e = cudaFuncSetAttribute(k_forward_eval_tc<true>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_forward_eval_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kSmemBytes);
}

void launch_forward_eval_tc(const uint64_t* A, int64_t M, int nw_in, const uint64_t* W, int N,
                            int Kin, uint64_t* Aout, int nw_out, unsigned int* timeouts,
                            cudaStream_t st) {
  const dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
  const bool vec = (nw_in % 2 == 0) && (reinterpret_cast<uintptr_t>(A) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(W) % 16 == 0);
  if (vec)
    k_forward_eval_tc<true><<<grid, THREADS, kSmemBytes, st>>>(A, M, nw_in, W, N, Kin, Aout,
                                                                nw_out, timeouts);
  else
    k_forward_eval_tc<false><<<grid, THREADS, kSmemBytes, st>>>(A, M, nw_in, W, N, Kin, Aout,
                                                                 nw_out, timeouts);
}

}  // namespace bk
