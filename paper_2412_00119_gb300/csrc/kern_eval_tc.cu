// kern_eval_tc.cu -- tensor-core forward for forward-only evaluation
// (Sec. 3.1; Alg. 1 l.8-9 without the training side outputs).
//
// Same exact e4m3 formulation as the training forward (+-1 -> 0x38 / 0xB8,
// pads 0, fp32 sums exact), tiled for large batches.
//
// Tile.  A cluster of two CTAs computes 256 patterns x 512 neurons with
// tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 32), two MMAs per 32-element
// k-step, one per N half (neurons n0 .. n0 + 255 and n0 + 256 .. n0 + 511):
// CTA r of the pair stages activation rows m0 + 128 r .. + 127 and, for half
// h, weight rows n0 + 256 h + 128 r .. + 127; the even CTA issues the MMAs,
// which read the A and B halves of both CTAs at the same shared-memory
// offsets, and CTA r's TMEM receives D rows 128 r .. + 127 for all 512
// neurons (all 512 columns; column c is neuron n0 + c).  Each CTA stages 384
// rows per 128 x 512 outputs, against 384 per 128 x 256 with one CTA: the
// expansion, not the tensor core, sets the pace.
//   - producer warps: kRowSplit threads per stage row (128 activation rows,
//     then 256 weight rows); per 128-element k-block a thread loads its
//     16 / kRowSplit bytes of bits (kStages blocks ahead, in registers) and
//     expands them into its chunks of the 4-stage ring of 48 KB stages;
//     every producer warp arrives on its own CTA's "full" barrier;
//   - in the odd CTA one relay thread waits on that barrier and forwards one
//     arrival (cluster release) to the even CTA's, so no thread with bit
//     loads in flight executes a cluster-scope release;
//   - the even CTA's MMA thread waits on "full" (cluster acquire), issues the
//     eight MMAs of the stage and commits to the "empty" barrier of both CTAs
//     (multicast);
//   - the epilogue: producer warps 0..7 read TMEM (warp w: lanes 32 (w % 4) ..,
//     column blocks w / 4, w / 4 + 2, ..) and write the sign bits of their
//     patterns as 32-bit pieces of the packed rows (pad bits 0);
//   - both CTAs pass a cluster barrier after initialisation (no remote arrive
//     or commit reaches an uninitialised barrier) and before releasing TMEM.
// Every mbarrier wait is bounded; the first expiry stops every other wait of
// the CTA and the kernel counts it in *timeouts, releases TMEM and returns.
#include "tc_common.cuh"

namespace bk {
namespace {

using namespace tc;

constexpr int TM = 128;                  // pattern rows per CTA (MMA M = 256 per pair)
constexpr int kHalves = 2;               // N = 256 MMAs per k-step (TMEM column ranges)
constexpr int TN = 256 * kHalves;        // neurons per pair
constexpr int TB = 128 * kHalves;        // weight rows per CTA
constexpr int kStages = 4;
constexpr int kRowSplit = 1;             // producer threads per stage row
constexpr int kProducers = (TM + TB) * kRowSplit;
constexpr int kProdWarps = kProducers / 32;
constexpr int THREADS = kProducers + 32;
constexpr int A_BYTES = TM * KB;         // 16 KB
constexpr int B_BYTES = TB * KB;         // 32 KB: 16 KB per N half
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = TN;
constexpr uint32_t kIdesc = idesc_f8(2 * TM, 256);

struct __align__(8) EvShared {
  unsigned long long full[kStages];
  unsigned long long empty[kStages];
  unsigned long long done;
  uint32_t tmem_base;
  int failed;
};

constexpr size_t kSmemBytes = 1024 + kStages * STAGE_BYTES + sizeof(EvShared);

// -------- the pair kernel -----------------------------------------------------
__device__ __forceinline__ uint32_t pair_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void pair_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}

// Bounded wait with cluster-scope acquire (the barrier collects an arrival
// from the peer CTA).
__device__ __forceinline__ bool mbar_wait_cluster(unsigned long long* bar, uint32_t parity,
                                                  volatile int* failed) {
  const uint32_t a = smem_u32(bar);
  const unsigned long long t0 = clock64();
  while (true) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok) : "r"(a), "r"(parity) : "memory");
    if (ok) return true;
    if (*failed) return false;
    if (clock64() - t0 > kWaitCycles) {
      *failed = 1;
      return false;
    }
  }
}

// Arrive on the barrier at the same offset in CTA 0 of the cluster.
__device__ __forceinline__ void mbar_arrive_rank0(unsigned long long* bar) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(remote) : "r"(smem_u32(bar)));
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote) : "memory");
}

__device__ __forceinline__ void mma_f8_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n}"
      ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate));
}

// Arrive once on the barrier at this offset in both CTAs of the pair when the
// MMAs issued so far complete.
__device__ __forceinline__ void mma_commit_pair(unsigned long long* bar) {
  const uint16_t mask = 0x3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
      ::"r"(smem_u32(bar)), "h"(mask) : "memory");
}

// kVec: nw even and both operands 16-byte aligned (every row then is); with
// one thread per row its two words of a k-block are then one 16-byte load
template <bool kVec>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    k_forward_eval_tc(const uint64_t* __restrict__ A, int64_t M, int nw,
                      const uint64_t* __restrict__ W, int N, int Kin, uint64_t* __restrict__ Aout,
                      int nw_out, unsigned int* __restrict__ timeouts) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  EvShared* sh = reinterpret_cast<EvShared*>(base + kStages * STAGE_BYTES);
  const uint32_t rank = pair_rank();
  // neuron tiles vary fastest: the pairs in flight share a tile of patterns,
  // and the layer's packed W (8 MB at 8192 x 8192) stays in L2
  const int64_t m0 = (int64_t)blockIdx.y * (2 * TM) + (int64_t)rank * TM;  // this CTA's patterns
  const int MR = (int)max((int64_t)0, min((int64_t)TM, M - m0));
  const int n0 = (int)(blockIdx.x >> 1) * TN;                               // the pair's neurons
  // weight row q of this CTA (block q / 128 of the B stage) is neuron
  // n0 + 256 (q / 128) + 128 rank + q % 128: half h of the pair's MMAs covers
  // neurons n0 + 256 h .. + 255, 128 from each CTA
  auto neuron_of = [&](int q) { return n0 + 256 * (q >> 7) + 128 * (int)rank + (q & 127); };
  const int nkb = (Kin + KB - 1) / KB;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* failed = &sh->failed;

  for (int s = 0; s < kStages; ++s) {
    uint4* a4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES);
    for (int i = MR * (KB / 16) + threadIdx.x; i < TM * (KB / 16); i += THREADS)
      a4[i] = make_uint4(0, 0, 0, 0);
    uint4* b4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES + A_BYTES);
    for (int i = threadIdx.x; i < TB * (KB / 16); i += THREADS)
      if (neuron_of(i / (KB / 16)) >= N) b4[i] = make_uint4(0, 0, 0, 0);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      // the producer warps and, on the even CTA, the odd CTA's relayed arrival
      mbar_init(&sh->full[s], kProdWarps + (rank == 0 ? 1 : 0));
      mbar_init(&sh->empty[s], 1);
    }
    mbar_init(&sh->done, 1);
    sh->failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&sh->tmem_base)), "r"(TMEM_COLS) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  pair_sync();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = sh->tmem_base;

  if (threadIdx.x < kProducers) {
    // stage row p (activation row p < TM, else weight row p - TM), part `part`
    // of its 128 K-elements per k-block: chunks kCh part .. kCh part + kCh - 1
    constexpr int kCh = 8 / kRowSplit;          // 16-byte chunks per thread and stage
    constexpr int kWords = 2 / kRowSplit > 0 ? 2 / kRowSplit : 1;
    const int p = threadIdx.x / kRowSplit, part = threadIdx.x % kRowSplit;
    const bool isA = p < TM;
    const int r = isA ? p : p - TM;
    const uint64_t* src = nullptr;
    if (isA && r < MR) src = A + (m0 + r) * nw;
    if (!isA && neuron_of(r) < N) src = W + (int64_t)neuron_of(r) * nw;
    const uint32_t row_off = (isA ? 0u : (uint32_t)A_BYTES) + (uint32_t)(r * KB);
    const int swz = r & 7;
    // bits of k-block kb for this thread: words 2 kb + kWords part .. (0 past nw)
    auto load = [&](int kb) -> uint4 {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (src == nullptr || kb >= nkb) return v;
      if (kVec && kWords == 2) return __ldg(reinterpret_cast<const uint4*>(src) + kb);
      const int w0 = 2 * kb + kWords * part;
      const uint64_t lo = w0 < nw ? __ldg(src + w0) : 0ull;
      v.x = (uint32_t)lo;
      v.y = (uint32_t)(lo >> 32);
      if (kWords == 2) {
        const uint64_t hi = w0 + 1 < nw ? __ldg(src + w0 + 1) : 0ull;
        v.z = (uint32_t)hi;
        v.w = (uint32_t)(hi >> 32);
      }
      return v;
    };
    uint4 pre[kStages];
#pragma unroll
    for (int d = 0; d < kStages; ++d) pre[d] = load(d);

    for (int kb0 = 0; kb0 < nkb; kb0 += kStages) {
#pragma unroll
      for (int d = 0; d < kStages; ++d) {  // the stage of k-block kb0 + d is d
        const int kb = kb0 + d;
        if (kb >= nkb) break;
        if (kb0 > 0 &&
            !__all_sync(kFull, mbar_wait(&sh->empty[d], (uint32_t)((kb0 / kStages - 1) & 1), failed)))
          break;
        if (src != nullptr) {
          uint8_t* row = base + d * STAGE_BYTES + row_off;
          const uint32_t x[4] = {pre[d].x, pre[d].y, pre[d].z, pre[d].w};
          const int valid = Kin - KB * kb - 16 * kCh * part;
          if (valid >= 16 * kCh) {
#pragma unroll
            for (int q = 0; q < kCh; ++q) {
              const int c = kCh * part + q;
              *reinterpret_cast<uint4*>(row + 16 * (c ^ swz)) = chunk16(x[q >> 1] >> (16 * (q & 1)));
            }
          } else {
#pragma unroll
            for (int q = 0; q < kCh; ++q) {
              const int c = kCh * part + q;
              *reinterpret_cast<uint4*>(row + 16 * (c ^ swz)) =
                  chunk16_masked(x[q >> 1] >> (16 * (q & 1)), valid - 16 * q);
            }
          }
        }
        pre[d] = load(kb + kStages);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->full[d]);
      }
      if (__any_sync(kFull, *failed != 0)) break;
    }
  } else if (threadIdx.x == kProducers && rank == 0) {
    // MMA issuer of the pair: lane 0 of the even CTA's last warp
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % kStages;
      if (!mbar_wait_cluster(&sh->full[s], (uint32_t)((kb / kStages) & 1), failed)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint8_t* sa = base + s * STAGE_BYTES;
      const uint64_t ad = smem_desc(smem_u32(sa));
#pragma unroll
      for (int j = 0; j < KB / 32; ++j)
#pragma unroll
        for (int h = 0; h < kHalves; ++h)
          mma_f8_pair(tmem + 256u * (uint32_t)h, ad + 2 * j,
                      smem_desc(smem_u32(sa + A_BYTES + h * (B_BYTES / kHalves))) + 2 * j,
                      (kb > 0 || j > 0) ? 1u : 0u);
      mma_commit_pair(&sh->empty[s]);
    }
    if (!*failed) mma_commit_pair(&sh->done);
  } else if (threadIdx.x == kProducers) {
    // relay of the odd CTA: its stage is full -> one arrival on the even CTA's
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % kStages;
      if (!mbar_wait(&sh->full[s], (uint32_t)((kb / kStages) & 1), failed)) break;
      mbar_arrive_rank0(&sh->full[s]);
    }
  }

  // epilogue: this CTA's 128 rows of D, all TN neurons (TMEM column c = neuron n0 + c)
  bool go = false;
  if (warp < 8) {
    go = !*failed && mbar_wait(&sh->done, 0, failed);
    go = __all_sync(0xffffffffu, go);
  }
  if (go) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int sub = warp & 3;
    const int m = 32 * sub + lane;
    for (int cb = warp >> 2; cb < TN / 32; cb += 2) {
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
  pair_sync();   // no CTA releases TMEM or leaves while its peer may still use the pair
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (threadIdx.x == 0 && *failed) atomicAdd(timeouts, 1u);
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
}

// Failure-path probe: the bounded mbarrier wait of the kernels above on a
// barrier whose phase completes only if `arrive` (one arrival before the wait).
__global__ void k_wait_probe(unsigned int* __restrict__ timeouts, int arrive,
                             unsigned long long limit) {
  __shared__ unsigned long long bar;
  __shared__ int failed;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (arrive) mbar_arrive(&bar);
    if (!mbar_wait(&bar, 0, &failed, limit)) atomicAdd(timeouts, 1u);
  }
}

}  // namespace

void launch_wait_probe(unsigned int* timeouts, int arrive, unsigned long long limit_cycles,
                       cudaStream_t st) {
  k_wait_probe<<<1, 32, 0, st>>>(timeouts, arrive, limit_cycles);
}

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
  const dim3 grid((unsigned)(2 * ((N + TN - 1) / TN)), (unsigned)((M + 2 * TM - 1) / (2 * TM)));
  const bool vec = (nw_in % 2 == 0) && (reinterpret_cast<uintptr_t>(A) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(W) % 16 == 0);
  if (vec)
    k_forward_eval_tc<true><<<grid, THREADS, kSmemBytes, st>>>(A, M, nw_in, W, N, Kin, Aout, nw_out,
                                                                timeouts);
  else
    k_forward_eval_tc<false><<<grid, THREADS, kSmemBytes, st>>>(A, M, nw_in, W, N, Kin, Aout, nw_out,
                                                                 timeouts);
}

}  // namespace bk
