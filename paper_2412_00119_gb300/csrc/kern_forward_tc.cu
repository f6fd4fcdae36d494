// kern_forward_tc.cu -- tensor-core forward contraction of the BMLP
// (Alg. 1 l.8-9) on sm_103a with tcgen05.
//
//   z^mu_k = sum_i a^mu_i w_ik,  a, w in {-1, +1}
//
// is computed exactly as an e4m3 x e4m3 -> fp32 matrix product: +-1 are exact
// in e4m3 (0x38 / 0xB8), pad elements are 0x00, and every partial sum is an
// integer of magnitude <= K_in < 2^24, exact in fp32 whatever the order.
// One CTA owns TN = 64 neurons and all (<= 128) patterns of the mini-batch.
// The A operand of layers l >= 2 arrives pre-expanded: the epilogue of layer
// l - 1 also writes its activations as e4m3 in the swizzled stage image (one
// 16 KB tile per 128 K-elements, DevLayer::AE), and one producer pulls each
// tile into the stage with a single cp.async.bulk that completes on the
// stage's "full" mbarrier.  For layer 1 (the caller's bit-packed input) and in
// general:
//   - 16 producer warps expand the bit-packed activations (A, patterns x
//     words) and visible weights (W, neurons x words), 128 K-elements per row
//     per stage, into the K-major SWIZZLE_128B layout the MMA reads (16-byte
//     chunk c of row r stored at chunk c ^ (r % 8)).  The stage's 16-byte
//     chunks are dealt round-robin to the 512 producer threads (three per
//     thread for A + B, one for B alone in tile mode); their 16-bit pieces of
//     bits are loaded kPrefetch stages ahead into registers.  Each producer
//     warp arrives once on the stage's "full" mbarrier, after every lane's
//     proxy fence.
//   - 1 MMA warp waits on "full", issues tcgen05.mma.kind::f8f6f4 (M = 128,
//     N = 64, K = 32) four times per stage into a 128-lane x 64-column fp32
//     accumulator in TMEM, and commits to the stage's "empty" mbarrier, on
//     which producers wait before overwriting the stage (kStages-deep ring).
//   - the epilogue reads the accumulator with tcgen05.ld (warp w % 4 owns TMEM
//     lanes 32 (w % 4) .., 16 columns per warp), converts to int, stores z
//     (int16) and packs the sign bits of 16 neurons per thread directly into
//     the activation words.
// Every mbarrier wait is bounded; the first expiry sets a shared flag that
// stops every other wait, the kernel counts the failure in the control block
// (host: BMLP_ETIMEOUT), releases its TMEM and returns.
#include "tc_common.cuh"

namespace bk {
namespace {

using namespace tc;

constexpr int TM = 128;           // MMA M: patterns (rows >= bsz are zero)
constexpr int TN = 64;            // MMA N: neurons per CTA
constexpr int kStages = 4;
constexpr int kPrefetch = 8;      // stages of bit-words held in registers ahead
constexpr int kProducers = 512;   // 16 warps: one (row, half) item per thread
constexpr int THREADS = kProducers + 32;
constexpr int A_BYTES = TM * KB;  // 16 KB
constexpr int B_BYTES = TN * KB;  // 8 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 64;

struct __align__(8) TcShared {
  unsigned long long full[kStages];   // the producers filled stage s
  unsigned long long empty[kStages];  // the MMAs that read stage s completed
  unsigned long long done;            // all MMAs completed
  uint32_t tmem_base;
  int failed;
};

constexpr size_t kSmemBytes = 1024 /*alignment slack*/ + kStages * STAGE_BYTES + sizeof(TcShared);

constexpr uint32_t kIdesc = tc::idesc_f8(TM, TN);

template <bool kTiles>
__global__ void __launch_bounds__(THREADS, 1) k_train_forward_tc(const StepParams* __restrict__ P, int l);

}  // namespace

size_t train_forward_tc_smem() { return kSmemBytes; }

cudaError_t prepare_train_forward_tc() {
  cudaError_t e = cudaFuncSetAttribute(k_train_forward_tc<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_train_forward_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kSmemBytes);
}

void launch_train_forward_tc(bool tiles, int Kout, cudaStream_t st, const StepParams* P, int l) {
  const dim3 grid((unsigned)((Kout + TN - 1) / TN));
  if (tiles)
    k_train_forward_tc<true><<<grid, THREADS, kSmemBytes, st>>>(P, l);
  else
    k_train_forward_tc<false><<<grid, THREADS, kSmemBytes, st>>>(P, l);
}

size_t act_tile_bytes(int K) { return (size_t)((K + KB - 1) / KB) * A_BYTES; }

namespace {

template <bool kTiles>
__global__ void __launch_bounds__(THREADS, 1) k_train_forward_tc(const StepParams* __restrict__ P, int l) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  TcShared* sh = reinterpret_cast<TcShared*>(base + kStages * STAGE_BYTES);
  const DevLayer& Ly = P->layer[l - 1];
  const int64_t start = (int64_t)P->ctrl->s * P->bs;
  const int64_t rem = P->n - start;
  const int M = (int)(rem < P->bs ? rem : P->bs);
  const uint64_t* A = (l == 1) ? P->x + start * P->nw0 : P->layer[l - 2].A;
  const int n0 = blockIdx.x * TN;
  const int N = Ly.Kout, Kin = Ly.Kin, nw = Ly.nw_in;
  const int NB = min(TN, N - n0);   // neuron rows of this CTA
  const int nkb = (Kin + KB - 1) / KB;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* failed = &sh->failed;

  // zero the pattern rows >= M and neuron rows >= NB of every stage once; the
  // producers never write them, so they stay zero (0 * anything = 0)
  for (int s = 0; s < kStages; ++s) {
    uint4* a4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES);
    for (int i = M * (KB / 16) + threadIdx.x; i < TM * (KB / 16); i += THREADS)
      a4[i] = make_uint4(0, 0, 0, 0);
    uint4* b4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES + A_BYTES);
    for (int i = NB * (KB / 16) + threadIdx.x; i < TN * (KB / 16); i += THREADS)
      b4[i] = make_uint4(0, 0, 0, 0);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      // one arrival per producer warp, plus (kTiles) the tile copy's
      // expect_tx arrival
      mbar_init(&sh->full[s], kProducers / 32 + (kTiles ? 1 : 0));
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
    // ---------------- producers ----------------
    // items: the 16-byte chunks of A rows [0, M) (only without tiles), then
    // of B rows [0, NB); item i belongs to thread i % kProducers
    constexpr int kItems = kTiles ? 8 * TN / kProducers : 8 * (TM + TN) / kProducers;
    const int nA = kTiles ? 0 : 8 * M, nItems = nA + 8 * NB;
    Chunk ch[kItems];
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      const int i = threadIdx.x + j * kProducers;
      if (i < nA) {
        ch[j] = make_chunk(A + (int64_t)(i >> 3) * nw, 0, i >> 3, i & 7);
      } else if (i < nItems) {
        const int b = i - nA;
        ch[j] = make_chunk(Ly.W + (int64_t)(n0 + (b >> 3)) * nw, A_BYTES, b >> 3, b & 7);
      } else {
        ch[j] = Chunk{nullptr, 0u, 0};
      }
    }
    uint32_t pre[kPrefetch][kItems];
#pragma unroll
    for (int d = 0; d < kPrefetch; ++d)
#pragma unroll
      for (int j = 0; j < kItems; ++j) pre[d][j] = load_chunk(ch[j], d, nw);

    for (int kb0 = 0; kb0 < nkb; kb0 += kPrefetch) {
#pragma unroll
      for (int d = 0; d < kPrefetch; ++d) {
        const int kb = kb0 + d;
        if (kb >= nkb) break;
        const int s = kb % kStages;
        if (kb >= kStages &&
            !__all_sync(kFull, mbar_wait(&sh->empty[s], (uint32_t)((kb / kStages - 1) & 1), failed)))
          break;
        uint8_t* stage = base + s * STAGE_BYTES;
        if (kTiles && threadIdx.x == 0) {
          // A: the pre-expanded activation tile of this k-block
          mbar_arrive_tx(&sh->full[s], A_BYTES);
          bulk_g2s(stage, P->layer[l - 2].AE + (size_t)kb * A_BYTES, A_BYTES, &sh->full[s]);
        }
#pragma unroll
        for (int j = 0; j < kItems; ++j) {
          if (ch[j].src != nullptr) store_chunk(stage, ch[j], pre[d][j], kb, Kin);
          pre[d][j] = load_chunk(ch[j], kb + kPrefetch, nw);
        }
        // every writer orders its stores for the async proxy; one arrival per warp
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->full[s]);
      }
      if (__any_sync(kFull, *failed != 0)) break;
    }
  } else if (threadIdx.x == kProducers) {
    // ---------------- MMA issuer (lane 0 of the last warp) ----------------
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % kStages;
      if (!mbar_wait(&sh->full[s], (uint32_t)((kb / kStages) & 1), failed)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint8_t* sa = base + s * STAGE_BYTES;
      const uint64_t ad = smem_desc(smem_u32(sa));
      const uint64_t bd = smem_desc(smem_u32(sa + A_BYTES));
#pragma unroll
      for (int j = 0; j < KB / 32; ++j)   // K = 32 bytes per MMA: +2 in the address field
        mma_f8<kIdesc>(tmem, ad + 2 * j, bd + 2 * j, (kb > 0 || j > 0) ? 1u : 0u);
      mma_commit(&sh->empty[s]);
    }
    if (!*failed) mma_commit(&sh->done);
  }

  // ---------------- epilogue (producer warps) ----------------
  // tcgen05.ld is warp-collective: the go / no-go decision is made per warp
  bool go = false;
  if (threadIdx.x < kProducers) {
    go = !*failed && mbar_wait(&sh->done, 0, failed);
    go = __all_sync(0xffffffffu, go);
  }
  if (go) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int sub = warp & 3;            // TMEM lanes 32 sub .. 32 sub + 31
    const int col0 = 16 * (warp >> 2);   // accumulator columns col0 .. col0 + 15
    uint32_t v[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
          "=r"(v[14]), "=r"(v[15])
        : "r"(tmem + ((uint32_t)(32 * sub) << 16) + (uint32_t)col0));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
    const int m = 32 * sub + lane;
    if (m < M) {
      int16_t* zrow = Ly.Z + (int64_t)m * N;
      uint32_t bits = 0;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int n = n0 + col0 + j;
        const int z = __float2int_rn(__uint_as_float(v[j]));
        if (n < N) {
          zrow[n] = (int16_t)z;
          if (z >= 0) bits |= 1u << j;
        }
      }
      reinterpret_cast<uint16_t*>(Ly.A + (int64_t)m * Ly.nw_out + (n0 >> 6))[col0 >> 4] = (uint16_t)bits;
      if (Ly.AE != nullptr) {
        // the same 16 activations as e4m3 (+1 0x38, -1 0xB8, past N 0x00) in the
        // swizzled tile image that the next layer's stages copy verbatim
        const int nf = n0 + col0;
        uint32_t q[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          uint32_t word = 0;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int jj = 4 * b + j;
            const uint32_t e = (nf + jj < N) ? (((bits >> jj) & 1u) ? 0x38u : 0xB8u) : 0u;
            word |= e << (8 * j);
          }
          q[b] = word;
        }
        const int c = (nf % KB) / 16;
        uint8_t* dst = Ly.AE + (size_t)(nf / KB) * A_BYTES + (size_t)m * KB + 16 * (c ^ (m & 7));
        *reinterpret_cast<uint4*>(dst) = make_uint4(q[0], q[1], q[2], q[3]);
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (threadIdx.x == 0 && *failed) atomicAdd(&P->ctrl->timeouts, 1u);
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
}

}  // namespace
}  // namespace bk
