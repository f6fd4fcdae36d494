// kern_forward_tc.cu -- tensor-core forward contraction of the BMLP
// (Alg. 1 l.8-9) on sm_103a with tcgen05, for one training mini-batch.
//
//   z^mu_k = sum_i a^mu_i w_ik,  a, w in {-1, +1}
//
// is computed exactly as an e4m3 x e4m3 -> fp32 matrix product: +-1 are exact
// in e4m3 (0x38 / 0xB8), padded weight elements are 0x00, and every partial
// sum is an integer of magnitude <= K_in < 2^24, exact in fp32 in any order.
//
// Tiling.  A tile is the whole mini-batch (MMA M = 128 rows; rows >= bs are
// computed and never read) x TN = 256 neurons.  The K range is split across a
// cluster of kSplit = 4 CTAs so that every SM has work with only K_out / 256
// tiles: CTA r of the cluster accumulates k-blocks [r nkb / 4, (r+1) nkb / 4)
// (128 K-elements each) in TMEM.
//
// Operands.  The tensor core can take the A operand from tensor memory, and
// that is where the activations go; only the weights pass through shared
// memory.  A pipeline that stages both operands in shared memory writes and
// reads every byte of both there, and on this shape shared-memory bandwidth,
// not the tensor core, sets the pace.  Per k-block:
//   - 16 producer warps in two groups of eight take alternate k-blocks; in a
//     group, thread t expands the packed visible weights of neuron row t of
//     the tile (128 K-elements) into a 32 KB stage in the 128B-swizzled
//     K-major layout the MMA reads (16-byte chunk c of row r at chunk
//     c ^ (r % 8)), and 64 K-elements of one pattern row into TMEM with
//     tcgen05.st: warp w writes the lanes 32 (w % 4) .. 32 (w % 4) + 31 that
//     its lane quarter may access and K-elements 64 (w / 4) .. + 63 of the
//     block, i.e. 16 TMEM columns (four e4m3 per 32-bit column) from one
//     64-bit word of bits;
//   - bit words are loaded kPrefetch k-blocks ahead into registers (each
//     group holds its own k-blocks);
//   - each producer warp waits for its TMEM stores, fences its shared-memory
//     stores for the async proxy and arrives once on the stage's "full"
//     mbarrier (eight arrivals complete a stage);
//   - one MMA thread waits on "full" and issues four tcgen05.mma.kind::f8f6f4
//     (M = 128, N = 256, K = 32; A from TMEM, B from the stage) into the
//     128 x 256 fp32 accumulator, then commits to the stage's "empty" mbarrier.
//   TMEM: accumulator in columns 0 .. 255, kStages activation stages of 32
//   columns above it.  Shared memory: kStages weight stages.
// Epilogue.  tcgen05.ld -> partials in shared memory (offset 16-bit lanes,
// two per word, so that 32-bit adds sum two elements at once), laid out by the
// CTA that owns each 64-column slice (CTA r of the cluster finalises neurons
// 64 r .. 64 r + 63 of the tile); one cluster barrier; then each CTA pushes
// its three foreign slices into their owners' slices with bulk reduce-adds
// (cp.reduce.async.bulk .add, shared::cta -> shared::cluster), which complete
// on the owner's mbarrier; the owner waits for the three, and writes z
// (int16) and the packed sign bits of its 64 neurons.  A CTA leaves only after
// its outgoing bulk reads have completed and its own slice has received all
// three adds, so no second cluster barrier is needed.
// Every mbarrier wait is bounded; the first expiry sets a shared flag that
// stops every other wait, the kernel counts the failure in the control block
// (host: BMLP_ETIMEOUT), still passes the cluster barrier, releases its TMEM
// and returns.
#include "tc_common.cuh"

namespace bk {
namespace {

using namespace tc;

constexpr int TM = 128;           // MMA M: patterns (rows >= bsz unused)
constexpr int TN = 256;           // MMA N: neurons per tile
constexpr int kSplit = 4;         // CTAs per cluster, each a quarter of K
constexpr int kStages = 6;        // weight stages in shared memory, activation stages in TMEM
constexpr int kPrefetch = 8;      // k-blocks of bit words held in registers ahead
constexpr int kProducers = 512;   // 16 warps
constexpr int THREADS = kProducers + 32;
constexpr int B_BYTES = TN * KB;  // 32 KB weight stage
constexpr int kAccCols = TN;      // fp32 accumulator columns
constexpr int kStageCols = KB / 4;  // TMEM columns of one activation stage (4 e4m3 per column)
constexpr int TMEM_COLS = 512;
static_assert(kAccCols + kStages * kStageCols <= TMEM_COLS, "TMEM budget");
constexpr int kCols = TN / kSplit;  // neurons finalised by one CTA
static_assert(kCols == 64, "one CTA writes one packed activation word per row");
// A CTA's partial covers at most ceil(ceil(K_in / 128) / 4) <= 64 k-blocks of
// 128 elements (K_in <= 32767), so it is an integer in [-8192, 8192]; stored
// with the offset kOff = 8192 in a 16-bit lane, two lanes per 32-bit word, the
// kSplit = 4 offset partials of an element sum to z + 4 kOff, which lies in
// [1, 65535] because |z| <= K_in <= 32767 -- so 32-bit adds of the packed
// words never carry from one lane into the next.
constexpr uint32_t kOff = 8192;
constexpr int kSliceRow = 2 * kCols + 16;  // bytes per pattern row of a partial slice (+16: banks)
constexpr int kSliceBytes = TM * kSliceRow;
static_assert(kSplit * kSliceBytes <= kStages * B_BYTES, "partials must fit in the stages");
static_assert(kSliceRow % 16 == 0, "bulk copies move multiples of 16 bytes");

struct __align__(8) TcShared {
  unsigned long long full[kStages];   // the producers filled stage s
  unsigned long long empty[kStages];  // the MMAs that read stage s completed
  unsigned long long done;            // all MMAs completed
  unsigned long long red;             // the three peers' slices were added into ours
  uint32_t tmem_base;
  int failed;
  int red_failed;                     // only the wait on `red` sets this one
};

constexpr size_t kSmemBytes = 1024 /*alignment slack*/ + kStages * B_BYTES + sizeof(TcShared);

constexpr uint32_t kIdesc = tc::idesc_f8(TM, TN);

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}

__device__ __forceinline__ uint32_t peer_addr(uint32_t local_addr, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(local_addr), "r"(rank));
  return a;
}

// MMA with the A operand in tensor memory (lane = row, four e4m3 per column).
__device__ __forceinline__ void mma_f8_tmem_a(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n}"
      ::"r"(tmem_d), "r"(tmem_a), "l"(bdesc), "r"(kIdesc), "r"(accumulate));
}

// 64 K-elements of one row (bits 0..63 of x) as sixteen TMEM columns of e4m3.
__device__ __forceinline__ void tmem_store_row64(uint32_t taddr, uint64_t x) {
  uint32_t v[16];
  const uint32_t lo = (uint32_t)x, hi = (uint32_t)(x >> 32);
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    v[c] = e4m3_quad<0>(lo >> (4 * c));
    v[8 + c] = e4m3_quad<0>(hi >> (4 * c));
  }
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15, %16};"
      ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]),
        "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15]) : "memory");
}

__global__ void __cluster_dims__(kSplit, 1, 1) __launch_bounds__(THREADS, 1)
    k_train_forward_tc(const StepParams* __restrict__ P, int l);

}  // namespace

size_t train_forward_tc_smem() { return kSmemBytes; }

cudaError_t prepare_train_forward_tc() {
  return cudaFuncSetAttribute(k_train_forward_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kSmemBytes);
}

cudaError_t launch_train_forward_tc(int Kout, cudaStream_t st, bool pdl, const StepParams* P, int l) {
  const dim3 grid((unsigned)(((Kout + TN - 1) / TN) * kSplit));
  return launch_kernel(k_train_forward_tc, grid, dim3(THREADS), kSmemBytes, st, pdl, P, l);
}

namespace {

__global__ void __cluster_dims__(kSplit, 1, 1) __launch_bounds__(THREADS, 1)
    k_train_forward_tc(const StepParams* __restrict__ P, int l) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  TcShared* sh = reinterpret_cast<TcShared*>(base + kStages * B_BYTES);
  const DevLayer& Ly = P->layer[l - 1];
  const uint32_t rank = cluster_rank();
  const int n0 = (int)(blockIdx.x / kSplit) * TN;
  const int N = Ly.Kout, Kin = Ly.Kin, nw = Ly.nw_in;
  const int NB = min(TN, N - n0);   // neuron rows of this tile
  const int nkb = (Kin + KB - 1) / KB;
  const int kb0 = (int)((nkb * rank) / kSplit);
  const int nk = (int)((nkb * (rank + 1)) / kSplit) - kb0;  // k-blocks of this CTA (may be 0)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* failed = &sh->failed;

  // weight rows >= NB of every stage are zero (never written by the producers)
  for (int s = 0; s < kStages; ++s) {
    uint4* b4 = reinterpret_cast<uint4*>(base + s * B_BYTES);
    for (int i = NB * (KB / 16) + threadIdx.x; i < TN * (KB / 16); i += THREADS)
      b4[i] = make_uint4(0, 0, 0, 0);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh->full[s], kProducers / 64);   // one arrival per warp of the owning group
      mbar_init(&sh->empty[s], 1);
    }
    mbar_init(&sh->done, 1);
    mbar_init(&sh->red, 1);
    sh->failed = 0;
    sh->red_failed = 0;
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

  // ---------------- producer roles ----------------
  // Two groups of eight warps take alternate k-blocks (group g: k = g, g + 2,
  // ...; with an even kStages each stage slot belongs to one group), so one
  // group's store fences and barrier arrival overlap the other group's
  // expansion.  Within a group, thread t = 32 w + lane (w = warp % 8) expands
  // weight row t of the tile (128 K-elements, eight 16-byte chunks) and 64
  // K-elements (half w / 4) of activation row 32 (w % 4) + lane, the TMEM lane
  // its warp may access.
  const int grp = (warp >> 3) & 1, gw = warp & 7;
  const int r = 32 * gw + lane;
  const int q = gw & 3, j2 = gw >> 2;
  const int m = 32 * q + lane;
  const uint64_t* wsrc = (warp < 16 && r < NB) ? Ly.W + (int64_t)(n0 + r) * nw : nullptr;
  const bool wvec = (nw % 2 == 0) && (reinterpret_cast<uintptr_t>(Ly.W) % 16 == 0);
  const uint64_t* aprev = (l == 1) ? P->x : P->layer[l - 2].A;
  const int bs = P->bs;
  const int64_t ncall = P->n;
  auto load_w = [&](int kb) -> uint4 {
    if (wsrc == nullptr || kb >= kb0 + nk) return make_uint4(0, 0, 0, 0);
    if (wvec) return __ldg(reinterpret_cast<const uint4*>(wsrc) + kb);
    const uint64_t lo = 2 * kb < nw ? __ldg(wsrc + 2 * kb) : 0ull;
    const uint64_t hi = 2 * kb + 1 < nw ? __ldg(wsrc + 2 * kb + 1) : 0ull;
    return make_uint4((uint32_t)lo, (uint32_t)(lo >> 32), (uint32_t)hi, (uint32_t)(hi >> 32));
  };
  constexpr int kPf = kPrefetch / 2;   // own k-blocks held ahead (every other k-block)
  uint4 pw[kPf];
  // Layers >= 2: the weights (the previous step's update), the batch index
  // and every pointer were written two or more launches back, so they are
  // read before waiting for the previous layer, whose activations are read
  // after.  Layer 1 waits first: its weights and batch index come from the
  // update launched just before it.
  int64_t start = 0;
  int M = 0;
  if (l > 1) {
    start = (int64_t)P->ctrl->s * bs;
    M = (int)min((int64_t)bs, ncall - start);
#pragma unroll
    for (int i = 0; i < kPf; ++i) pw[i] = load_w(kb0 + grp + 2 * i);
  }
  pdl_wait();
  if (l == 1) {
    start = (int64_t)P->ctrl->s * bs;
    M = (int)min((int64_t)bs, ncall - start);
#pragma unroll
    for (int i = 0; i < kPf; ++i) pw[i] = load_w(kb0 + grp + 2 * i);
  }
  pdl_trigger();
  const uint64_t* A = (l == 1) ? aprev + start * P->nw0 : aprev;

  if (threadIdx.x < kProducers) {
    // ---------------- producers ----------------
    const uint64_t* asrc = (m < M) ? A + (int64_t)m * nw : nullptr;
    auto load_a = [&](int kb) -> uint64_t {
      const int ai = 2 * kb + j2;
      return (asrc != nullptr && kb < kb0 + nk && ai < nw) ? __ldg(asrc + ai) : 0ull;
    };
    uint64_t pa[kPf];
#pragma unroll
    for (int i = 0; i < kPf; ++i) pa[i] = load_a(kb0 + grp + 2 * i);
    const uint32_t alane = (uint32_t)(32 * q) << 16;
    const uint32_t woff = (uint32_t)(r * KB);
    const int swz = r & 7;
    for (int i0 = 0; grp + 2 * i0 < nk; i0 += kPf) {
#pragma unroll
      for (int d = 0; d < kPf; ++d) {
        const int k = grp + 2 * (i0 + d);
        if (k >= nk) break;
        const int kb = kb0 + k;
        const int s = k % kStages;
        if (k >= kStages &&
            !__all_sync(kFull, mbar_wait(&sh->empty[s], (uint32_t)((k / kStages - 1) & 1), failed)))
          break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // activation row m, K-elements 64 j2 .. 64 j2 + 63 -> 16 TMEM columns
        // (rows >= M hold whatever: their outputs are never read; K-elements
        // past K_in meet zero weights)
        tmem_store_row64(tmem + alane + (uint32_t)(kAccCols + kStageCols * s + 16 * j2), pa[d]);
        // weight row r -> shared memory; elements at K >= K_in are 0
        if (wsrc != nullptr) {
          uint8_t* row = base + s * B_BYTES + woff;
          const uint32_t x[4] = {pw[d].x, pw[d].y, pw[d].z, pw[d].w};
          const int valid = Kin - KB * kb;
          if (valid >= KB) {
#pragma unroll
            for (int c = 0; c < 8; ++c)
              *reinterpret_cast<uint4*>(row + 16 * (c ^ swz)) = chunk16(x[c >> 1] >> (16 * (c & 1)));
          } else {
#pragma unroll
            for (int c = 0; c < 8; ++c)
              *reinterpret_cast<uint4*>(row + 16 * (c ^ swz)) =
                  chunk16_masked(x[c >> 1] >> (16 * (c & 1)), valid - 16 * c);
          }
        }
        pw[d] = load_w(kb + 2 * kPf);
        pa[d] = load_a(kb + 2 * kPf);
        // TMEM stores complete, shared-memory stores ordered for the async
        // proxy, then one arrival per warp
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->full[s]);
      }
      if (__any_sync(kFull, *failed != 0)) break;
    }
  } else if (threadIdx.x == kProducers) {
    // ---------------- MMA issuer (lane 0 of the last warp) ----------------
    for (int k = 0; k < nk; ++k) {
      const int s = k % kStages;
      if (!mbar_wait(&sh->full[s], (uint32_t)((k / kStages) & 1), failed)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint64_t bd = smem_desc(smem_u32(base + s * B_BYTES));
      const uint32_t ta = tmem + (uint32_t)(kAccCols + kStageCols * s);
#pragma unroll
      for (int j = 0; j < KB / 32; ++j)   // K = 32 per MMA: 8 TMEM columns, +2 in the B address field
        mma_f8_tmem_a(tmem, ta + 8 * j, bd + 2 * j, (k > 0 || j > 0) ? 1u : 0u);
      mma_commit(&sh->empty[s]);
    }
    if (nk > 0 && !*failed) mma_commit(&sh->done);
  }

  // ---------------- partial accumulator -> shared-memory slices ----------------
  // (the stages are free: every MMA that read them has completed).  Slice r
  // holds columns 64 r .. 64 r + 63 of every pattern row as 16-bit lanes
  // offset by kOff, two per 32-bit word.
  uint8_t* slices = base;
  if (threadIdx.x == 0 && M > 0)
    mbar_arrive_tx(&sh->red, (uint32_t)((kSplit - 1) * M * kSliceRow));
  if (threadIdx.x < kProducers) {
    bool go = nk > 0 && !*failed && mbar_wait(&sh->done, 0, failed);
    go = __all_sync(kFull, go);   // tcgen05.ld is warp-collective
    if (go) asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int sub = warp & 3;     // TMEM lanes 32 sub .. 32 sub + 31
    const int mrow = 32 * sub + lane;
    const int dst = warp >> 2;    // this warp's 64 columns belong to cluster CTA dst
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int col0 = 64 * dst + 32 * hh;
      uint32_t v[32];
      if (go) {
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
            "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
              "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
              "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),
              "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
              "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),
              "=r"(v[31])
            : "r"(tmem + ((uint32_t)(32 * sub) << 16) + (uint32_t)col0));
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = 0u;  // empty K range (or a failed wait): 0
      }
      if (mrow < M) {
        uint32_t pk[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          pk[j] = (((uint32_t)__float2int_rn(__uint_as_float(v[2 * j])) + kOff) & 0xFFFFu) |
                  (((uint32_t)__float2int_rn(__uint_as_float(v[2 * j + 1])) + kOff) << 16);
        uint4* out = reinterpret_cast<uint4*>(slices + dst * kSliceBytes + mrow * kSliceRow +
                                              2 * (32 * hh));
#pragma unroll
        for (int c = 0; c < 4; ++c) out[c] = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
      }
    }
  }
  // the slices are visible to the bulk-copy proxy, and every CTA of the
  // cluster has written its own slice before anyone adds into it
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  cluster_sync_all();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

  // ---------------- push the three foreign slices to their owners ----------------
  // (one thread in each of three warps, so the three bulk copies are issued
  // together)
  if (lane == 0 && warp >= 1 && warp < kSplit && M > 0) {
    {
      const uint32_t peer = (rank + (uint32_t)warp) % kSplit;
      const uint32_t src = smem_u32(slices + peer * kSliceBytes);
      const uint32_t dstp = peer_addr(src, peer);  // the owner's own slice, same offset
      const uint32_t bar = peer_addr(smem_u32(&sh->red), peer);
      asm volatile(
          "cp.reduce.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes.add.u32 "
          "[%0], [%1], %2, [%3];"
          ::"r"(dstp), "r"(src), "r"((uint32_t)(M * kSliceRow)), "r"(bar) : "memory");
    }
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
  }

  // ---------------- this CTA's 64 neurons: z, sign bits ----------------
  if (threadIdx.x < kProducers) {
    // waited for even after a failure elsewhere: the peers always push their
    // three slices, and this CTA must outlive those writes into its memory
    const bool ok = M > 0 && mbar_wait(&sh->red, 0, &sh->red_failed) && !*failed;
    const int mrow = threadIdx.x >> 2;             // pattern row
    const int c16 = 16 * (threadIdx.x & 3);        // 16 of the slice's 64 columns
    const int nf = n0 + kCols * (int)rank + c16;   // first neuron of the 16
    if (ok && mrow < M) {
      const uint4* in = reinterpret_cast<const uint4*>(slices + rank * kSliceBytes + mrow * kSliceRow +
                                                       2 * c16);
      int zz[16];
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const uint4 v = in[c];
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          zz[8 * c + 2 * e] = (int)(w4[e] & 0xFFFFu) - (int)(kSplit * kOff);
          zz[8 * c + 2 * e + 1] = (int)(w4[e] >> 16) - (int)(kSplit * kOff);
        }
      }
      int16_t* zrow = Ly.Z + (int64_t)mrow * N;
      uint32_t bits = 0, zp[8];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int z = zz[j];
        if (nf + j < N && z >= 0) bits |= 1u << j;
        if (j & 1) zp[j >> 1] |= (uint32_t)(z & 0xFFFF) << 16;
        else zp[j >> 1] = (uint32_t)(z & 0xFFFF);
      }
      if ((N & 7) == 0 && nf + 16 <= N) {
        // the 16 pre-activations are 32 contiguous, 16-byte aligned bytes
        uint4* zv = reinterpret_cast<uint4*>(zrow + nf);
        zv[0] = make_uint4(zp[0], zp[1], zp[2], zp[3]);
        zv[1] = make_uint4(zp[4], zp[5], zp[6], zp[7]);
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (nf + j < N) zrow[nf + j] = (int16_t)(zp[j >> 1] >> (16 * (j & 1)));
      }
      if ((nf >> 4) < 4 * Ly.nw_out)   // pad groups of the last word get 0 bits
        reinterpret_cast<uint16_t*>(Ly.A + (int64_t)mrow * Ly.nw_out)[nf >> 4] = (uint16_t)bits;
    }
  }
  // outgoing bulk reads done before the shared memory goes away
  if (lane == 0 && warp >= 1 && warp < kSplit && M > 0)
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (threadIdx.x == 0 && (*failed || sh->red_failed)) atomicAdd(&P->ctrl->timeouts, 1u);
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
}

}  // namespace
}  // namespace bk
