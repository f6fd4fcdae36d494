// kern_forward_tc.cu -- tensor-core forward contraction of the BMLP
// (Alg. 1 l.8-9) on sm_103a with tcgen05.
//
//   z^mu_k = sum_i a^mu_i w_ik,  a, w in {-1, +1}
//
// is computed exactly as an e4m3 x e4m3 -> fp32 matrix product: +-1 are exact
// in e4m3 (0x38 / 0xB8), pad elements are 0x00, and every partial sum is an
// integer of magnitude <= K_in <= 2^20 < 2^24, exact in fp32 whatever the
// accumulation order.  One CTA owns TN = 64 neurons and all (<= 128) patterns:
//   - the bit-packed activations (A, patterns x words) and visible weights (W,
//     neurons x words) are expanded in shared memory, 128 K-elements (two
//     64-bit words) per row per stage, into the K-major SWIZZLE_128B layout the
//     MMA reads (16-byte chunk c of row r stored at chunk c ^ (r % 8));
//   - one thread issues tcgen05.mma.kind::f8f6f4 (M = 128, N = 64, K = 32) four
//     times per stage into a 128-lane x 64-column fp32 accumulator in TMEM and
//     commits to the stage's mbarrier, so the expansion of the next stages
//     overlaps the MMAs of the previous ones (4-stage ring);
//   - the epilogue reads the accumulator with tcgen05.ld (warp w % 4 owns TMEM
//     lanes 32 (w % 4) ..), converts to int, stores z (int16) and packs the sign
//     bits of 32 neurons per thread directly into the activation words.
// Every mbarrier wait is bounded; on expiry the kernel records the failure in
// the control block (host: BMLP_ETIMEOUT), releases its TMEM and returns.
#include "bmlp_internal.cuh"

namespace bk {
namespace {

constexpr int TM = 128;           // MMA M: patterns (rows >= bsz are zero)
constexpr int TN = 64;            // MMA N: neurons per CTA
constexpr int KB = 128;           // K elements (bytes) per stage and row
constexpr int STAGES = 4;
constexpr int THREADS = 256;
constexpr int A_BYTES = TM * KB;  // 16 KB
constexpr int B_BYTES = TN * KB;  // 8 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 64;
constexpr unsigned long long kWaitCycles = 4000000000ull;  // ~2 s at 2 GHz

struct __align__(8) TcShared {
  unsigned long long empty[STAGES];  // MMAs that read stage s completed
  unsigned long long done;           // all MMAs completed
  uint32_t tmem_base;
  int failed;
};

constexpr size_t kSmemBytes = 1024 /*alignment slack*/ + STAGES * STAGE_BYTES + sizeof(TcShared);

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(unsigned long long* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

// Bounded wait for the phase with the given parity; false on expiry.
__device__ __forceinline__ bool mbar_wait(unsigned long long* bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  const unsigned long long t0 = clock64();
  while (true) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok) : "r"(a), "r"(parity) : "memory");
    if (ok) return true;
    if (clock64() - t0 > kWaitCycles) return false;
  }
}

// Shared-memory matrix descriptor: K-major, SWIZZLE_128B, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);           // start address
  d |= (uint64_t)1 << 16;                              // leading byte offset (unused for SW128 K-major)
  d |= (uint64_t)(1024 >> 4) << 32;                    // stride byte offset
  d |= (uint64_t)1 << 46;                              // descriptor version (sm_100 family)
  d |= (uint64_t)2 << 61;                              // swizzle: 128B
  return d;
}

// Instruction descriptor, kind::f8f6f4: D fp32, A = B = e4m3, both K-major.
constexpr uint32_t kIdesc = (1u << 4)                  // D format: f32
                            | (0u << 7) | (0u << 10)   // A, B format: e4m3
                            | ((uint32_t)(TN >> 3) << 17)
                            | ((uint32_t)(TM >> 4) << 24);

__device__ __forceinline__ void mma_f8(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}"
      ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate));
}

__device__ __forceinline__ void mma_commit(unsigned long long* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
               ::"r"(smem_u32(bar)) : "memory");
}

// 4 activation bits -> 4 e4m3 bytes (+1 = 0x38, -1 = 0xB8).  Byte j of the
// product keeps bit j; adding (0x80 - 2^j) per byte moves it to bit 7 without
// carries between bytes.
__device__ __forceinline__ uint32_t expand4(uint32_t nib) {
  const uint32_t m = (nib * 0x01010101u) & 0x08040201u;
  const uint32_t t = m + 0x787C7E7Fu;
  return (t & 0x80808080u) ^ 0xB8B8B8B8u;
}

// Expand one 64-bit word (64 K-elements) into 64 bytes = four 16-byte chunks
// of a swizzled row.  `valid` = number of valid elements in the word (0..64).
__device__ __forceinline__ void expand_word(uint8_t* row_base, int r, int chunk0, uint64_t w,
                                            int valid) {
  const uint32_t lo = (uint32_t)w, hi = (uint32_t)(w >> 32);
#pragma unroll
  for (int q = 0; q < 4; ++q) {        // chunk q: elements 16q .. 16q+15
    const uint32_t bits = (q < 2 ? lo : hi) >> (16 * (q & 1));
    uint4 v;
    v.x = expand4(bits & 0xF);
    v.y = expand4((bits >> 4) & 0xF);
    v.z = expand4((bits >> 8) & 0xF);
    v.w = expand4((bits >> 12) & 0xF);
    if (valid < 64) {
      const int e0 = 16 * q;
      uint32_t* vv = &v.x;
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int n_ok = valid - (e0 + 4 * b);  // valid elements in this 4-byte group
        const uint32_t keep = n_ok >= 4 ? 0xFFFFFFFFu : (n_ok <= 0 ? 0u : ((1u << (8 * n_ok)) - 1u));
        vv[b] &= keep;
      }
    }
    const int c = chunk0 + q;
    *reinterpret_cast<uint4*>(row_base + 16 * (c ^ (r & 7))) = v;
  }
}

// Expand rows [0, rows) of a bit-packed matrix (row stride nw words) for the
// K-block starting at element k0 into a swizzled stage of `cap` rows.
__device__ __forceinline__ void expand_block(uint8_t* stage, const uint64_t* __restrict__ src,
                                             int64_t rows, int nw, int k0, int Kin) {
  const int w0 = k0 >> 6;  // first of the block's two words
  for (int idx = threadIdx.x; idx < rows * 2; idx += THREADS) {
    const int r = idx >> 1, half = idx & 1;
    const int wi = w0 + half;
    const int valid = min(64, max(0, Kin - 64 * wi));
    const uint64_t w = (wi < nw && valid > 0) ? __ldg(src + (int64_t)r * nw + wi) : 0ull;
    expand_word(stage + r * KB, r, 4 * half, w, valid);
  }
}

}  // namespace

size_t train_forward_tc_smem() { return kSmemBytes; }
dim3 train_forward_tc_grid(int Kout) { return dim3((unsigned)((Kout + TN - 1) / TN)); }
dim3 train_forward_tc_block() { return dim3(THREADS); }

__global__ void __launch_bounds__(THREADS, 1) k_train_forward_tc(const StepParams* __restrict__ P, int l) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  TcShared* sh = reinterpret_cast<TcShared*>(base + STAGES * STAGE_BYTES);
  const DevLayer& Ly = P->layer[l - 1];
  const int64_t start = (int64_t)P->ctrl->s * P->bs;
  const int64_t rem = P->n - start;
  const int M = (int)(rem < P->bs ? rem : P->bs);
  const uint64_t* A = (l == 1) ? P->x + start * P->nw0 : P->layer[l - 2].A;
  const int n0 = blockIdx.x * TN;
  const int N = Ly.Kout, Kin = Ly.Kin, nw = Ly.nw_in;
  const int nkb = (Kin + KB - 1) / KB;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const int NB = min(TN, N - n0);  // neuron rows of this CTA
  // zero the pattern rows >= M and neuron rows >= NB of every stage once; the
  // expansion never writes them, so they stay zero (0 * anything = 0)
  for (int s = 0; s < STAGES; ++s) {
    uint4* a4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES);
    for (int i = M * (KB / 16) + threadIdx.x; i < TM * (KB / 16); i += THREADS)
      a4[i] = make_uint4(0, 0, 0, 0);
    uint4* b4 = reinterpret_cast<uint4*>(base + s * STAGE_BYTES + A_BYTES);
    for (int i = NB * (KB / 16) + threadIdx.x; i < TN * (KB / 16); i += THREADS)
      b4[i] = make_uint4(0, 0, 0, 0);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(&sh->empty[s], 1);
    mbar_init(&sh->done, 1);
    sh->failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&sh->tmem_base)), "r"(TMEM_COLS) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = sh->tmem_base;

  bool ok = true;
  for (int kb = 0; kb < nkb; ++kb) {
    const int s = kb % STAGES;
    uint8_t* sa = base + s * STAGE_BYTES;
    uint8_t* sb = sa + A_BYTES;
    if (kb >= STAGES) {
      if (!mbar_wait(&sh->empty[s], (uint32_t)((kb / STAGES - 1) & 1))) ok = false;
    }
    if (__syncthreads_or(!ok)) { ok = false; break; }
    expand_block(sa, A, M, nw, kb * KB, Kin);
    expand_block(sb, Ly.W + (int64_t)n0 * nw, NB, nw, kb * KB, Kin);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint64_t ad = smem_desc(smem_u32(sa));
      const uint64_t bd = smem_desc(smem_u32(sb));
#pragma unroll
      for (int j = 0; j < KB / 32; ++j)   // K = 32 bytes per MMA: +2 in the address field
        mma_f8(tmem, ad + 2 * j, bd + 2 * j, (kb > 0 || j > 0) ? 1u : 0u);
      mma_commit(&sh->empty[s]);
    }
  }
  if (threadIdx.x == 0 && ok) mma_commit(&sh->done);
  if (ok && !mbar_wait(&sh->done, 0)) ok = false;
  if (__syncthreads_or(!ok)) {
    if (threadIdx.x == 0) atomicAdd(&P->ctrl->timeouts, 1u);
  } else {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    // epilogue: warp w reads lanes 32 (w % 4) .., columns 32 (w / 4) ..
    const int sub = warp & 3;
    const int col0 = 32 * (warp >> 2);
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
    const int m = 32 * sub + lane;
    uint32_t bits = 0;
    if (m < M) {
      int16_t* zrow = Ly.Z + (int64_t)m * N;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const int n = n0 + col0 + j;
        const int z = __float2int_rn(__uint_as_float(v[j]));
        if (n < N) {
          zrow[n] = (int16_t)z;
          if (z >= 0) bits |= 1u << j;
        }
      }
      reinterpret_cast<uint32_t*>(Ly.A + (int64_t)m * Ly.nw_out + (n0 >> 6))[col0 >> 5] = bits;
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
}

}  // namespace bk
