// kern_forward.cu -- CUDA-core forward contraction of the BMLP (Alg. 1 l.8-9).
//
//   z^mu_k = sum_i a^mu_i w_ik = K_in - 2 popcount(A[mu] XOR W[k])   (+-1 dot product)
//   a^mu_k = sign(z^mu_k), sign(0) = +1, packed 64 neurons per word.
//
// Both operands are bit-packed rows (A: patterns x words, W: neurons x words),
// pad bits 0 in both, so pads never count in the XOR.  One CTA computes a
// 64-pattern x 64-neuron tile; K is streamed in chunks of 16 words through a
// double-buffered, k-major shared-memory stage (stride 65 words, so that both
// the transposing stores and the broadcast loads are free of bank conflicts).
// Thread (ty, tx) owns patterns ty + 16 r and neurons tx + 16 c (r, c < 4), so
// a warp reads 16 consecutive W words and 2 A words per k step.  The epilogue
// writes Z (int16) and the sign bits: the 16 lanes that share a pattern OR
// their nibbles together with shuffles and one lane stores the 64-bit word.
#include "bmlp_internal.cuh"

namespace bk {
namespace {

constexpr int TM = 64;   // patterns per CTA tile
constexpr int TN = 64;   // neurons per CTA tile (one packed output word)
constexpr int KC = 16;   // words per K chunk
constexpr int NT = 256;  // threads
constexpr int SLD = 65;  // shared stride (words) of one k row of the stage

struct Stage {
  uint64_t a[KC][SLD];
  uint64_t w[KC][SLD];
};

__device__ __forceinline__ void load_chunk(const uint64_t* __restrict__ A, int64_t M, int nw,
                                           const uint64_t* __restrict__ W, int N, int64_t m0,
                                           int n0, int kc0, uint64_t (&ra)[4], uint64_t (&rw)[4]) {
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int v = threadIdx.x + NT * j;  // 0..511
    const int row = v >> 3;
    const int col = (v & 7) * 2;
    const int64_t gm = m0 + row;
    const int gn = n0 + row;
    const int gk = kc0 + col;
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const bool kin = (gk + e) < nw;
      ra[2 * j + e] = (gm < M && kin) ? __ldg(A + gm * nw + gk + e) : 0ull;
      rw[2 * j + e] = (gn < N && kin) ? __ldg(W + (int64_t)gn * nw + gk + e) : 0ull;
    }
  }
}

__device__ __forceinline__ void store_chunk(Stage& st, const uint64_t (&ra)[4],
                                            const uint64_t (&rw)[4]) {
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int v = threadIdx.x + NT * j;
    const int row = v >> 3;
    const int col = (v & 7) * 2;
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      st.a[col + e][row] = ra[2 * j + e];
      st.w[col + e][row] = rw[2 * j + e];
    }
  }
}

__device__ __forceinline__ int popc64(uint64_t x) {
  return __popc((uint32_t)x) + __popc((uint32_t)(x >> 32));
}

// One 64 x 64 output tile.  Z may be null (evaluation).
__device__ __forceinline__ void xnor_popc_tile(const uint64_t* __restrict__ A, int64_t M, int nw,
                                               const uint64_t* __restrict__ W, int N, int Kin,
                                               int16_t* __restrict__ Z, int ldz,
                                               uint64_t* __restrict__ Aout, int ldo, int64_t m0,
                                               int n0, Stage* st) {
  const int tx = threadIdx.x & 15;
  const int ty = threadIdx.x >> 4;
  int acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0;

  uint64_t ra[4], rw[4];
  const int nchunks = (nw + KC - 1) / KC;
  load_chunk(A, M, nw, W, N, m0, n0, 0, ra, rw);
  store_chunk(st[0], ra, rw);
  __syncthreads();
  for (int ch = 0; ch < nchunks; ++ch) {
    const int buf = ch & 1;
    if (ch + 1 < nchunks) load_chunk(A, M, nw, W, N, m0, n0, (ch + 1) * KC, ra, rw);
#pragma unroll
    for (int kk = 0; kk < KC; ++kk) {
      uint64_t a[4], w[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) a[r] = st[buf].a[kk][ty + 16 * r];
#pragma unroll
      for (int c = 0; c < 4; ++c) w[c] = st[buf].w[kk][tx + 16 * c];
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] += popc64(a[r] ^ w[c]);
    }
    if (ch + 1 < nchunks) store_chunk(st[buf ^ 1], ra, rw);
    __syncthreads();
  }

  // epilogue: z = K - 2 popc, sign bits packed per pattern
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int64_t m = m0 + ty + 16 * r;
    uint64_t bits = 0;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int n = n0 + tx + 16 * c;
      const int z = Kin - 2 * acc[r][c];
      if (n < N) {
        if (z >= 0) bits |= 1ull << (tx + 16 * c);
        if (Z != nullptr && m < M) Z[m * ldz + n] = (int16_t)z;
      }
    }
#pragma unroll
    for (int off = 1; off < 16; off <<= 1) bits |= __shfl_xor_sync(0xffffffffu, bits, off);
    if (tx == 0 && m < M) Aout[m * ldo + (n0 >> 6)] = bits;
  }
}

}  // namespace

dim3 train_forward_grid(int bs, int Kout) {
  return dim3((unsigned)((bs + TM - 1) / TM), (unsigned)((Kout + TN - 1) / TN));
}
dim3 train_forward_block() { return dim3(NT); }
dim3 eval_forward_grid(int64_t M, int Kout) {
  return dim3((unsigned)((M + TM - 1) / TM), (unsigned)((Kout + TN - 1) / TN));
}
dim3 eval_forward_block() { return dim3(NT); }

__global__ void __launch_bounds__(NT) k_train_forward(const StepParams* __restrict__ P, int l) {
  __shared__ Stage st[2];
  const DevLayer& Ly = P->layer[l - 1];
  const int64_t start = (int64_t)P->ctrl->s * P->bs;
  const int64_t rem = P->n - start;
  const int64_t bsz = rem < P->bs ? rem : P->bs;
  const uint64_t* A = (l == 1) ? P->x + start * P->nw0 : P->layer[l - 2].A;
  xnor_popc_tile(A, bsz, Ly.nw_in, Ly.W, Ly.Kout, Ly.Kin, Ly.Z, Ly.Kout, Ly.A, Ly.nw_out,
                 (int64_t)blockIdx.x * TM, (int)blockIdx.y * TN, st);
}

__global__ void __launch_bounds__(NT) k_forward_eval(const uint64_t* __restrict__ A, int64_t M,
                                                     int nw_in, const uint64_t* __restrict__ W,
                                                     int N, int Kin, uint64_t* __restrict__ Aout,
                                                     int nw_out) {
  __shared__ Stage st[2];
  xnor_popc_tile(A, M, nw_in, W, N, Kin, nullptr, 0, Aout, nw_out, (int64_t)blockIdx.x * TM,
                 (int)blockIdx.y * TN, st);
}

}  // namespace bk
