// bmlp_internal.cuh -- device-side data layout and shared device helpers of the
// BMLP library (fully binary training rule of arXiv 2412.00119, Alg. 1-3).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/bmlp.h"

namespace bk {

// ---------------------------------------------------------------------------
// HBM layout of one layer l (K_in = K_{l-1}, K_out = K_l):
//   H    uint32 [K_out][ldh]     hidden weights, neuron-major, bit-sliced: a weight h
//                                 (odd, |h| <= h_max) is stored as its lattice index
//                                 u = (h + h_max)/2 in [0, h_max], a CP or R event
//                                 moves u by +-1 with clamping, and h > 0 iff
//                                 u >= (h_max + 1)/2.  Inputs are grouped by 32:
//                                 group g of row k (inputs 32 g .. 32 g + 31) is
//                                 nplanes words, word p holding bit p of u of the 32
//                                 weights (bit j <-> input 32 g + j); nbits planes are
//                                 used (the bits of h_max), nplanes = nbits rounded
//                                 up to a power of two (unused planes 0); ldh =
//                                 ngrp * nplanes rounded up to a multiple of 4 words
//                                 (16-byte rows).  Inputs i >= K_in hold u = 0 and
//                                 are never stepped
//   W    uint64 [K_out][nw_in]    packed sign(H), bit (i%64) of word i/64 = (h_ik > 0)
//   PT   uint64 [c][nw_out]       packed P_l^T, bit (k%64) of word k/64 = (rho_kj > 0)
//   rho  int8  [K_out][c]         P_l itself, for the stability rho_{k,y}
//   rhoT int8  [c][K_out]         the same, class-major
//   Z    int16 [bs][K_out]        pre-activations of the current mini-batch
//   A    uint64 [bs][nw_out]      packed activations a_l of the current mini-batch
//   mark uint8 [bs]               1 iff the pattern is in M_l
//   sel  int16 [G][bs]            selected neuron per (group, pattern), -1 = none
// ---------------------------------------------------------------------------
struct DevLayer {
  uint32_t* H;
  uint64_t* W;
  uint64_t* PT;
  int8_t* rho;
  int8_t* rhoT;       // [c][K_out]: rho transposed (class-major), for the selection
  int16_t* Z;
  uint64_t* A;
  uint8_t* mark;
  int16_t* sel;       // [G][bs] selected neuron per group and pattern, or -1 (group-major)
  int16_t* member;    // [K_out] group order (neuron at position j), or null: contiguous groups
  int16_t* group_of;  // [K_out] group of neuron k (with member)
  int32_t Kin, Kout, nw_in, nw_out, ldh, gamma, G;
  int32_t ngrp;          // groups of 32 inputs per neuron row (ceil(K_in / 32))
  int32_t ev_cta_base;   // first CTA of this layer in the event-draw grid
  int32_t row_base;      // first row of this layer in the update's row numbering
  int32_t nblk;          // blocks of 64 inputs per neuron row (ceil(K_in / 64))
  uint64_t* EV;          // [K_out][ev_stride] reinforcement events of the current step,
                         // bit i % 64 of word i / 64 = input i reinforced
  int32_t ev_stride;     // words per EV row: nblk rounded up to even (16-byte rows)
};

// Device-resident step control.  The update kernel's last CTA advances t and s
// and clears the per-step flags, so that one captured graph replays step after
// step without host involvement.
struct Ctrl {
  unsigned long long t;         // global mini-batch counter since creation
  unsigned long long err;       // last-layer 01-loss count since the last epoch end
  unsigned long long bad_labels;// labels outside 0..c-1 seen by the kernels
  uint32_t s;                   // mini-batch index within the current train call
  uint32_t done;                // CTAs of the update kernel finished this step
  uint32_t timeouts;            // bounded device waits that expired (BMLP_ETIMEOUT)
  uint32_t upd_next;            // next row for the update kernel's warps this step
  uint32_t any_mark[BMLP_MAX_LAYERS];
  // update-kernel statistics, accumulated until read with reset
  unsigned long long upd_rows;       // neuron rows visited (layers with M_l non-empty)
  unsigned long long upd_streamed;   // rows streamed (at least one CP tuple)
  unsigned long long upd_bytes;      // algorithmic bytes: H read + write and W write of the
                                     // streamed rows, the planes of a group read + written
                                     // per group with an event of a row without tuple
  unsigned long long layer_err[BMLP_MAX_LAYERS];  // local 01-loss count of each layer
};

// Thresholds of the reinforcement sampler of one layer (Alg. 3 l.5-12): the
// events of a neuron row are drawn per block of 64 inputs (the last block
// holds K_in mod 64 when that is not 0).  For a block of n inputs:
//   any      = thr(1 - (1-q)^n)        at least one event iff the block draw < any
//   first[j] = thr((1 - (1-q)^(j+1)) / (1 - (1-q)^n))   first event: least j with V < first[j]
//   gap[g]   = thr(1 - (1-q)^(g+1))    next event p + 1 + g: least g <= n-2-p with V < gap[g]
// thr(x) = ceil(x 2^32) (0 for x <= 0, 2^32 for x >= 1); (1-q)^m a left-to-right
// IEEE product.  Index [0]: n = 64, [1]: the last, shorter block.
struct RTables {
  unsigned long long any[2];
  unsigned long long first[2][64];
  unsigned long long gap[64];       // entries g < 63 (independent of n)
};

struct StepParams {
  DevLayer layer[BMLP_MAX_LAYERS];
  const uint64_t* x;            // packed inputs of the current train call
  const int32_t* y;             // labels of the current train call
  int64_t n;                    // patterns in the current train call
  const RTables* rt;            // [L] reinforcement sampler thresholds
  int32_t nblk_max;             // max over layers of ceil(K_in / 64)
  Ctrl* ctrl;
  int32_t L, c, bs, h_max, r_num, r_den, nw0, upd_ctas_total, ev_ctas_total;
  int32_t rows_total;           // sum of K_l over the layers (update rows)
  int32_t nbits, nplanes;       // bit-planes of H used / stored per group (see H above)
  uint32_t key0, key1;          // Philox key = (seed mod 2^32, seed div 2^32)
};


constexpr int kClsThreads = 512;

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), device version.
// Counter layout of the library's random streams (purpose tag in c2):
//   initial h_ik of layer l : (i/4, k, 1*2^16 + l, 0)   word i%4, +1 iff bit 31
//   rho_kj of P_l           : (j/4, k, 2*2^16 + l, 0)   word j%4, +1 iff bit 31
//   block draw U of block b (inputs 64b .. 64b+63) of neuron k at step t:
//                             (b/4, k, 3*2^16 + l, t)   word b%4
//   event draws V_0, V_1, .. of that block: words 0..3 of (b, k, (4+r)*2^16 + l, t),
//                             r = 0, 1, ..
//   group-order key u_k of neuron k: (k/4, 0, 32*2^16 + l, t')   word k%4
//   expansion weight e_ki   : (i/4, k, 33*2^16, 0)      word i%4, +1 iff bit 31
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 ctr, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)0xD2511F53u * ctr.x;  // one wide multiply each
    const uint64_t p1 = (uint64_t)0xCD9E8D57u * ctr.z;
    ctr = make_uint4((uint32_t)(p1 >> 32) ^ ctr.y ^ (k0 + (uint32_t)r * 0x9E3779B9u), (uint32_t)p1,
                     (uint32_t)(p0 >> 32) ^ ctr.w ^ (k1 + (uint32_t)r * 0xBB67AE85u), (uint32_t)p0);
  }
  return ctr;
}

// Programmatic dependent launch: a kernel launched with the
// programmatic-stream-serialization attribute may start while the kernel
// before it in the stream is still running.  pdl_wait() returns once that
// kernel has completed and its memory is visible (at once without the
// attribute); pdl_trigger() lets the next kernel start launching.  Every
// kernel that triggers does so only after its own wait, so when a kernel
// starts, every kernel two or more launches before it has completed.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch with or without the programmatic-stream-serialization attribute.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                          bool pdl, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k, args...);
}

__device__ __forceinline__ int clip_h(int h, int h_max) {
  return h > h_max ? h_max : (h < -h_max ? -h_max : h);
}

// ---------------------------------------------------------------------------
// Kernels
// ---------------------------------------------------------------------------
// Forward of layer l (1-based) for the current training mini-batch.
__global__ void k_train_forward(const StepParams* P, int l);
// Local classifier, 01-loss, margin, marks, and the group selection, all layers.
__global__ void k_cls_select(const StepParams* P);
// Group order of every layer with a random partition (DevLayer::member /
// group_of); redraw: keyed by the current step (else by step 0).
cudaError_t prepare_group_order(int max_K);  // shared-memory attribute, once
cudaError_t launch_group_order(int L, int max_K, bool redraw, cudaStream_t st, const StepParams* P);
// Reinforcement events of every neuron row of every layer for the current
// step into DevLayer::EV (Alg. 3 l.5-12); grid = P->ev_ctas_total CTAs.
void launch_r_events(unsigned grid, cudaStream_t st, const StepParams* P, uint32_t key0,
                     uint32_t key1);
constexpr int kEvRowsPerCta = 4;   // one warp per row
constexpr int kEvThreads = 32 * kEvRowsPerCta;
// Generic forward for evaluation: A (M x nw_in) against W -> Aout (M x nw_out).
__global__ void k_forward_eval(const uint64_t* __restrict__ A, int64_t M, int nw_in,
                               const uint64_t* __restrict__ W, int N, int Kin,
                               uint64_t* __restrict__ Aout, int nw_out);
// Final classifier argmax for evaluation.
__global__ void k_predict_out(const uint64_t* __restrict__ A, int64_t M, int nw,
                              const uint64_t* __restrict__ PT, int c, int K,
                              int32_t* __restrict__ out);
// Initialisation of H, W of one layer and rho, PT.
__global__ void k_init_hw(uint32_t* H, uint64_t* W, int Kin, int Kout, int ldh, int ngrp, int nplanes,
                          int l, uint32_t key0, uint32_t key1, int h_max);
__global__ void k_init_rho(int8_t* rho, int Kout, int c, int l, uint32_t key0, uint32_t key1);
__global__ void k_pack_pt(const int8_t* rho, uint64_t* PT, int Kout, int c, int nw_out);
__global__ void k_transpose_rho(const int8_t* rho, int8_t* rhoT, int Kout, int c);
// Re-derive W from H for one layer (after set_state).
__global__ void k_repack_w(const uint32_t* H, uint64_t* W, int Kin, int Kout, int ldh, int ngrp,
                           int nplanes, int h_max);
// Tensor-core forward (tcgen05, +-1 as e4m3, exact fp32 sums), training layer l;
// needs bs <= 128.  The activations of layer l - 1 (the inputs for l = 1) are
// read as packed bits.
size_t train_forward_tc_smem();
cudaError_t prepare_train_forward_tc();
// pdl: launched with the programmatic-stream-serialization attribute.
cudaError_t launch_train_forward_tc(int Kout, cudaStream_t st, bool pdl, const StepParams* P, int l);
// Median binarisation of n x K fp32 patterns into n x nw packed words.
void launch_binarize_median(const float* x, int64_t n, int K, int nw, uint64_t* out,
                            cudaStream_t st);
// Expansion layer for uint8 inputs: E (K x ceil(D/64) words) from the
// expansion-weight stream, and out = packed sign(x E^T) (n x ceil(K/64)).
void launch_expand_weights(uint64_t seed, int K, int D, uint64_t* E, cudaStream_t st);
void launch_expand_sign(const uint8_t* x, int64_t n, int D, const uint64_t* E, int K,
                        uint64_t* out, cudaStream_t st);
// Tensor-core forward for evaluation: A (M x nw_in) against W -> Aout
// (M x nw_out), 256-pattern x 256-neuron tiles per CTA pair; an expired
// bounded wait adds one to *timeouts.
cudaError_t prepare_forward_eval_tc();
// One CTA waiting (bounded by limit_cycles) on an mbarrier that completes only
// with arrive != 0; an expired wait adds one to *timeouts.
void launch_wait_probe(unsigned int* timeouts, int arrive, unsigned long long limit_cycles,
                       cudaStream_t st);
void launch_forward_eval_tc(const uint64_t* A, int64_t M, int nw_in, const uint64_t* W, int N,
                            int Kin, uint64_t* Aout, int nw_out, unsigned int* timeouts,
                            cudaStream_t st);

// One layer on the b1 mma.sync path (kern_forward_b1.cu): Aout (M x nw_out)
// = packed sign(A W^T), sign(0) = +1, pad bits 0.
cudaError_t launch_forward_b1(const uint64_t* A, int64_t M, int nw_in, const uint64_t* W, int N,
                              int Kin, uint64_t* Aout, int nw_out, cudaStream_t st);
// CP + R + repack of every layer with a non-empty M_l, then advance the step
// (kern_update_ws.cu): bulk copies into a ring of shared-memory slots, the
// bit-sliced steps by consumer warps; one CTA per SM (grid = the SM count).
// pdl: launched with the programmatic-stream-serialization attribute.
// nplanes: DevLayer's planes per group (StepParams::nplanes); bs: the
// mini-batch size (the tuple lists of the slot ring).
size_t update_ws_smem(int nplanes, int bs);
cudaError_t prepare_update_ws();
cudaError_t launch_update_ws(int nplanes, int h_max, int bs, unsigned grid, cudaStream_t st, bool pdl,
                             const StepParams* P);
// Attributes of the update kernel: fails when the library holds no sm_103a image.
cudaError_t update_kernel_image(cudaFuncAttributes* fa);
// Peak-rate kernel of one contraction engine (BMLP_FWD_*): launches it on
// `sms` SMs' worth of CTAs and returns the bit-pairs (MACs) it performs.
cudaError_t launch_engine_peak(int engine, int64_t iters, int sms, int* sink, unsigned int* timeouts,
                               cudaStream_t st, double* bitpairs);

// Launch helpers implemented in the kernel files (grid shapes live next to the
// kernels they describe).
dim3 train_forward_grid(int bs, int Kout);
dim3 train_forward_block();
dim3 eval_forward_grid(int64_t M, int Kout);
dim3 eval_forward_block();

}  // namespace bk
