/*
 * bmlp.h -- C-ABI of the GB300 (sm_103a) library that trains and evaluates
 * binary multi-layer perceptrons (BMLPs) with the fully binary, gradient-free
 * rule of "Training multi-layer binary neural networks with random local binary
 * error signals" (arXiv 2412.00119).
 *
 * What the library computes (paper notation; layers l = 1..L, widths K_0..K_L,
 * c classes):
 *   - H_l (K_{l-1} x K_l) integer "hidden metaplastic" weights, W_l = sign(H_l)
 *     the visible binary weights, P_l (K_l x c) a fixed random +-1 local
 *     classifier per layer (Sec. 3.1);
 *   - per mini-batch of bs patterns (Alg. 1): z_l = a_{l-1} W_l, a_l = sign(z_l),
 *     yhat_l = a_l P_l, the 01-loss of Eq. 1 and the robustness margin tau of
 *     Alg. 1 l.13-15 marking the patterns M_l to learn from;
 *   - the layer-level selection of Alg. 2: per group of gamma neurons the
 *     perceptron with the negative stability z_k rho_{k,y} closest to 0;
 *   - the perceptron-level CP + R rule of Alg. 3 with hidden weights clipped to
 *     [-h_max, h_max], W_l re-derived and re-packed in the same pass;
 *   - the end-of-epoch rescale p_r <- p_r sqrt(E^e) (Alg. 1 l.21);
 *   - forward-only evaluation: argmax of a_L P_L (Sec. 3.1).
 * Conventions where the paper is silent: sign(0) = +1; argmax ties go to the
 * lowest class; groups are contiguous (neuron k in group k / gamma); tuples are
 * applied in ascending pattern order with clipping after each; LayerUpdate runs
 * only when M_l is non-empty; the reinforcement events are drawn per block
 * of 64 inputs from 32-bit Philox4x32-10 draws against integer thresholds
 * (bmlp_reinforce_tables).  Every result is an integer or a bit and is
 * reproducible bit for bit.
 *
 * Data formats
 *   packed +-1 vectors: a vector of K values is ceil(K/64) little-endian uint64
 *     words; bit j of word w is element 64 w + j; a set bit means +1; pad bits
 *     must be 0.  A batch of n vectors is n such rows, row after row.
 *   labels: int32 in 0..c-1.
 *   H (state export): int16, K_l rows of K_{l-1} (neuron-major: element
 *     [k * K_{l-1} + i] is h_{ik}), odd values in [-h_max, h_max].
 *   W (state export): uint64, K_l rows of ceil(K_{l-1}/64) words, bit = (h > 0).
 *   P (state export): int8, K_l rows of c values rho_{kj} in {-1, +1}.
 *
 * Pointers and streams
 *   Batch inputs and outputs (x_packed, labels, labels_out) may be device or
 *   host pointers; the library asks the CUDA runtime which.  Host buffers are
 *   staged through library-owned device buffers with cudaMemcpyAsync on the
 *   given stream (pinned host memory makes the copies asynchronous).  The
 *   caller owns every buffer it passes in and must keep it alive until the
 *   work on `cuda_stream` has completed; the library owns the model state.
 *   `cuda_stream` is a cudaStream_t (NULL = the legacy default stream).
 *   Calls are asynchronous on that stream, except those that return host
 *   values (n_errors_out, BMLP_EPOCH_END, bmlp_get_state, bmlp_set_state),
 *   which synchronise it.
 *
 * Errors
 *   Every int-returning call returns BMLP_OK (0) or a negative BMLP_E* code and
 *   never throws or aborts; bmlp_last_error() gives a one-line reason.  Labels
 *   outside 0..c-1 in device memory are not read out of bounds: the kernels
 *   count them, and the next call that synchronises returns BMLP_EINVAL.
 *
 * One handle is used by one host thread at a time.
 */
#ifndef BMLP_H_
#define BMLP_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BMLP_OK 0
#define BMLP_EINVAL (-1)   /* bad argument or bad label values */
#define BMLP_ENOMEM (-2)   /* device or host allocation failed */
#define BMLP_ECUDA (-3)    /* a CUDA runtime call or kernel launch failed */
#define BMLP_ETIMEOUT (-4) /* a bounded device-side wait gave up */
#define BMLP_ESTATE (-5)   /* state blob inconsistent with the model */
#define BMLP_ENODEV (-6)   /* no usable sm_103 device */

#define BMLP_MAX_LAYERS 16
#define BMLP_MAX_BS 1024
#define BMLP_MAX_CLASSES 1024

/* bmlp_train flags */
#define BMLP_EPOCH_END 1u  /* after these n patterns, close the epoch (Alg. 1 l.21) */

/* forward-contraction engines (hparams.fwd_impl) */
#define BMLP_FWD_AUTO 0     /* library's choice */
#define BMLP_FWD_POPC 1     /* CUDA-core XOR + popcount */
#define BMLP_FWD_TCGEN05 2  /* 5th-gen tensor cores, +-1 as e4m3, fp32 accumulate (exact) */
/* Further contraction units, measured by bmlp_engine_peak (and, for B1MMA,
 * bmlp_layer_forward_engine) for the engine comparison; training uses POPC or
 * TCGEN05.  tcgen05.mma.kind::i8 does not exist on sm_103a, so +-1 as int8 on
 * tensor cores is the legacy mma.sync path (S8MMA). */
#define BMLP_FWD_B1MMA 3    /* mma.sync m16n8k256 .b1 xor.popc (legacy tensor path) */
#define BMLP_FWD_S8MMA 4    /* mma.sync m16n8k32 .s8, +-1 as int8 (legacy tensor path) */

typedef struct bmlp bmlp_t;

/* Hyperparameters (Alg. 1 header).  Zero-initialise and set what you need:
 * a zero / negative field selects the paper's setting of Sec. 4.2. */
typedef struct bmlp_hparams {
  int32_t bs;            /* mini-batch size, 1..BMLP_MAX_BS; 0 -> 100 */
  int32_t r_num, r_den;  /* robustness r = r_num / r_den; r_den == 0 -> r = 1/4 */
  double p_r0;           /* initial reinforcement probability; < 0 -> 0.5 */
  const int32_t* gamma;  /* L group sizes, each dividing K_l; NULL -> Sec. 4.3 rule */
  int32_t fwd_impl;      /* BMLP_FWD_*; 0 -> auto */
  int32_t group_mode;    /* BMLP_GROUPS_*: group membership of Alg. 2 (Sec. 4.3); 0 -> contiguous */
} bmlp_hparams;

/* Group membership (Sec. 4.3: by the permutation symmetry of a hidden layer
 * its groups may be any fixed random partition, or one redrawn at every
 * step).  CONTIGUOUS: group g = neurons g*gamma .. (g+1)*gamma - 1.  FIXED /
 * RESHUFFLED: order the neurons k of layer l by the key u_k = word k%4 of
 * Philox4x32-10 at counter (k/4, 0, 32*2^16 + l, t') with the model's key,
 * ties to the smaller k; group g = the neurons at positions g*gamma ..
 * (g+1)*gamma - 1 of that order, with t' = 0 (FIXED) or t' = the step counter
 * (RESHUFFLED, a new partition every mini-batch).  Within a group the easiest
 * neuron is chosen with ties to the lowest neuron index.  FIXED and
 * RESHUFFLED need every K_l <= 16384. */
#define BMLP_GROUPS_CONTIGUOUS 0
#define BMLP_GROUPS_FIXED 1
#define BMLP_GROUPS_RESHUFFLED 2

/* Create a model and initialise H_l, P_l uniformly on {+-1} from `seed`
 * (Alg. 1 l.2).  widths: K_0..K_L (n_widths = L + 1, 2..BMLP_MAX_LAYERS + 1,
 * each 1..32767); classes: 2..BMLP_MAX_CLASSES; h_max: odd, 1..16383 (255 = 8-bit
 * hidden weights, Table 4); hp may be NULL (paper defaults).  Allocates the
 * model state on the current CUDA device.  On success *out owns it. */
int bmlp_create(const int32_t* widths, int32_t n_widths, int32_t classes, int16_t h_max,
                uint64_t seed, const bmlp_hparams* hp, bmlp_t** out);

/* Free the model (synchronises the device first).  NULL is accepted. */
void bmlp_destroy(bmlp_t* h);

/* One pass of NetworkUpdate (Alg. 1 l.4-20) over n patterns in the given
 * order, in mini-batches of bs (a last shorter batch is processed as a batch of
 * its own size).  x_packed: n packed rows of K_0 bits; labels: n int32.
 * flags & BMLP_EPOCH_END: afterwards set E = (last-layer 01-loss count since the
 * previous epoch end) / (patterns since then) and p_r <- p_r sqrt(E).
 * n_errors_out (host, may be NULL): last-layer 01-loss count of these n
 * patterns, measured in the training forward pass.  n == 0 is a no-op.
 * If a bounded device-side wait of a training forward pass expires (tensor-
 * core engine), that mini-batch and every later one until the expiry is
 * reported change neither H nor W (no marks, no update; the step counter
 * still advances); the next call that synchronises returns BMLP_ETIMEOUT. */
int bmlp_train(bmlp_t* h, const uint64_t* x_packed, const int32_t* labels, int64_t n,
               uint32_t flags, void* cuda_stream, int64_t* n_errors_out);

/* Forward-only evaluation (Sec. 3.1): labels_out[mu] = argmax_j (a_L P_L)_{mu j}
 * (lowest index on ties) for n packed rows of K_0 bits.  Does not change state.
 * With device x_packed and labels_out the call does not synchronise, and an
 * expired bounded device wait (tensor-core engine) is reported by the next
 * call that does (BMLP_ETIMEOUT). */
int bmlp_predict(bmlp_t* h, const uint64_t* x_packed, int64_t n, int32_t* labels_out,
                 void* cuda_stream);

/* Early-exit evaluation (Sec. 3.1: after training, the intermediate random
 * classifiers P_l may serve early-exit strategies).  For every layer
 * l = 1..L: labels_out[(l-1) n + mu] = argmax_j of yhat_l = a_l P_l for
 * pattern mu (ties to the lowest class), a_l from the same forward pass as
 * bmlp_predict; row L equals bmlp_predict's output.  x_packed: as for
 * bmlp_predict; labels_out: L x n int32, layer-major, caller-owned, host or
 * device.  Asynchronous on cuda_stream when both pointers are device
 * pointers; synchronises otherwise.  Errors as bmlp_predict. */
int bmlp_predict_layers(bmlp_t* h, const uint64_t* x_packed, int64_t n, int32_t* labels_out,
                        void* cuda_stream);

/* Local error counts (Eq. 1 for every layer, Alg. 1 l.12): errs_out[l-1] =
 * the number of training patterns whose layer-l local 01-loss was 1 in their
 * training forward pass (the weights of their mini-batch before its update),
 * counted since creation or the last reset; errs_out[L-1] counts what
 * bmlp_train's n_errors_out reports.  errs_out: host, L values.  Synchronises
 * the device; reset != 0 sets the counters to 0 after reading them.  The
 * counters are not part of the state that bmlp_get_state / bmlp_set_state
 * carry. */
int bmlp_layer_errors(bmlp_t* h, int64_t* errs_out, int32_t reset);

/* MedianBinarization (Alg. 1 l.5; Sec. 3.2: the median value is the
 * threshold) of real-valued patterns, for data that is not already +-1:
 * bit i of pattern mu is 1 (+1) iff x[mu][i] > m_mu, where m_mu is the
 * ceil(K/2)-th smallest of the pattern's K values (its lower median) and the
 * comparison is made in fp32 (-0 and +0 are equal); else 0 (-1).  Pad bits
 * are 0, so the output is bmlp_train / bmlp_predict input for K_0 = K.
 *   x: device, n x K fp32, row-major, 4-byte aligned, finite values (a NaN
 *      ranks by its bit pattern and compares false); caller-owned.
 *   out: device, n x ceil(K/64) words, 8-byte aligned, caller-owned.
 * Needs no handle (errors read with bmlp_last_error(NULL)); asynchronous on
 * cuda_stream.  BMLP_EINVAL for n < 0, K < 1, NULL, host or misaligned
 * pointers; BMLP_ECUDA if the launch fails. */
int bmlp_binarize_median(const float* x, int64_t n, int32_t K, uint64_t* out, void* cuda_stream);

/* Weights of a fixed random expansion layer (Sec. 3.2, footnote to the
 * binarisation step: a fixed random input layer with weights in {+-1} and
 * sign activation lets the BMLP take non-binary inputs directly):
 * e_k,i = +1 iff bit 31 of word i%4 of Philox4x32-10 at counter
 * (i/4, k, 33*2^16, 0) with key (seed mod 2^32, seed div 2^32), else -1.
 *   E_out: device, K x ceil(D/64) words (bit i % 64 of word i / 64 of row k
 *          = 1 <-> e_k,i = +1; pad bits 0), 8-byte aligned, caller-owned.
 * No handle (errors: bmlp_last_error(NULL)); asynchronous on cuda_stream.
 * BMLP_EINVAL for K < 1, D < 1, D > 2^23, NULL, host or misaligned E_out. */
int bmlp_expand_weights(uint64_t seed, int32_t K, int32_t D, uint64_t* E_out, void* cuda_stream);

/* The expansion layer itself, for unsigned 8-bit inputs (pixel
 * intensities): bit k of pattern mu is 1 (+1) iff
 * sum_i x[mu][i] e_k,i >= 0 (sign(0) = +1, as for every activation), the
 * sum taken exactly in integers; else 0 (-1).  Pad bits are 0, so the output
 * is bmlp_train / bmlp_predict input for K_0 = K.
 *   x: device, n x D uint8, row-major (row mu at x + mu D), caller-owned;
 *      any alignment.
 *   E: device, K x ceil(D/64) words as written by bmlp_expand_weights (any
 *      +-1 matrix in that layout; pad bits ignored), 8-byte aligned.
 *   out: device, n x ceil(K/64) words, 8-byte aligned, caller-owned.
 * No handle (errors: bmlp_last_error(NULL)); asynchronous on cuda_stream.
 * BMLP_EINVAL for n < 0, K < 1, D < 1, D > 2^23 (the int32 sum bound),
 * NULL, host or misaligned pointers; BMLP_ECUDA if the launch fails. */
int bmlp_expand_sign(const uint8_t* x, int64_t n, int32_t D, const uint64_t* E, int32_t K,
                     uint64_t* out, void* cuda_stream);

/* One layer of forward-only evaluation (Sec. 3.1; Alg. 1 l.8-9):
 * a_out = sign(a_in W_l), sign(0) = +1, for n packed rows.  a_in: n rows of
 * ceil(K_{l-1}/64) words (pad bits 0); a_out: n rows of ceil(K_l/64) words,
 * written with pad bits 0.  Both must be device pointers (else BMLP_EINVAL).
 * Runs the engine bmlp_predict uses for this handle; asynchronous on
 * cuda_stream.  An expired bounded device wait (tensor-core engine) is
 * reported by the next call that synchronises (BMLP_ETIMEOUT). */
int bmlp_layer_forward(bmlp_t* h, int32_t layer, const uint64_t* a_in, int64_t n,
                       uint64_t* a_out, void* cuda_stream);

/* bmlp_layer_forward on an engine chosen per call (the engine comparison of
 * the forward contraction, Alg. 1 l.8-9; Table 3 counts its XNOR/popcount
 * work): engine BMLP_FWD_POPC, BMLP_FWD_TCGEN05 or BMLP_FWD_B1MMA, whatever
 * the handle's own engine.  Same arguments, layouts and results as
 * bmlp_layer_forward (every engine gives the same bits); BMLP_EINVAL for
 * another engine (BMLP_FWD_S8MMA has no layer kernel). */
int bmlp_layer_forward_engine(bmlp_t* h, int32_t layer, int32_t engine, const uint64_t* a_in,
                              int64_t n, uint64_t* a_out, void* cuda_stream);

/* Copy layer `layer` (1..L) to host buffers (each may be NULL; formats above),
 * plus the current p_r and step counter t (mini-batches since creation). */
int bmlp_get_state(const bmlp_t* h, int32_t layer, int16_t* H_out, uint64_t* W_out,
                   int8_t* P_out, double* p_r_out, int64_t* step_out);

/* Resume: load H of layer `layer` (host, format above; NULL keeps it) and
 * re-derive W from it; set p_r and the step counter (step < 0 keeps both).
 * Values must be odd and within [-h_max, h_max], else BMLP_ESTATE and nothing
 * changes.  The epoch's error and pattern counters restart at 0. */
int bmlp_set_state(bmlp_t* h, int32_t layer, const int16_t* H_in, double p_r, int64_t step);

/* Model shape: any output may be NULL.  widths_out: L + 1 values; gamma_out: L. */
int bmlp_get_info(const bmlp_t* h, int32_t* n_layers, int32_t* widths_out, int32_t* classes,
                  int32_t* gamma_out, int32_t* bs, int32_t* fwd_impl);

/* One-line description of the last error on this handle ("" if none).  With
 * h == NULL: the last error of a call that had no handle (e.g. bmlp_create). */
const char* bmlp_last_error(const bmlp_t* h);

/* Group size chosen by the rule of Sec. 4.3 for a layer of K neurons: the
 * divisor of K closest to [75, 105], the largest among equally close ones;
 * -1 for K < 1.  Host only. */
int32_t bmlp_gamma_rule(int32_t K);

/* Thresholds of the reinforcement sampler (Alg. 3 l.5-12) for a block of n
 * inputs (1 <= n <= 64) of a layer of width K at p_r.  Each hidden weight is
 * reinforced independently with probability q = p_r sqrt(2 / (pi K)) (IEEE
 * double; >= 1 taken as 1).  The events of a neuron row are drawn per block
 * of 64 consecutive inputs (the last block shorter): the block has an event
 * iff its 32-bit draw U < any_out; its first event is at the least j with
 * V < first_out[j]; after an event at p the next is at p + 1 + g for the
 * least g <= n - 2 - p with V < gap_out[g], none if there is no such g (V the
 * block's successive 32-bit draws).  With thr(x) = ceil(x 2^32) (0 for
 * x <= 0, 2^32 for x >= 1) and (1-q)^m a left-to-right IEEE product:
 *   any_out = thr(1 - (1-q)^n), first_out[j] = thr((1 - (1-q)^(j+1)) /
 *   (1 - (1-q)^n)) for j < n, gap_out[g] = thr(1 - (1-q)^(g+1)) for g < n - 1.
 * first_out holds n values and gap_out n - 1 (caller-owned).  Host only;
 * BMLP_EINVAL for K < 1, n outside 1..64 or a NULL output. */
int bmlp_reinforce_tables(double p_r, int32_t K, int32_t n, uint64_t* any_out,
                          uint64_t* first_out, uint64_t* gap_out);

/* Debug view of the most recent training mini-batch (synchronises): for layer
 * `layer`, Z (bs x K_l int16 pre-activations), A (bs x ceil(K_l/64) packed
 * activations), mark (bs uint8, 1 = pattern in M_l), sel (bs x G_l int16,
 * selected neuron per group or -1).  Rows beyond the batch's size are stale.
 * Any output may be NULL. */
int bmlp_debug_last_step(const bmlp_t* h, int32_t layer, int16_t* Z, uint64_t* A,
                         uint8_t* mark, int16_t* sel);

/* Failure-path probe of the bounded device waits (no counterpart in the
 * paper): one CTA initialises an mbarrier and waits on its first phase with
 * the same bounded wait the tensor-core kernels use, limited to `seconds`
 * (0 < seconds <= 10) of SM clock.  arrive > 0: one arrival completes the
 * phase first, so the wait succeeds.  arrive <= 0: nothing arrives, the wait
 * gives up when the limit expires, the kernel counts it as a timeout and
 * returns (no trap, no fault; the context stays usable).  Synchronises; then,
 * for arrive >= 0, returns BMLP_ETIMEOUT if any timeout is pending (and clears
 * it), else BMLP_OK; for arrive < 0 returns BMLP_OK and leaves the expiry
 * pending, as an expired wait inside a training step would (the next call
 * that synchronises reports it). */
int bmlp_debug_wait_probe(bmlp_t* h, int32_t arrive, double seconds);

/* Per-kernel timing.  every = 0: off.  every = S > 0: every S-th training
 * mini-batch (counted by the step counter t) and every evaluation launch is
 * enqueued kernel by kernel between two CUDA events on the caller's stream; the
 * other mini-batches replay the captured step graph as usual.  Per kernel kind
 * the library accumulates the launch count and the summed device time when
 * the call ends (which then synchronises the stream).  kinds: 0 forward
 * (train), 1 local classifier + selection, 2 update (CP + R + repack),
 * 3 forward (predict), 4 predict output, 5 host-buffer copies, 6 drawing of
 * the reinforcement events (in the replayed step graph this kernel runs beside
 * the forward passes; in a sampled mini-batch it runs first, alone).
 * bmlp_launch_count: kernels this handle has launched since creation (graph
 * replays count each node). */
int bmlp_set_profiling(bmlp_t* h, int32_t every);
int bmlp_get_profile(const bmlp_t* h, int32_t kind, int64_t* launches, double* total_ms);
int bmlp_reset_profile(bmlp_t* h);
int64_t bmlp_launch_count(const bmlp_t* h);

/* Update-kernel statistics accumulated since creation or the last reset
 * (synchronises): neuron rows visited (layers with a non-empty M_l), rows
 * streamed (rows with at least one CP tuple; a row without tuple changes only
 * at its reinforcement events and keeps its W), and the algorithmic bytes the
 * rule touched: per streamed row its hidden weights read and written as the
 * library stores them (bit-sliced: the bits of h_max rounded up to a power of
 * two per weight, rows padded to 16 bytes) and its W row written, per group of
 * 32 weights with a reinforcement event in a row without tuple the group's
 * planes read and written.  Any output may be NULL; reset != 0 zeroes the
 * counters after reading them. */
int bmlp_update_stats(bmlp_t* h, int64_t* rows_out, int64_t* streamed_out, int64_t* bytes_out,
                      int32_t reset);

/* Failure injection for the allocation paths (no counterpart in the paper;
 * it tests the library's clean-up without a GPU fault).  After
 * bmlp_debug_fail_alloc(n), n >= 1, the n-th memory allocation the library
 * makes from then on -- counting every cudaMalloc of a device buffer and the
 * pinned host block of bmlp_create, in any handle of the process -- fails as
 * if memory were exhausted: the call that needed it returns BMLP_ENOMEM
 * ("... (injected)"), a half-built handle is freed whole, and the injection
 * disarms itself.  n = 0 disarms it.  BMLP_EINVAL for n < 0.
 * bmlp_debug_alloc_stats: the number of allocations the library holds now,
 * over every live handle of the process, and their bytes (either output may
 * be NULL); a failed bmlp_create leaves both where they were.  Host only;
 * neither call touches the device. */
int bmlp_debug_fail_alloc(int64_t nth);
int bmlp_debug_alloc_stats(int64_t* live_allocs, int64_t* live_bytes);

/* Peak rate of one contraction unit on the current device (the engine
 * comparison for the forward XNOR/popcount term of Table 3; Alg. 1 l.8):
 * a kernel that keeps its operands on chip and issues only that unit's
 * instruction, `iters` iterations per thread (or per MMA-issuing thread),
 * timed between CUDA events after one untimed launch.  engine: BMLP_FWD_POPC
 * (32-bit XOR + popcount on CUDA cores, 32 bit-pairs each), BMLP_FWD_TCGEN05
 * (tcgen05.mma kind::f8f6f4 e4m3, M128 N256 K32), BMLP_FWD_B1MMA
 * (mma.sync m16n8k256 b1 xor.popc), BMLP_FWD_S8MMA (mma.sync m16n8k32 s8).
 * *bitpairs_per_s: multiply-accumulates (bit-pairs) per second over the whole
 * device; *ms_out (may be NULL): the timed launch.  Synchronises the device;
 * allocates a few bytes.  No handle (errors: bmlp_last_error(NULL));
 * BMLP_EINVAL for an unknown engine or iters outside 1..2^31; BMLP_ETIMEOUT
 * if the tcgen05 kernel's bounded completion wait expired. */
int bmlp_engine_peak(int32_t engine, int64_t iters, double* bitpairs_per_s, double* ms_out);

/* Forward-only evaluation that allocates no memory.  The paper has no
 * counterpart: this is bmlp_predict with its scratch moved into the library,
 * for callers that cannot call cudaMalloc -- code running in a host callback,
 * a real-time loop with a fixed memory plan, or a process whose device
 * allocator belongs to another runtime.  bmlp_predict allocates its
 * inter-layer activation buffers on first use; this call instead uses one
 * fixed 16 MiB device array inside the library (two buffers of 2^20 64-bit
 * words), which every GPU that loads the library holds until the process
 * exits.  Results equal bmlp_predict's.
 *   n * ceil(max_l K_l / 64) must not exceed 1,048,576 (n <= 8192 for
 *   8192-wide layers); a larger n returns BMLP_EINVAL before any work.
 *   x_packed and labels_out must be device pointers on the current device
 *   (or managed memory): staging host buffers would allocate; host pointers
 *   and other devices' pointers return BMLP_EINVAL.
 *   The first call on a device looks up the array's device address once
 *   (cudaGetSymbolAddress); make that first call before any stream capture.
 *   Every call shares the array and it keeps the last call's contents (each
 *   call writes every word it reads); calls whose GPU work overlaps -- on
 *   different streams, or from different handles -- race on it.
 *   Calls no cudaMalloc, cudaFree or allocating library routine. */
int bmlp_predict_noalloc(bmlp_t* h, const uint64_t* x_packed, int64_t n, int32_t* labels_out,
                         void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* BMLP_H_ */
