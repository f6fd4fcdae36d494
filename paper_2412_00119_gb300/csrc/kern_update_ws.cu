// kern_update_ws.cu -- the hidden-weight update of one training step (Alg. 3:
// clipped perceptron, then reinforcement; Sec. 3.1: W = sign(H) re-packed in
// the same pass), with its memory traffic driven by bulk copies.
//
// The hidden weights are bit-sliced (DevLayer::H, update_common.cuh): a group
// of 32 inputs of a neuron row is kP words, word p holding bit p of the
// lattice index u = (h + h_max)/2 of the 32 weights.  A clipped step of +-1
// is a ripple of word operations through the planes, on 32 weights at once.
// The perceptron step of a tuple (mu, rho) moves weight i up where
// a^mu_i rho_{k,y^mu} = +1 and down elsewhere, so its direction word is the
// group's activation word, complemented when rho = -1; reinforcement moves
// the weights of its events away from 0, so its direction word is the
// group's h > 0 lanes, which is also the group's W word (a step away from 0
// never flips a sign).
//
// The update streams every hidden weight of every neuron row that received a
// CP tuple: read, the steps, write.
//   - kSched scheduler warps take rows from the step's row counter, find the
//     row's CP tuples (Alg. 2's selections of the neuron's group; labels in
//     shared memory), and fill one slot of a shared-memory ring per segment
//     of the row: bulk copies (cp.async.bulk, completing on the slot's "full"
//     mbarrier) of the segment's planes, of its part of the reinforcement-
//     event bitmap and of the first tuples' activation words, plus the tuple
//     list and a header;
//   - consumer group j (kPerGroup warps) takes the slots of scheduler j in
//     order: each lane holds two groups of 32 weights at a time in
//     registers, applies the tuples in ascending mu, then the reinforcement
//     events (Alg. 3 applies R after CP), and writes the planes and the W
//     word to global memory; each warp releases the slot ("empty") when it
//     has read its part, without waiting for the other warps.
// A row without tuple occupies a slot with its event bitmap only: its groups
// with an event are stepped in place in global memory, and its W is
// unchanged.  Layers with an empty M_l are skipped (no CP, no R).  Every
// mbarrier wait is bounded; an expiry stops the CTA's loops, waits (bounded)
// for the copies it issued, and is counted in the control block.  The last
// CTA to finish advances the step counters.
#include "tc_common.cuh"
#include "update_common.cuh"

namespace bk {
namespace {

using namespace upd;

constexpr int kSched = 8;                     // scheduler warps
constexpr int kPerGroup = 2;                  // consumer warps per group; group j serves scheduler j
constexpr int kCons = kSched * kPerGroup;
constexpr int kThreads = 32 * (kSched + kCons);
constexpr int kGroupLanes = 32 * kPerGroup;
constexpr int kGroupsInFlight = 2;            // groups of 32 weights per consumer lane at once (kP <= 8)
constexpr int kMaxT = BMLP_MAX_BS;            // CP tuples of one row at most
constexpr int kMaxSlots = 24;
constexpr int kSmemLimit = 232448;            // dynamic shared memory of one CTA at most

enum SlotType : int { kSlotRow = 0, kSlotSparse = 1, kSlotEnd = 2 };

struct SlotMeta {
  uint32_t* hrow;          // the segment's first plane word in global memory
  uint32_t* wrow;          // the W word (32 bits) of the segment's first group
  const uint32_t* aprev;   // pattern 0's activation word of the segment's first group
  int type, n_t;           // slot type, CP tuples of the row
  int ng;                  // groups of the segment
  uint32_t last_mask;      // valid inputs of the segment's last group
  int arow_words;          // 32-bit words per activation row
  int nstage;              // tuples whose activation words are staged in the slot
  int nwords;              // stored plane words of the segment (row padding included)
  int pad;
};

// Slot layout for kP planes per group: planes, event bits, staged activation
// words, tuple list (uint16: mu | 0x8000 when rho = -1; 2 bs bytes), header.
template <int kP>
struct Geo {
  static constexpr int kSegG = (2048 / kP) < 1024 ? (2048 / kP) : 1024;  // groups per segment
  static constexpr int kHBytes = 4 * kP * kSegG;
  static constexpr int kEvBytes = 4 * kSegG;
  static constexpr int kActBytes = 4 * kSegG;                   // one pattern's words of a segment
  static constexpr int kActT = 4096 / kActBytes > 1 ? 4096 / kActBytes : 1;  // tuples staged at most
  static constexpr int kOffEv = kHBytes;
  static constexpr int kOffAct = kOffEv + kEvBytes;
  static constexpr int kOffTup = kOffAct + kActT * kActBytes;
};

// What the schedulers read of a layer, copied to shared memory at the start
// (the parameter block's cache lines do not survive in the small L1 that the
// slot ring leaves, and every row reads several of them in sequence).
struct LayerSh {
  uint32_t* H;
  uint64_t* W;
  const uint64_t* EV;
  const int16_t* sel;
  const int8_t* rho;
  const int16_t* group_of;
  const uint32_t* aprev;   // the layer's input activations of this mini-batch, row 0
  int row_base, gamma, ngrp, ldh, nw_in, ev_stride, Kin, pad;
};

struct __align__(16) WsShared {
  LayerSh lay[BMLP_MAX_LAYERS];
  unsigned long long full[kMaxSlots];
  unsigned long long empty[kMaxSlots];
  int16_t y[kMaxT];                   // labels of the mini-batch (bad ones as 0)
  unsigned long long stats[3];        // rows visited, rows streamed, algorithmic bytes
  int issued[kMaxSlots];              // last use of each slot with copies issued (-1: none)
  int failed;
};

// The ring for a mini-batch size: as many slots as fit in the shared memory
// (a multiple of kSched, at most kMaxSlots), followed by the schedulers' tuple
// scans (kSched lists of bs entries) and WsShared; the host sizes the launch
// with the same function.
struct Ring {
  int slot_bytes, nslots, off_meta;
  int list_bytes;   // one scheduler's tuple scan
  size_t smem;      // dynamic shared memory of the launch (128 bytes of alignment slack)
};

template <int kP>
__host__ __device__ __forceinline__ Ring ring_of(int bs) {
  Ring r;
  const int tup = (2 * bs + 15) & ~15;
  r.off_meta = Geo<kP>::kOffTup + tup;
  r.slot_bytes = (r.off_meta + (int)sizeof(SlotMeta) + 127) & ~127;
  r.list_bytes = tup;
  const int fixed = 128 + kSched * r.list_bytes + (int)sizeof(WsShared);
  int n = (kSmemLimit - fixed) / r.slot_bytes;
  n = n < kMaxSlots ? n : kMaxSlots;
  r.nslots = n / kSched * kSched;
  r.smem = (size_t)fixed + (size_t)r.nslots * r.slot_bytes;
  return r;
}

__device__ __forceinline__ uint8_t* slot_ptr(uint8_t* ring, int s, int slot_bytes) {
  return ring + (size_t)s * slot_bytes;
}

// ---------------------------------------------------------------------------
// Scheduler warp j: rows -> slots j, j + kSched, ... (sequence numbers
// j, j + kSched, ...).  Rows are pipelined one deep: while row r is turned
// into slots, the selections of row r + 1 (its ticket taken one row earlier)
// are in flight, and the ticket of row r + 2 is taken.
// ---------------------------------------------------------------------------
struct RowFetch {
  int gr;          // global row number (>= rows_total: none)
  int li, k;       // layer index, neuron
  int sv[4];       // this lane's selections of patterns 32 q + lane (the first 128)
  int rho_lane;    // rho_{k, lane} for c <= 32
  bool skip;       // M_l empty, or the step's forward pass failed: no CP, no R
};

template <int kP>
__device__ __forceinline__ void ws_scheduler(const StepParams* __restrict__ P, WsShared* sh,
                                             uint8_t* ring, const Ring R, int j, int lane, int bsz,
                                             bool step_failed) {
  using G = Geo<kP>;
  const uint32_t nslots = (uint32_t)R.nslots;
  Ctrl* ctrl = P->ctrl;
  volatile int* failed = &sh->failed;
  const int c = P->c;
  const int L = P->L;
  const int bs = P->bs;
  const int rows_total = P->rows_total;
  uint16_t* list = reinterpret_cast<uint16_t*>(ring + (size_t)R.nslots * R.slot_bytes + (size_t)j * R.list_bytes);
  uint32_t seq = (uint32_t)j;
  uint64_t st_rows = 0, st_streamed = 0, st_bytes = 0;
  // lane i < L holds layer i's first row and its "M_l non-empty" flag
  const int rb_lane = lane < L ? sh->lay[lane].row_base : 0;
  const unsigned am_lane = lane < L ? ctrl->any_mark[lane] : 0u;
  // acquire the slot of sequence number q (its previous use released)
  auto acquire = [&](uint32_t q) -> bool {
    const uint32_t u = q / nslots;
    if (u == 0) return true;
    return __all_sync(kFull, tc::mbar_wait(&sh->empty[q % nslots], (u - 1) & 1u, failed));
  };
  // issue the loads of row gr (consumed one row later)
  auto fetch = [&](int gr) -> RowFetch {
    RowFetch f;
    f.gr = gr;
    f.li = __popc(__ballot_sync(kFull, lane >= 1 && lane < L && gr >= rb_lane));
    f.skip = gr >= rows_total || step_failed || __shfl_sync(kFull, am_lane, f.li) == 0u;
    f.k = 0;
    f.rho_lane = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) f.sv[q] = -1;
    if (!f.skip) {
      const LayerSh& Ly = sh->lay[f.li];
      f.k = gr - Ly.row_base;
      const int g = Ly.group_of ? (int)Ly.group_of[f.k] : f.k / Ly.gamma;
      const int16_t* selg = Ly.sel + (int64_t)g * bs;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int m = 32 * q + lane;
        if (m < bsz) f.sv[q] = (int)selg[m];
      }
      if (c <= 32 && lane < c) f.rho_lane = (int)Ly.rho[(int64_t)f.k * c + lane];
    }
    return f;
  };
  // tuples from selections sv of patterns m0 + 32 q + lane, appended to list
  auto scan4 = [&](const RowFetch& f, const int (&sv)[4], int m0, int n_t) -> int {
    const LayerSh& Ly = sh->lay[f.li];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int m = m0 + 32 * q + lane;
      const bool hit = sv[q] == f.k;
      const unsigned bal = __ballot_sync(kFull, hit);
      if (bal != 0u) {
        const int yv = hit ? (int)sh->y[m] : 0;
        const int rs = __shfl_sync(kFull, f.rho_lane, yv & 31);
        if (hit) {
          const int rho = (c <= 32) ? rs : (int)Ly.rho[(int64_t)f.k * c + yv];
          list[n_t + __popc(bal & ((1u << lane) - 1u))] = (uint16_t)(m | ((rho > 0) ? 0 : 0x8000));
        }
      }
      n_t += __popc(bal);
    }
    return n_t;
  };
  int ticket = 0;
  if (lane == 0) ticket = (int)atomicAdd(&ctrl->upd_next, 1u);
  RowFetch cur = fetch(__shfl_sync(kFull, ticket, 0));
  if (lane == 0) ticket = (int)atomicAdd(&ctrl->upd_next, 1u);
#pragma unroll 1
  while (cur.gr < rows_total && !*failed) {
    const RowFetch nxt = fetch(__shfl_sync(kFull, ticket, 0));
    if (lane == 0) ticket = (int)atomicAdd(&ctrl->upd_next, 1u);
    if (cur.skip) {
      cur = nxt;
      continue;
    }
    const LayerSh& Ly = sh->lay[cur.li];
    const int k = cur.k;
    // ---- CP tuples of neuron k, ascending mu: the patterns whose selection
    // in its group is k ----
    int n_t = scan4(cur, cur.sv, 0, 0);
    if (bsz > 128) {
      const int g = Ly.group_of ? (int)Ly.group_of[k] : k / Ly.gamma;
      const int16_t* selg = Ly.sel + (int64_t)g * bs;
#pragma unroll 1
      for (int m0 = 128; m0 < bsz; m0 += 128) {
        int sv[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int m = m0 + 32 * q + lane;
          sv[q] = (m < bsz) ? (int)selg[m] : -1;
        }
        n_t = scan4(cur, sv, m0, n_t);
      }
    }
    __syncwarp();
    st_rows += 1;
    const int ngrp = Ly.ngrp;
    const uint32_t* aprev = Ly.aprev;
    const int arow_words = 2 * Ly.nw_in;
    const bool act_ok = (arow_words % 4 == 0) && (reinterpret_cast<uintptr_t>(aprev) % 16u == 0);
    if (n_t > 0) {
      st_streamed += 1;
      st_bytes += 8ull * (uint64_t)Ly.ldh + 8ull * (uint64_t)Ly.nw_in;   // H read + write, W write
    }
    const uint32_t* evrow = reinterpret_cast<const uint32_t*>(Ly.EV + (int64_t)k * Ly.ev_stride);
    // ---- one slot per segment of kSegG groups ----
#pragma unroll 1
    for (int g0 = 0; g0 < ngrp; g0 += G::kSegG) {
      if (!acquire(seq)) break;
      const int s = (int)(seq % nslots);
      uint8_t* sl = slot_ptr(ring, s, R.slot_bytes);
      SlotMeta* meta = reinterpret_cast<SlotMeta*>(sl + R.off_meta);
      const int ng = min(G::kSegG, ngrp - g0);
      const int nwords = min(G::kSegG * kP, Ly.ldh - g0 * kP);              // a multiple of 4
      const uint32_t ev_bytes = (uint32_t)min(4 * G::kSegG, 8 * Ly.ev_stride - 4 * g0);
      const uint32_t act_bytes = (uint32_t)min(G::kActBytes, 4 * arow_words - 4 * g0);
      const int nstage = (n_t > 0 && act_ok) ? min(n_t, G::kActT) : 0;
      for (int q = lane; q < n_t; q += 32) reinterpret_cast<uint16_t*>(sl + G::kOffTup)[q] = list[q];
      if (lane == 0) {
        meta->hrow = Ly.H + (int64_t)k * Ly.ldh + (int64_t)g0 * kP;
        meta->wrow = reinterpret_cast<uint32_t*>(Ly.W + (int64_t)k * Ly.nw_in) + g0;
        meta->aprev = aprev + g0;
        meta->type = n_t > 0 ? kSlotRow : kSlotSparse;
        meta->n_t = n_t;
        meta->ng = ng;
        meta->last_mask = (g0 + ng == ngrp) ? group_mask(ngrp - 1, Ly.Kin) : kFull;
        meta->arow_words = arow_words;
        meta->nstage = nstage;
        meta->nwords = nwords;
      }
      __syncwarp();
      if (lane == 0) {
        const uint32_t h_bytes = n_t > 0 ? 4u * (uint32_t)nwords : 0u;
        tc::mbar_arrive_tx(&sh->full[s], ev_bytes + h_bytes + (uint32_t)nstage * act_bytes);
        sh->issued[s] = (int)(seq / nslots);
        tc::bulk_g2s(sl + G::kOffEv, evrow + g0, ev_bytes, &sh->full[s]);
        if (n_t > 0) tc::bulk_g2s(sl, meta->hrow, h_bytes, &sh->full[s]);
        for (int q = 0; q < nstage; ++q)
          tc::bulk_g2s(sl + G::kOffAct + q * G::kActBytes,
                       aprev + (size_t)(list[q] & 0x7FFF) * arow_words + g0, act_bytes, &sh->full[s]);
      }
      seq += kSched;
    }
    cur = nxt;
  }
  // no more rows: an END slot for consumer group j (released by nobody)
  if (acquire(seq)) {
    const int s = (int)(seq % nslots);
    if (lane == 0) {
      reinterpret_cast<SlotMeta*>(slot_ptr(ring, s, R.slot_bytes) + R.off_meta)->type = kSlotEnd;
      tc::mbar_arrive(&sh->full[s]);
    }
  }
  if (lane == 0) {
    atomicAdd(&sh->stats[0], st_rows);
    atomicAdd(&sh->stats[1], st_streamed);
    atomicAdd(&sh->stats[2], st_bytes);
  }
}

// ---------------------------------------------------------------------------
// Consumer warp ci of group ci / kPerGroup: the slots of its scheduler ->
// hidden weights and W.  The segment's groups are dealt to the group's
// kGroupLanes lanes, two per lane at a time (g and g + kGroupLanes), so the
// tuple loop is shared.  The warps of a group do not wait for one another:
// each reads its part of the slot, releases it (the slot's "empty" barrier
// counts the group's warps), and writes planes and W words to global memory
// from registers.
// ---------------------------------------------------------------------------
template <int kP, bool kOnes>
__device__ __forceinline__ void ws_consumer(const StepParams* __restrict__ P, WsShared* sh,
                                            uint8_t* ring, const Ring R, int ci, int lane) {
  using G = Geo<kP>;
  const uint32_t nslots = (uint32_t)R.nslots;
  constexpr int kPerLane = (G::kSegG + kGroupLanes - 1) / kGroupLanes;   // groups of a segment per lane at most
  // groups a lane holds in registers at once (more give the dependent step
  // chains of different groups to interleave)
  constexpr int kInFlight = kP <= 8 ? kGroupsInFlight : 2;
  volatile int* failed = &sh->failed;
  const Sliced<kP, kOnes> S(P->h_max);
  const int grp = ci / kPerGroup, wi = ci % kPerGroup;
  const int ti = wi * 32 + lane;
  uint64_t sparse_bytes = 0;
#pragma unroll 1
  for (uint32_t seq = (uint32_t)grp;; seq += kSched) {
    const int s = (int)(seq % nslots);
    if (!__all_sync(kFull, tc::mbar_wait(&sh->full[s], (seq / nslots) & 1u, failed))) break;
    uint8_t* sl = slot_ptr(ring, s, R.slot_bytes);
    const SlotMeta meta = *reinterpret_cast<const SlotMeta*>(sl + R.off_meta);
    if (meta.type == kSlotEnd) break;
    const uint32_t* ev = reinterpret_cast<const uint32_t*>(sl + G::kOffEv);
    const int ng = meta.ng;
    if (meta.type == kSlotSparse) {
      // a row without tuple: the event words are read and the slot released,
      // then the groups with an event are stepped in global memory
      uint32_t evs[kPerLane];
#pragma unroll
      for (int q = 0; q < kPerLane; ++q) {
        const int gi = ti + q * kGroupLanes;
        evs[q] = gi < ng ? ev[gi] & (gi == ng - 1 ? meta.last_mask : kFull) : 0u;
      }
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sh->empty[s]);
      // two groups at a time, both loads first, so that their latencies overlap
#pragma unroll
      for (int q0 = 0; q0 < kPerLane; q0 += 2) {
        uint32_t u[2][kP];
#pragma unroll
        for (int d = 0; d < 2 && q0 + d < kPerLane; ++d)
          if (evs[q0 + d] != 0u)
            load_planes<kP>(u[d], meta.hrow + (size_t)(ti + (q0 + d) * kGroupLanes) * kP);
#pragma unroll
        for (int d = 0; d < 2 && q0 + d < kPerLane; ++d) {
          if (evs[q0 + d] == 0u) continue;
          S.step(u[d], S.positive(u[d]), evs[q0 + d]);
          store_planes<kP>(meta.hrow + (size_t)(ti + (q0 + d) * kGroupLanes) * kP, u[d]);
          sparse_bytes += 8ull * kP;
        }
      }
      continue;
    }
    const int n_t = meta.n_t;
    const uint16_t* tl = reinterpret_cast<const uint16_t*>(sl + G::kOffTup);
    const uint32_t* act = reinterpret_cast<const uint32_t*>(sl + G::kOffAct);
    const uint32_t* aseg = meta.aprev;
    const int arow_words = meta.arow_words;
    const int nstage = meta.nstage;
    const uint32_t* hs = reinterpret_cast<const uint32_t*>(sl);
#pragma unroll 1
    for (int g0 = ti; g0 < ng; g0 += kInFlight * kGroupLanes) {
      // kInFlight groups of this lane: g0 + i kGroupLanes
      uint32_t u[kInFlight][kP], en[kInFlight], r[kInFlight];
#pragma unroll
      for (int i = 0; i < kInFlight; ++i) {
        const int g = g0 + i * kGroupLanes;
        const bool live = g < ng;
        en[i] = live ? (g == ng - 1 ? meta.last_mask : kFull) : 0u;
        if (live) load_planes<kP>(u[i], hs + (size_t)g * kP);
        else {
#pragma unroll
          for (int p = 0; p < kP; ++p) u[i][p] = 0u;
        }
        r[i] = live ? ev[g] & en[i] : 0u;
      }
      // ---- CP tuples, ascending mu ----
#pragma unroll 1
      for (int q = 0; q < n_t; ++q) {
        const uint32_t e = tl[q];
        const uint32_t xm = (e & 0x8000u) ? kFull : 0u;   // rho = -1: complement
        const uint32_t* arow = q < nstage ? act + q * (G::kActBytes / 4)
                                          : aseg + (size_t)(e & 0x7FFFu) * arow_words;
#pragma unroll
        for (int i = 0; i < kInFlight; ++i) {
          const int g = g0 + i * kGroupLanes;
          const uint32_t a = en[i] ? arow[g] : 0u;
          S.step(u[i], a ^ xm, en[i]);
        }
      }
      // ---- R: the events step away from 0; W = the lanes with h > 0 ----
#pragma unroll
      for (int i = 0; i < kInFlight; ++i) {
        const int g = g0 + i * kGroupLanes;
        const uint32_t pos = S.positive(u[i]) & en[i];
        S.step(u[i], pos, r[i]);
        if (en[i]) {
          meta.wrow[g] = pos;
          store_planes<kP>(meta.hrow + (size_t)g * kP, u[i]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) tc::mbar_arrive(&sh->empty[s]);
  }
  if (sparse_bytes) atomicAdd(&sh->stats[2], sparse_bytes);
}

template <int kP, bool kOnes>
__global__ void __launch_bounds__(kThreads, 1) k_update_ws(const StepParams* __restrict__ P) {
  const Ring R = ring_of<kP>(P->bs);
  const int nslots = R.nslots;
  extern __shared__ uint8_t ws_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(ws_raw) + 127) &
                                             ~static_cast<uintptr_t>(127));
  WsShared* sh = reinterpret_cast<WsShared*>(ring + (size_t)nslots * R.slot_bytes + (size_t)kSched * R.list_bytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  Ctrl* ctrl = P->ctrl;
  // barriers: independent of every earlier kernel
  if (threadIdx.x < nslots) sh->issued[threadIdx.x] = -1;
  if (threadIdx.x == 0) {
    for (int q = 0; q < nslots; ++q) {
      tc::mbar_init(&sh->full[q], 1);
      tc::mbar_init(&sh->empty[q], kPerGroup);
    }
    sh->stats[0] = sh->stats[1] = sh->stats[2] = 0ull;
    sh->failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_wait();
  pdl_trigger();
  const unsigned long long t = ctrl->t;
  const uint32_t sidx = ctrl->s;
  const int64_t start = (int64_t)sidx * P->bs;
  const int64_t rem = P->n - start;
  const int bsz = (int)(rem < P->bs ? rem : P->bs);
  // an expired bounded wait in this step's forward pass: no CP, no R (the
  // selection kernel marked nothing either); the counters still advance
  const bool step_failed = ctrl->timeouts != 0u;
  if (threadIdx.x < P->L) {
    const int li = threadIdx.x;
    const DevLayer& D = P->layer[li];
    LayerSh& o = sh->lay[li];
    o.H = D.H; o.W = D.W; o.EV = D.EV; o.sel = D.sel; o.rho = D.rho; o.group_of = D.group_of;
    o.aprev = li == 0 ? reinterpret_cast<const uint32_t*>(P->x + start * P->nw0)
                      : reinterpret_cast<const uint32_t*>(P->layer[li - 1].A);
    o.row_base = D.row_base; o.gamma = D.gamma; o.ngrp = D.ngrp; o.ldh = D.ldh; o.nw_in = D.nw_in;
    o.ev_stride = D.ev_stride; o.Kin = D.Kin; o.pad = 0;
  }
  for (int i = threadIdx.x; i < bsz; i += kThreads) {
    const int yv = P->y[start + i];
    sh->y[i] = (int16_t)((yv < 0 || yv >= P->c) ? 0 : yv);   // memory-safe stand-in; the host reports bad labels
  }
  __syncthreads();
  if (warp < kSched)
    ws_scheduler<kP>(P, sh, ring, R, warp, lane, bsz, step_failed);
  else
    ws_consumer<kP, kOnes>(P, sh, ring, R, warp - kSched, lane);
  __syncthreads();
  if (sh->failed && threadIdx.x < nslots && sh->issued[threadIdx.x] >= 0) {
    // after an expired wait: the copies issued into this slot land before the
    // CTA's shared memory goes away (a wait of its own, bounded)
    int own = 0;
    (void)tc::mbar_wait(&sh->full[threadIdx.x], (uint32_t)sh->issued[threadIdx.x] & 1u, &own);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    atomicAdd(&ctrl->upd_rows, sh->stats[0]);
    atomicAdd(&ctrl->upd_streamed, sh->stats[1]);
    atomicAdd(&ctrl->upd_bytes, sh->stats[2]);
    if (sh->failed) atomicAdd(&ctrl->timeouts, 1u);
    // step completion: the last CTA to finish advances the counters
    __threadfence();
    const unsigned prev = atomicAdd(&ctrl->done, 1u);
    if (prev == gridDim.x - 1) {
      ctrl->t = t + 1;
      ctrl->s = sidx + 1;
      for (int i = 0; i < P->L; ++i) ctrl->any_mark[i] = 0u;
      ctrl->upd_next = 0u;
      ctrl->done = 0u;
      __threadfence();
    }
  }
}

template <int kP, bool kOnes>
cudaError_t set_smem() {
  return cudaFuncSetAttribute(k_update_ws<kP, kOnes>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kSmemLimit);
}

template <int kP, bool kOnes>
cudaError_t launch_one(unsigned grid, size_t smem, cudaStream_t st, bool pdl, const StepParams* P) {
  return launch_kernel(k_update_ws<kP, kOnes>, dim3(grid), dim3(kThreads), smem, st, pdl, P);
}

}  // namespace

size_t update_ws_smem(int nplanes, int bs) {
  switch (nplanes) {
    case 1: return ring_of<1>(bs).smem;
    case 2: return ring_of<2>(bs).smem;
    case 4: return ring_of<4>(bs).smem;
    case 8: return ring_of<8>(bs).smem;
    default: return ring_of<16>(bs).smem;
  }
}

cudaError_t prepare_update_ws() {
  cudaError_t e;
  if ((e = set_smem<1, true>()) != cudaSuccess || (e = set_smem<2, true>()) != cudaSuccess ||
      (e = set_smem<4, true>()) != cudaSuccess || (e = set_smem<4, false>()) != cudaSuccess ||
      (e = set_smem<8, true>()) != cudaSuccess || (e = set_smem<8, false>()) != cudaSuccess ||
      (e = set_smem<16, false>()) != cudaSuccess)
    return e;
  return cudaSuccess;
}

cudaError_t update_kernel_image(cudaFuncAttributes* fa) {
  return cudaFuncGetAttributes(fa, k_update_ws<8, true>);
}

cudaError_t launch_update_ws(int nplanes, int h_max, int bs, unsigned grid, cudaStream_t st, bool pdl,
                             const StepParams* P) {
  const bool ones = h_max == (1 << nplanes) - 1;
  const size_t smem = update_ws_smem(nplanes, bs);
  switch (nplanes) {
    case 1: return launch_one<1, true>(grid, smem, st, pdl, P);
    case 2: return launch_one<2, true>(grid, smem, st, pdl, P);
    case 4: return ones ? launch_one<4, true>(grid, smem, st, pdl, P)
                        : launch_one<4, false>(grid, smem, st, pdl, P);
    case 8: return ones ? launch_one<8, true>(grid, smem, st, pdl, P)
                        : launch_one<8, false>(grid, smem, st, pdl, P);
    case 16: return launch_one<16, false>(grid, smem, st, pdl, P);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace bk
