// kern_update_ws.cu -- the hidden-weight update of one training step (Alg. 3:
// clipped perceptron and reinforcement; Sec. 3.1: W = sign(H) re-packed in
// the same pass) with its memory traffic driven by bulk copies.
//
// The update streams every hidden weight of every neuron row that received a
// CP tuple: read, a few integer steps, write.  In a kernel where each warp
// loads its own row, the loads it can keep in flight bound the memory rate,
// and the CP arithmetic delays them.  Here the two are split between warps:
//   - kWsSched scheduler warps take rows from the step's row counter, find the
//     row's CP tuples (Alg. 2's selections of the neuron's group; labels in
//     shared memory), and fill one slot of a shared-memory ring per segment
//     of kSegW hidden weights: bulk copies (cp.async.bulk, completing on the
//     slot's "full" mbarrier) of the segment's hidden weights, of its part of
//     the reinforcement-event bitmap, and of the first kActT tuples'
//     activation bytes, plus the tuple list and a header;
//   - kWsCons consumer warps, in kWsGroups groups that take different slots
//     at once (group g the slots of schedulers g, g + kWsGroups, ...): each
//     lane applies the tuples to its chunks of 8 weights in the slot and
//     writes the chunk's W byte (reinforcement never flips a sign, so W is
//     final after CP); after a group barrier the lanes apply the segment's few
//     reinforcement events in the slot; one bulk copy writes the segment's H
//     back to global memory, and the warps release the slot ("empty").
// A row without tuple occupies a slot with its event bitmap only; its events
// are applied as single-weight read-modify-writes and its W is unchanged
// (reinforcement never flips a sign).  Slots are used in sequence order,
// scheduler j filling sequence numbers j, j + kWsSched, ...; a scheduler that
// finds no more rows fills one END slot, after which the consumers skip its
// numbers.  The per-chunk arithmetic is that of k_update (update_common.cuh).
// Every mbarrier wait is bounded; an expiry stops the CTA's loops, waits
// (bounded) for the copies it issued, and is counted in the control block.
// The last CTA to finish advances the step counters.
#include "tc_common.cuh"
#include "update_common.cuh"

namespace bk {
namespace {

using namespace upd;

constexpr int kWsSched = 4;                  // scheduler warps
constexpr int kWsCons = 24;                  // consumer warps
constexpr int kWsGroups = 4;                 // consumer groups, each on its own slots
constexpr int kWsPerGroup = kWsCons / kWsGroups;
static_assert(kWsSched % kWsGroups == 0, "group g takes the slots of schedulers g, g + kWsGroups, ...");
constexpr int kWsThreads = 32 * (kWsSched + kWsCons);
constexpr int kWsSlots = 8;                  // ring slots, a multiple of kWsSched
static_assert(kWsSlots % kWsSched == 0, "each slot belongs to one scheduler warp");
constexpr int kSegW = 8192;                  // hidden weights per segment (one slot)
constexpr int kActT = 4;                     // tuples whose activation bytes are staged
constexpr int kMaxT = 128;                   // tuples per row at most (mini-batches <= 128)

enum SlotType : int { kSlotRow = 0, kSlotSparse = 1, kSlotEnd = 2 };

struct SlotMeta {
  int16_t* hrow;         // the segment's first hidden weight in global memory
  uint8_t* wrow;         // its first W byte
  const uint8_t* aprev;  // the layer's input activations (row 0, byte 0 of the segment)
  int type, n_t;         // slot type, CP tuples of the row
  int nin;               // real inputs of the segment
  int ch0;               // chunk offset of the segment in its row
  int arow_bytes;        // bytes per activation row
  int act_smem;          // activation bytes of the first min(n_t, kActT) tuples staged
  int nseg;              // stored hidden weights of the segment (row padding included)
  int pad;
};

constexpr int kOffH = 0;                              // kSegW int16
constexpr int kOffEv = kOffH + 2 * kSegW;             // kSegW / 64 uint64
constexpr int kOffAct = kOffEv + kSegW / 8;           // kActT x kSegW / 8 bytes
constexpr int kOffTup = kOffAct + kActT * (kSegW / 8);  // kMaxT int32
constexpr int kOffMeta = kOffTup + 4 * kMaxT;
constexpr int kSlotBytes = (kOffMeta + (int)sizeof(SlotMeta) + 127) & ~127;

struct __align__(16) WsShared {
  unsigned long long full[kWsSlots];
  unsigned long long empty[kWsSlots];
  uint4 db[256];                   // packed CP steps per activation byte (rho = +1)
  int y[kMaxT];                    // labels of the mini-batch (bad ones as 0)
  int list[kWsSched][kMaxT];       // a scheduler's tuple scan
  unsigned long long stats[3];     // rows visited, rows streamed, algorithmic bytes
  int issued[kWsSlots];            // last use of each slot with copies issued (-1: none)
  int failed;
};

constexpr size_t kWsSmemBytes = 128 /*alignment slack*/ + (size_t)kWsSlots * kSlotBytes + sizeof(WsShared);

__device__ __forceinline__ uint8_t* slot_ptr(uint8_t* ring, int s) { return ring + (size_t)s * kSlotBytes; }

// barrier of the kWsPerGroup warps of consumer group g (named barriers 1..)
__device__ __forceinline__ void group_sync(int g) {
  asm volatile("bar.sync %0, %1;" ::"r"(1 + g), "r"(32 * kWsPerGroup) : "memory");
}

// ---------------------------------------------------------------------------
// Scheduler warp: rows -> slots.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void ws_scheduler(const StepParams* __restrict__ P, WsShared* sh,
                                             uint8_t* ring, int j, int lane, int64_t start, int bsz,
                                             bool step_failed) {
  Ctrl* ctrl = P->ctrl;
  volatile int* failed = &sh->failed;
  const int c = P->c;
  const int rows_total = P->rows_total;
  int* list = sh->list[j];
  uint32_t seq = (uint32_t)j;
  uint64_t st_rows = 0, st_streamed = 0, st_bytes = 0;
  // acquire the slot of sequence number seq (wait until the consumers released its previous use)
  auto acquire = [&](uint32_t q) -> bool {
    const uint32_t u = q / kWsSlots;
    if (u == 0) return true;
    return __all_sync(kFull, tc::mbar_wait(&sh->empty[q % kWsSlots], (u - 1) & 1u, failed));
  };
  // the ticket of the next row is taken while the current row is scanned
  int next = 0;
  if (lane == 0) next = (int)atomicAdd(&ctrl->upd_next, 1u);
  next = __shfl_sync(kFull, next, 0);
#pragma unroll 1
  while (true) {
    const int gr = next;
    if (gr >= rows_total || *failed) break;
    if (lane == 0) next = (int)atomicAdd(&ctrl->upd_next, 1u);
    int li = 0;
    while (li + 1 < P->L && gr >= P->layer[li + 1].row_base) ++li;
    if (step_failed || ctrl->any_mark[li] == 0u) {   // M_l empty: no CP, no R
      next = __shfl_sync(kFull, next, 0);
      continue;
    }
    const DevLayer& Ly = P->layer[li];
    const int k = gr - Ly.row_base;
    const int g = Ly.group_of ? (int)Ly.group_of[k] : k / Ly.gamma;
    // ---- CP tuples of neuron k, ascending mu ----
    // the group's selections of all (<= 128) patterns and, for c <= 32, the
    // neuron's row of P_l are loaded together: one round trip
    int n_t = 0;
    const int16_t* selg = Ly.sel + (int64_t)g * P->bs;
    const int rho_lane = (c <= 32 && lane < c) ? (int)Ly.rho[(int64_t)k * c + lane] : 0;
    int sv[kMaxT / 32];
#pragma unroll
    for (int q = 0; q < kMaxT / 32; ++q) {
      const int m = 32 * q + lane;
      sv[q] = (m < bsz) ? (int)selg[m] : -1;
    }
#pragma unroll
    for (int q = 0; q < kMaxT / 32; ++q) {
      const int m = 32 * q + lane;
      const bool hit = sv[q] == k;
      const unsigned bal = __ballot_sync(kFull, hit);
      if (bal != 0u) {
        const int yv = hit ? sh->y[m] : 0;
        const int rs = __shfl_sync(kFull, rho_lane, yv & 31);
        if (hit) {
          const int rho = (c <= 32) ? rs : (int)Ly.rho[(int64_t)k * c + yv];
          list[n_t + __popc(bal & ((1u << lane) - 1u))] = m | ((rho > 0) ? 0 : 0x10000);
        }
      }
      n_t += __popc(bal);
    }
    __syncwarp();
    st_rows += 1;
    const int Kin = Ly.Kin;
    const uint8_t* aprev = (li == 0) ? reinterpret_cast<const uint8_t*>(P->x + start * P->nw0)
                                     : reinterpret_cast<const uint8_t*>(P->layer[li - 1].A);
    const uint32_t arow_bytes = (uint32_t)Ly.nw_in * 8u;
    const bool act_ok = (arow_bytes % 16u == 0) && (reinterpret_cast<uintptr_t>(aprev) % 16u == 0);
    if (n_t > 0) {
      st_streamed += 1;
      st_bytes += 4ull * (uint64_t)Ly.ldh + 8ull * (uint64_t)Ly.nw_in;
    }
    // ---- one slot per segment of kSegW hidden weights ----
    for (int w0 = 0; w0 < Kin; w0 += kSegW) {
      if (!acquire(seq)) break;
      const int s = (int)(seq % kWsSlots);
      uint8_t* sl = slot_ptr(ring, s);
      SlotMeta* meta = reinterpret_cast<SlotMeta*>(sl + kOffMeta);
      const int nseg = min(kSegW, Ly.ldh - w0);                 // stored weights (multiple of 64)
      const int nevw = min(kSegW / 64, Ly.ev_stride - w0 / 64);  // event words (even)
      const int nact = min(kSegW / 8, (int)arow_bytes - w0 / 8); // activation bytes
      const int nstage = (n_t > 0 && act_ok) ? min(n_t, kActT) : 0;
      for (int q = lane; q < n_t; q += 32) reinterpret_cast<int*>(sl + kOffTup)[q] = list[q];
      if (lane == 0) {
        meta->hrow = Ly.H + (int64_t)k * Ly.ldh + w0;
        meta->wrow = reinterpret_cast<uint8_t*>(Ly.W + (int64_t)k * Ly.nw_in) + w0 / 8;
        meta->aprev = aprev + w0 / 8;
        meta->type = n_t > 0 ? kSlotRow : kSlotSparse;
        meta->n_t = n_t;
        meta->nin = min(kSegW, Kin - w0);
        meta->ch0 = w0 / 8;
        meta->arow_bytes = (int)arow_bytes;
        meta->act_smem = nstage > 0 ? 1 : 0;
        meta->nseg = nseg;
      }
      __syncwarp();
      if (lane == 0) {
        const uint32_t ev_bytes = 8u * (uint32_t)nevw;
        const uint32_t h_bytes = n_t > 0 ? 2u * (uint32_t)nseg : 0u;
        const uint32_t a_bytes = (uint32_t)nstage * (uint32_t)((nact + 15) & ~15);
        tc::mbar_arrive_tx(&sh->full[s], ev_bytes + h_bytes + a_bytes);
        sh->issued[s] = (int)(seq / kWsSlots);
        tc::bulk_g2s(sl + kOffEv, Ly.EV + (int64_t)k * Ly.ev_stride + w0 / 64, ev_bytes, &sh->full[s]);
        if (n_t > 0)
          tc::bulk_g2s(sl + kOffH, Ly.H + (int64_t)k * Ly.ldh + w0, h_bytes, &sh->full[s]);
        for (int q = 0; q < nstage; ++q)
          tc::bulk_g2s(sl + kOffAct + q * (kSegW / 8),
                       aprev + (size_t)(list[q] & 0xFFFF) * arow_bytes + w0 / 8,
                       (uint32_t)((nact + 15) & ~15), &sh->full[s]);
      }
      seq += kWsSched;
    }
    next = __shfl_sync(kFull, next, 0);
  }
  // no more rows: an END slot for the consumers (released by nobody)
  if (acquire(seq)) {
    const int s = (int)(seq % kWsSlots);
    if (lane == 0) {
      reinterpret_cast<SlotMeta*>(slot_ptr(ring, s) + kOffMeta)->type = kSlotEnd;
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
// Consumer warp ci: slots -> hidden weights and W.  Each slot's chunks of 8
// weights are dealt to the kWsCons x 32 consumer lanes, two per lane at a
// time (chunks c and c + kWsCons * 32), so the tuple loop is shared.
// ---------------------------------------------------------------------------
template <int kHb>
__device__ __forceinline__ void ws_consumer(const StepParams* __restrict__ P, WsShared* sh,
                                            uint8_t* ring, int ci, int lane) {
  volatile int* failed = &sh->failed;
  Enc E;
  E.h_max = P->h_max;
  E.hb = P->hb;
  E.base = 1 << P->hb;
  Lanes<kHb> LN;
  LN.hb_rt = P->hb;
  LN.over_pair = (uint32_t)(E.base + E.h_max + 1) * kLaneOne;
  LN.pos_pair = (uint32_t)(E.base + (E.h_max + 1) / 2) * kLaneOne;
  const uint32_t pos_from = (uint32_t)(E.base + (E.h_max + 1) / 2);  // lattice index of h = +1
  const uint32_t v_top = (uint32_t)(E.base + E.h_max);
  constexpr int kStride = kWsPerGroup * 32;   // chunk distance between a lane's two chunks
  const int grp = ci / kWsPerGroup, wi = ci % kWsPerGroup;
  // the schedulers whose slots this group takes: grp, grp + kWsGroups, ...
  unsigned mine = 0;
  for (int j = grp; j < kWsSched; j += kWsGroups) mine |= 1u << j;
  uint64_t sparse_bytes = 0;
  unsigned finished = 0;
#pragma unroll 1
  for (uint32_t seq = (uint32_t)grp; finished != mine; seq += kWsGroups) {
    const int j = (int)(seq % kWsSched);
    if ((finished >> j) & 1u) continue;
    const int s = (int)(seq % kWsSlots);
    if (!__all_sync(kFull, tc::mbar_wait(&sh->full[s], (seq / kWsSlots) & 1u, failed))) break;
    uint8_t* sl = slot_ptr(ring, s);
    const SlotMeta meta = *reinterpret_cast<const SlotMeta*>(sl + kOffMeta);
    if (meta.type == kSlotEnd) {
      finished |= 1u << j;
      continue;
    }
    int16_t* hrow = meta.hrow;
    const uint64_t* ev = reinterpret_cast<const uint64_t*>(sl + kOffEv);
    if (meta.type == kSlotSparse) {
      // a row without tuple: its reinforcement events as single-weight RMWs
      const int nblk = (meta.nin + 63) / 64;
      for (int b = wi * 32 + lane; b < nblk; b += kStride) {
        uint64_t mask = ev[b];
        sparse_bytes += 4ull * (uint64_t)__popcll(mask);
#pragma unroll 1
        while (mask != 0ull) {
          const int bit = __ffsll((long long)mask) - 1;
          mask &= mask - 1ull;
          int16_t* hp = hrow + 64 * b + bit;
          const uint32_t v = (uint16_t)*hp;
          *hp = (int16_t)((v >= pos_from) ? min(v + 1u, v_top) : max(v - 1u, (uint32_t)E.base));
        }
      }
    } else {
      const int n_t = meta.n_t;
      const int32_t* tl = reinterpret_cast<const int32_t*>(sl + kOffTup);
      const uint8_t* act = sl + kOffAct;
      const int nin = meta.nin;                    // real inputs of the segment
      const int nch = (nin + 7) >> 3;              // chunks holding at least one input
      const int full = nin >> 3;                   // chunks of 8 real inputs
      const int ch0 = meta.ch0;                    // chunk offset of the segment in the row
      const uint32_t arow_bytes = (uint32_t)meta.arow_bytes;
      const uint8_t* aseg = meta.aprev;            // activation row 0 at the segment's first byte
      const uint8_t* aprev = aseg - ch0;           // ... at the row's first byte
      const int nstage = meta.act_smem ? min(n_t, kActT) : 0;
      uint8_t* wrow = meta.wrow;
      const uint4* hs = reinterpret_cast<const uint4*>(sl + kOffH);
#pragma unroll 1
      for (int cb = wi * 32; cb < nch; cb += 2 * kStride) {
        int chv[2];
        bool live[2];
        uint4 w[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          chv[u] = cb + u * kStride + lane;
          live[u] = chv[u] < nch;
          w[u] = live[u] ? hs[chv[u]] : make_uint4(0, 0, 0, 0);
        }
        const uint4 w_in[2] = {w[0], w[1]};
        // ---- CP tuples, ascending mu ----
#pragma unroll 1
        for (int q = 0; q < n_t; ++q) {
          const int e = tl[q];
          const uint32_t xm = (e & 0x10000) ? 0xFFu : 0u;   // rho = -1: ~byte
          const uint8_t* arow = aseg + (size_t)(e & 0xFFFF) * arow_bytes;
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            uint32_t byte = 0u;
            if (live[u]) byte = q < nstage ? act[q * (kSegW / 8) + chv[u]] : arow[chv[u]];
            const uint4 d = sh->db[(byte ^ xm) & 0xFFu];
            w[u].x = LN.clip(w[u].x + d.x);
            w[u].y = LN.clip(w[u].y + d.y);
            w[u].z = LN.clip(w[u].z + d.z);
            w[u].w = LN.clip(w[u].w + d.w);
          }
        }
        // ---- W bytes (reinforcement never flips a sign, so W is final
        // after CP), H back into the slot ----
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          if (!live[u]) continue;
          uint32_t wbyte = LN.w_byte(w[u]);
          if (chv[u] >= full) {
            // the partly padded last chunk of the row: CP per weight, from the row as loaded
            const ChunkOut o = chunk_scalar(w_in[u], ch0 + chv[u], nin - 8 * chv[u], tl, n_t, aprev,
                                            arow_bytes, E, 0u);
            w[u] = o.w;
            wbyte = o.wbyte;
          }
          reinterpret_cast<uint4*>(sl + kOffH)[chv[u]] = w[u];
          wrow[chv[u]] = (uint8_t)wbyte;
        }
      }
      // ---- R, after every CP of the segment: the row's few events, applied in
      // the slot (lanes take event words) ----
      group_sync(grp);
      {
        int16_t* hseg = reinterpret_cast<int16_t*>(sl + kOffH);
        const int nblk = (nin + 63) / 64;
        for (int b = wi * 32 + lane; b < nblk; b += kStride) {
          uint64_t mask = ev[b];
#pragma unroll 1
          while (mask != 0ull) {
            const int bit = __ffsll((long long)mask) - 1;
            mask &= mask - 1ull;
            int16_t* hp = hseg + 64 * b + bit;
            const uint32_t v = (uint16_t)*hp;
            *hp = (int16_t)((v >= pos_from) ? min(v + 1u, v_top) : max(v - 1u, (uint32_t)E.base));
          }
        }
      }
      // the slot's H to global memory in one bulk copy (the generic-proxy
      // writes above are fenced for the copy engine by every writer)
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      group_sync(grp);
      if (wi == 0 && lane == 0) {
        asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
                     ::"l"(hrow), "r"(tc::smem_u32(sl + kOffH)), "r"((uint32_t)(2 * meta.nseg)) : "memory");
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");   // the slot may be refilled
      }
    }
    __syncwarp();
    if (lane == 0) tc::mbar_arrive(&sh->empty[s]);
  }
  // the group's bulk stores of H complete before the kernel ends
  if (wi == 0 && lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  if (sparse_bytes) atomicAdd(&sh->stats[2], sparse_bytes);
}

template <int kHb>
__global__ void __launch_bounds__(kWsThreads, 1) k_update_ws(const StepParams* __restrict__ P) {
  extern __shared__ uint8_t ws_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(ws_raw) + 127) &
                                             ~static_cast<uintptr_t>(127));
  WsShared* sh = reinterpret_cast<WsShared*>(ring + (size_t)kWsSlots * kSlotBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  Ctrl* ctrl = P->ctrl;
  // tables and barriers: independent of every earlier kernel
  if (threadIdx.x < 256) {
    // db[b]: the +-1 lattice steps of the 8 weights of a chunk whose activation
    // byte is b, for rho = +1 (rho = -1 indexes with ~b), two lanes per word
    // (d_lo + 2^16 d_hi: one 32-bit add steps both lanes)
    const int b = threadIdx.x;
    uint32_t wv[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int d0 = ((b >> (2 * q)) & 1) ? 1 : -1, d1 = ((b >> (2 * q + 1)) & 1) ? 1 : -1;
      wv[q] = (uint32_t)(d0 + 65536 * d1);
    }
    sh->db[b] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
  if (threadIdx.x < kWsSlots) sh->issued[threadIdx.x] = -1;
  if (threadIdx.x == 0) {
    for (int q = 0; q < kWsSlots; ++q) {
      tc::mbar_init(&sh->full[q], 1);
      tc::mbar_init(&sh->empty[q], kWsPerGroup);
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
  for (int i = threadIdx.x; i < bsz; i += kWsThreads) {
    const int yv = P->y[start + i];
    sh->y[i] = (yv < 0 || yv >= P->c) ? 0 : yv;   // memory-safe stand-in; the host reports bad labels
  }
  __syncthreads();
  if (warp < kWsSched)
    ws_scheduler(P, sh, ring, warp, lane, start, bsz, step_failed);
  else
    ws_consumer<kHb>(P, sh, ring, warp - kWsSched, lane);
  __syncthreads();
  if (sh->failed && threadIdx.x < kWsSlots && sh->issued[threadIdx.x] >= 0) {
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

}  // namespace

size_t update_ws_smem() { return kWsSmemBytes; }

cudaError_t prepare_update_ws() {
  cudaError_t e = cudaFuncSetAttribute(k_update_ws<8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kWsSmemBytes);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_update_ws<-1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)kWsSmemBytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_update_ws<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kWsSmemBytes);
}

cudaError_t launch_update_ws(int hb_mode, unsigned grid, cudaStream_t st, bool pdl, const StepParams* P) {
  if (hb_mode == 8)
    return launch_kernel(k_update_ws<8>, dim3(grid), dim3(kWsThreads), kWsSmemBytes, st, pdl, P);
  if (hb_mode != 0)
    return launch_kernel(k_update_ws<-1>, dim3(grid), dim3(kWsThreads), kWsSmemBytes, st, pdl, P);
  return launch_kernel(k_update_ws<0>, dim3(grid), dim3(kWsThreads), kWsSmemBytes, st, pdl, P);
}

}  // namespace bk
