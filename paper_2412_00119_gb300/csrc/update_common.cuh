// update_common.cuh -- per-chunk arithmetic of the hidden-weight update
// (Alg. 3: clipped perceptron, reinforcement, and the repack of W = sign(H),
// Sec. 3.1) shared by the update kernels.  A chunk is 8 consecutive hidden
// weights of one neuron row (16 bytes of int16 lattice indices v = (h +
// h_max)/2 + 2^hb, two 16-bit lanes per 32-bit word; see DevLayer::H).
#pragma once

#include "bmlp_internal.cuh"

namespace bk {
namespace upd {

constexpr uint32_t kLaneTop = 0x80008000u;
constexpr uint32_t kLaneOne = 0x00010001u;
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ uint32_t lane_v(const uint4& w, int j) {
  const uint32_t word = (j < 2) ? w.x : (j < 4) ? w.y : (j < 6) ? w.z : w.w;
  return (word >> (16 * (j & 1))) & 0xFFFFu;
}

__device__ __forceinline__ void set_lane_v(uint4& w, int j, uint32_t v) {
  const int sh = 16 * (j & 1);
  const uint32_t m = ~(0xFFFFu << sh), x = (v & 0xFFFFu) << sh;
  if (j < 2) w.x = (w.x & m) | x;
  else if (j < 4) w.y = (w.y & m) | x;
  else if (j < 6) w.z = (w.z & m) | x;
  else w.w = (w.w & m) | x;
}

struct ChunkOut {
  uint4 w;
  uint32_t wbyte;
};

struct Enc {
  int h_max, hb, base;  // v = (h + h_max)/2 + base, base = 2^hb
  __device__ __forceinline__ int dec(uint32_t v) const { return 2 * ((int)v - base) - h_max; }
  __device__ __forceinline__ uint32_t enc(int h) const { return (uint32_t)((h + h_max) / 2 + base); }
};

// Per-weight path (rule as printed, on decoded h): CP, then R for the inputs
// whose bit of `fire` is set, and W, for the first `nvalid` weights of the
// chunk.  Taken only by the ragged last chunk of a row; its loops stay rolled.
__device__ __forceinline__ ChunkOut chunk_scalar(uint4 w, int ch, int nvalid, const int32_t* list,
                                                 int n_t, const uint8_t* aprev, uint32_t arow_bytes,
                                                 Enc E, uint32_t fire) {
#pragma unroll 1
  for (int q = 0; q < n_t; ++q) {
    const int e = list[q];
    const int m = e & 0xFFFF;
    const int rho = (e & 0x10000) ? -1 : 1;
    const uint32_t byte = aprev[(size_t)m * arow_bytes + ch];
#pragma unroll 1
    for (int j = 0; j < nvalid; ++j) {
      const int step = ((byte >> j) & 1u) ? rho : -rho;
      set_lane_v(w, j, E.enc(clip_h(E.dec(lane_v(w, j)) + 2 * step, E.h_max)));
    }
  }
  ChunkOut out;
  out.wbyte = 0;
#pragma unroll 1
  for (int j = 0; j < nvalid; ++j) {
    int h = E.dec(lane_v(w, j));
    if ((fire >> j) & 1u) {
      h = clip_h(h + (h > 0 ? 2 : -2), E.h_max);
      set_lane_v(w, j, E.enc(h));
    }
    out.wbyte |= (h > 0 ? 1u : 0u) << j;
  }
  out.w = w;
  return out;
}

// bit 15 of every lane of w equal to the lane value of cpair (exact, carry-free)
__device__ __forceinline__ uint32_t eq_flags(uint32_t w, uint32_t cpair) {
  const uint32_t x = w ^ cpair;
  return ~(((x & 0x7FFF7FFFu) + 0x7FFF7FFFu) | x) & kLaneTop;
}

// Gather bit 15 of the 8 lanes into a byte (lane j -> bit j).
__device__ __forceinline__ uint32_t gather_top(uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  const uint32_t p0 = __byte_perm(a, b, 0x7531) & 0x80808080u;
  const uint32_t p1 = __byte_perm(c, d, 0x7531) & 0x80808080u;
  return ((p0 * 0x00204081u) >> 28) | (((p1 * 0x00204081u) >> 28) << 4);
}

// kHb > 0: h_max + 1 = 2^kHb, a compile-time exponent; kHb = -1: h_max + 1 a
// power of two given at run time; kHb = 0: any odd h_max.
template <int kHb>
struct Lanes {
  static constexpr bool kPow2 = kHb != 0;
  int hb_rt;
  __device__ __forceinline__ int hb() const { return kHb > 0 ? kHb : hb_rt; }
  uint32_t over_pair;  // pair(2^hb + h_max + 1), used when !kPow2
  uint32_t pos_pair;   // pair(2^hb + (h_max + 1)/2), used when !kPow2
  // lanes that left [2^hb, 2^hb + h_max] by one step go back
  __device__ __forceinline__ uint32_t clip(uint32_t v) const {
    if (kPow2) {
      const uint32_t t = (v >> hb()) & 0x00030003u;  // 0 under, 1 inside, 2 over
      return v + kLaneOne - t;
    } else {
      const uint32_t under = (~v >> hb()) & kLaneOne;
      return v + under - (eq_flags(v, over_pair) >> 15);
    }
  }
  // bit 15 of each lane = (h > 0)
  __device__ __forceinline__ uint32_t pos_top(uint32_t v) const {
    if (kPow2) return (v << (16 - hb())) & kLaneTop;
    return ((v | kLaneTop) - pos_pair) & kLaneTop;
  }
  // lanes with f = 1 (f: 0 or 1 per lane) step away from 0, then clip
  __device__ __forceinline__ uint32_t reinforce(uint32_t v, uint32_t f) const {
    const uint32_t p = pos_top(v) >> 15;
    return clip(v + (f & p) - (f & ~p));
  }
  // W byte of a chunk (lane j -> bit j = h_j > 0)
  __device__ __forceinline__ uint32_t w_byte(const uint4& w) const {
    if (kPow2) {
      // move each lane's sign bit (bit hb - 1) to bit 7 of the lane's low byte;
      // the low bytes of the 8 lanes then hold the 8 sign bits at bit 7
      const int sh = 8 - hb();
      const uint32_t x = sh >= 0 ? w.x << sh : w.x >> -sh, y = sh >= 0 ? w.y << sh : w.y >> -sh;
      const uint32_t z = sh >= 0 ? w.z << sh : w.z >> -sh, u = sh >= 0 ? w.w << sh : w.w >> -sh;
      const uint32_t p0 = __byte_perm(x, y, 0x6420) & 0x80808080u;
      const uint32_t p1 = __byte_perm(z, u, 0x6420) & 0x80808080u;
      return ((p0 * 0x00204081u) >> 28) | (((p1 * 0x00204081u) >> 28) << 4);
    }
    return gather_top(pos_top(w.x), pos_top(w.y), pos_top(w.z), pos_top(w.w));
  }
};

__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) {
  return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

}  // namespace upd
}  // namespace bk
