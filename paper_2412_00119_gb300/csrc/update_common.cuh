// update_common.cuh -- bit-sliced arithmetic on the hidden weights, shared by
// the update, initialisation and repack kernels (Alg. 3: the clipped
// perceptron and reinforcement steps; Sec. 3.1: W = sign(H)).
//
// A group is 32 weights of one neuron row held as kP 32-bit planes u[0..kP):
// bit j of u[p] is bit p of the lattice index u_j = (h_j + h_max)/2 of weight
// j (DevLayer::H).  h_j moves by 2 per event, so u_j moves by 1, clipped to
// [0, h_max]; h_j > 0 iff u_j >= (h_max + 1)/2.  One step of +-1 on all 32
// weights is a ripple through the planes: the lanes that move flip plane 0,
// and a lane's carry (moving up) or borrow (moving down) reaches plane p + 1
// while its bit p was 1 (up) or 0 (down).  The clip removes from the moving
// lanes those already at h_max (moving up) or at 0 (moving down): no lane
// leaves [0, h_max], so no carry passes the top plane.
#pragma once

#include "bmlp_internal.cuh"

namespace bk {
namespace upd {

constexpr unsigned kFull = 0xffffffffu;

// Planes used by the lattice index of h_max (the bits of h_max) and stored per
// group (that count rounded up to a power of two: 1, 2, 4, 8 or 16).
__host__ __device__ inline int bits_of(int h_max) {
  int b = 1;
  while ((1 << b) <= h_max) ++b;
  return b;
}
__host__ __device__ inline int planes_of(int nbits) {
  int p = 1;
  while (p < nbits) p <<= 1;
  return p;
}

// A constant broadcast to 32 lanes, plane by plane: m[p] = all ones where
// bit p of v is set.
template <int kP>
struct PlaneConst {
  uint32_t m[kP];
  __device__ __forceinline__ explicit PlaneConst(int v) {
#pragma unroll
    for (int p = 0; p < kP; ++p) m[p] = ((v >> p) & 1) ? kFull : 0u;
  }
};

// kOnes: h_max = 2^kP - 1, every stored plane is used, the upper bound is
// all ones and h > 0 is the top plane.
template <int kP, bool kOnes>
struct Sliced {
  PlaneConst<kP> hm;  // h_max
  PlaneConst<kP> pm;  // (h_max + 1)/2, the lattice index of h = +1
  __device__ __forceinline__ explicit Sliced(int h_max) : hm(h_max), pm((h_max + 1) / 2) {}

  // lanes with u == h_max
  __device__ __forceinline__ uint32_t at_top(const uint32_t (&u)[kP]) const {
    uint32_t r = kFull;
#pragma unroll
    for (int p = 0; p < kP; ++p) r &= kOnes ? u[p] : ~(u[p] ^ hm.m[p]);
    return r;
  }
  // lanes with u > 0
  __device__ __forceinline__ uint32_t nonzero(const uint32_t (&u)[kP]) const {
    uint32_t r = 0u;
#pragma unroll
    for (int p = 0; p < kP; ++p) r |= u[p];
    return r;
  }
  // The lanes of en step: up where d is set, down elsewhere; a lane at the
  // bound in its direction stays.
  __device__ __forceinline__ void step(uint32_t (&u)[kP], uint32_t d, uint32_t en) const {
    const uint32_t top = at_top(u), nz = nonzero(u);
    uint32_t k = en & ((d & ~top) | (~d & nz));
    const uint32_t nd = ~d;
#pragma unroll
    for (int p = 0; p < kP; ++p) {
      const uint32_t nk = k & (u[p] ^ nd);  // carry on 1 (up) / borrow on 0 (down)
      u[p] ^= k;
      k = nk;
    }
  }
  // lanes with h > 0, i.e. u >= (h_max + 1)/2
  __device__ __forceinline__ uint32_t positive(const uint32_t (&u)[kP]) const {
    if (kOnes) return u[kP - 1];
    uint32_t gt = 0u, eq = kFull;
#pragma unroll
    for (int p = kP - 1; p >= 0; --p) {
      gt |= eq & u[p] & ~pm.m[p];
      eq &= ~(u[p] ^ pm.m[p]);
    }
    return gt | eq;
  }
};

// The kP planes of one group (16-byte aligned for kP >= 4).
template <int kP>
__device__ __forceinline__ void load_planes(uint32_t (&u)[kP], const uint32_t* src) {
  if constexpr (kP >= 4) {
#pragma unroll
    for (int q = 0; q < kP / 4; ++q) {
      const uint4 v = reinterpret_cast<const uint4*>(src)[q];
      u[4 * q] = v.x; u[4 * q + 1] = v.y; u[4 * q + 2] = v.z; u[4 * q + 3] = v.w;
    }
  } else if constexpr (kP == 2) {
    const uint2 v = *reinterpret_cast<const uint2*>(src);
    u[0] = v.x; u[1] = v.y;
  } else {
    u[0] = *src;
  }
}

template <int kP>
__device__ __forceinline__ void store_planes(uint32_t* dst, const uint32_t (&u)[kP]) {
  if constexpr (kP >= 4) {
#pragma unroll
    for (int q = 0; q < kP / 4; ++q)
      reinterpret_cast<uint4*>(dst)[q] = make_uint4(u[4 * q], u[4 * q + 1], u[4 * q + 2], u[4 * q + 3]);
  } else if constexpr (kP == 2) {
    *reinterpret_cast<uint2*>(dst) = make_uint2(u[0], u[1]);
  } else {
    *dst = u[0];
  }
}

__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) {
  return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// Valid-input mask of group g of a row of Kin inputs.
__host__ __device__ __forceinline__ uint32_t group_mask(int g, int Kin) {
  const int n = Kin - 32 * g;
  return n >= 32 ? 0xffffffffu : (n <= 0 ? 0u : ((1u << n) - 1u));
}

}  // namespace upd
}  // namespace bk
