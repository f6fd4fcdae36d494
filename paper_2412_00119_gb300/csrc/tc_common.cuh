// tc_common.cuh -- device helpers shared by the tcgen05 forward kernels:
// mbarrier waits (bounded), shared-memory matrix descriptors, the
// tcgen05.mma kind::f8f6f4 issue and commit, and the expansion of bit-packed
// +-1 vectors into e4m3 bytes in the 128B-swizzled K-major stage layout.
#pragma once

#include "bmlp_internal.cuh"

namespace bk {
namespace tc {

constexpr unsigned kFull = 0xffffffffu;
constexpr int KB = 128;  // K elements (bytes of e4m3) per stage row
constexpr unsigned long long kWaitCycles = 4000000000ull;  // ~2 s at 2 GHz

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(unsigned long long* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_arrive(unsigned long long* bar) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}"
               ::"r"(smem_u32(bar)) : "memory");
}

// Bounded wait for the phase with the given parity; false on expiry (after
// `limit` SM clock cycles) or when another thread already recorded a failure.
__device__ __forceinline__ bool mbar_wait(unsigned long long* bar, uint32_t parity,
                                          volatile int* failed,
                                          unsigned long long limit = kWaitCycles) {
  const uint32_t a = smem_u32(bar);
  const unsigned long long t0 = clock64();
  while (true) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok) : "r"(a), "r"(parity) : "memory");
    if (ok) return true;
    if (*failed) return false;
    if (clock64() - t0 > limit) {
      *failed = 1;
      return false;
    }
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

// Instruction descriptor, kind::f8f6f4: D fp32, A = B = e4m3, both K-major,
// M x N per instruction (K = 32).
constexpr uint32_t idesc_f8(int M, int N) {
  return (1u << 4)                        // D format: f32
         | (0u << 7) | (0u << 10)         // A, B format: e4m3
         | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

template <uint32_t kIdesc>
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

// 8 bits -> 8 e4m3 bytes (+1 = 0x38, -1 = 0xB8) as two words.  Byte j of the
// replicated value keeps bit j of b; adding (0x80 - 2^j) per byte moves it to
// bit 7 without carries between bytes.
__device__ __forceinline__ uint2 expand8(uint32_t b) {
  const uint32_t rep = b * 0x01010101u;
  const uint32_t lo = (rep & 0x08040201u) + 0x787C7E7Fu;
  const uint32_t hi = (rep & 0x80402010u) + 0x00406070u;
  return make_uint2((lo & 0x80808080u) ^ 0xB8B8B8B8u, (hi & 0x80808080u) ^ 0xB8B8B8B8u);
}

__device__ __forceinline__ void mbar_arrive_tx(unsigned long long* bar, uint32_t bytes) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}"
               ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

// 1-D bulk copy global -> this CTA's shared memory, completing on `bar`
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         unsigned long long* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// A producer item: one 16-byte chunk of one row of a stage, i.e. 16
// K-elements (two bytes of bits) -> 16 e4m3 bytes.  The chunk's logical index
// c (K-elements 16c .. 16c + 15 of the stage's 128) is stored at physical
// chunk c ^ (r % 8) of row r (SWIZZLE_128B).
struct Chunk {
  const uint16_t* src;  // the row's bits as 16-bit pieces; null: no item
  uint32_t dst;         // byte offset of the chunk inside a stage
  int c;                // logical chunk 0..7
};

// Item for row r (of a matrix whose rows start `soff` bytes into the stage).
__device__ __forceinline__ Chunk make_chunk(const uint64_t* row, int soff, int r, int c) {
  return Chunk{reinterpret_cast<const uint16_t*>(row),
               (uint32_t)(soff + r * KB + 16 * (c ^ (r & 7))), c};
}

// The item's 16 bits for k-block kb (0 past the row's nw words).
__device__ __forceinline__ uint32_t load_chunk(const Chunk& ch, int kb, int nw) {
  const int pi = 8 * kb + ch.c;
  return (ch.src != nullptr && pi < 4 * nw) ? (uint32_t)__ldg(ch.src + pi) : 0u;
}

// Bytes of a 4-byte group to keep when n_ok of its elements are real.
__device__ __forceinline__ uint32_t keep_mask(int n_ok) {
  return n_ok >= 4 ? 0xFFFFFFFFu : (n_ok <= 0 ? 0u : ((1u << (8 * n_ok)) - 1u));
}

// Four K-elements, bits P .. P + 3 of x (P = 0 or 4), as four e4m3 bytes
// (bit 1 -> 0x38 = +1, bit 0 -> 0xB8 = -1): the product places bit P + j at
// bit 8 j + 7; its four shifted copies of the masked nibble do not overlap,
// so it carries nothing.
template <int P>
__device__ __forceinline__ uint32_t e4m3_quad(uint32_t x) {
  static_assert(P == 0 || P == 4, "nibble position");
  constexpr uint32_t kMul = P == 0 ? 0x10204080u : 0x01020408u;
  return ((x & (0xFu << P)) * kMul & 0x80808080u) ^ 0xB8B8B8B8u;
}

// 16 K-elements (bits 0..15 of h) -> one 16-byte chunk.
__device__ __forceinline__ uint4 chunk16(uint32_t h) {
  return make_uint4(e4m3_quad<0>(h), e4m3_quad<4>(h), e4m3_quad<0>(h >> 8), e4m3_quad<4>(h >> 8));
}

// The same with the elements at index >= valid set to 0 (ragged K only).
__device__ __forceinline__ uint4 chunk16_masked(uint32_t h, int valid) {
  uint4 v = chunk16(h);
  v.x &= keep_mask(valid);
  v.y &= keep_mask(valid - 4);
  v.z &= keep_mask(valid - 8);
  v.w &= keep_mask(valid - 12);
  return v;
}

// Expand the item's bits into its stage chunk; elements at K >= Kin are 0.
__device__ __forceinline__ void store_chunk(uint8_t* stage, const Chunk& ch, uint32_t bits, int kb,
                                            int Kin) {
  const uint2 e0 = expand8(bits & 0xFFu);
  const uint2 e1 = expand8(bits >> 8);
  uint4 v = make_uint4(e0.x, e0.y, e1.x, e1.y);
  const int valid = Kin - (KB * kb + 16 * ch.c);
  if (valid < 16) {
    v.x &= keep_mask(valid);
    v.y &= keep_mask(valid - 4);
    v.z &= keep_mask(valid - 8);
    v.w &= keep_mask(valid - 12);
  }
  *reinterpret_cast<uint4*>(stage + ch.dst) = v;
}

// A producer item of 64 K-elements: one (row, half) of a stage row, i.e. one
// 64-bit word of bits -> four 16-byte chunks (chunks 4 half .. 4 half + 3).
struct Item {
  const uint64_t* src;  // row start (bit words), or null when the thread has no item
  uint32_t dst;         // byte offset of the row inside a stage
  int r;                // row index inside its matrix (for the swizzle)
  int half;             // which of the stage's two words
};

__device__ __forceinline__ uint64_t load_word(const Item& it, int kb, int nw) {
  const int wi = 2 * kb + it.half;
  return (it.src != nullptr && wi < nw) ? __ldg(it.src + wi) : 0ull;
}

// Expand the item's word for k-block kb into its four chunks; elements at
// K >= Kin are 0.
__device__ __forceinline__ void store_word(uint8_t* stage, const Item& it, uint64_t w, int kb,
                                           int Kin) {
  const int valid = Kin - (KB * kb + 64 * it.half);
#pragma unroll
  for (int q = 0; q < 4; ++q) {  // chunk 4 half + q: elements 16 q .. 16 q + 15 of the word
    const uint32_t bits = (uint32_t)(w >> (16 * q)) & 0xFFFFu;
    const uint2 e0 = expand8(bits & 0xFFu);
    const uint2 e1 = expand8(bits >> 8);
    uint4 v = make_uint4(e0.x, e0.y, e1.x, e1.y);
    if (valid < 64) {
      const int n = valid - 16 * q;
      v.x &= keep_mask(n);
      v.y &= keep_mask(n - 4);
      v.z &= keep_mask(n - 8);
      v.w &= keep_mask(n - 12);
    }
    const int c = 4 * it.half + q;
    *reinterpret_cast<uint4*>(stage + it.dst + 16 * (c ^ (it.r & 7))) = v;
  }
}

}  // namespace tc
}  // namespace bk
