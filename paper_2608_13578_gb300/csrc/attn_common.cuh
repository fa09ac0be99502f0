// Shared-memory helpers of the tcgen05 attention kernels.
#pragma once

#include "common.cuh"
#include "tc.cuh"

namespace bcmt {
namespace attn {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Writes 16-byte unit `u` (keys 8u .. 8u+7) of row r of a 128 x 128 bf16
// K-major operand stored as two 128-row swizzle-128 atoms (keys 0-63, 64-127).
__device__ __forceinline__ void put_unit(uint8_t* base, int r, int u, uint4 val) {
  *reinterpret_cast<uint4*>(base + (u >> 3) * 16384 + tc::sw128_offset(r, u & 7)) = val;
}

// 2^x by the ex2.approx.ftz instruction (relative error near 2^-22, 2^-inf =
// +0): for probabilities that are rounded to bf16 or summed in fp32.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}

__device__ __forceinline__ uint4 pack8(const float* v) {
  return make_uint4(pack2(v[0], v[1]), pack2(v[2], v[3]), pack2(v[4], v[5]), pack2(v[6], v[7]));
}

// A 128-row x DH bf16 tile (DH in {16, 32, 64}) as TMA writes it with the
// swizzle whose span is one row (DH * 2 bytes: 32, 64 or 128), and the MMA
// operand descriptors that read it.
template <int DH>
struct Geo {
  static constexpr uint32_t span = DH * 2;    // bytes per tile row
  static constexpr uint32_t tile = 128 * span;  // one 128-row tile
  static constexpr uint32_t sbo = 8 * span;   // 8-row atom
  static constexpr uint32_t layout = DH == 64 ? 2u : DH == 32 ? 4u : 6u;
  // K-major [rows x DH] operand at row offset `row0`, K step kk (16 columns)
  static __device__ __forceinline__ uint64_t kmaj(const uint8_t* t, int row0, int kk) {
    return tc::sdesc_sw(tc::smem_u32(t) + row0 * span + kk * 32, 16, sbo, layout);
  }
  // the same tile read MN-major (DH contiguous = N), K = rows from row0, step kk
  static __device__ __forceinline__ uint64_t mnmaj(const uint8_t* t, int row0, int kk) {
    return tc::sdesc_sw(tc::smem_u32(t) + (row0 + kk * 16) * span, tile, sbo, layout);
  }
  // byte offset of 16-byte unit u (columns 8u .. 8u+7) of row r: the unit
  // index is XORed with address bits 7.. of the unswizzled offset (1, 2 or 3
  // bits for the 32-, 64- and 128-byte swizzles)
  static __device__ __forceinline__ uint32_t unit(int r, int u) {
    const uint32_t o = (uint32_t)r * span + (uint32_t)u * 16u;
    constexpr uint32_t mask = DH == 64 ? 7u : DH == 32 ? 3u : 1u;
    return o ^ (((o >> 7) & mask) << 4);
  }
};

// A [128 x 128] bf16 operand in two 64-column swizzle-128 halves (put_unit's
// layout), read K-major from column 64*half, K step kk.  A single 64-column
// half buffer is read with half = 0 and kk < 4.
__device__ __forceinline__ uint64_t p_kmaj(const uint8_t* p, int half, int kk) {
  return tc::sdesc(tc::smem_u32(p) + half * 16384 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
}

// Loads TMEM columns col .. col+DH-1 of the warp's lane quarter (thread = row).
template <int DH>
__device__ __forceinline__ void tmem_row(uint32_t taddr, float* v) {
  uint32_t r[2][32];
  tc::tmem_ld32_issue(taddr, r[0]);
  if (DH > 32) tc::tmem_ld32_issue(taddr + 32u, r[1]);
  tc::tmem_wait();
#pragma unroll
  for (int c = 0; c < DH; ++c) v[c] = __uint_as_float(r[c >> 5][c & 31]);
}

template <int DH>
__device__ __forceinline__ void store_row(bf16* dst, const float* v, float mul) {
#pragma unroll
  for (int u = 0; u < DH / 8; ++u) {
    float t[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) t[e] = v[8 * u + e] * mul;
    *reinterpret_cast<uint4*>(dst + 8 * u) = pack8(t);
  }
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Number of 32-key chunks, counted from the warp's first readable key column
// wbs, up to the last key any of the warp's 32 query rows (warp*32 .. +31)
// can see in a diagonal tile.
__device__ __forceinline__ int chunks_needed(int warp, int wbs) { return (warp * 32 - wbs) / 32 + 1; }

}  // namespace attn
}  // namespace bcmt
