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

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Number of 32-key chunks, counted from the warp's first readable key column
// wbs, up to the last key any of the warp's 32 query rows (warp*32 .. +31)
// can see in a diagonal tile.
__device__ __forceinline__ int chunks_needed(int warp, int wbs) { return (warp * 32 - wbs) / 32 + 1; }

}  // namespace attn
}  // namespace bcmt
