// Intra-block causal attention on the tcgen05 tensor cores (Sec. 3.3), bf16
// operands, head width DH in {16, 32, 64}, block size L in {16, 32, 64, 128}.
//
// One CTA per (128-token tile, head, batch); 128 % L == 0, so a tile holds
// 128 / L whole blocks and its keys are its own 128 tokens.  The attention
// pattern inside the tile is block-diagonal causal: query r sees keys
// [blockstart(r), r].  TMA brings the Q, K, V head slices of the tile into
// shared memory (the swizzle whose span is one DH-wide row; a 3-D tensor map
// per operand zero-fills tokens past the end of the sequence), tcgen05.mma
// computes the scores into TMEM, each thread owns one query row for the
// masked softmax (the whole row fits in TMEM, so there is no online
// rescaling), writes P in bf16 back to shared memory as the A operand of
// P V, and the normalised output leaves
// through a TMA store.  The backward recomputes P from the saved log-sum-exp
// and runs the five products S = Q K^T, dP = dO V^T, dV = P^T dO,
// dQ = dS K, dK = dS^T Q on the tensor cores, reading the same shared tiles
// K-major or MN-major as each product needs.
#include "attn_common.cuh"
#include "common.cuh"
#include "internal.h"
#include "tc.cuh"
#include "tmap.h"

namespace bcmt {
using namespace attn;

namespace {
constexpr int kTile = 128;
}  // namespace

// Both kernels are instantiated for NCH = the number of 32-key chunks of a
// block that one warp's 32 query rows can reach (1 for L <= 32, L / 32
// otherwise); a warp reads only the chunks up to its own last row's key, the
// rest of its P and dS rows are causal zeros.

// Stores one DH-wide fp32 row as bf16 into row r of a 128 x DH swizzled tile
// (the TMA store layout).
template <int DH>
__device__ __forceinline__ void stage_row(uint8_t* tile, int r, const float* v) {
#pragma unroll
  for (int u = 0; u < DH / 8; ++u)
    *reinterpret_cast<uint4*>(tile + Geo<DH>::unit(r, u)) = pack8(v + 8 * u);
}

// ====================================================================== forward
// For head widths DH in {16, 32, 64}.  At DH = 64 the P tile (32 KB) covers
// the Q and K tiles once S = Q K^T has consumed them; at DH = 16 / 32 it
// follows the three tiles.  The output is staged in the Q tile.
template <int DH> constexpr int fwd_smem_bytes() {
  return (DH == 64 ? 3 * Geo<DH>::tile : 3 * Geo<DH>::tile + 32768) + 1024 + 64;
}

template <int NCH, int DH>
__global__ void __launch_bounds__(128)
    attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mK,
                       const __grid_constant__ CUtensorMap mV, const __grid_constant__ CUtensorMap mO,
                       float* __restrict__ lse, int Tlen, int H, int L, float scale,
                       unsigned* status) {
  using G = Geo<DH>;
  constexpr uint32_t kT = G::tile;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem;            // Q; then the output staging tile
  uint8_t* sK = smem + kT;       // K
  uint8_t* sV = smem + 2 * kT;   // V
  uint8_t* sP = DH == 64 ? sQ : smem + 3 * kT;  // P (32 KB)
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + (DH == 64 ? 3 * kT : 3 * kT + 32768));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;

  // Setup overlaps the previous kernel (before pdl_wait); the loads go out
  // first after it, so the TMEM allocation and the block barrier overlap them.
  if (tid == 0) {
    for (int i = 0; i < 3; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar[0], 3 * kT);
    tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sK, &mK, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sV, &mV, &bar[0], h * DH, t0, b);
  }
  __syncwarp();
  if (warp == 0) {
    tc::tmem_alloc(tslot, 128);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);

  if (tid == 0) {
    const bool ok = tc::mbar_wait(&bar[0], 0, status);
    tc::fence_after_sync();
    if (ok) {
      constexpr uint32_t idS = tc::idesc_bf16(128, 128, 0, 0);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)
        tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK, 0, kk), idS, kk > 0 ? 1u : 0u);
    }
    tc::mma_commit(&bar[1]);
  }
  __syncwarp();

  bool ok = tc::mbar_wait(&bar[1], 0, status);
  tc::fence_after_sync();

  // ---- masked softmax, thread = query row r of the tile: the row's scores
  // (at most 128 keys) come out of TMEM in one batch of loads
  const int r = warp * 32 + lane;
  const int wbs = L < 32 ? warp * 32 : ((warp * 32) / L) * L;  // first key column read
  const int nld = chunks_needed(warp, wbs);                    // 32-column chunks read
  const int rbs = (r / L) * L;                              // first key row r may see
  const float sl2 = scale * kLog2e;
  uint32_t sr[NCH][32];
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci)
    if (ci < nld) tc::tmem_ld32_issue(trow + (uint32_t)(wbs + ci * 32), sr[ci]);
  tc::tmem_wait();
  // the max and the sum run in independent partials (short dependency chains)
  float mxp[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci)
    if (ci < nld) {
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const int kk = wbs + ci * 32 + j;
        if (kk >= rbs && kk <= r) mxp[j & 3] = fmaxf(mxp[j & 3], __uint_as_float(sr[ci][j]));
      }
    }
  const float mx = fmaxf(fmaxf(mxp[0], mxp[1]), fmaxf(mxp[2], mxp[3]));
  const float nm = -mx * sl2;
  float ps[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci)
    if (ci < nld) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        float v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int kk = wbs + ci * 32 + u * 8 + e;
          v[e] = (kk >= rbs && kk <= r) ? ex2(fmaf(__uint_as_float(sr[ci][u * 8 + e]), sl2, nm))
                                        : 0.f;
          ps[e & 3] += v[e];
        }
        put_unit(sP, r, (wbs + ci * 32) / 8 + u, pack8(v));
      }
    }
  const float sum = (ps[0] + ps[1]) + (ps[2] + ps[3]);
  const uint4 zero = make_uint4(0, 0, 0, 0);
  for (int u = 0; u < 16; ++u)
    if (u * 8 < wbs || u * 8 >= wbs + nld * 32) put_unit(sP, r, u, zero);
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();

  if (tid == 0) {
    tc::fence_after_sync();
    constexpr uint32_t idO = tc::idesc_bf16(128, DH, 0, 1);
#pragma unroll
    for (int kk = 0; kk < kTile / 16; ++kk)
      tc::mma_bf16(tmem, p_kmaj(sP, 0, kk), G::mnmaj(sV, 0, kk), idO, kk > 0 ? 1u : 0u);
    tc::mma_commit(&bar[2]);
  }
  __syncwarp();
  ok = tc::mbar_wait(&bar[2], 0, status) && ok;
  tc::fence_after_sync();

  // ---- epilogue: O = (P V) / sum, staged in the (now free) Q/P tile
  const float inv = 1.0f / sum;
  {
    float o[DH];
    tmem_row<DH>(trow, o);
#pragma unroll
    for (int c = 0; c < DH; ++c) o[c] *= inv;
    stage_row<DH>(sQ, r, o);
  }
  if (ok && t0 + r < Tlen) lse[((long)b * H + h) * Tlen + t0 + r] = mx * scale + logf(sum);
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0 && ok) {
    tc::tma_store_3d(&mO, sQ, h * DH, t0, b);
    tc::tma_store_commit();
    tc::tma_store_wait_read<0>();  // the staging is read; the writes finish with the grid
  }
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 128);
}

// ===================================================================== backward
// For head widths DH in {16, 32, 64}.  Shared memory: the Q, K, dO, V and O
// tiles (128 x DH, TMA-swizzled with a one-row span) and a 32 KB region that
// holds P (for dV = P^T dO), then scale * dS (for dK and dQ): dS waits in
// registers until the dV product has consumed P.  At DH = 64 the P region
// covers V and the 16 KB after it (96 KB per CTA: two CTAs per SM); at
// DH = 16 / 32 it follows the five tiles (52 / 72 KB).  O comes in by TMA
// with the other tiles (for Drow = dO . O).  The gradients leave through the
// Q, K, dO tiles as staging, in the same layout, by TMA stores.
template <int DH> constexpr int bwd_smem_bytes() {
  return (DH == 64 ? 6 * Geo<DH>::tile : 5 * Geo<DH>::tile + 32768) + 1024 + 64;
}

template <int NCH, int DH>
__global__ void __launch_bounds__(128)
    attn_bwd_tc_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mK,
                       const __grid_constant__ CUtensorMap mV, const __grid_constant__ CUtensorMap mdO,
                       const __grid_constant__ CUtensorMap mdQ, const __grid_constant__ CUtensorMap mdK,
                       const __grid_constant__ CUtensorMap mdV, const __grid_constant__ CUtensorMap mO,
                       const float* __restrict__ lse, int Tlen, int H, int L, float scale,
                       unsigned* status) {
  using G = Geo<DH>;
  constexpr uint32_t kT = G::tile;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem;              // Q; then dQ staging
  uint8_t* sK = smem + kT;         // K; then dK staging
  uint8_t* sdO = smem + 2 * kT;    // dO; then dV staging
  uint8_t* sV = smem + 3 * kT;     // V
  uint8_t* sO = smem + (DH == 64 ? 5 : 4) * kT;  // O
  uint8_t* sP = DH == 64 ? sV : smem + 5 * kT;    // P, then scale * dS (32 KB)
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + (DH == 64 ? 6 * kT : 5 * kT + 32768));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;

  if (tid == 0) {
    for (int i = 0; i < 4; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
    tc::prefetch_tmap(&mdO);
    tc::prefetch_tmap(&mO);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar[0], 5 * kT);
    tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sK, &mK, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sV, &mV, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sO, &mO, &bar[0], h * DH, t0, b);
  }
  __syncwarp();
  if (warp == 0) {
    tc::tmem_alloc(tslot, 256);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);

  if (tid == 0) {
    const bool ok = tc::mbar_wait(&bar[0], 0, status);
    tc::fence_after_sync();
    if (ok) {
      constexpr uint32_t id128 = tc::idesc_bf16(128, 128, 0, 0);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // S = Q K^T -> TMEM columns 0..127
        tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK, 0, kk), id128, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // dP = dO V^T -> TMEM columns 128..255
        tc::mma_bf16(tmem + 128, G::kmaj(sdO, 0, kk), G::kmaj(sV, 0, kk), id128,
                     kk > 0 ? 1u : 0u);
    }
    tc::mma_commit(&bar[1]);
  }
  __syncwarp();

  const int r = warp * 32 + lane;
  const bool row_ok = (t0 + r) < Tlen;
  const float lr = row_ok ? lse[((long)b * H + h) * Tlen + t0 + r] : 0.f;
  bool ok = tc::mbar_wait(&bar[0], 0, status);
  float drow = 0.f;  // Drow = dO_r . O_r from the staged tiles
  if (row_ok) {
#pragma unroll
    for (int u = 0; u < DH / 8; ++u) {
      const uint4 gv = *reinterpret_cast<const uint4*>(sdO + G::unit(r, u));
      const uint4 ov = *reinterpret_cast<const uint4*>(sO + G::unit(r, u));
      const bf16* gp = reinterpret_cast<const bf16*>(&gv);
      const bf16* op = reinterpret_cast<const bf16*>(&ov);
#pragma unroll
      for (int e = 0; e < 8; ++e) drow = fmaf(__bfloat162float(gp[e]), __bfloat162float(op[e]), drow);
    }
  }
  ok = tc::mbar_wait(&bar[1], 0, status) && ok;
  tc::fence_after_sync();

  // ---- P = exp(S*scale - lse) to shared memory; scale * P * (dP - Drow) kept
  // packed in registers (up to 128 keys: 64 words)
  const int wbs = L < 32 ? warp * 32 : ((warp * 32) / L) * L;
  const int nld = chunks_needed(warp, wbs);
  const int rbs = (r / L) * L;
  const float sl2 = scale * kLog2e, nl2 = -lr * kLog2e, ndr = -drow * scale;
  uint32_t dsp[NCH * 16];
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci) {
    if (ci < nld) {
      const int c = ci * 32;
      float s[32], dp[32];
      {
        uint32_t rs[32], rd[32];
        tc::tmem_ld32_issue(trow + (uint32_t)(wbs + c), rs);
        tc::tmem_ld32_issue(trow + 128u + (uint32_t)(wbs + c), rd);
        tc::tmem_wait();
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          s[j] = __uint_as_float(rs[j]);
          dp[j] = __uint_as_float(rd[j]);
        }
      }
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const int kk = wbs + c + j;
        const float p = (row_ok && kk >= rbs && kk <= r) ? ex2(fmaf(s[j], sl2, nl2)) : 0.f;
        s[j] = p;
        dp[j] = p * fmaf(dp[j], scale, ndr);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        uint4 q;
        q.x = pack2(s[8 * u + 0], s[8 * u + 1]);
        q.y = pack2(s[8 * u + 2], s[8 * u + 3]);
        q.z = pack2(s[8 * u + 4], s[8 * u + 5]);
        q.w = pack2(s[8 * u + 6], s[8 * u + 7]);
        put_unit(sP, r, (wbs + c) / 8 + u, q);
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) dsp[ci * 16 + j] = pack2(dp[2 * j], dp[2 * j + 1]);
    }
  }
  const uint4 zero = make_uint4(0, 0, 0, 0);
  for (int u = 0; u < 16; ++u)
    if (u * 8 < wbs || u * 8 >= wbs + nld * 32) put_unit(sP, r, u, zero);
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();

  if (tid == 0) {
    tc::fence_after_sync();
    // dV = P^T dO -> columns 0.. (A = P read MN-major: M = keys, K = queries)
    constexpr uint32_t idMN = tc::idesc_bf16(128, DH, 1, 1);
#pragma unroll
    for (int kk = 0; kk < kTile / 16; ++kk)
      tc::mma_bf16(tmem, tc::sdesc(tc::smem_u32(sP) + kk * 2048, 16384, 1024),
                   G::mnmaj(sdO, 0, kk), idMN, kk > 0 ? 1u : 0u);
    tc::mma_commit(&bar[2]);
  }
  __syncwarp();
  // P consumed: overwrite it with scale * dS
  ok = tc::mbar_wait(&bar[2], 0, status) && ok;
  tc::fence_after_sync();
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci) {
    if (ci < nld) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint4 d = make_uint4(dsp[ci * 16 + 4 * u], dsp[ci * 16 + 4 * u + 1],
                                   dsp[ci * 16 + 4 * u + 2], dsp[ci * 16 + 4 * u + 3]);
        put_unit(sP, r, (wbs + ci * 32) / 8 + u, d);
      }
    }
  }
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();

  if (tid == 0) {
    tc::fence_after_sync();
    const uint32_t adS = tc::smem_u32(sP);
    // dK = dS^T Q -> columns 64..
    constexpr uint32_t idMN = tc::idesc_bf16(128, DH, 1, 1);
#pragma unroll
    for (int kk = 0; kk < kTile / 16; ++kk)
      tc::mma_bf16(tmem + 64, tc::sdesc(adS + kk * 2048, 16384, 1024), G::mnmaj(sQ, 0, kk), idMN,
                   kk > 0 ? 1u : 0u);
    // dQ = dS K -> columns 128.. (A = dS K-major, B = K read MN-major)
    constexpr uint32_t idKM = tc::idesc_bf16(128, DH, 0, 1);
#pragma unroll
    for (int kk = 0; kk < kTile / 16; ++kk)
      tc::mma_bf16(tmem + 128, p_kmaj(sP, 0, kk), G::mnmaj(sK, 0, kk), idKM, kk > 0 ? 1u : 0u);
    tc::mma_commit(&bar[3]);
  }
  __syncwarp();
  ok = tc::mbar_wait(&bar[3], 0, status) && ok;
  tc::fence_after_sync();

  // ---- epilogue: rows of dV, dK (key r) and dQ (query r) through staging tiles
  {
    uint8_t* const dst[3] = {sdO, sK, sQ};  // dV, dK, dQ staging tiles
#pragma unroll
    for (int q = 0; q < 3; ++q) {
      float v[DH];
      tmem_row<DH>(trow + (uint32_t)(64 * q), v);
      stage_row<DH>(dst[q], r, v);
    }
  }
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  if (tid == 0 && ok) {
    tc::tma_store_3d(&mdQ, sQ, h * DH, t0, b);
    tc::tma_store_3d(&mdK, sK, h * DH, t0, b);
    tc::tma_store_3d(&mdV, sdO, h * DH, t0, b);
    tc::tma_store_commit();
    tc::tma_store_wait_read<0>();  // the staging is read; the writes finish with the grid
  }
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 256);
}

// ========================================================================= host
bool attn_tc_supported(int dtype, int dh, int L) {
  return dtype == 1 && (dh == 16 || dh == 32 || dh == 64) &&
         (L == 16 || L == 32 || L == 64 || L == 128) && tmap_encoder() != nullptr;
}

// 128-token x DH boxes of one head, with the swizzle whose span is one row
static bool head_map(CUtensorMap* m, const void* base, long ld, int D, int T, int B, int dh) {
  const uint64_t dims[3] = {(uint64_t)D, (uint64_t)T, (uint64_t)B};
  const uint64_t st[2] = {(uint64_t)ld * 2, (uint64_t)ld * 2 * (uint64_t)T};
  const uint32_t box[3] = {(uint32_t)dh, kTile, 1};
  const CUtensorMapSwizzle sw = dh == 64   ? CU_TENSOR_MAP_SWIZZLE_128B
                                : dh == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                           : CU_TENSOR_MAP_SWIZZLE_32B;
  return make_tmap_bf16(m, base, 3, dims, st, box, sw);
}


static int chunks_for(int L) { return L <= 32 ? 1 : L / 32; }

template <int NCH, int DH>
static cudaError_t fwd_launch(const Launch& lc, const AttnArgs& a, const CUtensorMap* m) {
  static std::atomic<unsigned long long> opted{0};
  auto kern = attn_fwd_tc_kernel<NCH, DH>;
  constexpr int smem = fwd_smem_bytes<DH>();
  if (cudaError_t e = smem_opt_in(kern, smem, &opted); e != cudaSuccess) return e;
  dim3 grid((a.T + kTile - 1) / kTile, a.H, a.B);
  cudaError_t e = launch_k(kern, grid, dim3(128), smem, lc.stream, m[0], m[1], m[2], m[3], a.lse,
                           a.T, a.H, a.L, 1.0f / sqrtf((float)a.dh), lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int DH>
static cudaError_t fwd_dh(const Launch& lc, const AttnArgs& a) {
  const int D = a.H * DH;
  CUtensorMap m[4];
  if (!head_map(&m[0], a.Q, a.ld_qkv, D, a.T, a.B, DH) ||
      !head_map(&m[1], a.K, a.ld_qkv, D, a.T, a.B, DH) ||
      !head_map(&m[2], a.V, a.ld_qkv, D, a.T, a.B, DH) ||
      !head_map(&m[3], a.O, a.ld_o, D, a.T, a.B, DH))
    return cudaErrorInvalidValue;
  switch (chunks_for(a.L)) {
    case 1: return fwd_launch<1, DH>(lc, a, m);
    case 2: return fwd_launch<2, DH>(lc, a, m);
    default: return fwd_launch<4, DH>(lc, a, m);
  }
}

cudaError_t attn_fwd_tc(const Launch& lc, const AttnArgs& a) {
  if (!attn_tc_supported(1, a.dh, a.L)) return cudaErrorNotSupported;
  switch (a.dh) {
    case 16: return fwd_dh<16>(lc, a);
    case 32: return fwd_dh<32>(lc, a);
    default: return fwd_dh<64>(lc, a);
  }
}

template <int NCH, int DH>
static cudaError_t bwd_launch(const Launch& lc, const AttnBwdArgs& a, const CUtensorMap* m) {
  const AttnArgs& f = a.f;
  static std::atomic<unsigned long long> opted{0};
  auto kern = attn_bwd_tc_kernel<NCH, DH>;
  constexpr int smem = bwd_smem_bytes<DH>();
  if (cudaError_t e = smem_opt_in(kern, smem, &opted); e != cudaSuccess) return e;
  dim3 grid((f.T + kTile - 1) / kTile, f.H, f.B);
  cudaError_t e = launch_k(kern, grid, dim3(128), smem, lc.stream, m[0], m[1], m[2], m[3], m[4],
                           m[5], m[6], m[7], f.lse, f.T, f.H, f.L, 1.0f / sqrtf((float)f.dh),
                           lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int DH>
static cudaError_t bwd_dh(const Launch& lc, const AttnBwdArgs& a) {
  const AttnArgs& f = a.f;
  const int D = f.H * DH;
  CUtensorMap m[8];
  if (!head_map(&m[0], f.Q, f.ld_qkv, D, f.T, f.B, DH) ||
      !head_map(&m[1], f.K, f.ld_qkv, D, f.T, f.B, DH) ||
      !head_map(&m[2], f.V, f.ld_qkv, D, f.T, f.B, DH) ||
      !head_map(&m[3], a.dO, f.ld_o, D, f.T, f.B, DH) ||
      !head_map(&m[4], a.dQ, a.ld_dqkv, D, f.T, f.B, DH) ||
      !head_map(&m[5], a.dK, a.ld_dqkv, D, f.T, f.B, DH) ||
      !head_map(&m[6], a.dV, a.ld_dqkv, D, f.T, f.B, DH) ||
      !head_map(&m[7], f.O, f.ld_o, D, f.T, f.B, DH))
    return cudaErrorInvalidValue;
  switch (chunks_for(f.L)) {
    case 1: return bwd_launch<1, DH>(lc, a, m);
    case 2: return bwd_launch<2, DH>(lc, a, m);
    default: return bwd_launch<4, DH>(lc, a, m);
  }
}

cudaError_t attn_bwd_tc(const Launch& lc, const AttnBwdArgs& a) {
  const AttnArgs& f = a.f;
  if (!attn_tc_supported(1, f.dh, f.L)) return cudaErrorNotSupported;
  switch (f.dh) {
    case 16: return bwd_dh<16>(lc, a);
    case 32: return bwd_dh<32>(lc, a);
    default: return bwd_dh<64>(lc, a);
  }
}

}  // namespace bcmt
