// Intra-block causal attention on the tcgen05 tensor cores (Sec. 3.3) that
// walks key tiles: head widths DH in {16, 32, 64} and block sizes L that
// divide 128 or are multiples of 128 (up to 1024), bf16 operands.  The layer
// uses it for blocks longer than one 128-token tile (L >= 256); for L <= 128
// it takes the single-tile kernels of attn_tc.cu.
//
// A CTA owns a 128-token tile of one head and walks the key tiles its rows
// can see: for L >= 128 the tiles of its block from the block start up to the
// diagonal tile, for L < 128 the diagonal tile alone (whose mask is then
// block-diagonal).  Q/K/V/dO tiles are [128 tokens x DH] slices brought in by
// TMA with the swizzle whose span is one row (DH * 2 bytes: 32, 64 or 128),
// so every operand is a canonical swizzled layout the MMA reads K-major or
// MN-major.  Scores and products accumulate in TMEM.
//
//  * forward: per key tile S = Q K^T (N = 128), online softmax with the
//    thread owning one query row (running max and sum in registers), P in
//    bf16 to shared memory, P V into TMEM, O rescaled and accumulated in
//    registers; O and the log-sum-exp are stored at the end.  At L > 128
//    the layer runs the half-tile form (64-key halves, 128 TMEM columns per
//    CTA, more CTAs per SM).
//  * backward, two kernels (no atomics, fixed summation order):
//      dQ:  per query tile, Drow = dO . O, then per key tile and 64-key half
//           S, dP (N = 64), dS = P (dP - Drow) scale, dQ += dS K (TMEM);
//      dKV: per key tile, per query tile and 64-query half S^T = K Q^T,
//           dP^T = V dO^T, dV += P^T dO, dK += dS^T Q (TMEM), with the query
//           tile's log-sum-exp and Drow staged in shared memory; the second
//           half's S^T and dP^T are issued ahead of the first half's dV/dK.
//    For head widths up to 32 both walk 32-key / 32-query quarters instead
//    (128 TMEM columns per CTA: three or four CTAs per SM).
#include "attn_common.cuh"
#include "common.cuh"
#include "internal.h"
#include "tc.cuh"
#include "tmap.h"

namespace bcmt {
using namespace attn;

namespace {
constexpr int kTile = 128;

// max(a, b, c) in one instruction (three-input max.f32, sm_100 and later)
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// First key of the key-tile walk of the query tile at t0, and the tile count.
__device__ __forceinline__ void key_walk(int t0, int L, int& kstart, int& nkt) {
  kstart = L >= kTile ? (t0 / L) * L : t0;
  nkt = (t0 - kstart) / kTile + 1;
}
}  // namespace

// ====================================================================== forward
// Pipelined over the key tiles: K is double-buffered, so the score product of
// tile kt+1 is issued as soon as every thread has read tile kt's scores out of
// TMEM and runs under tile kt's softmax; K of tile kt+2 streams in meanwhile.
// V (single buffer) is reloaded once tile kt's P V product has completed.
// NCH = the 32-key chunks a warp's rows can reach (1 or 2 for L < 128, else
// 4); ONE: every query tile sees one key tile (L <= 128), so O can take the
// columns of the consumed scores and the CTA needs 128 TMEM columns, not 256
// (with fewer registers for NCH <= 2, three to four CTAs share an SM).
template <int DH, int NCH, bool ONE>
__global__ void __launch_bounds__(128, NCH <= 2 ? 3 : 2)
    attn_fwd_fl_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mK,
                       const __grid_constant__ CUtensorMap mV, bf16* __restrict__ O, long ld_o,
                       float* __restrict__ lse, int Tlen, int H, int L, float scale,
                       unsigned* status) {
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sP = smem;                       // 32 KB: P [128 queries x 128 keys]
  uint8_t* sQ = smem + 32768;
  uint8_t* sK0 = sQ + G::tile;              // K, two buffers
  uint8_t* sV = sK0 + 2 * G::tile;
  // barriers: K buffer 0/1 loaded (buffer 0 also counts Q), V loaded, S ready, P V done
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + G::tile);
  uint64_t* bar_k = bar;
  uint64_t* bar_v = bar + 2;
  uint64_t* bar_s = bar + 3;
  uint64_t* bar_o = bar + 4;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 5);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;
  int kstart, nkt;
  key_walk(t0, L, kstart, nkt);

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar_k[0], 2 * G::tile);
    tc::tma_load_3d(sQ, &mQ, &bar_k[0], h * DH, t0, b);
    tc::tma_load_3d(sK0, &mK, &bar_k[0], h * DH, kstart, b);
    tc::mbar_arrive_expect_tx(bar_v, G::tile);
    tc::tma_load_3d(sV, &mV, bar_v, h * DH, kstart, b);
    if (nkt > 1) {
      tc::mbar_arrive_expect_tx(&bar_k[1], G::tile);
      tc::tma_load_3d(sK0 + G::tile, &mK, &bar_k[1], h * DH, kstart + kTile, b);
    }
  }
  __syncwarp();
  constexpr uint32_t kCols = ONE ? 128 : 256;  // S; O at kOcol
  constexpr uint32_t kOcol = ONE ? 0 : 128;
  if (warp == 0) {
    tc::tmem_alloc(tslot, kCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  constexpr uint32_t idS = tc::idesc_bf16(128, 128, 0, 0);
  constexpr uint32_t idO = tc::idesc_bf16(128, DH, 0, 1);

  if (tid == 0) {  // S of the first key tile
    const bool okk = tc::mbar_wait(&bar_k[0], 0, status);
    tc::fence_after_sync();
    if (okk) {
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)
        tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK0, 0, kk), idS, kk > 0 ? 1u : 0u);
    }
    tc::mma_commit(bar_s);
  }
  __syncwarp();

  const int r = warp * 32 + lane;
  const float sl2 = scale * kLog2e;
  float m = -INFINITY, l = 0.f;
  float oacc[DH];
#pragma unroll
  for (int c = 0; c < DH; ++c) oacc[c] = 0.f;
  bool ok = true;

  for (int kt = 0; kt < nkt; ++kt) {
    const bool diag = kt == nkt - 1;
    ok = tc::mbar_wait(bar_s, kt & 1, status) && ok;
    tc::fence_after_sync();

    // ---- this tile's scores out of TMEM (thread = query row r)
    int wbs = 0, nld = 4, rbs = 0;
    if (diag) {
      if (L < kTile) {
        wbs = L < 32 ? warp * 32 : ((warp * 32) / L) * L;
        rbs = (r / L) * L;
      }
      nld = chunks_needed(warp, wbs);
    }
    uint32_t sr[NCH][32];
#pragma unroll
    for (int ci = 0; ci < NCH; ++ci)
      if (ci < nld) tc::tmem_ld32_issue(trow + (uint32_t)(wbs + ci * 32), sr[ci]);
    tc::tmem_wait();
    tc::fence_before_sync();
    __syncthreads();  // every thread has its scores: the S columns are free
    if (tid == 0) {
      tc::fence_after_sync();
      if (kt + 1 < nkt) {  // next tile's scores, under this tile's softmax
        const int nb = (kt + 1) & 1;
        const bool okk = tc::mbar_wait(&bar_k[nb], ((kt + 1) >> 1) & 1, status);
        tc::fence_after_sync();
        if (okk) {
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk)
            tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK0 + nb * G::tile, 0, kk), idS,
                         kk > 0 ? 1u : 0u);
        }
        tc::mma_commit(bar_s);
      }
      if (kt + 2 < nkt) {  // K buffer kt & 1 was read by tile kt's (completed) product
        const int cb = kt & 1;
        tc::mbar_arrive_expect_tx(&bar_k[cb], G::tile);
        tc::tma_load_3d(sK0 + cb * G::tile, &mK, &bar_k[cb], h * DH, kstart + (kt + 2) * kTile, b);
      }
    }

    // ---- online softmax (P to shared memory; the previous P V has completed).
    // Tiles left of the diagonal need no mask: their max, exponentials and
    // sum run with independent partial accumulators.  For L <= 128 (one
    // tile) the masked branch below serves.
    float m_new, psum;
    if (!ONE && diag) {
      // the diagonal tile of a walk (L > 128: no block offset, wbs = rbs = 0)
      // goes through the unmasked code below with its hidden scores set to
      // -inf (exp2 gives 0): one softmax body keeps the kernel's code small
      // (with a masked copy of it, instruction fetch was the top stall)
#pragma unroll
      for (int ci = 0; ci < NCH; ++ci)
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (ci >= nld || ci * 32 + j > r) sr[ci][j] = __float_as_uint(-INFINITY);
    }
    if (!ONE) {
      // three-input max, and the exponent arguments and the partial sums as
      // packed fp32 pairs: about a third fewer instructions per score
      float mx[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = -INFINITY;
#pragma unroll
      for (int ci = 0; ci < NCH; ++ci)
#pragma unroll
        for (int j = 0; j < 32; j += 2)
          mx[(j >> 1) & 7] = max3f(mx[(j >> 1) & 7], __uint_as_float(sr[ci][j]),
                                   __uint_as_float(sr[ci][j + 1]));
      const float mt = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[5]),
                             fmaxf(mx[6], mx[7]));
      m_new = fmaxf(m, mt * sl2);
      const float2 sl2x2 = make_float2(sl2, sl2), nm2 = make_float2(-m_new, -m_new);
      float2 ps[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
      for (int u = 0; u < 4 * NCH; ++u) {
        float v[8];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          const float2 a = __ffma2_rn(
              make_float2(__uint_as_float(sr[u >> 2][(u & 3) * 8 + e]),
                          __uint_as_float(sr[u >> 2][(u & 3) * 8 + e + 1])),
              sl2x2, nm2);
          v[e] = ex2(a.x);
          v[e + 1] = ex2(a.y);
          ps[(e >> 1) & 1] = __fadd2_rn(ps[(e >> 1) & 1], make_float2(v[e], v[e + 1]));
        }
        put_unit(sP, r, u, pack8(v));
      }
      psum = (ps[0].x + ps[0].y) + (ps[1].x + ps[1].y);
    } else {
      float mt = -INFINITY;
#pragma unroll
      for (int ci = 0; ci < NCH; ++ci)
        if (ci < nld) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int kk = wbs + ci * 32 + j;
            if (kk >= rbs && kk <= r) mt = fmaxf(mt, __uint_as_float(sr[ci][j]));
          }
        }
      m_new = fmaxf(m, mt * sl2);
      const float nm = -m_new;
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
              v[e] = (kk >= rbs && kk <= r)
                         ? ex2(fmaf(__uint_as_float(sr[ci][u * 8 + e]), sl2, nm))
                         : 0.f;
              ps[e & 3] += v[e];
            }
            put_unit(sP, r, (wbs + ci * 32) / 8 + u, pack8(v));
          }
        }
      psum = (ps[0] + ps[1]) + (ps[2] + ps[3]);
      const uint4 zero = make_uint4(0, 0, 0, 0);
      for (int u = 0; u < 16; ++u)
        if (u * 8 < wbs || u * 8 >= wbs + nld * 32) put_unit(sP, r, u, zero);
    }
    const float alpha = ex2(m - m_new);  // 0 on the first tile (m = -inf)
    l = l * alpha + psum;
    m = m_new;
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    __syncthreads();

    if (tid == 0) {
      tc::fence_after_sync();
      const bool okv = tc::mbar_wait(bar_v, kt & 1, status);
      tc::fence_after_sync();
      if (okv) {
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk)
          tc::mma_bf16(tmem + kOcol, p_kmaj(sP, 0, kk), G::mnmaj(sV, 0, kk), idO, kk > 0 ? 1u : 0u);
      }
      tc::mma_commit(bar_o);
    }
    __syncwarp();
    ok = tc::mbar_wait(bar_o, kt & 1, status) && ok;
    tc::fence_after_sync();
    // V and P are free: fetch the next tile's V while this P V is folded in
    if (tid == 0 && kt + 1 < nkt) {
      tc::mbar_arrive_expect_tx(bar_v, G::tile);
      tc::tma_load_3d(sV, &mV, bar_v, h * DH, kstart + (kt + 1) * kTile, b);
    }
    float o[DH];
    tmem_row<DH>(trow + kOcol, o);
#pragma unroll
    for (int c = 0; c < DH; ++c) oacc[c] = fmaf(oacc[c], alpha, o[c]);
  }

  const int t = t0 + r;
  if (ok && t < Tlen) {
    store_row<DH>(O + ((long)b * Tlen + t) * ld_o + h * DH, oacc, 1.0f / l);
    lse[((long)b * H + h) * Tlen + t] = m * kLn2 + logf(l);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, kCols);
}

// The forward at L > 128, with each 128-key tile taken as two 64-key halves
// in turn: S of a half (N = 64) and O need at most 128 TMEM columns and P one
// 16 KB half, so a CTA allocates 128 columns and three or four CTAs share an
// SM (more warps than the kernel above, whose per-score chains are
// latency-bound).  Per half: S = Q K_h^T, online softmax of its 64 scores (the
// diagonal tile's hidden keys set to -inf first), P_h in bf16 to shared
// memory, P_h V_h into TMEM, folded into O in registers.  The next half's S is
// issued as soon as every thread has read this half's scores and runs under
// its softmax.  Up to width 32, K is double-buffered across tiles (K of tile
// kt+2 streams in once tile kt's second half has its scores); at width 64 one
// K buffer (66 KB per CTA: three per SM) takes tile kt+1's K at that point
// and its first S waits for it.  V is reloaded once tile kt's second P V has
// completed.
template <int DH>
__global__ void __launch_bounds__(128, DH <= 16 ? 4 : 3)
    attn_fwd_fl_half_kernel(const __grid_constant__ CUtensorMap mQ,
                            const __grid_constant__ CUtensorMap mK,
                            const __grid_constant__ CUtensorMap mV, bf16* __restrict__ O,
                            long ld_o, float* __restrict__ lse, int Tlen, int H, int L,
                            float scale, unsigned* status) {
  static_assert(DH <= 64, "a 64-key S half and O fit 128 TMEM columns for DH <= 64");
  constexpr int NKB = DH <= 32 ? 2 : 1;  // K buffers
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sP = smem;                       // 16 KB: P of one half [128 queries x 64 keys]
  uint8_t* sQ = smem + 16384;
  uint8_t* sK0 = sQ + G::tile;              // K, NKB buffers
  uint8_t* sV = sK0 + NKB * G::tile;
  // barriers: K buffer 0/1 loaded (buffer 0 also counts Q), V loaded, S ready, P V done
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + G::tile);
  uint64_t* bar_k = bar;
  uint64_t* bar_v = bar + 2;
  uint64_t* bar_s = bar + 3;
  uint64_t* bar_o = bar + 4;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 5);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;
  int kstart, nkt;
  key_walk(t0, L, kstart, nkt);

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar_k[0], 2 * G::tile);
    tc::tma_load_3d(sQ, &mQ, &bar_k[0], h * DH, t0, b);
    tc::tma_load_3d(sK0, &mK, &bar_k[0], h * DH, kstart, b);
    tc::mbar_arrive_expect_tx(bar_v, G::tile);
    tc::tma_load_3d(sV, &mV, bar_v, h * DH, kstart, b);
    if (NKB == 2 && nkt > 1) {
      tc::mbar_arrive_expect_tx(&bar_k[NKB - 1], G::tile);
      tc::tma_load_3d(sK0 + (NKB - 1) * G::tile, &mK, &bar_k[NKB - 1], h * DH, kstart + kTile, b);
    }
  }
  __syncwarp();
  constexpr uint32_t kCols = 128, kOcol = 64;  // S half at 0..63, O at 64..
  if (warp == 0) {
    tc::tmem_alloc(tslot, kCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  constexpr uint32_t idS = tc::idesc_bf16(128, 64, 0, 0);
  constexpr uint32_t idO = tc::idesc_bf16(128, DH, 0, 1);
  // S of half hh of the key tile in K buffer kb
  auto issue_s = [&](int kb, int hh) {
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk)
      tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK0 + kb * G::tile, 64 * hh, kk), idS,
                   kk > 0 ? 1u : 0u);
    tc::mma_commit(bar_s);
  };

  if (tid == 0) {
    const bool okk = tc::mbar_wait(&bar_k[0], 0, status);
    tc::fence_after_sync();
    if (okk) issue_s(0, 0);
    else tc::mma_commit(bar_s);
  }
  __syncwarp();

  const int r = warp * 32 + lane;
  const float sl2 = scale * kLog2e;
  float m = -INFINITY, l = 0.f;
  float oacc[DH];
#pragma unroll
  for (int c = 0; c < DH; ++c) oacc[c] = 0.f;
  bool ok = true;
  int ns = 0, no = 0;  // S and P V commits consumed

  for (int kt = 0; kt < nkt; ++kt) {
    const bool diag = kt == nkt - 1;
    const int kb = NKB == 2 ? (kt & 1) : 0;
    if constexpr (NKB == 1) {
      if (kt > 0 && tid == 0) {  // this tile's K (loaded during the last tile)
        const bool okk = tc::mbar_wait(&bar_k[0], kt & 1, status);
        tc::fence_after_sync();
        if (okk && ok) issue_s(0, 0);
        else tc::mma_commit(bar_s);
      }
      __syncwarp();
    }
    for (int hh = 0; hh < 2; ++hh) {
      ok = tc::mbar_wait(bar_s, ns & 1, status) && ok;
      ++ns;
      tc::fence_after_sync();
      uint32_t sr[2][32];
      tc::tmem_ld32_issue(trow, sr[0]);
      tc::tmem_ld32_issue(trow + 32u, sr[1]);
      tc::tmem_wait();
      tc::fence_before_sync();
      __syncthreads();  // every thread has this half's scores: the S columns are free
      if (tid == 0) {
        tc::fence_after_sync();
        if (hh == 0) {  // the tile's second half
          if (ok) issue_s(kb, 1);
          else tc::mma_commit(bar_s);
        } else if (NKB == 2 && kt + 1 < nkt) {  // the next tile's first half (K prefetched)
          const int nb = (kt + 1) & 1;
          const bool okk = tc::mbar_wait(&bar_k[nb], ((kt + 1) >> 1) & 1, status);
          tc::fence_after_sync();
          if (okk && ok) issue_s(nb, 0);
          else tc::mma_commit(bar_s);
        }
        // K buffer kb: both halves' scores are read (tile kt done with it)
        if (hh == 1 && kt + NKB < nkt) {
          tc::mbar_arrive_expect_tx(&bar_k[kb], G::tile);
          tc::tma_load_3d(sK0 + kb * G::tile, &mK, &bar_k[kb], h * DH,
                          kstart + (kt + NKB) * kTile, b);
        }
      }
      if (diag) {  // keys past the query row (L > 128: no block offset in the tile)
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (64 * hh + 32 * c + j > r) sr[c][j] = __float_as_uint(-INFINITY);
      }
      // online softmax of the half's 64 scores (P to shared memory; the
      // previous P V has completed)
      float mx[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = -INFINITY;
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int j = 0; j < 32; j += 2)
          mx[(j >> 1) & 7] = max3f(mx[(j >> 1) & 7], __uint_as_float(sr[c][j]),
                                   __uint_as_float(sr[c][j + 1]));
      const float mt = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[5]),
                             fmaxf(mx[6], mx[7]));
      const float m_new = fmaxf(m, mt * sl2);
      const float2 sl2x2 = make_float2(sl2, sl2), nm2 = make_float2(-m_new, -m_new);
      float2 ps[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        float v[8];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          const float2 a = __ffma2_rn(make_float2(__uint_as_float(sr[u >> 2][(u & 3) * 8 + e]),
                                                  __uint_as_float(sr[u >> 2][(u & 3) * 8 + e + 1])),
                                      sl2x2, nm2);
          v[e] = ex2(a.x);
          v[e + 1] = ex2(a.y);
          ps[(e >> 1) & 1] = __fadd2_rn(ps[(e >> 1) & 1], make_float2(v[e], v[e + 1]));
        }
        put_unit(sP, r, u, pack8(v));
      }
      const float psum = (ps[0].x + ps[0].y) + (ps[1].x + ps[1].y);
      const float alpha = ex2(m - m_new);  // 0 on the first half (m = -inf)
      l = l * alpha + psum;
      m = m_new;
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncthreads();

      if (tid == 0) {
        tc::fence_after_sync();
        const bool okv = tc::mbar_wait(bar_v, kt & 1, status);
        tc::fence_after_sync();
        if (okv && ok) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // O_h = P_h V[64 hh .., :]
            tc::mma_bf16(tmem + kOcol, p_kmaj(sP, 0, kk), G::mnmaj(sV, 64 * hh, kk), idO,
                         kk > 0 ? 1u : 0u);
        }
        tc::mma_commit(bar_o);
      }
      __syncwarp();
      ok = tc::mbar_wait(bar_o, no & 1, status) && ok;
      ++no;
      tc::fence_after_sync();
      // V is free after the tile's second P V: fetch the next tile's V while
      // this product is folded in
      if (tid == 0 && hh == 1 && kt + 1 < nkt) {
        tc::mbar_arrive_expect_tx(bar_v, G::tile);
        tc::tma_load_3d(sV, &mV, bar_v, h * DH, kstart + (kt + 1) * kTile, b);
      }
      float o[DH];
      tmem_row<DH>(trow + kOcol, o);
#pragma unroll
      for (int c = 0; c < DH; ++c) oacc[c] = fmaf(oacc[c], alpha, o[c]);
    }
  }

  const int t = t0 + r;
  if (ok && t < Tlen) {
    store_row<DH>(O + ((long)b * Tlen + t) * ld_o + h * DH, oacc, 1.0f / l);
    lse[((long)b * H + h) * Tlen + t] = m * kLn2 + logf(l);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, kCols);
}

// ================================================================ backward: dQ
template <int DH>
__global__ void __launch_bounds__(128)
    attn_bwd_dq_fl_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mK,
                          const __grid_constant__ CUtensorMap mV, const __grid_constant__ CUtensorMap mdO,
                          const bf16* __restrict__ O, const bf16* __restrict__ dO, long ld_o,
                          const float* __restrict__ lse, float* __restrict__ Drow,
                          bf16* __restrict__ dQ, long ld_d, int Tlen, int H, int L, float scale,
                          unsigned* status) {
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sdS = smem;                      // 2 x 16 KB: scale * dS of the two 64-key halves
  uint8_t* sQ = smem + 32768;
  uint8_t* sdO = sQ + G::tile;
  uint8_t* sK = sdO + G::tile;
  uint8_t* sV = sK + G::tile;
  // K/V loaded; S/dP done; dQ product of half 0 / half 1 done
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + G::tile);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;
  int kstart, nkt;
  key_walk(t0, L, kstart, nkt);

  if (tid == 0) {
    for (int i = 0; i < 4; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
    tc::prefetch_tmap(&mdO);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar[0], 4 * G::tile);
    tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sK, &mK, &bar[0], h * DH, kstart, b);
    tc::tma_load_3d(sV, &mV, &bar[0], h * DH, kstart, b);
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

  // Drow_t = dO_t . O_t and the row's log-sum-exp (global rows)
  const int r = warp * 32 + lane;
  const int t = t0 + r;
  const bool row_ok = t < Tlen;
  float drow = 0.f, lse2 = 0.f;
  if (row_ok) {
    const bf16* orow = O + ((long)b * Tlen + t) * ld_o + h * DH;
    const bf16* grow = dO + ((long)b * Tlen + t) * ld_o + h * DH;
#pragma unroll
    for (int u = 0; u < DH / 8; ++u) {
      float ov[8], gv[8];
      load8(orow + 8 * u, ov);
      load8(grow + 8 * u, gv);
#pragma unroll
      for (int e = 0; e < 8; ++e) drow = fmaf(ov[e], gv[e], drow);
    }
    const long li = ((long)b * H + h) * Tlen + t;
    Drow[li] = drow;
    lse2 = lse[li] * kLog2e;
  }
  const float sl2 = scale * kLog2e;
  const float nl2 = -lse2, ndr = -drow * scale;
  const int rbs = L < kTile ? (r / L) * L : 0;
  bool ok = true;
  // S and dP of half hh of the loaded key tile into TMEM columns 0..127
  auto issue_sdp = [&](int hh) {
    if (ok) {
      constexpr uint32_t id64 = tc::idesc_bf16(128, 64, 0, 0);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // S half -> columns 0..63
        tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK, 64 * hh, kk), id64, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // dP half -> columns 64..127
        tc::mma_bf16(tmem + 64, G::kmaj(sdO, 0, kk), G::kmaj(sV, 64 * hh, kk), id64,
                     kk > 0 ? 1u : 0u);
    }
    tc::mma_commit(&bar[1]);
  };
  if (tid == 0) {
    ok = tc::mbar_wait(&bar[0], 0, status) && ok;
    tc::fence_after_sync();
    issue_sdp(0);
  }
  __syncwarp();
  int ns = 0;  // S/dP commits consumed so far

  // Per key tile, the two 64-key halves overlap: S and dP of half 1 run under
  // half 0's dS, and each half writes its own dS buffer (the one the dQ product
  // of the same half of the previous tile read).
  for (int kt = 0; kt < nkt; ++kt) {
    const bool diag = kt == nkt - 1;
    for (int hh = 0; hh < 2; ++hh) {
      ok = tc::mbar_wait(&bar[1], ns & 1, status) && ok;
      ++ns;
      tc::fence_after_sync();
      uint32_t rs[2][32], rd[2][32];
      tc::tmem_ld32_issue(trow, rs[0]);
      tc::tmem_ld32_issue(trow + 32u, rs[1]);
      tc::tmem_ld32_issue(trow + 64u, rd[0]);
      tc::tmem_ld32_issue(trow + 96u, rd[1]);
      tc::tmem_wait();
      tc::fence_before_sync();
      __syncthreads();  // every thread has this half's S and dP: the columns are free
      if (tid == 0 && hh == 0) {
        tc::fence_after_sync();
        issue_sdp(1);
      }
      uint8_t* sdSh = sdS + hh * 16384;
      if (kt > 0) {  // the previous tile's dQ product of this half read sdSh
        ok = tc::mbar_wait(&bar[2 + hh], (kt - 1) & 1, status) && ok;
        tc::fence_after_sync();
      }
      // dS = P (dP - Drow) scale; rows past the end see zero-filled Q and dO
      // (P finite, dP = Drow = 0), so only the diagonal tile needs a mask
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        float v[32];
        if (!diag) {
#pragma unroll
          for (int j = 0; j < 32; ++j)
            v[j] = ex2(fmaf(__uint_as_float(rs[c][j]), sl2, nl2)) *
                   fmaf(__uint_as_float(rd[c][j]), scale, ndr);
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int kk = 64 * hh + 32 * c + j;  // key column within the tile
            const bool valid = row_ok && kk >= rbs && kk <= r;
            v[j] = valid ? ex2(fmaf(__uint_as_float(rs[c][j]), sl2, nl2)) *
                               fmaf(__uint_as_float(rd[c][j]), scale, ndr)
                         : 0.f;
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) put_unit(sdSh, r, 4 * c + u, pack8(v + 8 * u));
      }
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncthreads();
      if (tid == 0) {
        tc::fence_after_sync();
        if (ok) {
          constexpr uint32_t idQ = tc::idesc_bf16(128, DH, 0, 1);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // dQ += dS[:, 64hh..] K[64hh.., :]
            tc::mma_bf16(tmem + 128, p_kmaj(sdSh, 0, kk), G::mnmaj(sK, 64 * hh, kk), idQ,
                         (kt > 0 || hh > 0 || kk > 0) ? 1u : 0u);
        }
        tc::mma_commit(&bar[2 + hh]);
      }
    }
    // the next key tile may overwrite K and V once this tile's products are
    // done (the half-1 commit covers every earlier product); then its half 0
    if (tid == 0 && kt + 1 < nkt) {
      ok = tc::mbar_wait(&bar[3], kt & 1, status) && ok;
      tc::mbar_arrive_expect_tx(&bar[0], 2 * G::tile);
      tc::tma_load_3d(sK, &mK, &bar[0], h * DH, kstart + (kt + 1) * kTile, b);
      tc::tma_load_3d(sV, &mV, &bar[0], h * DH, kstart + (kt + 1) * kTile, b);
      ok = tc::mbar_wait(&bar[0], (kt + 1) & 1, status) && ok;
      tc::fence_after_sync();
      issue_sdp(0);
    }
    __syncwarp();
  }
  ok = tc::mbar_wait(&bar[3], (nkt - 1) & 1, status) && ok;
  tc::fence_after_sync();
  float q[DH];
  tmem_row<DH>(trow + 128u, q);
  if (ok && row_ok) store_row<DH>(dQ + ((long)b * Tlen + t) * ld_d + h * DH, q, 1.0f);
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 256);
}

// The dQ kernel for head widths up to 32 with each key tile taken as four
// 32-key quarters in turn: S and dP of a quarter (N = 32 each) and the dQ
// accumulator need at most 96 TMEM columns, so a CTA allocates 128 and three
// or four CTAs share an SM (the kernel above, at 256 columns, runs two, and
// its per-half chains wait on barriers and TMEM).  Quarter q's scale * dS goes
// to columns 32 (q % 2) .. of the 64-key half buffer q / 2, which the dQ
// product of the same quarter of the previous tile read (bar[2 + q] tracks
// it); S and dP of the next quarter are issued as soon as every thread has
// read this quarter's and run under its elementwise pass.
template <int DH>
__global__ void __launch_bounds__(128, DH <= 16 ? 4 : 3)
    attn_bwd_dq_fl_q_kernel(const __grid_constant__ CUtensorMap mQ,
                            const __grid_constant__ CUtensorMap mK,
                            const __grid_constant__ CUtensorMap mV,
                            const __grid_constant__ CUtensorMap mdO, const bf16* __restrict__ O,
                            const bf16* __restrict__ dO, long ld_o, const float* __restrict__ lse,
                            float* __restrict__ Drow, bf16* __restrict__ dQ, long ld_d, int Tlen,
                            int H, int L, float scale, unsigned* status) {
  static_assert(DH <= 32, "S, dP quarters and dQ fit 128 TMEM columns for DH <= 64; smem for <= 32");
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sdS = smem;                      // 2 x 16 KB: scale * dS, quarters 0-1 / 2-3
  uint8_t* sQ = smem + 32768;
  uint8_t* sdO = sQ + G::tile;
  uint8_t* sK = sdO + G::tile;
  uint8_t* sV = sK + G::tile;
  // K/V loaded; S/dP of a quarter done; dQ product of quarter 0..3 done
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + G::tile);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 6);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;
  int kstart, nkt;
  key_walk(t0, L, kstart, nkt);

  if (tid == 0) {
    for (int i = 0; i < 6; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
    tc::prefetch_tmap(&mdO);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar[0], 4 * G::tile);
    tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, t0, b);
    tc::tma_load_3d(sK, &mK, &bar[0], h * DH, kstart, b);
    tc::tma_load_3d(sV, &mV, &bar[0], h * DH, kstart, b);
  }
  __syncwarp();
  constexpr uint32_t kCols = 128, kQcol = 64;  // S quarter 0..31, dP quarter 32..63, dQ 64..
  if (warp == 0) {
    tc::tmem_alloc(tslot, kCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);

  // Drow_t = dO_t . O_t and the row's log-sum-exp (global rows)
  const int r = warp * 32 + lane;
  const int t = t0 + r;
  const bool row_ok = t < Tlen;
  float drow = 0.f, lse2 = 0.f;
  if (row_ok) {
    const bf16* orow = O + ((long)b * Tlen + t) * ld_o + h * DH;
    const bf16* grow = dO + ((long)b * Tlen + t) * ld_o + h * DH;
#pragma unroll
    for (int u = 0; u < DH / 8; ++u) {
      float ov[8], gv[8];
      load8(orow + 8 * u, ov);
      load8(grow + 8 * u, gv);
#pragma unroll
      for (int e = 0; e < 8; ++e) drow = fmaf(ov[e], gv[e], drow);
    }
    const long li = ((long)b * H + h) * Tlen + t;
    Drow[li] = drow;
    lse2 = lse[li] * kLog2e;
  }
  const float sl2 = scale * kLog2e;
  const float nl2 = -lse2, ndr = -drow * scale;
  const int rbs = L < kTile ? (r / L) * L : 0;
  bool ok = true;
  // S and dP of quarter q of the loaded key tile into TMEM columns 0..63
  auto issue_sdp = [&](int q) {
    if (ok) {
      constexpr uint32_t id32 = tc::idesc_bf16(128, 32, 0, 0);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // S quarter -> columns 0..31
        tc::mma_bf16(tmem, G::kmaj(sQ, 0, kk), G::kmaj(sK, 32 * q, kk), id32, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // dP quarter -> columns 32..63
        tc::mma_bf16(tmem + 32, G::kmaj(sdO, 0, kk), G::kmaj(sV, 32 * q, kk), id32,
                     kk > 0 ? 1u : 0u);
    }
    tc::mma_commit(&bar[1]);
  };
  if (tid == 0) {
    ok = tc::mbar_wait(&bar[0], 0, status) && ok;
    tc::fence_after_sync();
    issue_sdp(0);
  }
  __syncwarp();
  int ns = 0;  // S/dP commits consumed so far

  for (int kt = 0; kt < nkt; ++kt) {
    const bool diag = kt == nkt - 1;
    for (int q = 0; q < 4; ++q) {
      ok = tc::mbar_wait(&bar[1], ns & 1, status) && ok;
      ++ns;
      tc::fence_after_sync();
      uint32_t rs[32], rd[32];
      tc::tmem_ld32_issue(trow, rs);
      tc::tmem_ld32_issue(trow + 32u, rd);
      tc::tmem_wait();
      tc::fence_before_sync();
      __syncthreads();  // every thread has this quarter's S and dP: the columns are free
      if (tid == 0 && q < 3) {
        tc::fence_after_sync();
        issue_sdp(q + 1);
      }
      uint8_t* sdSq = sdS + (q >> 1) * 16384;
      if (kt > 0) {  // the previous tile's dQ product of this quarter read its columns
        ok = tc::mbar_wait(&bar[2 + q], (kt - 1) & 1, status) && ok;
        tc::fence_after_sync();
      }
      // dS = P (dP - Drow) scale; rows past the end see zero-filled Q and dO
      // (P finite, dP = Drow = 0), so only the diagonal tile needs a mask
      float v[32];
      if (!diag) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          v[j] = ex2(fmaf(__uint_as_float(rs[j]), sl2, nl2)) *
                 fmaf(__uint_as_float(rd[j]), scale, ndr);
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int kk = 32 * q + j;  // key column within the tile
          const bool valid = row_ok && kk >= rbs && kk <= r;
          v[j] = valid ? ex2(fmaf(__uint_as_float(rs[j]), sl2, nl2)) *
                             fmaf(__uint_as_float(rd[j]), scale, ndr)
                       : 0.f;
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) put_unit(sdSq, r, 4 * (q & 1) + u, pack8(v + 8 * u));
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncthreads();
      if (tid == 0) {
        tc::fence_after_sync();
        if (ok) {
          constexpr uint32_t idQ = tc::idesc_bf16(128, DH, 0, 1);
#pragma unroll
          for (int kk = 0; kk < 2; ++kk)  // dQ += dS[:, 32q..] K[32q.., :]
            tc::mma_bf16(tmem + kQcol, p_kmaj(sdSq, 0, 2 * (q & 1) + kk),
                         G::mnmaj(sK, 32 * q, kk), idQ, (kt > 0 || q > 0 || kk > 0) ? 1u : 0u);
        }
        tc::mma_commit(&bar[2 + q]);
      }
    }
    // the next key tile may overwrite K and V once this tile's products are
    // done (the last quarter's commit covers every earlier product); then its
    // first quarter
    if (tid == 0 && kt + 1 < nkt) {
      ok = tc::mbar_wait(&bar[5], kt & 1, status) && ok;
      tc::mbar_arrive_expect_tx(&bar[0], 2 * G::tile);
      tc::tma_load_3d(sK, &mK, &bar[0], h * DH, kstart + (kt + 1) * kTile, b);
      tc::tma_load_3d(sV, &mV, &bar[0], h * DH, kstart + (kt + 1) * kTile, b);
      ok = tc::mbar_wait(&bar[0], (kt + 1) & 1, status) && ok;
      tc::fence_after_sync();
      issue_sdp(0);
    }
    __syncwarp();
  }
  ok = tc::mbar_wait(&bar[5], (nkt - 1) & 1, status) && ok;
  tc::fence_after_sync();
  float qv[DH];
  tmem_row<DH>(trow + kQcol, qv);
  if (ok && row_ok) store_row<DH>(dQ + ((long)b * Tlen + t) * ld_d + h * DH, qv, 1.0f);
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, kCols);
}

// =============================================================== backward: dKV
template <int DH>
__global__ void __launch_bounds__(128)
    attn_bwd_dkv_fl_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mK,
                           const __grid_constant__ CUtensorMap mV, const __grid_constant__ CUtensorMap mdO,
                           const float* __restrict__ lse, const float* __restrict__ Drow,
                           bf16* __restrict__ dK, bf16* __restrict__ dV, long ld_d, int Tlen, int H,
                           int L, float scale, unsigned* status) {
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sPt = smem;                      // 16 KB: P^T, one 64-query half
  uint8_t* sdSt = smem + 16384;             // 16 KB: scale * dS^T, the same half
  uint8_t* sK = smem + 32768;
  uint8_t* sV = sK + G::tile;
  uint8_t* sQ = sV + G::tile;
  uint8_t* sdO = sQ + G::tile;
  float* slse = reinterpret_cast<float*>(sdO + G::tile);  // [128] -lse * log2(e)
  float* sdr = slse + kTile;                               // [128] -Drow * scale
  uint64_t* bar = reinterpret_cast<uint64_t*>(sdr + kTile);  // kv, s, q
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 3);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int k0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;
  // queries that see this key tile: to the end of its block (L >= 128) or of
  // the tile itself (L < 128, block-diagonal mask)
  const int qend = min(L >= kTile ? (k0 / L + 1) * L : k0 + kTile, Tlen);
  const int nqt = (qend - k0 + kTile - 1) / kTile;

  if (tid == 0) {
    for (int i = 0; i < 3; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
    tc::prefetch_tmap(&mdO);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar[0], 4 * G::tile);
    tc::tma_load_3d(sK, &mK, &bar[0], h * DH, k0, b);
    tc::tma_load_3d(sV, &mV, &bar[0], h * DH, k0, b);
    tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, k0, b);
    tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, k0, b);
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

  const int r = warp * 32 + lane;  // key row
  const int key = k0 + r;
  const float sl2 = scale * kLog2e;
  // L < 128: key r's block ends at its block start + L (within the tile)
  const int kbe = L < kTile ? (r / L) * L + L : kTile;
  bool ok = true;
  int ns = 0, nq = 0;

  for (int qt = 0; qt < nqt; ++qt) {
    const int q0 = k0 + qt * kTile;
    const bool diag = qt == 0;
    {
      const int tq = q0 + tid;
      const long li = ((long)b * H + h) * Tlen + tq;
      slse[tid] = tq < Tlen ? -lse[li] * kLog2e : 0.f;
      sdr[tid] = tq < Tlen ? -Drow[li] * scale : 0.f;
    }
    if (tid == 0) {
      ok = tc::mbar_wait(&bar[0], qt & 1, status) && ok;
      tc::fence_after_sync();
    }
    __syncthreads();  // slse / sdr written
    // S^T and dP^T of query half hh -> TMEM columns 0..127 (tid 0)
    auto issue_scores = [&](int hh) {
      if (ok) {
        constexpr uint32_t id64 = tc::idesc_bf16(128, 64, 0, 0);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)  // S^T half -> columns 0..63
          tc::mma_bf16(tmem, G::kmaj(sK, 0, kk), G::kmaj(sQ, 64 * hh, kk), id64, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)  // dP^T half -> columns 64..127
          tc::mma_bf16(tmem + 64, G::kmaj(sV, 0, kk), G::kmaj(sdO, 64 * hh, kk), id64,
                       kk > 0 ? 1u : 0u);
      }
      tc::mma_commit(&bar[1]);
    };
    for (int hh = 0; hh < 2; ++hh) {
      // half 1's products were issued with half 0's dV/dK (below), ahead of them
      if (tid == 0 && hh == 0) issue_scores(0);
      __syncwarp();
      ok = tc::mbar_wait(&bar[1], ns & 1, status) && ok;
      ++ns;
      tc::fence_after_sync();
      uint32_t rs[2][32], rd[2][32];
      tc::tmem_ld32_issue(trow, rs[0]);
      tc::tmem_ld32_issue(trow + 32u, rs[1]);
      tc::tmem_ld32_issue(trow + 64u, rd[0]);
      tc::tmem_ld32_issue(trow + 96u, rd[1]);
      tc::tmem_wait();
      if (nq > 0) {  // the previous dV/dK products are done with P^T and dS^T
        ok = tc::mbar_wait(&bar[2], (nq - 1) & 1, status) && ok;
        tc::fence_after_sync();
      }
      // P^T and dS^T = P^T (dP^T - Drow) scale.  Query columns past the end
      // see zero-filled Q and dO (P finite, dO = dP = Drow = 0: no
      // contribution), so only the diagonal tile needs a mask.
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        float pv[32], dv[32];
        const float4* nl4 = reinterpret_cast<const float4*>(slse + 64 * hh + 32 * c);
        const float4* nd4 = reinterpret_cast<const float4*>(sdr + 64 * hh + 32 * c);
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {
          const float4 a = nl4[j4], d = nd4[j4];
          const float na[4] = {a.x, a.y, a.z, a.w}, nd[4] = {d.x, d.y, d.z, d.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int j = 4 * j4 + e;
            const int jq = 64 * hh + 32 * c + j;  // query column within the tile
            const bool valid = !diag || (q0 + jq < Tlen && jq >= r && jq < kbe);
            const float p = valid ? ex2(fmaf(__uint_as_float(rs[c][j]), sl2, na[e])) : 0.f;
            pv[j] = p;
            dv[j] = p * fmaf(__uint_as_float(rd[c][j]), scale, nd[e]);
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          put_unit(sPt, r, 4 * c + u, pack8(pv + 8 * u));
          put_unit(sdSt, r, 4 * c + u, pack8(dv + 8 * u));
        }
      }
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncthreads();
      if (tid == 0) {
        tc::fence_after_sync();
        // every thread has read this half's scores out of TMEM (the barrier
        // above): the next half's products go first, under this half's dV/dK
        // and the next elementwise pass
        if (hh == 0) issue_scores(1);
        if (ok) {
          constexpr uint32_t idKV = tc::idesc_bf16(128, DH, 0, 1);
          const uint32_t acc0 = (qt > 0 || hh > 0) ? 1u : 0u;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // dV += P^T[:, 64hh..] dO[64hh.., :]
            tc::mma_bf16(tmem + 128, p_kmaj(sPt, 0, kk), G::mnmaj(sdO, 64 * hh, kk), idKV,
                         (acc0 || kk > 0) ? 1u : 0u);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // dK += dS^T[:, 64hh..] Q[64hh.., :]
            tc::mma_bf16(tmem + 192, p_kmaj(sdSt, 0, kk), G::mnmaj(sQ, 64 * hh, kk), idKV,
                         (acc0 || kk > 0) ? 1u : 0u);
        }
        tc::mma_commit(&bar[2]);
      }
      ++nq;
    }
    if (tid == 0 && qt + 1 < nqt) {
      ok = tc::mbar_wait(&bar[2], (nq - 1) & 1, status) && ok;
      tc::mbar_arrive_expect_tx(&bar[0], 2 * G::tile);
      tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, q0 + kTile, b);
      tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, q0 + kTile, b);
    }
    __syncthreads();  // slse / sdr are rewritten next
  }
  ok = tc::mbar_wait(&bar[2], (nq - 1) & 1, status) && ok;
  tc::fence_after_sync();
  float v[DH];
  tmem_row<DH>(trow + 128u, v);
  if (ok && key < Tlen) store_row<DH>(dV + ((long)b * Tlen + key) * ld_d + h * DH, v, 1.0f);
  tmem_row<DH>(trow + 192u, v);
  if (ok && key < Tlen) store_row<DH>(dK + ((long)b * Tlen + key) * ld_d + h * DH, v, 1.0f);
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 256);
}

// The dK/dV kernel for head widths up to 32 with each query tile taken as
// four 32-query quarters in turn: S^T and dP^T of a quarter (N = 32 each), dV
// and dK need at most 128 TMEM columns, so three or four CTAs share an SM.
// Quarter n (counted over the walk) writes P^T and scale * dS^T to columns
// 32 (n % 2) .. of the 16 KB P^T / dS^T buffers, which quarter n - 2's dV/dK
// products read (bar[2 + n % 2] tracks them).
template <int DH>
__global__ void __launch_bounds__(128, 3)
    attn_bwd_dkv_fl_q_kernel(const __grid_constant__ CUtensorMap mQ,
                             const __grid_constant__ CUtensorMap mK,
                             const __grid_constant__ CUtensorMap mV,
                             const __grid_constant__ CUtensorMap mdO,
                             const float* __restrict__ lse, const float* __restrict__ Drow,
                             bf16* __restrict__ dK, bf16* __restrict__ dV, long ld_d, int Tlen,
                             int H, int L, float scale, unsigned* status) {
  static_assert(DH <= 32, "S^T, dP^T quarters, dV and dK fit 128 TMEM columns for DH <= 32");
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sPt = smem;                      // 16 KB: P^T, two 32-query quarters
  uint8_t* sdSt = smem + 16384;             // 16 KB: scale * dS^T, the same quarters
  uint8_t* sK = smem + 32768;
  uint8_t* sV = sK + G::tile;
  uint8_t* sQ = sV + G::tile;
  uint8_t* sdO = sQ + G::tile;
  float* slse = reinterpret_cast<float*>(sdO + G::tile);  // [128] -lse * log2(e)
  float* sdr = slse + kTile;                               // [128] -Drow * scale
  // tiles loaded; S^T/dP^T of a quarter done; dV/dK of even / odd quarters done
  uint64_t* bar = reinterpret_cast<uint64_t*>(sdr + kTile);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int k0 = blockIdx.x * kTile, h = blockIdx.y, b = blockIdx.z;
  const int qend = min(L >= kTile ? (k0 / L + 1) * L : k0 + kTile, Tlen);
  const int nqt = (qend - k0 + kTile - 1) / kTile;

  if (tid == 0) {
    for (int i = 0; i < 4; ++i) tc::mbar_init(&bar[i], 1);
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mQ);
    tc::prefetch_tmap(&mK);
    tc::prefetch_tmap(&mV);
    tc::prefetch_tmap(&mdO);
  }
  pdl_enter();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar[0], 4 * G::tile);
    tc::tma_load_3d(sK, &mK, &bar[0], h * DH, k0, b);
    tc::tma_load_3d(sV, &mV, &bar[0], h * DH, k0, b);
    tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, k0, b);
    tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, k0, b);
  }
  __syncwarp();
  constexpr uint32_t kCols = 128, kVcol = 64, kKcol = 64 + DH;
  if (warp == 0) {
    tc::tmem_alloc(tslot, kCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);

  const int r = warp * 32 + lane;  // key row
  const int key = k0 + r;
  const float sl2 = scale * kLog2e;
  const int kbe = L < kTile ? (r / L) * L + L : kTile;
  bool ok = true;
  int ns = 0, nq = 0;
  // S^T and dP^T of query quarter q -> TMEM columns 0..63 (tid 0)
  auto issue_scores = [&](int q) {
    if (ok) {
      constexpr uint32_t id32 = tc::idesc_bf16(128, 32, 0, 0);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // S^T quarter -> columns 0..31
        tc::mma_bf16(tmem, G::kmaj(sK, 0, kk), G::kmaj(sQ, 32 * q, kk), id32, kk > 0 ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk)  // dP^T quarter -> columns 32..63
        tc::mma_bf16(tmem + 32, G::kmaj(sV, 0, kk), G::kmaj(sdO, 32 * q, kk), id32,
                     kk > 0 ? 1u : 0u);
    }
    tc::mma_commit(&bar[1]);
  };

  for (int qt = 0; qt < nqt; ++qt) {
    const int q0 = k0 + qt * kTile;
    const bool diag = qt == 0;
    {
      const int tq = q0 + tid;
      const long li = ((long)b * H + h) * Tlen + tq;
      slse[tid] = tq < Tlen ? -lse[li] * kLog2e : 0.f;
      sdr[tid] = tq < Tlen ? -Drow[li] * scale : 0.f;
    }
    if (tid == 0) {
      ok = tc::mbar_wait(&bar[0], qt & 1, status) && ok;
      tc::fence_after_sync();
    }
    __syncthreads();  // slse / sdr written
    for (int q = 0; q < 4; ++q) {
      if (tid == 0 && q == 0) issue_scores(0);
      __syncwarp();
      ok = tc::mbar_wait(&bar[1], ns & 1, status) && ok;
      ++ns;
      tc::fence_after_sync();
      uint32_t rs[32], rd[32];
      tc::tmem_ld32_issue(trow, rs);
      tc::tmem_ld32_issue(trow + 32u, rd);
      tc::tmem_wait();
      const int qb = nq & 1;  // the column half of the P^T / dS^T buffers
      if (nq >= 2) {  // quarter nq - 2's dV/dK products are done with these columns
        ok = tc::mbar_wait(&bar[2 + qb], ((nq - 2) >> 1) & 1, status) && ok;
        tc::fence_after_sync();
      }
      // P^T and dS^T = P^T (dP^T - Drow) scale.  Query columns past the end
      // see zero-filled Q and dO (no contribution), so only the diagonal tile
      // needs a mask.
      float pv[32], dv[32];
      {
        const float4* nl4 = reinterpret_cast<const float4*>(slse + 32 * q);
        const float4* nd4 = reinterpret_cast<const float4*>(sdr + 32 * q);
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {
          const float4 a = nl4[j4], d = nd4[j4];
          const float na[4] = {a.x, a.y, a.z, a.w}, nd[4] = {d.x, d.y, d.z, d.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int j = 4 * j4 + e;
            const int jq = 32 * q + j;  // query column within the tile
            const bool valid = !diag || (q0 + jq < Tlen && jq >= r && jq < kbe);
            const float p = valid ? ex2(fmaf(__uint_as_float(rs[j]), sl2, na[e])) : 0.f;
            pv[j] = p;
            dv[j] = p * fmaf(__uint_as_float(rd[j]), scale, nd[e]);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        put_unit(sPt, r, 4 * qb + u, pack8(pv + 8 * u));
        put_unit(sdSt, r, 4 * qb + u, pack8(dv + 8 * u));
      }
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncthreads();
      if (tid == 0) {
        tc::fence_after_sync();
        // every thread has read this quarter's scores out of TMEM (the barrier
        // above): the next quarter's products go first, under this quarter's
        // dV/dK and the next elementwise pass
        if (q < 3) issue_scores(q + 1);
        if (ok) {
          constexpr uint32_t idKV = tc::idesc_bf16(128, DH, 0, 1);
          const uint32_t acc0 = (qt > 0 || q > 0) ? 1u : 0u;
#pragma unroll
          for (int kk = 0; kk < 2; ++kk)  // dV += P^T[:, 32q..] dO[32q.., :]
            tc::mma_bf16(tmem + kVcol, p_kmaj(sPt, 0, 2 * qb + kk), G::mnmaj(sdO, 32 * q, kk), idKV,
                         (acc0 || kk > 0) ? 1u : 0u);
#pragma unroll
          for (int kk = 0; kk < 2; ++kk)  // dK += dS^T[:, 32q..] Q[32q.., :]
            tc::mma_bf16(tmem + kKcol, p_kmaj(sdSt, 0, 2 * qb + kk), G::mnmaj(sQ, 32 * q, kk), idKV,
                         (acc0 || kk > 0) ? 1u : 0u);
        }
        tc::mma_commit(&bar[2 + qb]);
      }
      ++nq;
    }
    if (tid == 0 && qt + 1 < nqt) {  // every product of the tile is done with Q / dO
      ok = tc::mbar_wait(&bar[2 + ((nq - 1) & 1)], ((nq - 1) >> 1) & 1, status) && ok;
      tc::mbar_arrive_expect_tx(&bar[0], 2 * G::tile);
      tc::tma_load_3d(sQ, &mQ, &bar[0], h * DH, q0 + kTile, b);
      tc::tma_load_3d(sdO, &mdO, &bar[0], h * DH, q0 + kTile, b);
    }
    __syncthreads();  // slse / sdr are rewritten next
  }
  ok = tc::mbar_wait(&bar[2 + ((nq - 1) & 1)], ((nq - 1) >> 1) & 1, status) && ok;
  tc::fence_after_sync();
  float v[DH];
  tmem_row<DH>(trow + kVcol, v);
  if (ok && key < Tlen) store_row<DH>(dV + ((long)b * Tlen + key) * ld_d + h * DH, v, 1.0f);
  tmem_row<DH>(trow + kKcol, v);
  if (ok && key < Tlen) store_row<DH>(dK + ((long)b * Tlen + key) * ld_d + h * DH, v, 1.0f);
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, kCols);
}

// ========================================================================= host
bool attn_fl_supported(int dtype, int dh, int L) {
  const bool l_ok = (L >= 16 && kTile % L == 0) || (L % kTile == 0 && L <= 1024);
  return dtype == 1 && (dh == 16 || dh == 32 || dh == 64) && l_ok && tmap_encoder() != nullptr;
}

namespace {
template <int DH>
bool head_map_fl(CUtensorMap* m, const void* base, long ld, int D, int T, int B) {
  const uint64_t dims[3] = {(uint64_t)D, (uint64_t)T, (uint64_t)B};
  const uint64_t st[2] = {(uint64_t)ld * 2, (uint64_t)ld * 2 * (uint64_t)T};
  const uint32_t box[3] = {DH, kTile, 1};
  const CUtensorMapSwizzle sw = DH == 64   ? CU_TENSOR_MAP_SWIZZLE_128B
                                : DH == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                           : CU_TENSOR_MAP_SWIZZLE_32B;
  return make_tmap_bf16(m, base, 3, dims, st, box, sw);
}

// dynamic shared memory: 1 KB alignment slack + tiles + staging + barriers
template <int DH> constexpr int fwd_smem() { return 1024 + 32768 + 4 * Geo<DH>::tile + 64; }
template <int DH> constexpr int dq_smem() { return 1024 + 32768 + 4 * Geo<DH>::tile + 64; }
template <int DH> constexpr int dkv_smem() {
  return 1024 + 32768 + 4 * Geo<DH>::tile + 2 * kTile * 4 + 64;
}

template <int DH> constexpr int fwd_half_smem() {
  return 1024 + 16384 + (DH <= 32 ? 4 : 3) * Geo<DH>::tile + 64;
}

template <int DH>
cudaError_t fwd_fl_half_launch(const Launch& lc, const AttnArgs& a, const CUtensorMap* m) {
  static std::atomic<unsigned long long> opted{0};
  auto kern = attn_fwd_fl_half_kernel<DH>;
  cudaError_t e = smem_opt_in(kern, fwd_half_smem<DH>(), &opted);
  if (e != cudaSuccess) return e;
  dim3 grid((a.T + kTile - 1) / kTile, a.H, a.B);
  e = launch_k(kern, grid, dim3(128), fwd_half_smem<DH>(), lc.stream, m[0], m[1], m[2],
               (bf16*)a.O, a.ld_o, a.lse, a.T, a.H, a.L, 1.0f / sqrtf((float)DH), lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int DH, int NCH, bool ONE>
cudaError_t fwd_fl_launch(const Launch& lc, const AttnArgs& a, const CUtensorMap* m) {
  static std::atomic<unsigned long long> opted{0};
  auto kern = attn_fwd_fl_kernel<DH, NCH, ONE>;
  cudaError_t e = smem_opt_in(kern, fwd_smem<DH>(), &opted);
  if (e != cudaSuccess) return e;
  dim3 grid((a.T + kTile - 1) / kTile, a.H, a.B);
  e = launch_k(kern, grid, dim3(128), fwd_smem<DH>(), lc.stream, m[0], m[1], m[2], (bf16*)a.O,
               a.ld_o, a.lse, a.T, a.H, a.L, 1.0f / sqrtf((float)DH), lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int DH>
cudaError_t fwd_fl(const Launch& lc, const AttnArgs& a) {
  const int D = a.H * DH;
  CUtensorMap m[3];
  if (!head_map_fl<DH>(&m[0], a.Q, a.ld_qkv, D, a.T, a.B) ||
      !head_map_fl<DH>(&m[1], a.K, a.ld_qkv, D, a.T, a.B) ||
      !head_map_fl<DH>(&m[2], a.V, a.ld_qkv, D, a.T, a.B))
    return cudaErrorInvalidValue;
  if (a.L > kTile) return fwd_fl_half_launch<DH>(lc, a, m);
  if (a.L <= 32) return fwd_fl_launch<DH, 1, true>(lc, a, m);
  if (a.L == 64) return fwd_fl_launch<DH, 2, true>(lc, a, m);
  return fwd_fl_launch<DH, 4, true>(lc, a, m);
}

template <int DH>
cudaError_t bwd_fl(const Launch& lc, const AttnBwdArgs& a) {
  const AttnArgs& f = a.f;
  const int D = f.H * DH;
  CUtensorMap mq, mk, mv, mdo;
  if (!head_map_fl<DH>(&mq, f.Q, f.ld_qkv, D, f.T, f.B) ||
      !head_map_fl<DH>(&mk, f.K, f.ld_qkv, D, f.T, f.B) ||
      !head_map_fl<DH>(&mv, f.V, f.ld_qkv, D, f.T, f.B) ||
      !head_map_fl<DH>(&mdo, a.dO, f.ld_o, D, f.T, f.B))
    return cudaErrorInvalidValue;
  static std::atomic<unsigned long long> opted_q{0}, opted_kv{0};
  // head widths up to 32: the dQ kernel that walks 32-key quarters
  auto dq_kern = DH <= 32 ? attn_bwd_dq_fl_q_kernel<DH <= 32 ? DH : 32> : attn_bwd_dq_fl_kernel<DH>;
  cudaError_t e = smem_opt_in(dq_kern, dq_smem<DH>(), &opted_q);
  auto dkv_kern =
      DH <= 32 ? attn_bwd_dkv_fl_q_kernel<DH <= 32 ? DH : 32> : attn_bwd_dkv_fl_kernel<DH>;
  if (e == cudaSuccess) e = smem_opt_in(dkv_kern, dkv_smem<DH>(), &opted_kv);
  if (e != cudaSuccess) return e;
  const float scale = 1.0f / sqrtf((float)DH);
  dim3 grid((f.T + kTile - 1) / kTile, f.H, f.B);
  e = launch_k(dq_kern, grid, dim3(128), dq_smem<DH>(), lc.stream, mq, mk, mv,
               mdo, (const bf16*)f.O, (const bf16*)a.dO, f.ld_o, (const float*)f.lse, a.Drow,
               (bf16*)a.dQ, a.ld_dqkv, f.T, f.H, f.L, scale, lc.status);
  if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
  e = launch_k(dkv_kern, grid, dim3(128), dkv_smem<DH>(), lc.stream, mq, mk, mv,
               mdo, (const float*)f.lse, (const float*)a.Drow, (bf16*)a.dK, (bf16*)a.dV,
               a.ld_dqkv, f.T, f.H, f.L, scale, lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}
}  // namespace

cudaError_t attn_fwd_fl(const Launch& lc, const AttnArgs& a) {
  if (!attn_fl_supported(1, a.dh, a.L)) return cudaErrorNotSupported;
  switch (a.dh) {
    case 16: return fwd_fl<16>(lc, a);
    case 32: return fwd_fl<32>(lc, a);
    default: return fwd_fl<64>(lc, a);
  }
}

cudaError_t attn_bwd_fl(const Launch& lc, const AttnBwdArgs& a) {
  if (!attn_fl_supported(1, a.f.dh, a.f.L)) return cudaErrorNotSupported;
  switch (a.f.dh) {
    case 16: return bwd_fl<16>(lc, a);
    case 32: return bwd_fl<32>(lc, a);
    default: return bwd_fl<64>(lc, a);
  }
}

}  // namespace bcmt
