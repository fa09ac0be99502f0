// Dense GEMMs of the BCMT layer: the Q/K/V, W_O, W_g and W_m projections of
// Sec. 3.3-3.8 and their backward products.
//
//  * gemm_tc: bf16 inputs on the tcgen05 tensor cores.  One CTA computes a
//    128 x BN output tile with the fp32 accumulator in TMEM.  Warp 0 (one lane)
//    streams 64-deep K slices of A and B into a STAGES-deep shared-memory ring
//    with TMA (128-byte swizzle); warp 1 (one lane) issues tcgen05.mma into
//    one of two TMEM accumulators and releases each slot with tcgen05.commit;
//    warps 2-9 (two per TMEM lane quarter, each half of the tile's columns)
//    read the other accumulator back with tcgen05.ld (thread = output row) and
//    run the fused epilogue.  Every mbarrier wait is bounded.
//  * gemm_simt: true-fp32 FMA, used for fp32 tensors (a TF32 tensor-core
//    product cannot meet a 1e-4 absolute error bound).
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <type_traits>
#include <vector>

#include "common.cuh"
#include "epilogues.cuh"
#include "internal.h"
#include "tc.cuh"
#include "tmap.h"

namespace bcmt {

int effective_splits(int K, int splits) {
  const int nkb = (K + 63) / 64;
  if (splits < 1) splits = 1;
  if (splits > nkb) splits = nkb;
  const int kps = (nkb + splits - 1) / splits;
  return (nkb + kps - 1) / kps;
}

// ======================================================================== SIMT
template <class TI, class Epi>
__global__ void __launch_bounds__(256) gemm_simt_kernel(int M, int N, int K, const TI* __restrict__ A,
                                                        long sam, long sak,
                                                        const TI* __restrict__ B, long sbk,
                                                        long sbn, Epi epi, int kps) {
  pdl_enter();
  __shared__ float As[16][64 + 4];
  __shared__ float Bs[16][64 + 4];
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64, z = blockIdx.z;
  const int kb = z * kps, ke = min(K, kb + kps);
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = kb; k0 < ke; k0 += 16) {
    for (int e = tid; e < 16 * 64; e += 256) {
      int mm, ka;
      if (sak == 1) { ka = e % 16; mm = e / 16; } else { mm = e % 64; ka = e / 64; }
      const int m = m0 + mm, k = k0 + ka;
      As[ka][mm] = (m < M && k < ke) ? to_f(A[(long)m * sam + (long)k * sak]) : 0.f;
      int nn, kb2;
      if (sbn == 1) { nn = e % 64; kb2 = e / 64; } else { kb2 = e % 16; nn = e / 16; }
      const int n = n0 + nn, k2 = k0 + kb2;
      Bs[kb2][nn] = (n < N && k2 < ke) ? to_f(B[(long)k2 * sbk + (long)n * sbn]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const int col = n0 + tx * 4;
  if (col >= N) return;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = m0 + ty * 4 + i;
    if (row < M) epi(row, col, acc[i], 4, z);
  }
}

template <class TI, class Epi>
static cudaError_t simt_launch(const Launch& lc, int M, int N, int K, const void* A, long sam,
                               long sak, const void* B, long sbk, long sbn, const Epi& epi,
                               int splits) {
  const int nkb = (K + 63) / 64;
  const int kps = ((nkb + splits - 1) / splits) * 64;
  dim3 grid((N + 63) / 64, (M + 63) / 64, splits);
  launch_k(gemm_simt_kernel<TI, Epi>, dim3(grid), dim3(256), 0, lc.stream,

      M, N, K, static_cast<const TI*>(A), sam, sak, static_cast<const TI*>(B), sbk, sbn, epi, kps);
  return cudaGetLastError();
}

template <class TI>
static cudaError_t simt_typed(const Launch& lc, int dtype_out, int M, int N, int K, const void* A,
                              long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                              const EpiArgs& ea, int splits) {
  switch (epi) {
    case EPI_STORE:
      if (dtype_out == 0)
        return simt_launch<TI>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                               EpiStoreF<float>{(float*)ea.out, ea.ldo, 0}, 1);
      return simt_launch<TI>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                             EpiStoreF<bf16>{(bf16*)ea.out, ea.ldo, 0}, 1);
    case EPI_PARTIAL:
      return simt_launch<TI>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                             EpiStoreF<float>{(float*)ea.out, ea.ldo, ea.split_stride}, splits);
    case EPI_GATE:
      return simt_launch<TI>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                             EpiGateF<TI>{(TI*)ea.out, ea.ldo}, 1);
    case EPI_STORE_SCORE:
      if (dtype_out == 0)
        return simt_launch<TI>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                               EpiStoreScoreF<float>{(float*)ea.out, ea.ldo,
                                                     (const float*)ea.w_p, ea.spart, M},
                               1);
      return simt_launch<TI>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                             EpiStoreScoreF<bf16>{(bf16*)ea.out, ea.ldo, (const bf16*)ea.w_p,
                                                  ea.spart, M},
                             1);
  }
  return cudaErrorInvalidValue;
}

cudaError_t gemm_simt(const Launch& lc, int dtype, int dtype_out, int M, int N, int K,
                      const void* A, long sam, long sak, const void* B, long sbk, long sbn,
                      EpiKind epi, const EpiArgs& ea, int splits) {
  if (N % 64 != 0) return cudaErrorInvalidValue;
  splits = (epi == EPI_PARTIAL) ? effective_splits(K, splits) : 1;
  if (dtype == 0)
    return simt_typed<float>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  return simt_typed<bf16>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
}

// ===================================================================== tcgen05
namespace {
constexpr int kBM = 128, kBK = 64;
constexpr int kEpiWarps = 8;
constexpr int kOutStage = 4096;  // per epilogue warp: two 32x32 bf16 or one 32x32 fp32 chunk

// Output tile of a persistent GEMM's tile index: K split z slowest; within a
// split, bands of kBand m-blocks, and within a band m fastest, so that the
// tiles running at one time share a few rows of A and columns of B in L2
// instead of sweeping all of A for every column block.
constexpr int kBand = 8;
__device__ __forceinline__ void tile_mnz(int tile, int tiles_m, int tiles_n, int& m_blk,
                                         int& n_blk, int& z) {
  const int per_z = tiles_m * tiles_n;
  z = tile / per_z;
  const int t = tile - z * per_z;
  const int band = t / (kBand * tiles_n);
  const int m0 = band * kBand;
  const int gm = min(kBand, tiles_m - m0);
  const int r = t - band * kBand * tiles_n;
  m_blk = m0 + r % gm;
  n_blk = r / gm;
}

__device__ __forceinline__ uint4 pack8_bf16(const float* v) {
  uint4 q;
  __nv_bfloat162 t0 = __floats2bfloat162_rn(v[0], v[1]), t1 = __floats2bfloat162_rn(v[2], v[3]);
  __nv_bfloat162 t2 = __floats2bfloat162_rn(v[4], v[5]), t3 = __floats2bfloat162_rn(v[6], v[7]);
  q.x = *reinterpret_cast<uint32_t*>(&t0);
  q.y = *reinterpret_cast<uint32_t*>(&t1);
  q.z = *reinterpret_cast<uint32_t*>(&t2);
  q.w = *reinterpret_cast<uint32_t*>(&t3);
  return q;
}

// Epilogue output of one warp: 32 rows (thread = row) x 32 columns, after the
// functor's in-place transform.  TMA-stored epilogues stage the chunk in the
// warp's shared buffer in the swizzled layout of the output tensor map (64-byte
// swizzle for bf16 rows of 64 bytes, 128-byte swizzle for fp32 rows of 128) and
// lane 0 stores it with one bulk copy; bf16 chunks alternate between two
// buffers.  Other epilogues store from registers.
// apply: this thread's row is valid; store: lane 0 issues the chunk's store
// (rows past M are clipped by the tensor map).  Called by the whole warp.
// col: the chunk's column in the product; scol: its column in the output
// tensor map mC (col, or col - n_split in the second output of a dual
// epilogue).
template <class Epi>
__device__ __forceinline__ void epi_chunk(const Epi& epi, const CUtensorMap* mC, uint8_t* sbuf,
                                          int& nout, int lane, int row, int row0, int col,
                                          int scol, int z, float* v,
                                          const typename Epi::Pre& pre, bool apply, bool store) {
  if constexpr (Epi::kTma) {
    using OT = typename Epi::OutT;
    // a warp-wide epilogue (lane shuffles) runs on every lane of a valid tile
    if (Epi::kWarpWide ? store : apply) epi.apply(row, col, v, pre, z);
    constexpr bool kBf = sizeof(OT) == 2;
    uint8_t* buf = sbuf + (kBf ? (nout & 1) * 2048 : 0);
    if (lane == 0) {
      if (kBf)
        tc::tma_store_wait_read<1>();
      else
        tc::tma_store_wait_read<0>();
    }
    __syncwarp();

    if (kBf) {
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<uint4*>(buf + lane * 64 + ((u ^ ((lane >> 1) & 3)) << 4)) =
            pack8_bf16(v + 8 * u);
    } else {
#pragma unroll
      for (int u = 0; u < 8; ++u)
        *reinterpret_cast<float4*>(buf + lane * 128 + ((u ^ (lane & 7)) << 4)) =
            make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
    }
    tc::fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0 && store) {
      tc::tma_store_3d(mC, buf, scol, row0, z);
      tc::tma_store_commit();
    }
    ++nout;
  } else {
    (void)mC;
    (void)sbuf;
    (void)nout;
    (void)row0;
    (void)scol;
    (void)store;
    if (apply) epi.apply(row, col, v, pre, z);
  }
}

template <int BN, int STAGES>
struct TcCfg {
  static constexpr int A_BYTES = kBM * kBK * 2;
  static constexpr int B_BYTES = BN * kBK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int OUT_OFF = STAGES * STAGE_BYTES;          // output staging
  static constexpr int BAR_OFF = OUT_OFF + kEpiWarps * kOutStage;
  static constexpr int SMEM = BAR_OFF + 1024 + 256;
  static constexpr int TMEM_COLS = 2 * BN;  // two accumulators
};

int sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
      n = 1;
  }
  return n;
}
}  // namespace

// Persistent, warp-specialised tcgen05 GEMM.  Tiles are 128 x BN output
// blocks (optionally one K-split each), taken round-robin by the CTAs, m
// fastest.  Warp 0 / lane 0 streams 64-deep K slices of A and B into a
// STAGES-deep ring with TMA; warp 1 / lane 0 issues the MMAs into one of two
// TMEM accumulators; warps 2-9 drain the other accumulator through the
// epilogue at the same time (two warps per TMEM lane quarter, each taking
// half of the tile's columns), so a tile's epilogue overlaps the next tile's
// main loop.
constexpr int kGemmThreads = 320;

// The rest of a launch's description, beside product 0 (the kernel's own
// arguments):
//  * mB2, mC2: for a dual epilogue (Epi::kDual), the B operand and the output
//    of the columns from epi.n_split on (their own tensors, columns counted
//    from n_split);
//  * a second product with the same operand layouts and a plain store
//    epilogue of its own (has1, the kernel's Epi1): its n_tiles1 tiles follow
//    product 0's in the round-robin order, so a small product fills the idle
//    slots of a large one's last wave.
struct TcAux {
  CUtensorMap mB2, mC2;
  CUtensorMap mA1, mB1, mC1;
  int M1, N1, kps1, nkb1, tiles_m1, tiles_n1, n_tiles1;
  int has1;
};

// Where one tile of a launch reads and writes: its product's tensor maps,
// shape and K range, and its origin.
struct TcTile {
  const CUtensorMap *a, *b, *c;
  int M, N, m0, n0, nb0, nc0, z, kb0, nk;
  bool p1;  // a tile of the second product
};
template <int BN, class Epi>
__device__ __forceinline__ TcTile tc_tile(int tile, const CUtensorMap& mA, const CUtensorMap& mB,
                                          const CUtensorMap& mC, const TcAux& aux, int M, int N,
                                          int kps, int nkb, int tiles_m, int tiles_n, int n_tiles,
                                          const Epi& epi) {
  TcTile t;
  const bool p1 = tile >= n_tiles;
  const int tl = p1 ? tile - n_tiles : tile;
  const int tm = p1 ? aux.tiles_m1 : tiles_m, tn = p1 ? aux.tiles_n1 : tiles_n;
  const int ks = p1 ? aux.kps1 : kps, nb = p1 ? aux.nkb1 : nkb;
  int m_blk, n_blk;
  tile_mnz(tl, tm, tn, m_blk, n_blk, t.z);
  t.p1 = p1;
  t.a = p1 ? &aux.mA1 : &mA;
  t.b = p1 ? &aux.mB1 : &mB;
  t.c = p1 ? &aux.mC1 : &mC;
  t.M = p1 ? aux.M1 : M;
  t.N = p1 ? aux.N1 : N;
  t.m0 = m_blk * kBM;
  t.n0 = n_blk * BN;
  t.nb0 = t.nc0 = t.n0;
  if constexpr (Epi::kDual) {
    if (!p1 && t.n0 >= epi.n_split) {
      t.b = &aux.mB2;
      t.c = &aux.mC2;
      t.nb0 = t.nc0 = t.n0 - epi.n_split;
    }
  }
  t.kb0 = t.z * ks;
  t.nk = min(nb, t.kb0 + ks) - t.kb0;
  return t;
}

// One tile's epilogue (warps 2..9): warp w reads TMEM lanes 32*(w%4) .. +31
// and the columns of half (w-2)/4 of the tile, transforms and stores them.
template <int BN, class Epi>
__device__ __forceinline__ bool tc_epilogue(const Epi& epi, const TcTile& t, int warp, int lane,
                                            uint32_t tmem, int acc, int use, uint64_t* tfull,
                                            uint8_t* sbuf, int& nout, unsigned* status) {
  const int q = warp & 3;
  const int c_beg = ((warp - 2) >> 2) * (BN / 2);
  const int z = t.z, N = t.N;
  const int row0 = t.m0 + q * 32;
  const int row = row0 + lane;
  const int n0 = t.n0;
  const bool row_ok = row < t.M;
  // the output map and column of this tile (a dual epilogue's second part
  // and a second product have their own)
  const int soff = t.n0 - t.nc0;
  // The epilogue's own inputs do not depend on the accumulator: fetch the
  // first chunk's before waiting for it, and each next chunk's one ahead.
  constexpr int NCH = BN / 64;  // 32-column chunks per epilogue warp
  typename Epi::Pre pre[2];
  if (row_ok && n0 + c_beg < N) epi.load(row, n0 + c_beg, pre[0]);
  const bool ok = tc::mbar_wait(&tfull[acc], use & 1, status);
  tc::fence_after_sync();
  const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci) {
    const int c = c_beg + ci * 32;
    if (ci + 1 < NCH && row_ok && n0 + c + 32 < N) epi.load(row, n0 + c + 32, pre[(ci + 1) & 1]);
    float v[32];
    tc::tmem_ld32(base + (uint32_t)c, v);
    if (n0 + c < N)
      epi_chunk(epi, t.c, sbuf, nout, lane, row, row0, n0 + c, n0 + c - soff, z, v, pre[ci & 1],
                ok && row_ok, ok);
  }
  return ok;
}

template <int BN, int STAGES, bool A_MN, bool B_MN, class Epi, class Epi1 = EpiStoreF<bf16>>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB,
                   const __grid_constant__ CUtensorMap mC, const __grid_constant__ TcAux aux,
                   int M, int N, int kps, int nkb, int tiles_m, int tiles_n, int n_tiles, Epi epi,
                   Epi1 epi1, unsigned* status) {
  const int total = n_tiles + (aux.has1 ? aux.n_tiles1 : 0);
  using Cfg = TcCfg<BN, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Cfg::BAR_OFF);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;   // accumulator ready for the epilogue
  uint64_t* tempty = tfull + 2;       // accumulator drained by the epilogue
  uint32_t* tslot = reinterpret_cast<uint32_t*>(tempty + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (warp == 0 && lane == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(&tfull[a], 1);
      tc::mbar_init(&tempty[a], 8);
    }
    tc::fence_mbar_init();
    tc::prefetch_tmap(&mA);
    tc::prefetch_tmap(&mB);
    if (Epi::kDual) tc::prefetch_tmap(&aux.mB2);
    if (aux.has1) {
      tc::prefetch_tmap(&aux.mA1);
      tc::prefetch_tmap(&aux.mB1);
    }
  }
  if (warp == 1) {
    tc::tmem_alloc(tslot, Cfg::TMEM_COLS);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  pdl_enter();  // setup above overlapped the previous kernel

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer
      int it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
        const TcTile t = tc_tile<BN>(tile, mA, mB, mC, aux, M, N, kps, nkb, tiles_m, tiles_n,
                                     n_tiles, epi);
        const int m0 = t.m0, n0 = t.nb0, kb0 = t.kb0, nk = t.nk;
        for (int i = 0; i < nk; ++i, ++it) {
          const int s = it % STAGES;
          if (it >= STAGES && !tc::mbar_wait(&empty[s], ((it / STAGES) - 1) & 1, status)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + s * Cfg::STAGE_BYTES;
          uint8_t* sb = sa + Cfg::A_BYTES;
          tc::mbar_arrive_expect_tx(&full[s], Cfg::STAGE_BYTES);
          const int k0 = (kb0 + i) * kBK;
          if (!A_MN) {
            tc::tma_load_2d(sa, t.a, &full[s], k0, m0);
          } else {
            tc::tma_load_2d(sa, t.a, &full[s], m0, k0);
            tc::tma_load_2d(sa + 8192, t.a, &full[s], m0 + 64, k0);
          }
          if (!B_MN) {
            tc::tma_load_2d(sb, t.b, &full[s], k0, n0);
          } else {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j)
              tc::tma_load_2d(sb + j * 8192, t.b, &full[s], n0 + 64 * j, k0);
          }
        }
      }
      // No copy may still be in flight when the CTA exits.
      for (int i = (it > STAGES ? it - STAGES : 0); i < it; ++i)
        tc::mbar_wait(&full[i % STAGES], (i / STAGES) & 1, status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer
      constexpr uint32_t idesc = tc::idesc_bf16(kBM, BN, A_MN ? 1 : 0, B_MN ? 1 : 0);
      int it = 0, j = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x, ++j) {
        const TcTile t = tc_tile<BN>(tile, mA, mB, mC, aux, M, N, kps, nkb, tiles_m, tiles_n,
                                     n_tiles, epi);
        const int nk = t.nk;
        const int acc = j & 1, use = j >> 1;
        if (use > 0 && !tc::mbar_wait(&tempty[acc], (use - 1) & 1, status)) break;
        tc::fence_after_sync();
        const uint32_t d = tmem + (uint32_t)(acc * BN);
        for (int i = 0; i < nk; ++i, ++it) {
          const int s = it % STAGES;
          if (!tc::mbar_wait(&full[s], (it / STAGES) & 1, status)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
          const uint32_t sa = tc::smem_u32(smem + s * Cfg::STAGE_BYTES);
          const uint32_t sb = sa + Cfg::A_BYTES;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            const uint64_t ad = A_MN ? tc::sdesc(sa + kk * 2048, 8192, 1024)
                                     : tc::sdesc(sa + kk * 32, 16, 1024);
            const uint64_t bd = B_MN ? tc::sdesc(sb + kk * 2048, 8192, 1024)
                                     : tc::sdesc(sb + kk * 32, 16, 1024);
            tc::mma_bf16(d, ad, bd, idesc, (i | kk) != 0 ? 1u : 0u);
          }
          tc::mma_commit(&empty[s]);
        }
        tc::mma_commit(&tfull[acc]);
      }
    }
  } else {
    // ---- epilogue warps 2..9 (tc_epilogue), the second product's tiles
    // through its own epilogue
    uint8_t* sbuf = smem + Cfg::OUT_OFF + (warp - 2) * kOutStage;
    int j = 0, nout = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x, ++j) {
      const TcTile t = tc_tile<BN>(tile, mA, mB, mC, aux, M, N, kps, nkb, tiles_m, tiles_n,
                                   n_tiles, epi);
      const int acc = j & 1, use = j >> 1;
      const bool ok = t.p1 ? tc_epilogue<BN>(epi1, t, warp, lane, tmem, acc, use, tfull, sbuf,
                                             nout, status)
                           : tc_epilogue<BN>(epi, t, warp, lane, tmem, acc, use, tfull, sbuf,
                                             nout, status);
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&tempty[acc]);
      if (!ok) break;
    }
    if (lane == 0) tc::tma_store_wait_read<0>();  // staging read; the writes finish with the grid
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) tc::tmem_dealloc(tmem, Cfg::TMEM_COLS);
}

namespace {
bool g_tc_ok = true;
}

bool gemm_tc_available() { return g_tc_ok && tmap_encoder() != nullptr; }

// Tensor map of an epilogue's output for its TMA stores: [splits][M][N] with
// row stride ldo, 32 x 32 boxes (64-byte swizzle for bf16, 128-byte for fp32).
// The second output of a dual epilogue: [M][N - n_split], row stride ldo2.
template <class Epi>
static bool out_map2(CUtensorMap* m, const Epi& epi, int M, int N) {
  memset(m, 0, sizeof(*m));
  if constexpr (!Epi::kDual) {
    return true;
  } else {
    using OT = typename Epi::OutT;
    const uint64_t es = sizeof(OT);
    const uint64_t d[3] = {(uint64_t)(N - epi.n_split), (uint64_t)M, 1};
    const uint64_t st[2] = {(uint64_t)epi.ldo2 * es, (uint64_t)epi.ldo2 * es * (uint64_t)M};
    const uint32_t box[3] = {32, 32, 1};
    return make_tmap(m, es == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
                     epi.out2, 3, d, st, box,
                     es == 2 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B);
  }
}

template <class Epi>
static bool out_map(CUtensorMap* m, const Epi& epi, int M, int N, int splits) {
  memset(m, 0, sizeof(*m));
  if constexpr (!Epi::kTma) {
    return true;
  } else {
    using OT = typename Epi::OutT;
    const uint64_t es = sizeof(OT);
    const long ss = epi.split_stride > 0 ? epi.split_stride : (long)M * epi.ldo;
    const uint64_t d[3] = {(uint64_t)N, (uint64_t)M, (uint64_t)splits};
    const uint64_t st[2] = {(uint64_t)epi.ldo * es, (uint64_t)ss * es};
    const uint32_t box[3] = {32, 32, 1};
    return make_tmap(m, es == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
                     epi.out, 3, d, st, box,
                     es == 2 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B);
  }
}

// Operand tensor maps of the single-CTA kernel: A as 128 x 64 boxes (K-major)
// or 64 x 64 boxes (MN-major), B as BN x 64 (K-major) or 64 x 64 (MN-major).
template <bool A_MN>
static bool tc_a_map(CUtensorMap* m, const void* A, int M, int K, long sam, long sak) {
  if (!A_MN) {
    uint64_t d[2] = {(uint64_t)K, (uint64_t)M}, st[1] = {(uint64_t)sam * 2};
    uint32_t box[2] = {64, 128};
    return make_tmap_bf16(m, A, 2, d, st, box);
  }
  uint64_t d[2] = {(uint64_t)M, (uint64_t)K}, st[1] = {(uint64_t)sak * 2};
  uint32_t box[2] = {64, 64};
  return make_tmap_bf16(m, A, 2, d, st, box);
}
template <int BN, bool B_MN>
static bool tc_b_map(CUtensorMap* m, const void* B, int N, int K, long sbk, long sbn) {
  if (!B_MN) {
    uint64_t d[2] = {(uint64_t)K, (uint64_t)N}, st[1] = {(uint64_t)sbn * 2};
    uint32_t box[2] = {64, (uint32_t)BN};
    return make_tmap_bf16(m, B, 2, d, st, box);
  }
  uint64_t d[2] = {(uint64_t)N, (uint64_t)K}, st[1] = {(uint64_t)sbk * 2};
  uint32_t box[2] = {64, 64};
  return make_tmap_bf16(m, B, 2, d, st, box);
}

// One launch of the single-CTA kernel: product 0 (M, N, K, A, B, epi), for a
// dual epilogue the B operand b2 of its columns from epi.n_split on, and
// optionally a second product p1 stored as bf16 after product 0's tiles
// (plain-store epilogues only).
template <int BN, int STAGES, bool A_MN, bool B_MN, class Epi, class Epi1 = EpiStoreF<bf16>>
static cudaError_t tc_launch(const Launch& lc, int M, int N, int K, const void* A, long sam,
                             long sak, const void* B, long sbk, long sbn, const Epi& epi,
                             int splits, int max_ctas = 0, const void* b2 = nullptr,
                             const GemmProd* p1 = nullptr, const Epi1& epi1 = Epi1{}) {
  using Cfg = TcCfg<BN, STAGES>;
  CUtensorMap mA, mB, mC;
  TcAux aux;
  memset(&aux, 0, sizeof(aux));
  int nb = N;  // B columns of the first map
  if constexpr (Epi::kDual) nb = epi.n_split;
  if (!tc_a_map<A_MN>(&mA, A, M, K, sam, sak) || !tc_b_map<BN, B_MN>(&mB, B, nb, K, sbk, sbn))
    return cudaErrorInvalidValue;
  const int nkb = (K + kBK - 1) / kBK;
  const int kps = (nkb + splits - 1) / splits;
  const int tiles_m = (M + kBM - 1) / kBM, tiles_n = (N + BN - 1) / BN;
  const int n_tiles = tiles_m * tiles_n * splits;
  auto kern = gemm_tc_kernel<BN, STAGES, A_MN, B_MN, Epi, Epi1>;
  static std::atomic<unsigned long long> opted{0};
  if (cudaError_t e = smem_opt_in(kern, Cfg::SMEM, &opted); e != cudaSuccess) return e;
  if constexpr (Epi::kDual) {
    // every tile lies on one side of n_split
    if (epi.n_split % BN != 0 || epi.n_split <= 0 || epi.n_split >= N || !b2)
      return cudaErrorInvalidValue;
    if (!out_map(&mC, epi, M, epi.n_split, 1) || !out_map2(&aux.mC2, epi, M, N) ||
        !tc_b_map<BN, B_MN>(&aux.mB2, b2, N - epi.n_split, K, sbk, sbn))
      return cudaErrorInvalidValue;
  } else {
    if (!out_map(&mC, epi, M, N, splits)) return cudaErrorInvalidValue;
  }
  if (p1) {
    if (Epi::kDual || splits != 1) return cudaErrorInvalidValue;
    if (!tc_a_map<A_MN>(&aux.mA1, p1->A, p1->M, p1->K, p1->sam, p1->sak) ||
        !tc_b_map<BN, B_MN>(&aux.mB1, p1->B, p1->N, p1->K, p1->sbk, p1->sbn) ||
        !out_map(&aux.mC1, epi1, p1->M, p1->N, 1))
      return cudaErrorInvalidValue;
    aux.has1 = 1;
    aux.M1 = p1->M;
    aux.N1 = p1->N;
    aux.nkb1 = (p1->K + kBK - 1) / kBK;
    aux.kps1 = aux.nkb1;
    aux.tiles_m1 = (p1->M + kBM - 1) / kBM;
    aux.tiles_n1 = (p1->N + BN - 1) / BN;
    aux.n_tiles1 = aux.tiles_m1 * aux.tiles_n1;
  }
  const int total = n_tiles + (aux.has1 ? aux.n_tiles1 : 0);
  int grid = total < sm_count() ? total : sm_count();
  if (max_ctas > 0 && grid > max_ctas) grid = max_ctas;
  cudaError_t e = launch_k(kern, dim3(grid), dim3(kGemmThreads), Cfg::SMEM, lc.stream, mA, mB, mC,
                           aux, M, N, kps, nkb, tiles_m, tiles_n, n_tiles, epi, epi1, lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ============================================================ CTA-pair GEMM
// The same persistent, warp-specialised GEMM on pairs of CTAs (a cluster of
// two): one tcgen05.mma.cta_group::2 computes a 256 x BN tile, each CTA
// holding 128 rows of A and BN/2 of the N columns of B, so per SM a 64-deep K
// slice brings 128x64 + (BN/2)x64 operands for a 128 x BN product: with
// BN = 256 one and a half times the flops per byte of a single-CTA 128 x 256
// tile, and a 32 KB stage that allows a 6-deep ring.  Both CTAs stream their
// halves by TMA, counted on the even CTA's stage barrier; the even CTA issues
// the MMAs and its commits arrive on the stage and accumulator barriers of
// both CTAs; each CTA's epilogue warps drain their own 128 accumulator rows
// and report back to the even CTA.
//
// One launch may carry up to kTc2Max independent products (a group):
// product 0 with operand layouts and epilogue Op0, the others with Op1 (each
// with its own shape and tensor maps).  The products' tiles are numbered one
// product after the other and the pairs take the combined list round-robin,
// so products that would each leave SMs idle (dX and the K-split weight
// gradients at the end of the backward pass) share one wave.  A single
// product is a group of one.
template <int BN, int STAGES, int ACC>
struct Tc2Cfg {
  static constexpr int A_BYTES = kBM * kBK * 2;          // 16 KB
  static constexpr int B_BYTES = (BN / 2) * kBK * 2;     // this CTA's half of B
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int OUT_OFF = STAGES * STAGE_BYTES;
  static constexpr int BAR_OFF = OUT_OFF + kEpiWarps * kOutStage;
  static constexpr int SMEM = BAR_OFF + 1024 + 256;
  static constexpr int TMEM_COLS = ACC * BN;
};

// Compile-time half of one product of a group: operand layouts and epilogue.
template <bool A_MN_, bool B_MN_, class Epi_>
struct Tc2Op {
  static constexpr bool A_MN = A_MN_, B_MN = B_MN_;
  using Epi = Epi_;
};

// Run-time half: shape, K slices per split and tile counts (tiles_m counts
// 256-row pair tiles; n_tiles = tiles_m * tiles_n * splits).
struct Tc2Shape {
  int M, N, kps, nkb, tiles_m, tiles_n, n_tiles;
};

constexpr int kTc2Max = 4;
// A group's explicit schedule holds at most this many pairs and items.
constexpr int kTc2SchedPairs = 128;
constexpr int kTc2SchedItems = 512;
// Kernel parameter block of a group: tensor maps (A, B, output) and shape of
// each product, the epilogues, the number of products, and optionally the
// items of each pair: pair p takes items list[start[p] .. start[p+1]) of the
// combined numbering, in that order (npairs_sched == 0: round-robin).
template <class Op0, class Op1>
struct Tc2Params {
  CUtensorMap map[kTc2Max][3];
  Tc2Shape shape[kTc2Max];
  typename Op0::Epi epi0;
  typename Op1::Epi epi1[kTc2Max - 1];
  int count;
  int npairs_sched;
  uint16_t start[kTc2SchedPairs + 1];
  uint16_t list[kTc2SchedItems];
};

// TMA producer, one tile (both CTAs): this CTA's rows of A and half of B.
template <class Op, class Cfg, int BN, int STAGES>
__device__ __forceinline__ bool tc2_produce(const CUtensorMap* mA, const CUtensorMap* mB,
                                            const Tc2Shape& s, int tile, uint32_t rank,
                                            uint8_t* smem, uint64_t* full, uint64_t* empty,
                                            int& it, unsigned* status) {
  int m_blk, n_blk, z;
  tile_mnz(tile, s.tiles_m, s.tiles_n, m_blk, n_blk, z);
  const int m0 = m_blk * 2 * kBM + (int)rank * kBM;
  const int n0 = n_blk * BN + (int)rank * (BN / 2);
  const int kb0 = z * s.kps;
  const int nk = min(s.nkb, kb0 + s.kps) - kb0;
  for (int i = 0; i < nk; ++i, ++it) {
    const int st = it % STAGES;
    if (it >= STAGES && !tc::mbar_wait(&empty[st], ((it / STAGES) - 1) & 1, status)) return false;
    uint8_t* sa = smem + st * Cfg::STAGE_BYTES;
    uint8_t* sb = sa + Cfg::A_BYTES;
    const uint32_t fb = tc::mapa(tc::smem_u32(&full[st]), 0);
    if (rank == 0) tc::mbar_arrive_expect_tx(&full[st], 2 * Cfg::STAGE_BYTES);
    const int k0 = (kb0 + i) * kBK;
    if (!Op::A_MN) {
      tc::tma_load_2d_pair(sa, mA, fb, k0, m0);
    } else {
      tc::tma_load_2d_pair(sa, mA, fb, m0, k0);
      tc::tma_load_2d_pair(sa + 8192, mA, fb, m0 + 64, k0);
    }
    if (!Op::B_MN) {
      tc::tma_load_2d_pair(sb, mB, fb, k0, n0);
    } else {
#pragma unroll
      for (int j = 0; j < BN / 128; ++j)
        tc::tma_load_2d_pair(sb + j * 8192, mB, fb, n0 + 64 * j, k0);
    }
  }
  return true;
}

// MMA issuer, one tile (even CTA): the j-th tile of this pair goes to
// accumulator j % ACC once both CTAs' epilogues have drained its last use.
template <class Op, class Cfg, int BN, int STAGES, int ACC>
__device__ __forceinline__ bool tc2_mma(const Tc2Shape& s, int tile, int j, uint32_t tmem,
                                        uint8_t* smem, uint64_t* full, uint64_t* empty,
                                        uint64_t* tfull, uint64_t* tempty, int& it,
                                        unsigned* status) {
  constexpr uint32_t idesc = tc::idesc_bf16(2 * kBM, BN, Op::A_MN ? 1 : 0, Op::B_MN ? 1 : 0);
  const int z = (tile / s.tiles_m) / s.tiles_n;
  const int kb0 = z * s.kps, nk = min(s.nkb, kb0 + s.kps) - kb0;
  const int acc = j % ACC, use = j / ACC;
  if (use > 0 && !tc::mbar_wait_cluster(&tempty[acc], (use - 1) & 1, status)) return false;
  tc::fence_after_sync();
  const uint32_t d = tmem + (uint32_t)(acc * BN);
  bool ok = true;
  for (int i = 0; i < nk; ++i, ++it) {
    const int st = it % STAGES;
    if (!tc::mbar_wait_cluster(&full[st], (it / STAGES) & 1, status)) {
      ok = false;
      break;
    }
    tc::fence_after_sync();
    const uint32_t sa = tc::smem_u32(smem + st * Cfg::STAGE_BYTES);
    const uint32_t sb = sa + Cfg::A_BYTES;
#pragma unroll
    for (int kk = 0; kk < kBK / 16; ++kk) {
      const uint64_t ad = Op::A_MN ? tc::sdesc(sa + kk * 2048, 8192, 1024)
                                   : tc::sdesc(sa + kk * 32, 16, 1024);
      const uint64_t bd = Op::B_MN ? tc::sdesc(sb + kk * 2048, 8192, 1024)
                                   : tc::sdesc(sb + kk * 32, 16, 1024);
      tc::mma_bf16_pair(d, ad, bd, idesc, (i | kk) != 0 ? 1u : 0u);
    }
    tc::mma_commit_pair(&empty[st]);
  }
  tc::mma_commit_pair(&tfull[acc]);
  return ok;
}

// Epilogue, one tile (warps 2..9 of both CTAs): this CTA's 128 accumulator
// rows, warp w reading TMEM lane quarter w % 4 and half of the columns.
template <class Op, int BN, int ACC>
__device__ __forceinline__ bool tc2_epilogue(const typename Op::Epi& epi, const CUtensorMap* mC,
                                             const Tc2Shape& s, int tile, int j, uint32_t rank,
                                             int warp, int lane, uint32_t tmem, uint64_t* tfull,
                                             uint32_t te0, uint8_t* sbuf, int& nout,
                                             unsigned* status) {
  using Epi = typename Op::Epi;
  const int q = warp & 3;
  const int c_beg = ((warp - 2) >> 2) * (BN / 2);
  int m_blk, n_blk, z;
  tile_mnz(tile, s.tiles_m, s.tiles_n, m_blk, n_blk, z);
  const int acc = j % ACC, use = j / ACC;
  const int row0 = m_blk * 2 * kBM + (int)rank * kBM + q * 32;
  const int row = row0 + lane;
  const int n0 = n_blk * BN;
  const bool row_ok = row < s.M;
  constexpr int NCH = BN / 64;
  typename Epi::Pre pre[2];
  if (row_ok && n0 + c_beg < s.N) epi.load(row, n0 + c_beg, pre[0]);
  const bool ok = tc::mbar_wait(&tfull[acc], use & 1, status);
  tc::fence_after_sync();
  const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll
  for (int ci = 0; ci < NCH; ++ci) {
    const int c = c_beg + ci * 32;
    if (ci + 1 < NCH && row_ok && n0 + c + 32 < s.N) epi.load(row, n0 + c + 32, pre[(ci + 1) & 1]);
    float v[32];
    tc::tmem_ld32(base + (uint32_t)c, v);
    if (n0 + c < s.N)
      epi_chunk(epi, mC, sbuf, nout, lane, row, row0, n0 + c, n0 + c, z, v, pre[ci & 1],
                ok && row_ok, ok);
  }
  tc::fence_before_sync();
  __syncwarp();
  if (lane == 0) tc::mbar_arrive_cluster(te0 + (uint32_t)(acc * 8));
  return ok;
}

template <int BN, int STAGES, int ACC, class Op0, class Op1>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ Tc2Params<Op0, Op1> P, unsigned* status) {
  using Cfg = Tc2Cfg<BN, STAGES, ACC>;
  constexpr bool kSame = std::is_same<Op0, Op1>::value;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Cfg::BAR_OFF);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;   // accumulator ready for the epilogue
  uint64_t* tempty = tfull + ACC;     // accumulator drained by both CTAs' epilogues
  uint32_t* tslot = reinterpret_cast<uint32_t*>(tempty + ACC);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = tc::cluster_rank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  int total = 0;
  for (int q = 0; q < P.count; ++q) total += P.shape[q].n_tiles;
  // this pair's items: its list of the schedule, or every npairs-th item
  const int nmine = P.npairs_sched ? (int)P.start[pair + 1] - (int)P.start[pair]
                                   : (pair < total ? (total - 1 - pair) / npairs + 1 : 0);
  auto item_at = [&](int r) {
    return P.npairs_sched ? (int)P.list[P.start[pair] + r] : pair + r * npairs;
  };
  // product of a combined item index; *tile becomes the tile within it
  auto which = [&](int item, int* tile) {
    int q = 0;
    while (q + 1 < P.count && item >= P.shape[q].n_tiles) item -= P.shape[q++].n_tiles;
    *tile = item;
    return q;
  };

  if (warp == 0 && lane == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < ACC; ++a) {
      tc::mbar_init(&tfull[a], 1);
      tc::mbar_init(&tempty[a], 16);  // 8 epilogue warps in each CTA
    }
    tc::fence_mbar_init();
    for (int q = 0; q < P.count; ++q) {
      tc::prefetch_tmap(&P.map[q][0]);
      tc::prefetch_tmap(&P.map[q][1]);
    }
  }
  if (warp == 1) {
    tc::tmem_alloc_pair(tslot, Cfg::TMEM_COLS);
    tc::tmem_relinquish_pair();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::cluster_sync();  // both CTAs' barriers exist before any cross-CTA arrive
  tc::fence_after_sync();
  const uint32_t tmem = *tslot;
  pdl_enter();

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      for (int r = 0; r < nmine; ++r) {
        int tile;
        const int q = which(item_at(r), &tile);
        bool ok;
        if (kSame || q > 0)
          ok = tc2_produce<Op1, Cfg, BN, STAGES>(&P.map[q][0], &P.map[q][1], P.shape[q], tile, rank,
                                                 smem, full, empty, it, status);
        else
          ok = tc2_produce<Op0, Cfg, BN, STAGES>(&P.map[q][0], &P.map[q][1], P.shape[q], tile, rank,
                                                 smem, full, empty, it, status);
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      int it = 0;
      for (int j = 0; j < nmine; ++j) {
        int tile;
        const int q = which(item_at(j), &tile);
        bool ok;
        if (kSame || q > 0)
          ok = tc2_mma<Op1, Cfg, BN, STAGES, ACC>(P.shape[q], tile, j, tmem, smem, full, empty,
                                                  tfull, tempty, it, status);
        else
          ok = tc2_mma<Op0, Cfg, BN, STAGES, ACC>(P.shape[q], tile, j, tmem, smem, full, empty,
                                                  tfull, tempty, it, status);
        if (!ok) break;
      }
    }
  } else {
    const uint32_t te0 = tc::mapa(tc::smem_u32(&tempty[0]), 0);
    uint8_t* sbuf = smem + Cfg::OUT_OFF + (warp - 2) * kOutStage;
    int nout = 0, prev = -1;
    for (int j = 0; j < nmine; ++j) {
      int tile;
      const int q = which(item_at(j), &tile);
      bool ok;
      if constexpr (kSame) {
        ok = tc2_epilogue<Op1, BN, ACC>(q == 0 ? P.epi0 : P.epi1[q - 1], &P.map[q][2], P.shape[q],
                                        tile, j, rank, warp, lane, tmem, tfull, te0, sbuf, nout,
                                        status);
      } else {
        // the ops stage chunks of different sizes in the same buffer: the
        // first tile after a change of op waits until the other op's staged
        // chunks are read
        if (prev >= 0 && (q > 0) != (prev > 0) && lane == 0) tc::tma_store_wait_read<0>();
        ok = q > 0 ? tc2_epilogue<Op1, BN, ACC>(P.epi1[q - 1], &P.map[q][2], P.shape[q], tile, j,
                                                rank, warp, lane, tmem, tfull, te0, sbuf, nout,
                                                status)
                   : tc2_epilogue<Op0, BN, ACC>(P.epi0, &P.map[q][2], P.shape[q], tile, j, rank,
                                                warp, lane, tmem, tfull, te0, sbuf, nout, status);
      }
      prev = q;
      if (!ok) break;
    }
    if (lane == 0) tc::tma_store_wait_read<0>();  // staging read; the writes finish with the grid
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::cluster_sync();  // the peer no longer reads this CTA's shared memory or TMEM
  tc::fence_after_sync();
  if (warp == 1) tc::tmem_dealloc_pair(tmem, Cfg::TMEM_COLS);
}

// Operand tensor maps of one pair-kernel product (A: 128 x 64 boxes K-major,
// or two 64 x 64 boxes MN-major; B: BN/2 x 64 K-major or 64 x 64 MN-major).
template <int BN, bool A_MN, bool B_MN>
static bool tc2_operand_maps(CUtensorMap* mA, CUtensorMap* mB, int M, int N, int K, const void* A,
                             long sam, long sak, const void* B, long sbk, long sbn) {
  if (!A_MN) {
    uint64_t d[2] = {(uint64_t)K, (uint64_t)M}, st[1] = {(uint64_t)sam * 2};
    uint32_t box[2] = {64, 128};
    if (!make_tmap_bf16(mA, A, 2, d, st, box)) return false;
  } else {
    uint64_t d[2] = {(uint64_t)M, (uint64_t)K}, st[1] = {(uint64_t)sak * 2};
    uint32_t box[2] = {64, 64};
    if (!make_tmap_bf16(mA, A, 2, d, st, box)) return false;
  }
  if (!B_MN) {
    uint64_t d[2] = {(uint64_t)K, (uint64_t)N}, st[1] = {(uint64_t)sbn * 2};
    uint32_t box[2] = {64, (uint32_t)(BN / 2)};
    if (!make_tmap_bf16(mB, B, 2, d, st, box)) return false;
  } else {
    uint64_t d[2] = {(uint64_t)N, (uint64_t)K}, st[1] = {(uint64_t)sbk * 2};
    uint32_t box[2] = {64, 64};
    if (!make_tmap_bf16(mB, B, 2, d, st, box)) return false;
  }
  return true;
}

template <int BN>
static Tc2Shape tc2_shape(int M, int N, int K, int splits) {
  Tc2Shape s;
  s.M = M;
  s.N = N;
  s.nkb = (K + kBK - 1) / kBK;
  s.kps = (s.nkb + splits - 1) / splits;
  s.tiles_m = (M + 2 * kBM - 1) / (2 * kBM);
  s.tiles_n = (N + BN - 1) / BN;
  s.n_tiles = s.tiles_m * s.tiles_n * splits;
  return s;
}

template <int BN, int STAGES, int ACC, class Op0, class Op1>
static cudaError_t tc2_run(const Launch& lc, const Tc2Params<Op0, Op1>& P) {
  using Cfg = Tc2Cfg<BN, STAGES, ACC>;
  auto kern = gemm_tc2_kernel<BN, STAGES, ACC, Op0, Op1>;
  static std::atomic<unsigned long long> opted{0};
  if (cudaError_t e = smem_opt_in(kern, Cfg::SMEM, &opted); e != cudaSuccess) return e;
  int total = 0;
  for (int q = 0; q < P.count; ++q) total += P.shape[q].n_tiles;
  const int pairs =
      P.npairs_sched ? P.npairs_sched : (total < sm_count() / 2 ? total : sm_count() / 2);
  cudaError_t e = launch_k_cluster(kern, dim3(2 * pairs), dim3(kGemmThreads), Cfg::SMEM, lc.stream,
                                   2, P, lc.status);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int BN, int STAGES, int ACC, bool A_MN, bool B_MN, class Epi>
static cudaError_t tc2_launch(const Launch& lc, int M, int N, int K, const void* A, long sam,
                              long sak, const void* B, long sbk, long sbn, const Epi& epi,
                              int splits) {
  using Op = Tc2Op<A_MN, B_MN, Epi>;
  Tc2Params<Op, Op> P;
  memset(&P, 0, sizeof(P));
  if (!tc2_operand_maps<BN, A_MN, B_MN>(&P.map[0][0], &P.map[0][1], M, N, K, A, sam, sak, B, sbk,
                                        sbn))
    return cudaErrorInvalidValue;
  P.shape[0] = tc2_shape<BN>(M, N, K, splits);
  if (!out_map(&P.map[0][2], epi, M, N, splits)) return cudaErrorInvalidValue;
  P.epi0 = epi;
  P.count = 1;
  return tc2_run<BN, STAGES, ACC, Op, Op>(lc, P);
}

// Test path: the CTA-pair kernel with 256 x 256 tiles (plain and split-K stores).
cudaError_t gemm_tc_pair(const Launch& lc, int dtype_out, int M, int N, int K, const void* A,
                         long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                         const EpiArgs& ea, int splits) {
  if (N % 256 != 0 || M < 1 || K < 1) return cudaErrorInvalidValue;
  splits = (epi == EPI_PARTIAL) ? effective_splits(K, splits) : 1;
  const bool a_k = (sak == 1), b_k = (sbk == 1);
  constexpr int ST = 6, ACC = 2;
  auto go = [&](auto am, auto bm) -> cudaError_t {
    constexpr bool AM = decltype(am)::value, BM = decltype(bm)::value;
    if (epi == EPI_PARTIAL)
      return tc2_launch<256, ST, ACC, AM, BM>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                              EpiStoreF<float>{(float*)ea.out, ea.ldo, ea.split_stride},
                                              splits);
    if (dtype_out == 0)
      return tc2_launch<256, ST, ACC, AM, BM>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                              EpiStoreF<float>{(float*)ea.out, ea.ldo, 0}, 1);
    return tc2_launch<256, ST, ACC, AM, BM>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                            EpiStoreF<bf16>{(bf16*)ea.out, ea.ldo, 0}, 1);
  };
  using F = std::false_type;
  using T = std::true_type;
  // B_MN: B is N-contiguous (not K-major)
  if (a_k && !b_k) return go(F{}, T{});
  if (a_k && b_k) return go(F{}, F{});
  if (!a_k && !b_k) return go(T{}, T{});
  return go(T{}, F{});
}

bool tc2_group_schedule(const Tc2Shape* shape, int count, int max_pairs,
                        std::vector<std::vector<int>>* lists, long* makespan);

cudaError_t gemm_tc_pair_group(const Launch& lc, const PairProduct& p0, const PairProduct* w,
                               int nw) {
  if (nw < 1 || nw > kTc2Max - 1) return cudaErrorInvalidValue;
  auto valid = [](const PairProduct& q) { return q.N % 256 == 0 && q.M >= 1 && q.K >= 1; };
  if (!valid(p0) || p0.sak != 1 || p0.sbk != 1) return valid(p0) ? cudaErrorNotSupported
                                                                   : cudaErrorInvalidValue;
  for (int i = 0; i < nw; ++i) {
    if (!valid(w[i])) return cudaErrorInvalidValue;
    if (w[i].sam != 1 || w[i].sbn != 1) return cudaErrorNotSupported;
  }
  constexpr int ST = 6, ACC = 2;
  using Op0 = Tc2Op<false, false, EpiStoreF<bf16>>;
  using Op1 = Tc2Op<true, true, EpiStoreF<float>>;
  Tc2Params<Op0, Op1> P;
  memset(&P, 0, sizeof(P));
  P.epi0 = EpiStoreF<bf16>{(bf16*)p0.out, p0.ldo, 0};
  if (!tc2_operand_maps<256, false, false>(&P.map[0][0], &P.map[0][1], p0.M, p0.N, p0.K, p0.A,
                                           p0.sam, p0.sak, p0.B, p0.sbk, p0.sbn) ||
      !out_map(&P.map[0][2], P.epi0, p0.M, p0.N, 1))
    return cudaErrorInvalidValue;
  P.shape[0] = tc2_shape<256>(p0.M, p0.N, p0.K, 1);
  // the weight gradients: fp32 K-split partials, A and B MN-major
  for (int i = 0; i < nw; ++i) {
    const PairProduct& q = w[i];
    const int sp = effective_splits(q.K, q.splits);
    P.epi1[i] = EpiStoreF<float>{(float*)q.out, q.ldo, q.split_stride};
    P.shape[i + 1] = tc2_shape<256>(q.M, q.N, q.K, sp);
    if (!tc2_operand_maps<256, true, true>(&P.map[i + 1][0], &P.map[i + 1][1], q.M, q.N, q.K, q.A,
                                           q.sam, q.sak, q.B, q.sbk, q.sbn) ||
        !out_map(&P.map[i + 1][2], P.epi1[i], q.M, q.N, sp))
      return cudaErrorInvalidValue;
  }
  P.count = 1 + nw;
  // the pairs' item lists, longest first onto the least loaded pair
  std::vector<std::vector<int>> lists;
  if (tc2_group_schedule(P.shape, P.count, sm_count() / 2, &lists, nullptr)) {
    P.npairs_sched = (int)lists.size();
    int k = 0;
    for (int p = 0; p < P.npairs_sched; ++p) {
      P.start[p] = (uint16_t)k;
      for (int item : lists[p]) P.list[k++] = (uint16_t)item;
    }
    P.start[P.npairs_sched] = (uint16_t)k;
  }
  return tc2_run<256, ST, ACC, Op0, Op1>(lc, P);
}

// Two bf16 products with A K-major, B MN-major and plain bf16 stores in one
// CTA-pair launch (256 x 256 tiles, both N multiples of 256): product 0
// out[M, N] = A B, then p1; the items are scheduled longest first onto the
// least loaded pair (equal lengths: an even deal).
cudaError_t gemm_tc_pair_two(const Launch& lc, int M, int N, int K, const void* A, long sam,
                             long sak, const void* B, long sbk, long sbn, void* out, long ldo,
                             const GemmProd& p1) {
  if (!gemm_tc_available()) return cudaErrorNotSupported;
  if (N % 256 != 0 || p1.N % 256 != 0 || sak != 1 || sbn != 1 || p1.sak != 1 || p1.sbn != 1)
    return cudaErrorNotSupported;
  if (M < 1 || K < 1 || p1.M < 1 || p1.K < 1) return cudaErrorInvalidValue;
  constexpr int ST = 6, ACC = 2;
  using Op = Tc2Op<false, true, EpiStoreF<bf16>>;
  Tc2Params<Op, Op> P;
  memset(&P, 0, sizeof(P));
  P.epi0 = EpiStoreF<bf16>{(bf16*)out, ldo, 0};
  P.epi1[0] = EpiStoreF<bf16>{(bf16*)p1.out, p1.ldo, 0};
  if (!tc2_operand_maps<256, false, true>(&P.map[0][0], &P.map[0][1], M, N, K, A, sam, sak, B,
                                          sbk, sbn) ||
      !out_map(&P.map[0][2], P.epi0, M, N, 1) ||
      !tc2_operand_maps<256, false, true>(&P.map[1][0], &P.map[1][1], p1.M, p1.N, p1.K, p1.A,
                                          p1.sam, p1.sak, p1.B, p1.sbk, p1.sbn) ||
      !out_map(&P.map[1][2], P.epi1[0], p1.M, p1.N, 1))
    return cudaErrorInvalidValue;
  P.shape[0] = tc2_shape<256>(M, N, K, 1);
  P.shape[1] = tc2_shape<256>(p1.M, p1.N, p1.K, 1);
  P.count = 2;
  std::vector<std::vector<int>> lists;
  if (tc2_group_schedule(P.shape, P.count, sm_count() / 2, &lists, nullptr)) {
    P.npairs_sched = (int)lists.size();
    int k = 0;
    for (int q = 0; q < P.npairs_sched; ++q) {
      P.start[q] = (uint16_t)k;
      for (int item : lists[q]) P.list[k++] = (uint16_t)item;
    }
    P.start[P.npairs_sched] = (uint16_t)k;
  }
  return tc2_run<256, ST, ACC, Op, Op>(lc, P);
}

// Cost of one item of a CTA-pair product in 64-deep K slices of a 256 x 256
// tile, plus kTc2ItemOverhead for its share of pipeline fill and epilogue.
constexpr int kTc2ItemOverhead = 4;
static int tc2_item_cost(const Tc2Shape& s, int tile) {
  const int z = tile / (s.tiles_m * s.tiles_n);
  const int kb0 = z * s.kps;
  return std::min(s.nkb, kb0 + s.kps) - kb0 + kTc2ItemOverhead;
}

// Longest processing time first: the group's items, by decreasing cost (ties
// by item number), each onto the pair with the least load so far (ties to the
// lower pair); every pair's list is then put in item order, so the products
// follow each other in order within a pair.  Returns false when the group
// has more items or pairs than a schedule holds (round-robin then); fills
// *lists (one list per pair that has items) and *makespan (the largest
// pair load) when non-null.
bool tc2_group_schedule(const Tc2Shape* shape, int count, int max_pairs,
                        std::vector<std::vector<int>>* lists, long* makespan) {
  std::vector<std::pair<int, int>> items;  // (cost, item)
  int item = 0;
  for (int q = 0; q < count; ++q)
    for (int t = 0; t < shape[q].n_tiles; ++t, ++item)
      items.push_back({tc2_item_cost(shape[q], t), item});
  const int total = item;
  const int pairs = std::min(total, max_pairs);
  if (total > kTc2SchedItems || pairs > kTc2SchedPairs || pairs < 1) return false;
  std::stable_sort(items.begin(), items.end(),
                   [](const std::pair<int, int>& a, const std::pair<int, int>& b) {
                     return a.first > b.first;
                   });
  std::vector<long> load((size_t)pairs, 0);
  std::vector<std::vector<int>> out((size_t)pairs);
  for (const auto& it : items) {
    const size_t p = (size_t)(std::min_element(load.begin(), load.end()) - load.begin());
    load[p] += it.first;
    out[p].push_back(it.second);
  }
  for (auto& l : out) std::sort(l.begin(), l.end());
  if (makespan) *makespan = *std::max_element(load.begin(), load.end());
  if (lists) *lists = std::move(out);
  return true;
}

long tc2_group_makespan(int M0, int N0, int K0, const int* Mw, const int* Nw, const int* Kw,
                        const int* splits, int nw, int max_pairs) {
  Tc2Shape sh[kTc2Max];
  if (nw < 0 || nw > kTc2Max - 1) return -1;
  sh[0] = tc2_shape<256>(M0, N0, K0, 1);
  for (int i = 0; i < nw; ++i)
    sh[i + 1] = tc2_shape<256>(Mw[i], Nw[i], Kw[i], effective_splits(Kw[i], splits[i]));
  long ms = -1;
  if (tc2_group_schedule(sh, nw + 1, max_pairs, nullptr, &ms)) return ms;
  // too many items for a schedule: the launch deals them round-robin
  int total = 0;
  for (int q = 0; q <= nw; ++q) total += sh[q].n_tiles;
  const int pairs = std::max(1, std::min(total, max_pairs));
  std::vector<long> load((size_t)pairs, 0);
  int item = 0;
  for (int q = 0; q <= nw; ++q)
    for (int t = 0; t < sh[q].n_tiles; ++t, ++item) load[(size_t)(item % pairs)] += tc2_item_cost(sh[q], t);
  return *std::max_element(load.begin(), load.end());
}

// Output tile widths: 128 x 256 tiles move 48 KB per 64-deep K slice for
// 4.2 MFLOP (87 FLOP per L2 byte), 128 x 128 tiles 32 KB for 2.1 MFLOP (64).
// The wide tile is used when it still gives most SMs a tile; 128 x 64 tiles
// (an 8-deep ring) when even 128-wide tiles would leave most SMs idle.
template <int BN, bool A_MN, bool B_MN>
static cudaError_t tc_epi(const Launch& lc, int dtype_out, int M, int N, int K, const void* A,
                          long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                          const EpiArgs& ea, int splits) {
  constexpr int ST = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
  switch (epi) {
    case EPI_STORE:
      if (dtype_out == 0)
        return tc_launch<BN, ST, A_MN, B_MN>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                             EpiStoreF<float>{(float*)ea.out, ea.ldo, 0}, 1);
      return tc_launch<BN, ST, A_MN, B_MN>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                           EpiStoreF<bf16>{(bf16*)ea.out, ea.ldo, 0}, 1);
    case EPI_PARTIAL:
      return tc_launch<BN, ST, A_MN, B_MN>(
          lc, M, N, K, A, sam, sak, B, sbk, sbn,
          EpiStoreF<float>{(float*)ea.out, ea.ldo, ea.split_stride}, splits);
    default:
      break;
  }
  // fused epilogues, instantiated only for the operand layouts the layer uses
  if constexpr (!A_MN && B_MN) {
    switch (epi) {
      case EPI_GATE:
        return tc_launch<BN, ST, A_MN, B_MN>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                             EpiGateF<bf16>{(bf16*)ea.out, ea.ldo}, 1,
                                             ea.max_ctas);
      case EPI_STORE_SCORE:
        return tc_launch<BN, ST, A_MN, B_MN>(lc, M, N, K, A, sam, sak, B, sbk, sbn,
                                             EpiStoreScoreF<bf16>{(bf16*)ea.out, ea.ldo,
                                                                  (const bf16*)ea.w_p, ea.spart, M},
                                             1);
      case EPI_HGATE:
        return tc_launch<BN, ST, A_MN, B_MN>(
            lc, M, N, K, A, sam, sak, B, sbk, sbn,
            EpiHGateF<bf16>{(bf16*)ea.out, ea.ldo, (const bf16*)ea.w_p, ea.spart, M,
                            (bf16*)ea.out2, ea.ldo2, ea.n_split},
            1, 0, ea.b2);
      default:
        break;
    }
  }
  if constexpr (!A_MN && !B_MN) {
    if (epi == EPI_REVSCAN)
      return tc_launch<BN, ST, A_MN, B_MN>(
          lc, M, N, K, A, sam, sak, B, sbk, sbn,
          EpiRevScanT{(float*)ea.out, ea.ldo, ea.scan_zinv, ea.scan_decay, ea.scan_nb, N}, 1);
  }
  return cudaErrorNotSupported;
}

// Tile width forced by the test entry point (0: chosen per shape below).
int g_force_bn = 0;

template <bool A_MN, bool B_MN>
static cudaError_t tc_pick(const Launch& lc, int dtype_out, int M, int N, int K, const void* A,
                           long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                           const EpiArgs& ea, int splits) {
  if (g_force_bn == 64)
    return tc_epi<64, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  if (g_force_bn == 128)
    return tc_epi<128, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  if (g_force_bn == 256 && N % 256 == 0)
    return tc_epi<256, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  const long tm = (M + kBM - 1) / kBM;
  const long tiles256 = tm * ((N + 255) / 256) * splits;
  const long tiles128 = tm * ((N + 127) / 128) * splits;
  if (epi == EPI_HGATE) {  // the tile width must divide the first output's width
    if (N % 256 == 0 && ea.n_split % 256 == 0 && tiles256 * 4 >= (long)sm_count() * 3)
      return tc_epi<256, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, 1);
    if (ea.n_split % 128 == 0)
      return tc_epi<128, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, 1);
    return tc_epi<64, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, 1);
  }
  if (N % 256 == 0 && tiles256 * 4 >= (long)sm_count() * 3)
    return tc_epi<256, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea,
                                   splits);
  // few tiles (the memory stage's [B*Nb x D] products): narrow tiles spread the
  // operand traffic over more SMs
  if (tiles128 * 4 < (long)sm_count())
    return tc_epi<64, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea,
                                  splits);
  return tc_epi<128, A_MN, B_MN>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
}

// Long K or wide N: the CTA-pair kernel's 256 x 256 tiles need 2/3 of the
// operand bytes per flop of a single CTA's 128 x 256 tile (measured faster
// from K = 1024, or K = 768 with N >= 1024; no slower at K = 512).
static bool store_on_pair(int M, int N, int K) {
  return N % 256 == 0 && M >= 512 && (K >= 1024 || (K >= 768 && N >= 1024));
}

cudaError_t gemm_tc(const Launch& lc, int dtype_out, int M, int N, int K, const void* A, long sam,
                    long sak, const void* B, long sbk, long sbn, EpiKind epi, const EpiArgs& ea,
                    int splits) {
  if (M < 1 || K < 1) return cudaErrorInvalidValue;
  // the scan epilogue takes any column count (B*Nb); the others multiples of 64
  if (N % 64 != 0 && epi != EPI_REVSCAN) return cudaErrorInvalidValue;
  if (epi == EPI_REVSCAN && (ea.scan_nb < 1 || 32 % ea.scan_nb != 0)) return cudaErrorInvalidValue;
  if (epi == EPI_STORE && store_on_pair(M, N, K))
    return gemm_tc_pair(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, 1);
  splits = (epi == EPI_PARTIAL) ? effective_splits(K, splits) : 1;
  const bool a_k = (sak == 1), a_m = (sam == 1) && !a_k;
  const bool b_k = (sbk == 1), b_n = (sbn == 1) && !b_k;
  if (a_k && b_n) return tc_pick<false, true>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  if (a_k && b_k) return tc_pick<false, false>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  if (a_m && b_n) return tc_pick<true, true>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  if (a_m && b_k) return tc_pick<true, false>(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  return cudaErrorNotSupported;
}

cudaError_t gemm_tc_two(const Launch& lc, int M, int N, int K, const void* A, long sam, long sak,
                        const void* B, long sbk, long sbn, void* out, long ldo,
                        const GemmProd& p1) {
  if (!gemm_tc_available()) return cudaErrorNotSupported;
  if (N % 64 != 0 || M < 1 || K < 1 || p1.N % 64 != 0 || p1.M < 1 || p1.K < 1)
    return cudaErrorInvalidValue;
  // product 0 on the CTA-pair kernel, or other operand layouts: not here
  if (store_on_pair(M, N, K) || sak != 1 || sbn != 1 || p1.sak != 1 || p1.sbn != 1)
    return cudaErrorNotSupported;
  const EpiStoreF<bf16> epi{(bf16*)out, ldo, 0};
  const EpiStoreF<bf16> epi1{(bf16*)p1.out, p1.ldo, 0};
  const long tm = (M + kBM - 1) / kBM;
  // product 0 picks the tile width, as in tc_pick
  if (N % 256 == 0 && tm * (N / 256) * 4 >= (long)sm_count() * 3)
    return tc_launch<256, 4, false, true>(lc, M, N, K, A, sam, sak, B, sbk, sbn, epi, 1, 0,
                                          nullptr, &p1, epi1);
  if (tm * ((N + 127) / 128) * 4 < (long)sm_count())
    return tc_launch<64, 8, false, true>(lc, M, N, K, A, sam, sak, B, sbk, sbn, epi, 1, 0, nullptr,
                                         &p1, epi1);
  return tc_launch<128, 6, false, true>(lc, M, N, K, A, sam, sak, B, sbk, sbn, epi, 1, 0, nullptr,
                                        &p1, epi1);
}

cudaError_t gemm(const Launch& lc, int dtype, int dtype_out, int M, int N, int K, const void* A,
                 long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                 const EpiArgs& ea, int splits, const char** kernel_name) {
  if (dtype == 1 && gemm_tc_available()) {
    if (kernel_name) *kernel_name = "gemm_tc";
    cudaError_t e = gemm_tc(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
    if (e != cudaErrorNotSupported) return e;
  }
  if (kernel_name) *kernel_name = "gemm_simt";
  return gemm_simt(lc, dtype, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
}

// ============================================================ split reduction
// Up to kRedMax independent reductions (segments) in one launch: the first
// count_0 / 4 threads reduce segment 0, the next count_1 / 4 segment 1, ...
// Each thread sums its 4 elements over the splits in split order.
constexpr int kRedMax = 3;
template <class TO>
struct RedSegs {
  const float* part[kRedMax];
  TO* out[kRedMax];
  long count[kRedMax];
  int splits[kRedMax];
  int n;
};

template <class TO>
__global__ void reduce_splits_kernel(const __grid_constant__ RedSegs<TO> R) {
  pdl_enter();
  long i4 = ((long)blockIdx.x * blockDim.x + threadIdx.x) * 4;
  int q = 0;
  while (q < R.n && i4 >= R.count[q]) i4 -= R.count[q++];
  if (q >= R.n) return;
  const float* part = R.part[q];
  const long count = R.count[q];
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
  for (int s = 0; s < R.splits[q]; ++s) {
    float v[4];
    load4(part + (long)s * count + i4, v);
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[e] += v[e];
  }
  store4(R.out[q] + i4, acc);
}

template <class TO>
static cudaError_t reduce_typed(const Launch& lc, const SplitSum* segs, int n) {
  RedSegs<TO> R;
  memset(&R, 0, sizeof(R));
  long n4 = 0;
  for (int i = 0; i < n; ++i) {
    R.part[i] = segs[i].part;
    R.out[i] = static_cast<TO*>(segs[i].out);
    R.count[i] = segs[i].count;
    R.splits[i] = segs[i].splits;
    n4 += segs[i].count / 4;
  }
  R.n = n;
  const int threads = 256;
  const unsigned blocks = (unsigned)((n4 + threads - 1) / threads);
  launch_k(reduce_splits_kernel<TO>, dim3(blocks), dim3(threads), 0, lc.stream, R);
  return cudaGetLastError();
}

cudaError_t reduce_splits_n(const Launch& lc, const SplitSum* segs, int n, int dtype_out) {
  if (n < 1 || n > kRedMax) return cudaErrorInvalidValue;
  for (int i = 0; i < n; ++i)
    if (segs[i].count % 4 != 0) return cudaErrorInvalidValue;
  return dtype_out == 0 ? reduce_typed<float>(lc, segs, n) : reduce_typed<bf16>(lc, segs, n);
}

cudaError_t reduce_splits(const Launch& lc, const float* part, int splits, long count,
                          int dtype_out, void* out) {
  const SplitSum seg{part, splits, count, out};
  return reduce_splits_n(lc, &seg, 1, dtype_out);
}

}  // namespace bcmt
