// Adaptive block summaries (Sec. 3.4), the normalised exponential causal
// memory (Sec. 3.5), and the backward of these two stages and of the gated
// injection (Sec. 3.8): the O(T D) and O(N_b D) work of the layer, on CUDA
// cores.  (The memory's D x D projections run on the tensor cores, gemm.cu.)
// Every kernel reads rows with 16-byte vector loads, issues a batch's loads
// before its first use, and reduces in a fixed order (deterministic).
#include <algorithm>
#include <atomic>

#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace bcmt {

namespace {
constexpr int kMaxL = 1024;
constexpr int kThreads = 256;
}  // namespace

// 16-byte global -> shared copies that hold no registers while in flight
// (cp.async, cached in L2 only); a thread waits for its own copies.
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   (uint32_t)__cvta_generic_to_shared(smem_dst)),
               "l"(gmem_src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

// ======================================================== work items (device)
// Four or eight consecutive values of a row, held as loaded: bf16 stays packed
// until it is used, so that a batch of rows' loads can be in flight with few
// registers.
template <class T> struct Raw4 { float4 v; };
template <> struct Raw4<bf16> { uint2 v; };
__device__ __forceinline__ void ld_raw(const float* p, Raw4<float>& r) {
  r.v = *reinterpret_cast<const float4*>(p);
}
__device__ __forceinline__ void ld_raw(const bf16* p, Raw4<bf16>& r) {
  r.v = *reinterpret_cast<const uint2*>(p);
}
__device__ __forceinline__ void unraw(const Raw4<float>& r, float* v) {
  v[0] = r.v.x; v[1] = r.v.y; v[2] = r.v.z; v[3] = r.v.w;
}
__device__ __forceinline__ void unraw(const Raw4<bf16>& r, float* v) {
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.v.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.v.y));
  v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
}
template <class T> struct Raw8 { float4 lo, hi; };
template <> struct Raw8<bf16> { uint4 v; };
__device__ __forceinline__ void ld_raw(const float* p, Raw8<float>& r) {
  r.lo = *reinterpret_cast<const float4*>(p);
  r.hi = *reinterpret_cast<const float4*>(p + 4);
}
__device__ __forceinline__ void ld_raw(const bf16* p, Raw8<bf16>& r) {
  r.v = *reinterpret_cast<const uint4*>(p);
}
__device__ __forceinline__ void unraw(const Raw8<float>& r, float* v) {
  v[0] = r.lo.x; v[1] = r.lo.y; v[2] = r.lo.z; v[3] = r.lo.w;
  v[4] = r.hi.x; v[5] = r.hi.y; v[6] = r.hi.z; v[7] = r.hi.w;
}
__device__ __forceinline__ void unraw(const Raw8<bf16>& r, float* v) { unpack8(r.v, v); }

// The memory projection P = M W_m arrives as PS K-split fp32 partials,
// partial z of row r at Pm + z * pstride + r * D.  Sec. 3.5's shift makes the
// memory row of block i of batch b C_i = P_{i-1} (row b*Nb + i - 1) and
// C_0 = 0; N consecutive channels from c, all partials loaded first, then
// summed in split order.
template <int N, int PS>
__device__ __forceinline__ void mem_row(const float* __restrict__ Pm, long pstride, int b, int i,
                                        int Nb, int D, int c, float* v) {
#pragma unroll
  for (int e = 0; e < N; ++e) v[e] = 0.f;
  if (i == 0) return;
  const float* p = Pm + ((long)b * Nb + i - 1) * D + c;
  float4 q[PS][N / 4];
#pragma unroll
  for (int z = 0; z < PS; ++z)
#pragma unroll
    for (int e = 0; e < N / 4; ++e) q[z][e] = *reinterpret_cast<const float4*>(p + z * pstride + 4 * e);
#pragma unroll
  for (int z = 0; z < PS; ++z)
#pragma unroll
    for (int e = 0; e < N / 4; ++e) {
      v[4 * e] += q[z][e].x;
      v[4 * e + 1] += q[z][e].y;
      v[4 * e + 2] += q[z][e].z;
      v[4 * e + 3] += q[z][e].w;
    }
}

// Host: runs f(std::integral_constant<int, PS>) for the split count of the
// memory projections (1 to 4).
template <class F>
cudaError_t with_splits(int psplits, F&& f) {
  switch (psplits) {
    case 1: return f(std::integral_constant<int, 1>());
    case 2: return f(std::integral_constant<int, 2>());
    case 3: return f(std::integral_constant<int, 3>());
    case 4: return f(std::integral_constant<int, 4>());
    default: return cudaErrorInvalidValue;
  }
}

// Sec. 3.4 for block i of batch b, channels 256 z .. 256 z + 255: the pooling
// scores s = H w_p summed from the npart partial dot products the W_O epilogue
// wrote, alpha = softmax(s) over the block's tokens (stored by z == 0), and
// S_i = sum_t alpha_t H_t.  The first 64 rows' H loads are issued before the
// scores are known, so the block's H and score reads share one memory round
// trip.  Returns S_i[256 z + threadIdx.x] (0 past D).
template <class T>
__device__ float pool_block(float* sm, const T* __restrict__ Hm, const float* __restrict__ spart,
                            int npart, long n_tok, float* __restrict__ alpha, int Tlen, int D,
                            int L, int i, int b, int z) {
  float* sc = sm;                 // [kMaxL]
  float* red = sm + kMaxL;        // [2]
  float* part = sm + kMaxL + 4;   // [8][260]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const long row0 = (long)b * Tlen + t0;
  // 8 row groups (warps) x 32 threads of 8 channels
  const int c = z * 256 + lane * 8;
  const bool cin = c < D;
  const T* Hc = Hm + row0 * D + c;
  Raw8<T> h0[8];
#pragma unroll
  for (int u = 0; u < 8; ++u)
    if (cin && warp + 8 * u < n) ld_raw(Hc + (long)(warp + 8 * u) * D, h0[u]);
  for (int r = threadIdx.x; r < n; r += kThreads) {
    float s = 0.f;
#pragma unroll 16
    for (int j = 0; j < npart; ++j) s += spart[(long)j * n_tok + row0 + r];
    sc[r] = s;
  }
  __syncthreads();
  if (warp == 0) {
    float mx = -INFINITY;
    for (int r = lane; r < n; r += 32) mx = fmaxf(mx, sc[r]);
    mx = warp_max(mx);
    float sum = 0.f;
    for (int r = lane; r < n; r += 32) sum += expf(sc[r] - mx);
    sum = warp_sum(sum);
    if (lane == 0) {
      red[0] = mx;
      red[1] = 1.0f / sum;
    }
  }
  __syncthreads();
  const float mx = red[0], inv = red[1];
  for (int r = threadIdx.x; r < n; r += kThreads) {
    const float a = expf(sc[r] - mx) * inv;
    if (z == 0) alpha[row0 + r] = a;
    sc[r] = a;
  }
  __syncthreads();
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (cin) {
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (warp + 8 * u < n) {
        float h[8];
        unraw(h0[u], h);
        const float a = sc[warp + 8 * u];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = fmaf(a, h[e], acc[e]);
      }
    // blocks longer than 64 tokens: further batches of 64 rows, loads first
    for (int r0 = 64; r0 < n; r0 += 64) {
      Raw8<T> hb[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (r0 + warp + 8 * u < n) ld_raw(Hc + (long)(r0 + warp + 8 * u) * D, hb[u]);
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (r0 + warp + 8 * u < n) {
          float h[8];
          unraw(hb[u], h);
          const float a = sc[r0 + warp + 8 * u];
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[e] = fmaf(a, h[e], acc[e]);
        }
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) part[warp * 260 + lane * 8 + e] = acc[e];
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int g = 0; g < 8; ++g) t += part[g * 260 + threadIdx.x];
  return t;
}

// Sec. 3.8 reversed: item (x, i, b): kGateCh channels of block i of batch b
// (wide items: the whole backward gate fits in one wave of two CTAs per SM).
// For the block's tokens dU = dY * C_i * G * (1 - G) (through G = sigmoid(U)),
// and dC_i = sum_t dY_t * G_t (through Y = H + G * C_i) becomes dP[b, i-1]
// (C_i = P_{i-1}); block 0 writes the zero row dP[b, Nb-1].
constexpr int kGateCh = 256;
template <class T, int PS>
__device__ void gate_bwd_item(float* sm, const T* __restrict__ dY, const T* __restrict__ G,
                              const float* __restrict__ Pm, long pstride,
                              T* __restrict__ dU, float* dP, bf16* dPb, int Tlen, int D, int L,
                              int Nb, int x, int i, int b) {
  float* part = sm;                      // [8][kGateCh + 4]
  float* crow = sm + 8 * (kGateCh + 4);  // [kGateCh]: the block's memory row C_i
  const int rg = threadIdx.x >> 5, cq = threadIdx.x & 31;
  const int c = x * kGateCh + cq * 8;
  const bool cin = c < D;
  const int t0 = i * L, n = min(L, Tlen - t0);
  // rows rg, rg+8, ... in batches of RB (64 rows of the block in bf16, 32 in
  // fp32, whose rows take twice the registers; loads held packed): every
  // load of a batch is issued before its first store
  constexpr int RB = sizeof(T) == 2 ? 8 : 4;
  const long step = 8L * D;
  const long o0 = ((long)b * Tlen + t0 + rg) * D + c;
  const T* dyp = dY + o0;
  const T* gp = G + o0;
  T* dup = dU + o0;
  Raw8<T> rdy[RB], rgt[RB];
  // dY is an input of the call, complete before the layer's first kernel
  // started: its loads go out before the wait for the previous kernel (the
  // caller's pdl_enter is here)
#pragma unroll
  for (int u = 0; u < RB; ++u)
    if (cin && rg + 8 * u < n) ld_raw(dyp + u * step, rdy[u]);
  pdl_enter();
#pragma unroll
  for (int u = 0; u < RB; ++u)
    if (cin && rg + 8 * u < n) ld_raw(gp + u * step, rgt[u]);
  // meanwhile the memory row, one channel per thread, its K-split partials
  // summed in split order (C_0 = 0, C_i = P_{i-1})
  {
    const int cc = x * kGateCh + threadIdx.x;
    float v = 0.f;
    if (i > 0 && cc < D) {
      const float* p = Pm + ((long)b * Nb + i - 1) * D + cc;
      float q[PS];
#pragma unroll
      for (int z = 0; z < PS; ++z) q[z] = p[z * pstride];
#pragma unroll
      for (int z = 0; z < PS; ++z) v += q[z];
    }
    crow[threadIdx.x] = v;
  }
  __syncthreads();
  float acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = 0.f;
  if (cin) {
    float cm[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) cm[e] = crow[cq * 8 + e];
#pragma unroll 1
    for (int r0 = rg; r0 < n; r0 += 8 * RB, dyp += RB * step, gp += RB * step, dup += RB * step) {
      if (r0 != rg) {  // the block's next batch of rows
#pragma unroll
        for (int u = 0; u < RB; ++u)
          if (r0 + 8 * u < n) {
            ld_raw(dyp + u * step, rdy[u]);
            ld_raw(gp + u * step, rgt[u]);
          }
      }
#pragma unroll
      for (int u = 0; u < RB; ++u)
        if (r0 + 8 * u < n) {
          float dy[8], g[8], du[8];
          unraw(rdy[u], dy);
          unraw(rgt[u], g);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            du[e] = dy[e] * cm[e] * g[e] * (1.0f - g[e]);
            acc[e] = fmaf(dy[e], g[e], acc[e]);
          }
          store8(dup + u * step, du);
        }
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) part[rg * (kGateCh + 4) + cq * 8 + e] = acc[e];
  __syncthreads();
  if (threadIdx.x < kGateCh) {
    const int cc = x * kGateCh + threadIdx.x;
    if (cc < D) {
      float t = 0.f;
#pragma unroll
      for (int g = 0; g < 8; ++g) t += part[g * (kGateCh + 4) + threadIdx.x];
      const long o = (i > 0) ? ((long)b * Nb + i - 1) * D + cc : ((long)b * Nb + Nb - 1) * D + cc;
      dP[o] = (i > 0) ? t : 0.f;
      if (dPb) dPb[o] = __float2bfloat16_rn((i > 0) ? t : 0.f);
    }
  }
  __syncthreads();
}

// Sec. 3.5 reversed: item (x, b): channels 256x .. 256x+255.  With dM = dP W_m^T,
// the reverse decayed scan of M_i = N_i / Z_i,
//   R_i = dM_i / Z_i + a R_{i+1},  dS_i = R_i  (= sum_{i'>=i} a^(i'-i) dM_i' / Z_i').
// When da_part is non-null the same pass also differentiates the decay (the
// learned per-channel decay the paper names as future work, Sec. 5): with the
// adjoint of Z, Q_i = -dM_i M_i / Z_i + a Q_{i+1}, and N_{i-1} = M_{i-1} Z_{i-1},
//   d a = sum_{i>=1} (R_i N_{i-1} + Q_i Z_{i-1}) = sum_{i>=1} Z_{i-1} (R_i M_{i-1} + Q_i),
// written per batch row (da_part[b, c]) and summed over b by the caller.
template <int PS>
__device__ void scan_bwd_item(const float* dM, long mstride,
                              const float* __restrict__ decay, const float* __restrict__ Z,
                              const float* __restrict__ M, float* dS, float* __restrict__ da_part,
                              int Nb, int D, int x, int b) {
  const int c = x * blockDim.x + threadIdx.x;
  if (c >= D) return;
  const float a = decay[c];
  const long base = (long)b * Nb * D + c;
  float R = 0.f, Qz = 0.f, da = 0.f;
  constexpr int U = 16;
  for (int i1 = Nb; i1 > 0; i1 -= U) {
    float mv[U], zv[U], mi[U], mp[U], zp[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i1 - 1 - u;
      float dm[PS];  // dM from its K-split partials, loaded first, summed in split order
#pragma unroll
      for (int z = 0; z < PS; ++z) dm[z] = (i >= 0) ? __ldcg(dM + z * mstride + base + (long)i * D) : 0.f;
      mv[u] = 0.f;
#pragma unroll
      for (int z = 0; z < PS; ++z) mv[u] += dm[z];
      zv[u] = (i >= 0) ? Z[(long)i * D + c] : 1.f;
      if (da_part) {
        mi[u] = (i >= 0) ? M[base + (long)i * D] : 0.f;
        mp[u] = (i >= 1) ? M[base + (long)(i - 1) * D] : 0.f;
        zp[u] = (i >= 1) ? Z[(long)(i - 1) * D + c] : 0.f;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i1 - 1 - u;
      if (i >= 0) {
        const float g = mv[u] / zv[u];
        R = fmaf(a, R, g);
        dS[base + (long)i * D] = R;
        if (da_part) {
          Qz = fmaf(a, Qz, -g * mi[u]);
          da = fmaf(zp[u], fmaf(R, mp[u], Qz), da);
        }
      }
    }
  }
  if (da_part) da_part[(long)b * D + c] = da;
}

// Sec. 3.4 reversed: item (c, i, b), rows ROWS*c .. ROWS*c + ROWS-1 of block i of batch b.
// With S_i = sum_t alpha_t H_t and alpha = softmax(s): g_t = H_t . dS_i and
// ds_t = alpha_t (g_t - sum_u alpha_u g_u), where sum_u alpha_u g_u = S_i . dS_i
// (the forward's block summary), so every row chunk of a block is independent.
// The chunk's share of dW_p = sum_t ds_t H_t goes to dwp_part, and the same
// pass completes the gradient of H in place: dH_t += alpha_t dS_i + ds_t w_p
// (the pooling and score paths, added to dY + dU W_g^T already in dH).
// ROWS rows per item: 16, or 32 at narrow widths (D <= 256), where a 16-row
// item is too little work to cover its own latency.
template <class T, int ROWS>
__device__ void summary_bwd_item(float* sm, const T* __restrict__ Hm,
                                 const float* __restrict__ alpha, const float* __restrict__ Sb,
                                 const float* dS, const T* __restrict__ w_p,
                                 const T* __restrict__ dY, T* dH,
                                 float* __restrict__ ds_out, float* __restrict__ dwp_part,
                                 int Tlen, int D, int L, int Nb, int c, int i, int b) {
  float* g = sm;                  // [ROWS]
  float* red = sm + ROWS;         // [8]: per-warp partial sums of S_i . dS_i
  float* part = sm + ROWS + 8;    // [8][260]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int blen = min(L, Tlen - i * L);
  const int t0 = i * L + c * ROWS, n = min(ROWS, blen - c * ROWS);
  const T* Hb = Hm + ((long)b * Tlen + t0) * D;
  const float* dSi = dS + ((long)b * Nb + i) * D;
  const float* Si = Sb + ((long)b * Nb + i) * D;
  const float* ab = alpha + (long)b * Tlen + t0;
  // sum_u alpha_u g_u = S_i . dS_i
  float cp = 0.f;
  for (int k = threadIdx.x; k < D; k += kThreads) cp = fmaf(Si[k], __ldcg(dSi + k), cp);
  cp = warp_sum(cp);
  if (lane == 0) red[warp] = cp;
  // g_t = H_t . dS_i: warp w takes rows w, w+8; all the loads of a
  // 256-channel chunk for its rows go out together
  constexpr int RW = ROWS / 8;
  {
    float d[RW];
#pragma unroll
    for (int u = 0; u < RW; ++u) d[u] = 0.f;
#pragma unroll 2
    for (int k = lane * 8; k < D; k += 256) {
      float sv[8], h[RW][8];
      load8_cg(dSi + k, sv);
#pragma unroll
      for (int u = 0; u < RW; ++u)
        if (warp + 8 * u < n) load8(Hb + (long)(warp + 8 * u) * D + k, h[u]);
#pragma unroll
      for (int u = 0; u < RW; ++u)
        if (warp + 8 * u < n) {
#pragma unroll
          for (int e = 0; e < 8; ++e) d[u] = fmaf(h[u][e], sv[e], d[u]);
        }
    }
#pragma unroll
    for (int u = 0; u < RW; ++u) {
      const float t = warp_sum(d[u]);
      if (lane == 0 && warp + 8 * u < n) g[warp + 8 * u] = t;
    }
  }
  __syncthreads();
  float cd = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) cd += red[w];
  __syncthreads();  // everyone has read red before g is overwritten below
  if (threadIdx.x < n) {
    const int r = threadIdx.x;
    const float v = ab[r] * (g[r] - cd);
    ds_out[(long)b * Tlen + t0 + r] = v;
    g[r] = v;
  }
  __syncthreads();
  const int rg = warp, co = lane;
  T* dHb = dH + ((long)b * Tlen + t0) * D;
  const T* dYb = dY + ((long)b * Tlen + t0) * D;
  const long prow = ((long)b * Nb + i) * ((L + ROWS - 1) / ROWS) + c;
  for (int c0 = 0; c0 < D; c0 += 256) {
    const int k = c0 + co * 8;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (k < D) {
      float sv[8], wp[8];
      load8_cg(dSi + k, sv);
      load8(w_p + k, wp);
      // rows rg, rg+8: all their loads before the first store
      float h[RW][8], d[RW][8], yv[RW][8];
#pragma unroll
      for (int u = 0; u < RW; ++u)
        if (rg + 8 * u < n) {
          load8(Hb + (long)(rg + 8 * u) * D + k, h[u]);
          load8(dHb + (long)(rg + 8 * u) * D + k, d[u]);
          load8(dYb + (long)(rg + 8 * u) * D + k, yv[u]);
        }
#pragma unroll
      for (int u = 0; u < RW; ++u)
        if (rg + 8 * u < n) {
          const float w = g[rg + 8 * u], a = ab[rg + 8 * u];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            acc[e] = fmaf(w, h[u][e], acc[e]);
            d[u][e] += yv[u][e] + a * sv[e] + w * wp[e];
          }
          store8(dHb + (long)(rg + 8 * u) * D + k, d[u]);
        }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) part[rg * 260 + co * 8 + e] = acc[e];
    __syncthreads();
    const int cc = c0 + threadIdx.x;
    if (cc < D) {
      float t = 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q) t += part[q * 260 + threadIdx.x];
      dwp_part[prow * D + cc] = t;
    }
    __syncthreads();
  }
}

// The same pooling backward for bf16 at D <= 1024, item (c, i, b) = rows
// ROWS*c .. ROWS*c + ROWS-1 of block i of batch b with ROWS = 8*RW: warp w owns
// rows w, w+8, ..., lane l the channels 256 j + 8 l .. +7 (j < KC).  Every
// thread issues the loads of its rows of H and dH first; meanwhile the CTA
// stages dS_i and w_p in shared memory and forms S_i . dS_i.  The H rows stay
// in registers from the dot products g_t = H_t . dS_i to the update, so the
// item costs one memory round trip.  RW * KC <= 8 keeps the held rows within
// the registers of two CTAs per SM.
template <int RW, int KC>
__global__ void __launch_bounds__(kThreads, 2)
    summary_bwd_reg_kernel(const bf16* __restrict__ Hm, const float* __restrict__ alpha,
                           const float* __restrict__ Sb, const float* dS,
                           const bf16* __restrict__ w_p, const bf16* __restrict__ dY, bf16* dH,
                           float* __restrict__ ds_out, float* __restrict__ dwp_part, int Tlen,
                           int D, int L, int Nb) {
  constexpr int ROWS = 8 * RW;
  constexpr int PW = KC * 256 + 4;  // row-group stride of the dW_p partials
  __shared__ __align__(16) float dss[KC * 256];
  __shared__ __align__(16) float wps[KC * 256];
  __shared__ __align__(16) float part[8 * PW];
  __shared__ float red[8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x, i = blockIdx.y, b = blockIdx.z;
  const int blen = min(L, Tlen - i * L);
  const int t0 = i * L + c * ROWS, n = min(ROWS, blen - c * ROWS);
  const long prow = ((long)b * Nb + i) * gridDim.x + c;
  const long rowbase = (long)b * Tlen + t0;
  const bf16* Hb = Hm + rowbase * D;
  bf16* dHb = dH + rowbase * D;
  const bf16* dYb = dY + rowbase * D;
  // dY goes straight to shared memory (cp.async: no registers held while it
  // is in flight), each thread's own pieces, read back by the same thread.
  // dY is an input of the call, complete before the layer's first kernel
  // started, so its copies go out before the wait for the previous kernel.
  extern __shared__ __align__(16) uint8_t ys_raw[];  // [8 RW rows][KC * 256] bf16
  bf16* ys = reinterpret_cast<bf16*>(ys_raw);
#pragma unroll
  for (int u = 0; u < RW; ++u)
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      const int k = 256 * j + 8 * lane;
      if (warp + 8 * u < n && k < D)
        cp_async16(ys + ((warp + 8 * u) * KC + j) * 256 + 8 * lane,
                   dYb + (long)(warp + 8 * u) * D + k);
    }
  cp_async_commit();
  pdl_enter();
  if (n <= 0) {  // a ragged last block's empty chunk: zero partials of dW_p
    for (int k = threadIdx.x; k < D; k += kThreads) dwp_part[prow * D + k] = 0.f;
    return;
  }
  uint4 h[RW][KC], d[RW][KC];
#pragma unroll
  for (int u = 0; u < RW; ++u)
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      const int k = 256 * j + 8 * lane;
      if (warp + 8 * u < n && k < D) {
        const long o = (long)(warp + 8 * u) * D + k;
        load8_raw(Hb + o, h[u][j]);
        load8_raw(dHb + o, d[u][j]);
      }
    }
  float a[RW];
#pragma unroll
  for (int u = 0; u < RW; ++u) a[u] = (warp + 8 * u < n) ? alpha[rowbase + warp + 8 * u] : 0.f;
  // dS_i and w_p to shared memory; sum_u alpha_u g_u = S_i . dS_i
  const float* dSi = dS + ((long)b * Nb + i) * D;
  const float* Si = Sb + ((long)b * Nb + i) * D;
  float cp = 0.f;
  for (int k = 4 * threadIdx.x; k < D; k += 4 * kThreads) {
    const float4 dv = __ldcg(reinterpret_cast<const float4*>(dSi + k));
    const float4 sv = *reinterpret_cast<const float4*>(Si + k);
    float w[4];
    load4(w_p + k, w);
    *reinterpret_cast<float4*>(dss + k) = dv;
    *reinterpret_cast<float4*>(wps + k) = make_float4(w[0], w[1], w[2], w[3]);
    cp = fmaf(sv.x, dv.x, cp);
    cp = fmaf(sv.y, dv.y, cp);
    cp = fmaf(sv.z, dv.z, cp);
    cp = fmaf(sv.w, dv.w, cp);
  }
  cp = warp_sum(cp);
  if (lane == 0) red[warp] = cp;
  __syncthreads();
  float cd = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) cd += red[w];
  // g_t = H_t . dS_i and ds_t = alpha_t (g_t - S_i . dS_i) per row of the warp
  float dsr[RW];
#pragma unroll
  for (int u = 0; u < RW; ++u) {
    float g = 0.f;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      const int k = 256 * j + 8 * lane;
      if (warp + 8 * u < n && k < D) {
        float hv[8];
        unpack8(h[u][j], hv);
#pragma unroll
        for (int e = 0; e < 8; ++e) g = fmaf(hv[e], dss[k + e], g);
      }
    }
    g = warp_sum(g);
    dsr[u] = a[u] * (g - cd);
    if (lane == 0 && warp + 8 * u < n) ds_out[rowbase + warp + 8 * u] = dsr[u];
  }
  // dH_t = dY_t + (dU W_g^T)_t + alpha_t dS_i + ds_t w_p (the identity, gate
  // and pooling paths); the chunk's dW_p partial sum_t ds_t H_t
#pragma unroll
  for (int j = 0; j < KC; ++j) {
    const int k = 256 * j + 8 * lane;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (j == 0) cp_async_wait_all();  // this thread's dY pieces have landed
    if (k < D) {
#pragma unroll
      for (int u = 0; u < RW; ++u)
        if (warp + 8 * u < n) {
          float hv[8], dv[8], yv[8];
          unpack8(h[u][j], hv);
          unpack8(d[u][j], dv);
          unpack8(*reinterpret_cast<const uint4*>(ys + ((warp + 8 * u) * KC + j) * 256 + 8 * lane),
                  yv);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            acc[e] = fmaf(dsr[u], hv[e], acc[e]);
            dv[e] += yv[e] + a[u] * dss[k + e] + dsr[u] * wps[k + e];
          }
          store8(dHb + (long)(warp + 8 * u) * D + k, dv);
        }
    }

#pragma unroll
    for (int e = 0; e < 8; ++e) part[warp * PW + 256 * j + 8 * lane + e] = acc[e];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < D; k += kThreads) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += part[w * PW + k];
    dwp_part[prow * D + k] = t;
  }
}

// ======================================================== kernels (one per stage)
// Sec. 3.4: item (block i, batch b, chunk z) pools its block (pool_block)
// and stores S_i[256 z .. 256 z + 255].
template <class T>
__global__ void __launch_bounds__(kThreads)
    summary_fwd_kernel(const T* __restrict__ Hm, const float* __restrict__ spart, int npart,
                       long n_tok, float* __restrict__ alpha, float* __restrict__ S, int Tlen,
                       int D, int L, int Nb) {
  pdl_enter();
  extern __shared__ __align__(16) float sm[];
  const int i = blockIdx.x, b = blockIdx.y, z = blockIdx.z;
  const float Si = pool_block<T>(sm, Hm, spart, npart, n_tok, alpha, Tlen, D, L, i, b, z);
  const int c = z * 256 + threadIdx.x;
  if (c < D) S[((long)b * Nb + i) * D + c] = Si;
}

// Sec. 3.5 as a parallel scan over blocks: item (x, b) = channels
// 32x .. 32x+31 of batch b, 256 threads (8 warps).  The decayed sums
//   N_i = a N_{i-1} + S_i,  Z_i = a Z_{i-1} + 1,  M_i = N_i / Z_i
// (M_i = sum_{j<=i} a^(i-j) S_j / sum_{j<=i} a^(i-j)) compose associatively:
// a run of k blocks acts on the sums before it as (N, Z) -> (A N + n, A Z + z)
// with A = a^k and (n, z) the run's own sums from zero, and two runs combine
// as (A1, n1, z1) then (A2, n2, z2) = (A1 A2, A2 n1 + n2, A2 z1 + z2).  The
// blocks go in windows of up to kPsWin rows: the window's S rows come into
// shared memory with coalesced 16-byte loads; warp w takes channels w, w+8,
// w+16, w+24 in turn, lane l a run of ceil(rows / 32) consecutive blocks: the
// lane scans its run from zero, a warp-shuffle inclusive scan of the runs'
// (A, n, z) gives each lane the sums entering its run (with the previous
// windows' carry), and the lane walks its run again to form N, Z and M in
// shared memory; the window's M (fp32 and, when Mb is non-null, bf16) and,
// for batch 0, Z and 1 / Z leave as coalesced rows.
constexpr int kPsCh = 32;      // channels per CTA
constexpr int kPsThreads = 256;
constexpr int kPsWin = 256;    // blocks per shared-memory window
constexpr int kPsLd = kPsCh + 1;
__global__ void __launch_bounds__(kPsThreads)
    memory_scan_fwd_kernel(const float* __restrict__ S, const float* __restrict__ decay,
                           float* __restrict__ M, bf16* __restrict__ Mb, float* __restrict__ Z,
                           float* __restrict__ Zinv, int Nb, int D) {
  extern __shared__ __align__(16) float ps_sm[];
  const int win = min(Nb, kPsWin);
  float* Ss = ps_sm;                 // [win][kPsLd]: S, then M
  float* Zs = ps_sm + win * kPsLd;   // [win][kPsLd]: Z (batch 0)
  const int x = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c0 = x * kPsCh;
  pdl_enter();
  // the carry of the earlier windows, per channel this warp scans
  float cn[kPsCh / 8], cz[kPsCh / 8];
#pragma unroll
  for (int q = 0; q < kPsCh / 8; ++q) cn[q] = cz[q] = 0.f;
  float av[kPsCh / 8];
#pragma unroll
  for (int q = 0; q < kPsCh / 8; ++q) av[q] = decay[c0 + warp + 8 * q];
  for (int w0 = 0; w0 < Nb; w0 += kPsWin) {
    const int rows = min(kPsWin, Nb - w0);
    // S rows w0 .. w0+rows-1 of the chunk: 8 threads per row, 16 bytes each
    for (int o = threadIdx.x; o < rows * (kPsCh / 4); o += kPsThreads) {
      const int rr = o / (kPsCh / 4), p4 = o % (kPsCh / 4);
      const float4 v =
          *reinterpret_cast<const float4*>(S + ((long)b * Nb + w0 + rr) * D + c0 + 4 * p4);
      float* d = Ss + rr * kPsLd + 4 * p4;
      d[0] = v.x;
      d[1] = v.y;
      d[2] = v.z;
      d[3] = v.w;
    }
    __syncthreads();
    const int seg = (rows + 31) / 32;
    const int i0 = lane * seg, i1 = min(i0 + seg, rows);
#pragma unroll
    for (int q = 0; q < kPsCh / 8; ++q) {
      const int c = warp + 8 * q;
      const float a = av[q];
      // the lane's run from zero, and a^(run length)
      float n = 0.f, z = 0.f, A = 1.f;
      for (int i = i0; i < i1; ++i) {
        n = fmaf(a, n, Ss[i * kPsLd + c]);
        z = fmaf(a, z, 1.0f);
        A *= a;
      }
      // inclusive scan of the runs across the warp
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const float Ap = __shfl_up_sync(0xffffffffu, A, off);
        const float np = __shfl_up_sync(0xffffffffu, n, off);
        const float zp = __shfl_up_sync(0xffffffffu, z, off);
        if (lane >= off) {
          n = fmaf(A, np, n);
          z = fmaf(A, zp, z);
          A *= Ap;
        }
      }
      // the sums entering this lane's run: the earlier lanes (exclusive
      // prefix) applied to the earlier windows' carry
      float Ae = __shfl_up_sync(0xffffffffu, A, 1);
      float ne = __shfl_up_sync(0xffffffffu, n, 1);
      float ze = __shfl_up_sync(0xffffffffu, z, 1);
      if (lane == 0) {
        Ae = 1.f;
        ne = ze = 0.f;
      }
      float N = fmaf(Ae, cn[q], ne), Zz = fmaf(Ae, cz[q], ze);
      // the carry out of this window (lane 31's inclusive sums)
      const float At = __shfl_sync(0xffffffffu, A, 31);
      const float nt = __shfl_sync(0xffffffffu, n, 31);
      const float zt = __shfl_sync(0xffffffffu, z, 31);
      cn[q] = fmaf(At, cn[q], nt);
      cz[q] = fmaf(At, cz[q], zt);
      for (int i = i0; i < i1; ++i) {
        N = fmaf(a, N, Ss[i * kPsLd + c]);
        Zz = fmaf(a, Zz, 1.0f);
        Ss[i * kPsLd + c] = N / Zz;
        Zs[i * kPsLd + c] = Zz;
      }
    }
    __syncthreads();
    // the window's rows of M (and Mb; Z, 1/Z for batch 0)
    for (int o = threadIdx.x; o < rows * (kPsCh / 4); o += kPsThreads) {
      const int rr = o / (kPsCh / 4), p4 = o % (kPsCh / 4);
      const float* s = Ss + rr * kPsLd + 4 * p4;
      const long g = ((long)b * Nb + w0 + rr) * D + c0 + 4 * p4;
      *reinterpret_cast<float4*>(M + g) = make_float4(s[0], s[1], s[2], s[3]);
      if (Mb) {
        __nv_bfloat162 lo = __floats2bfloat162_rn(s[0], s[1]), hi = __floats2bfloat162_rn(s[2], s[3]);
        uint2 u;
        u.x = *reinterpret_cast<uint32_t*>(&lo);
        u.y = *reinterpret_cast<uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(Mb + g) = u;
      }
      if (b == 0) {
        const float* zz = Zs + rr * kPsLd + 4 * p4;
        const long gz = (long)(w0 + rr) * D + c0 + 4 * p4;
        *reinterpret_cast<float4*>(Z + gz) = make_float4(zz[0], zz[1], zz[2], zz[3]);
        *reinterpret_cast<float4*>(Zinv + gz) =
            make_float4(1.0f / zz[0], 1.0f / zz[1], 1.0f / zz[2], 1.0f / zz[3]);
      }
    }
    __syncthreads();  // the window's shared memory is reused
  }
}

// The reverse scan (memory_scan_bwd_kernel): kScanThreads threads per CTA
// spread the B * D chains over many SMs.
constexpr int kScanThreads = 64;

// ------------------------------------------------ warp-level bf16 products
// The memory's D x D projections at small shapes are [B*Nb, D] x [D, D]: a
// few tens of MFLOP, far too little for the tcgen05 GEMM's launch and ring
// fill.  Here one CTA per (column chunk, batch) multiplies the batch's Nb
// memory rows by a 32-column chunk of the weight with mma.sync m16n8k16
// (bf16 operands from shared memory through ldmatrix, fp32 accumulators):
// warp w takes columns 8 (w % 4) .. +7 and half w / 4 of the K range, and the
// two halves are added through shared memory.  Operand rows are padded by 8
// elements so that the 8 rows an ldmatrix reads fall in distinct banks.
// Copies rows of 16-byte pieces from global to shared memory, all threads of
// the CTA, up to eight loads of a thread in flight before their stores.
// copy_rows16<P>: `rows` rows of P pieces (src row stride lds elements, dst ldd).
// copy_rows16v: `rows` rows of `pieces` pieces, rows past `rows` up to `rows_pad`
// zero-filled.
template <int NT = kThreads>
__device__ __forceinline__ void copy_rows16v(bf16* dst, int ldd, const bf16* src, long lds,
                                             int rows, int pieces, int rows_pad) {
  const int total = rows_pad * pieces;
  for (int o0 = threadIdx.x; o0 < total; o0 += 8 * NT) {
    uint4 v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int o = o0 + j * NT;
      const int r = o / pieces, c = o % pieces;
      v[j] = make_uint4(0u, 0u, 0u, 0u);
      if (o < total && r < rows) v[j] = *reinterpret_cast<const uint4*>(src + r * lds + 8 * c);
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int o = o0 + j * NT;
      if (o < total)
        *reinterpret_cast<uint4*>(dst + (long)(o / pieces) * ldd + 8 * (o % pieces)) = v[j];
    }
  }
}
template <int P, int NT = kThreads>
__device__ __forceinline__ void copy_rows16(bf16* dst, int ldd, const bf16* src, long lds,
                                            int rows) {
  copy_rows16v<NT>(dst, ldd, src, lds, rows, P, rows);
}

constexpr int kProjNC = 32;   // output columns per CTA
constexpr int kProjPad = 8;   // bf16 elements of padding per shared-memory row
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t* r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t* r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];"
               : "=r"(r[0]), "=r"(r[1])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2_t(uint32_t addr, uint32_t* r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];"
               : "=r"(r[0]), "=r"(r[1])
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16_16816(float* d, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
// One warp's 16 x 8 product over K range [k0, k1) (multiples of 16): A rows
// r0 .. r0+15 of a row-major [.., lda] bf16 tile (K contiguous); B either
// [K][ldb] with N contiguous (kBT = false: ldmatrix .trans) or [N][ldb] with
// K contiguous (kBT = true), columns n0 .. n0+7.  acc: the mma C fragment.
template <bool kBT>
__device__ __forceinline__ void warp_mma_16x8(const bf16* A, int lda, int r0, const bf16* Bm,
                                              int ldb, int n0, int k0, int k1, float* acc) {
  const int lane = threadIdx.x & 31;
  const int mi = lane >> 3, rr = lane & 7;
  const uint32_t a_base = (uint32_t)__cvta_generic_to_shared(
      A + (long)(r0 + rr + 8 * (mi & 1)) * lda + 8 * (mi >> 1));
  // lanes 0-7 address B's k rows k .. k+7, lanes 8-15 rows k+8 .. k+15
  // (kBT: n rows n0 .. n0+7 at k and k+8)
  const int bl = lane & 15;
  const uint32_t b_base = kBT ? (uint32_t)__cvta_generic_to_shared(
                                    Bm + (long)(n0 + (bl & 7)) * ldb + 8 * (bl >> 3))
                              : (uint32_t)__cvta_generic_to_shared(Bm + (long)bl * ldb + n0);
  for (int k = k0; k < k1; k += 16) {
    uint32_t a[4], b[2];
    ldsm_x4(a_base + (uint32_t)(k * 2), a);
    if (kBT)
      ldsm_x2(b_base + (uint32_t)(k * 2), b);
    else
      ldsm_x2_t(b_base + (uint32_t)((long)k * ldb * 2), b);
    mma_bf16_16816(acc, a, b);
  }
}

// Sec. 3.5 and the memory projection in one launch (bf16), for shapes whose
// memory fits one CTA's shared memory: item (x, b) = output columns
// kProjNC*x .. kProjNC*x + kProjNC-1 of batch b, kProjThreads threads.  The
// weight chunk W_m[:, x] is fetched before the wait for the previous kernel
// (it is an input, not a product of the step).  After the wait the CTA
// copies the batch's summaries S [Nb, D] to shared memory and runs the
// decayed scan of every channel over the Nb blocks (thread t: channels t,
// t + kProjThreads; N_i = a N_{i-1} + S_i, Z_i = a Z_{i-1} + 1,
// M_i = N_i * (1 / Z_i)) into shared memory as bf16 (the operand the
// tensor-core path uses too), then P_i[c] = sum_k M_i[k] W_m[k][c] on the
// tensor cores: warp w takes columns 8 (w % 4) .. +7 and K quarter w / 4, the
// quarters added in order.  CTA x also stores M (fp32 and bf16) of its own
// kProjNC channels and, for batch 0, their Z and 1/Z.  P is stored unshifted
// [B*Nb, D]: its readers take C_i = P_{i-1}, C_0 = 0.
constexpr int kProjThreads = 512;
constexpr int kProjKQ = kProjThreads / 32 / 4;  // K ranges per column group
constexpr int kProjMaxCh = 4;                   // channels per thread (D <= 2048)
__global__ void __launch_bounds__(kProjThreads)
    memory_proj_fwd_kernel(const float* __restrict__ S, const float* __restrict__ decay,
                           const bf16* __restrict__ Wm, float* __restrict__ P,
                           float* __restrict__ M, bf16* __restrict__ Mb, float* __restrict__ Z,
                           float* __restrict__ Zinv, int Nb, int D) {
  extern __shared__ __align__(16) uint8_t smb[];
  const int Nr = (Nb + 15) & ~15;            // rows padded to the mma's 16
  const int lda = D + kProjPad, ldw = kProjNC + kProjPad;
  bf16* Ws = reinterpret_cast<bf16*>(smb);                         // [D][ldw]
  bf16* Ms = Ws + (long)D * ldw;                                   // [Nr][lda]
  float* red = reinterpret_cast<float*>(Ms + (long)Nr * lda);      // [KQ-1][4][16][8]
  float* Ss = red + (kProjKQ - 1) * 4 * 16 * 8;                    // [Nb][D]
  const int x = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the weight chunk: D rows of kProjNC columns (16 bytes per load, a batch
  // of loads in flight before their shared-memory stores)
  copy_rows16<kProjNC / 8, kProjThreads>(Ws, ldw, Wm + x * kProjNC, D, D);
  // the decay of this thread's channels (an input too)
  float apre[kProjMaxCh];
#pragma unroll
  for (int q = 0; q < kProjMaxCh; ++q) {
    const int k = threadIdx.x + q * kProjThreads;
    apre[q] = k < D ? decay[k] : 0.f;
  }
  pdl_enter();
  // the batch's summaries to shared memory in 16-byte pieces (all in flight
  // at once, no registers held)
  {
    const float* Sb = S + (long)b * Nb * D;
    for (int o = 4 * threadIdx.x; o < Nb * D; o += 4 * kProjThreads) cp_async16(Ss + o, Sb + o);
    cp_async_commit();
    cp_async_wait_all();
    __syncthreads();
  }
  // the scan, one channel per thread (a rolled loop: little code to fetch);
  // CTA x stores M, Mb (and for b == 0, Z and 1/Z) of its own 32 channels
#pragma unroll
  for (int q = 0; q < kProjMaxCh; ++q) {
    const int k = threadIdx.x + q * kProjThreads;
    if (k >= D) break;
    const float a = apre[q];
    const bool mine = k / kProjNC == x;
    float Nn = 0.f, Zz = 0.f;
#pragma unroll 4
    for (int i = 0; i < Nb; ++i) {
      Nn = fmaf(a, Nn, Ss[i * D + k]);
      Zz = fmaf(a, Zz, 1.0f);
      const float zi = __frcp_rn(Zz);
      const float m = Nn * zi;
      const bf16 mb = __float2bfloat16_rn(m);
      if (mine) {
        const long o = ((long)b * Nb + i) * D + k;
        M[o] = m;
        Mb[o] = mb;
        if (b == 0) {
          Z[(long)i * D + k] = Zz;
          Zinv[(long)i * D + k] = zi;
        }
      }
      Ms[(long)i * lda + k] = mb;
    }
    for (int i = Nb; i < Nr; ++i) Ms[(long)i * lda + k] = __float2bfloat16_rn(0.f);
  }
  __syncthreads();
  // warp w: columns 8 (w & 3) .. +7, K range w >> 2 of kProjKQ
  const int n0 = 8 * (warp & 3), kq = warp >> 2, kr = D / kProjKQ;
  const int fr = lane >> 2, fc = 2 * (lane & 3);
  for (int r0 = 0; r0 < Nr; r0 += 16) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    warp_mma_16x8<false>(Ms, lda, r0, Ws, ldw, n0, kq * kr, (kq + 1) * kr, acc);
    // C fragment: rows r0 + lane/4 (+8), columns n0 + 2 (lane % 4) (+1)
    if (kq > 0) {
      float* rw = red + (((kq - 1) * 4 + (warp & 3)) * 16) * 8;
      rw[fr * 8 + fc] = acc[0];
      rw[fr * 8 + fc + 1] = acc[1];
      rw[(fr + 8) * 8 + fc] = acc[2];
      rw[(fr + 8) * 8 + fc + 1] = acc[3];
    }
    __syncthreads();
    if (kq == 0) {
#pragma unroll
      for (int q = 1; q < kProjKQ; ++q) {
        const float* rw = red + (((q - 1) * 4 + (warp & 3)) * 16) * 8;
        acc[0] += rw[fr * 8 + fc];
        acc[1] += rw[fr * 8 + fc + 1];
        acc[2] += rw[(fr + 8) * 8 + fc];
        acc[3] += rw[(fr + 8) * 8 + fc + 1];
      }
      const long base = ((long)b * Nb + r0) * D + x * kProjNC + n0 + fc;
      if (r0 + fr < Nb) {
        P[base + (long)fr * D] = acc[0];
        P[base + (long)fr * D + 1] = acc[1];
      }
      if (r0 + fr + 8 < Nb) {
        P[base + (long)(fr + 8) * D] = acc[2];
        P[base + (long)(fr + 8) * D + 1] = acc[3];
      }
    }
    __syncthreads();
  }
}

template <class T, int PS>
__global__ void __launch_bounds__(kThreads, 2)
    gate_bwd_kernel(const T* __restrict__ dY, const T* __restrict__ G,
                    const float* __restrict__ Pm, long pstride, T* __restrict__ dU,
                    float* __restrict__ dP, bf16* __restrict__ dPb, int Tlen, int D, int L,
                    int Nb) {
  extern __shared__ __align__(16) float sm[];
  gate_bwd_item<T, PS>(sm, dY, G, Pm, pstride, dU, dP, dPb, Tlen, D, L, Nb, blockIdx.x,
                   blockIdx.y, blockIdx.z);
}

template <int PS>
__global__ void __launch_bounds__(kScanThreads)
    memory_scan_bwd_kernel(const float* __restrict__ dM, long mstride,
                           const float* __restrict__ decay, const float* __restrict__ Z,
                           const float* __restrict__ M, float* __restrict__ dS,
                           float* __restrict__ da_part, int Nb, int D) {
  pdl_enter();
  scan_bwd_item<PS>(dM, mstride, decay, Z, M, dS, da_part, Nb, D, blockIdx.x, blockIdx.y);
}

template <class T, int ROWS>
__global__ void __launch_bounds__(kThreads, 2)
    summary_bwd_kernel(const T* __restrict__ Hm, const float* __restrict__ alpha,
                       const float* __restrict__ Sb, const float* __restrict__ dS,
                       const T* __restrict__ w_p, const T* __restrict__ dY, T* dH,
                       float* __restrict__ ds, float* __restrict__ dwp_part, int Tlen, int D,
                       int L, int Nb) {
  pdl_enter();
  __shared__ __align__(16) float sm[ROWS + 8 + 8 * 260];
  // a ragged last block has fewer chunks than the grid's x extent: its empty
  // chunks contribute zero partials to dW_p
  if ((int)blockIdx.x * ROWS >= min(L, Tlen - (int)blockIdx.y * L)) {
    const long prow = ((long)blockIdx.z * Nb + blockIdx.y) * gridDim.x + blockIdx.x;
    for (int k = threadIdx.x; k < D; k += kThreads) dwp_part[prow * D + k] = 0.f;
    return;
  }
  summary_bwd_item<T, ROWS>(sm, Hm, alpha, Sb, dS, w_p, dY, dH, ds, dwp_part, Tlen, D, L, Nb,
                            blockIdx.x, blockIdx.y, blockIdx.z);
}

// Sec. 3.7-3.8: Y = H + G * C[b, t / L], the memory row of the token's block
// broadcast by index.  Item (run, row group, block i, batch b): 8 channels of
// kInjRows consecutive rows of one block, so the memory row (summed from the
// projection's K-split partials, shifted by one block) is read once for all
// of them; the rows' H and G loads are all issued before the first use.  The
// host sizes the grid so that every item's thread is resident at once (one
// wave): a second, partial wave would add a whole memory round trip.
// kInjRows rows per item in bf16 (4 in fp32, whose rows take twice the registers).
constexpr int kInjRows = 8;
__host__ __device__ constexpr int inj_rows(int elem_bytes) { return elem_bytes == 2 ? kInjRows : kInjRows / 2; }
template <class T, int PS>
__global__ void __launch_bounds__(kThreads, 2)
    inject_kernel(const T* __restrict__ Hm, const T* __restrict__ G, const float* __restrict__ Pm,
                  long pstride, T* __restrict__ Y, int B, int Tlen, int D, int L, int Nb) {
  pdl_enter();
  constexpr int kInjRows = inj_rows(sizeof(T));
  const int runs = D / 8, groups = (L + kInjRows - 1) / kInjRows;
  const long total = (long)B * Nb * groups * runs;
  for (long it = (long)blockIdx.x * kThreads + threadIdx.x; it < total;
       it += (long)gridDim.x * kThreads) {
    const int run = (int)(it % runs);
    long rest = it / runs;
    const int grp = (int)(rest % groups);
    rest /= groups;
    const int i = (int)(rest % Nb), b = (int)(rest / Nb);
    const int t0 = i * L + grp * kInjRows;
    const int nr = min(kInjRows, min((i + 1) * L, Tlen) - t0);
    if (nr <= 0) continue;
    const int cc = run * 8;
    const long o0 = ((long)b * Tlen + t0) * D + cc;
    Raw8<T> rh[kInjRows], rgt[kInjRows];
#pragma unroll
    for (int r = 0; r < kInjRows; ++r)
      if (r < nr) {
        ld_raw(Hm + o0 + (long)r * D, rh[r]);
        ld_raw(G + o0 + (long)r * D, rgt[r]);
      }
    float c[8];
    mem_row<8, PS>(Pm, pstride, b, i, Nb, D, cc, c);
#pragma unroll
    for (int r = 0; r < kInjRows; ++r)
      if (r < nr) {
        float h[8], g[8], y[8];
        unraw(rh[r], h);
        unraw(rgt[r], g);
#pragma unroll
        for (int e = 0; e < 8; ++e) y[e] = fmaf(g[e], c[e], h[e]);
        store8(Y + o0 + (long)r * D, y);
      }
  }
}

// ============================================================== host side
namespace {
// shared memory of the summary kernels: scores [kMaxL], two scalars, [8][260]
constexpr size_t kSummarySmem = (size_t)(kMaxL + 4 + 8 * 260) * sizeof(float);
constexpr size_t kGateSmem = (size_t)(8 * (kGateCh + 4) + kGateCh) * sizeof(float);
}  // namespace

cudaError_t summary_fwd(const Launch& lc, int dtype, const void* Hm, const float* spart, int npart,
                        float* alpha, float* S, int B, int T, int D, int L) {
  if (L > kMaxL) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  dim3 grid(Nb, B, (D + 255) / 256);
  const long n_tok = (long)B * T;
  cudaError_t e;
  if (dtype == 0)
    e = launch_k(summary_fwd_kernel<float>, grid, dim3(kThreads), kSummarySmem, lc.stream,
                 (const float*)Hm, spart, npart, n_tok, alpha, S, T, D, L, Nb);
  else
    e = launch_k(summary_fwd_kernel<bf16>, grid, dim3(kThreads), kSummarySmem, lc.stream,
                 (const bf16*)Hm, spart, npart, n_tok, alpha, S, T, D, L, Nb);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t memory_scan_fwd(const Launch& lc, const float* S, const float* decay, float* M,
                            void* Mb, float* Z, float* Zinv, int B, int Nb, int D) {
  if (D % kPsCh != 0) return cudaErrorInvalidValue;
  const size_t smem = (size_t)2 * std::min(Nb, kPsWin) * kPsLd * sizeof(float);
  static std::atomic<unsigned long long> opted{0};
  cudaError_t e = smem_opt_in(memory_scan_fwd_kernel, (int)((size_t)2 * kPsWin * kPsLd * sizeof(float)),
                              &opted);
  if (e != cudaSuccess) return e;
  dim3 grid(D / kPsCh, B);
  e = launch_k(memory_scan_fwd_kernel, grid, dim3(kPsThreads), smem, lc.stream, S, decay, M,
               (bf16*)Mb, Z, Zinv, Nb, D);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// The one-CTA-per-(column chunk, batch) memory kernel holds a batch's memory
// rows and a weight chunk in shared memory and runs the D x D projection with
// warp-level bf16 mma: taken for bf16 when that fits, Nb <= 16 (one row group
// of the mma) and the projection is small (B*Nb*D*D <= 2^28 multiply-adds),
// where the tcgen05 GEMM's launch and ring fill would dominate (measured: at
// Nb = 32, D = 1024 the scan kernel and tcgen05 projection were faster).
constexpr int kProjSmemMax = 200 * 1024;
static size_t proj_fwd_smem(int Nb, int D) {
  const size_t Nr = (size_t)((Nb + 15) & ~15);
  return ((size_t)D * (kProjNC + kProjPad) + Nr * (D + kProjPad)) * 2 +
         (size_t)(kProjKQ - 1) * 4 * 16 * 8 * 4 + (size_t)Nb * D * 4;
}
bool memory_proj_fits(int dtype, int B, int Nb, int D) {
  return dtype == 1 && D % 64 == 0 && D % (16 * kProjKQ) == 0 && Nb <= 16 &&
         D <= kProjMaxCh * kProjThreads &&
         proj_fwd_smem(Nb, D) <= (size_t)kProjSmemMax &&
         (double)B * Nb * D * D <= (double)(1 << 28);
}

cudaError_t memory_proj_fwd(const Launch& lc, const float* S, const float* decay, const void* Wm,
                            float* P, float* M, void* Mb, float* Z, float* Zinv, int B, int Nb,
                            int D) {
  if (!memory_proj_fits(1, B, Nb, D) || !Mb) return cudaErrorInvalidValue;
  // the limit is raised once per kernel and device, to the largest size any
  // accepted shape needs
  static std::atomic<unsigned long long> opted{0};
  cudaError_t e = smem_opt_in(memory_proj_fwd_kernel, kProjSmemMax, &opted);
  if (e != cudaSuccess) return e;
  e = launch_k(memory_proj_fwd_kernel, dim3(D / kProjNC, B), dim3(kProjThreads), proj_fwd_smem(Nb, D),
               lc.stream, S, decay, (const bf16*)Wm, P, M, (bf16*)Mb, Z, Zinv, Nb, D);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t gate_bwd(const Launch& lc, int dtype, const void* dY, const void* G, const float* Pm,
                     int psplits, void* dU, float* dP, void* dPb, int B, int T, int D, int L) {
  const int Nb = (T + L - 1) / L;
  const long pstride = (long)B * Nb * D;
  dim3 grid((D + kGateCh - 1) / kGateCh, Nb, B);
  cudaError_t e = with_splits(psplits, [&](auto ps) {
    constexpr int PS = decltype(ps)::value;
    if (dtype == 0)
      return launch_k(gate_bwd_kernel<float, PS>, grid, dim3(kThreads), kGateSmem, lc.stream,
                      (const float*)dY, (const float*)G, Pm, pstride, (float*)dU, dP, (bf16*)dPb,
                      T, D, L, Nb);
    return launch_k(gate_bwd_kernel<bf16, PS>, grid, dim3(kThreads), kGateSmem, lc.stream,
                    (const bf16*)dY, (const bf16*)G, Pm, pstride, (bf16*)dU, dP, (bf16*)dPb, T, D,
                    L, Nb);
  });
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t memory_scan_bwd(const Launch& lc, const float* dM, int msplits, const float* decay,
                            const float* Z, const float* M, float* dS, float* da_part, int B,
                            int Nb, int D) {
  dim3 grid((D + kScanThreads - 1) / kScanThreads, B);
  cudaError_t e = with_splits(msplits, [&](auto ms) {
    return launch_k(memory_scan_bwd_kernel<decltype(ms)::value>, grid, dim3(kScanThreads), 0,
                    lc.stream, dM, (long)B * Nb * D, decay, Z, M, dS, da_part, Nb, D);
  });
  return e != cudaSuccess ? e : cudaGetLastError();
}

// Rows per pooling-backward item: the register-held kernel (bf16, D <= 1024)
// takes 8 * RW rows with RW * ceil(D / 256) <= 8; the general kernel takes 16
// rows, or 32 when D <= 256.
static int summary_bwd_reg_rw(int dtype, int D) {
  if (dtype != 1 || D > 1024) return 0;
  const int kc = (D + 255) / 256;
  return kc == 1 ? 8 : kc == 2 ? 4 : 2;
}
static int summary_bwd_rows(int dtype, int D) {
  const int rw = summary_bwd_reg_rw(dtype, D);
  if (rw) return 8 * rw;
  return D <= 256 ? 32 : 16;
}
int summary_bwd_chunks(int dtype, int L, int D) {
  const int rows = summary_bwd_rows(dtype, D);
  return (L + rows - 1) / rows;
}

cudaError_t summary_bwd(const Launch& lc, int dtype, const void* Hm, const float* alpha,
                        const float* Sb, const float* dS, const void* w_p, const void* dY,
                        void* dH, float* ds, float* dwp_part, int B, int T, int D, int L) {
  if (L > kMaxL) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  dim3 grid(summary_bwd_chunks(dtype, L, D), Nb, B);
  const int rw = summary_bwd_reg_rw(dtype, D);
  cudaError_t e;
  if (rw) {
    const bf16 *H = (const bf16*)Hm, *wp = (const bf16*)w_p;
    bf16* dh = (bf16*)dH;
    const int kc = (D + 255) / 256;
    auto go = [&](auto rw, auto kcc) -> cudaError_t {
      constexpr int RW_ = decltype(rw)::value, KC_ = decltype(kcc)::value;
      // the dY staging buffer (dynamic shared memory beside the static arrays)
      constexpr int ys_bytes = 8 * RW_ * KC_ * 256 * 2;
      static std::atomic<unsigned long long> opted{0};
      cudaError_t r = smem_opt_in(summary_bwd_reg_kernel<RW_, KC_>, ys_bytes, &opted);
      if (r != cudaSuccess) return r;
      return launch_k(summary_bwd_reg_kernel<RW_, KC_>, grid, dim3(kThreads), ys_bytes, lc.stream,
                      H, alpha, Sb, dS, wp, (const bf16*)dY, dh, ds, dwp_part, T, D, L, Nb);
    };
    using I1 = std::integral_constant<int, 1>;
    using I2 = std::integral_constant<int, 2>;
    using I3 = std::integral_constant<int, 3>;
    using I4 = std::integral_constant<int, 4>;
    using I8 = std::integral_constant<int, 8>;
    e = kc == 1 ? go(I8(), I1()) : kc == 2 ? go(I4(), I2()) : kc == 3 ? go(I2(), I3()) : go(I2(), I4());
    return e != cudaSuccess ? e : cudaGetLastError();
  }
  auto go = [&](auto rows) {
    constexpr int R = decltype(rows)::value;
    if (dtype == 0)
      return launch_k(summary_bwd_kernel<float, R>, grid, dim3(kThreads), 0, lc.stream,
                      (const float*)Hm, alpha, Sb, dS, (const float*)w_p, (const float*)dY,
                      (float*)dH, ds, dwp_part, T, D, L, Nb);
    return launch_k(summary_bwd_kernel<bf16, R>, grid, dim3(kThreads), 0, lc.stream,
                    (const bf16*)Hm, alpha, Sb, dS, (const bf16*)w_p, (const bf16*)dY, (bf16*)dH,
                    ds, dwp_part, T, D, L, Nb);
  };
  e = summary_bwd_rows(dtype, D) == 32 ? go(std::integral_constant<int, 32>())
                                       : go(std::integral_constant<int, 16>());
  return e != cudaSuccess ? e : cudaGetLastError();
}

// Resident CTAs of `kern` (kThreads threads, no dynamic shared memory) on
// the whole device, looked up once per kernel.
template <class K>
static long resident_ctas(K kern) {
  static long n = 0;
  if (!n) {
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0) != cudaSuccess ||
        sms < 1 || per_sm < 1)
      return 148;
    n = (long)sms * per_sm;
  }
  return n;
}

cudaError_t inject(const Launch& lc, int dtype, const void* Hm, const void* G, const float* Pm,
                   int psplits, void* Y, int B, int T, int D, int L) {
  const int Nb = (T + L - 1) / L;
  const long pstride = (long)B * Nb * D;
  const int rows = inj_rows(dtype == 0 ? 4 : 2);
  const long items = (long)B * Nb * ((L + rows - 1) / rows) * (D / 8);
  const long want = (items + kThreads - 1) / kThreads;
  const long cap = dtype == 0 ? resident_ctas(inject_kernel<float, 4>)
                              : resident_ctas(inject_kernel<bf16, 4>);
  const int blocks = (int)std::max<long>(1, std::min<long>(want, cap));
  cudaError_t e = with_splits(psplits, [&](auto ps) {
    constexpr int PS = decltype(ps)::value;
    if (dtype == 0)
      return launch_k(inject_kernel<float, PS>, dim3(blocks), dim3(kThreads), 0, lc.stream,
                      (const float*)Hm, (const float*)G, Pm, pstride, (float*)Y, B, T, D, L, Nb);
    return launch_k(inject_kernel<bf16, PS>, dim3(blocks), dim3(kThreads), 0, lc.stream,
                    (const bf16*)Hm, (const bf16*)G, Pm, pstride, (bf16*)Y, B, T, D, L, Nb);
  });
  return e != cudaSuccess ? e : cudaGetLastError();
}

// Column sums in a fixed order: 8 row groups of 32 columns per CTA, then the
// group sums added in group order.
template <class TO>
__global__ void __launch_bounds__(256)
    reduce_rows_kernel(const float* __restrict__ in, int rows, int cols, TO* __restrict__ out) {
  pdl_enter();
  __shared__ float part[8][33];
  const int rg = threadIdx.x >> 5, cl = threadIdx.x & 31;
  const int c = blockIdx.x * 32 + cl;
  float acc = 0.f;
  if (c < cols)
    for (int r = rg; r < rows; r += 8) acc += in[(long)r * cols + c];
  part[rg][cl] = acc;
  __syncthreads();
  if (threadIdx.x < 32 && c < cols) {
    float t = 0.f;
#pragma unroll
    for (int g = 0; g < 8; ++g) t += part[g][threadIdx.x];
    out[c] = from_f<TO>(t);
  }
}

cudaError_t reduce_rows(const Launch& lc, const float* in, int rows, int cols, int dtype_out,
                        void* out) {
  const int blocks = (cols + 31) / 32;
  cudaError_t e;
  if (dtype_out == 0)
    e = launch_k(reduce_rows_kernel<float>, dim3(blocks), dim3(256), 0, lc.stream, in, rows, cols,
                 (float*)out);
  else
    e = launch_k(reduce_rows_kernel<bf16>, dim3(blocks), dim3(256), 0, lc.stream, in, rows, cols,
                 (bf16*)out);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t fill_zero(const Launch& lc, void* p, size_t bytes) {
  return cudaMemsetAsync(p, 0, bytes, lc.stream);
}

}  // namespace bcmt
