// Adaptive block summaries (Sec. 3.4), the normalised exponential causal
// memory with its projection and one-block shift (Sec. 3.5), and the backward
// of these two stages and of the gated injection (Sec. 3.8).
//
// These stages are HBM- or latency-bound (O(T D) and O(N_b D^2) work against
// O(T D^2) for the projections), so they run on CUDA cores with coalesced,
// vectorised row accesses and fixed-order (deterministic) reductions.
#include "common.cuh"
#include "internal.h"

namespace bcmt {

namespace {
constexpr int kMaxL = 1024;
}

// -------------------------------------------------------------- Sec. 3.4
// One CTA per (block i, batch b, 256 channels).  The pooling scores
// s_t = H_t . w_p arrive as npart partial dot products per token (written by
// the W_O GEMM epilogue over disjoint column ranges) and are summed here in a
// fixed order; alpha = softmax(s) over the block's tokens; S_i = sum_t alpha_t H_t
// for this CTA's channels.
template <class T>
__global__ void __launch_bounds__(256)
    summary_fwd_kernel(const T* __restrict__ Hm, const float* __restrict__ spart, int npart,
                       long n_tok, float* __restrict__ alpha, float* __restrict__ S, int Tlen,
                       int D, int L) {
  pdl_enter();
  __shared__ float sc[kMaxL];
  __shared__ float red[2];
  const int i = blockIdx.x, b = blockIdx.y, Nb = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const long row0 = (long)b * Tlen + t0;
  for (int r = threadIdx.x; r < n; r += blockDim.x) {
    float s = 0.f;
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
    if (lane == 0) { red[0] = mx; red[1] = 1.0f / sum; }
  }
  __syncthreads();
  const float mx = red[0], inv = red[1];
  for (int r = threadIdx.x; r < n; r += blockDim.x) {
    const float a = expf(sc[r] - mx) * inv;
    if (blockIdx.z == 0) alpha[row0 + r] = a;
    sc[r] = a;
  }
  __syncthreads();
  // S_i[c] = sum_t alpha_t H_t[c]: 8 row groups x 32 threads of 8 channels each,
  // then a fixed-order sum over the row groups.
  __shared__ float part[8][256 + 4];
  const int rg = threadIdx.x >> 5, co = threadIdx.x & 31;
  const int c = blockIdx.z * 256 + co * 8;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c < D) {
    const T* Hc = Hm + row0 * D + c;
    for (int r = rg; r < n; r += 8) {
      float h[8];
      load8(Hc + (long)r * D, h);
      const float a = sc[r];
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = fmaf(a, h[e], acc[e]);
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) part[rg][co * 8 + e] = acc[e];
  __syncthreads();
  const int cc = blockIdx.z * 256 + threadIdx.x;
  if (cc < D) {
    float t = 0.f;
#pragma unroll
    for (int g = 0; g < 8; ++g) t += part[g][threadIdx.x];
    S[((long)b * Nb + i) * D + cc] = t;
  }
}

cudaError_t summary_fwd(const Launch& lc, int dtype, const void* Hm, const float* spart, int npart,
                        float* alpha, float* S, int B, int T, int D, int L) {
  if (L > kMaxL) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  dim3 grid(Nb, B, (D + 255) / 256);
  const long n_tok = (long)B * T;
  if (dtype == 0)
    launch_k(summary_fwd_kernel<float>, dim3(grid), dim3(256), 0, lc.stream,
(const float*)Hm, spart, npart, n_tok,
                                                           alpha, S, T, D, L);
  else
    launch_k(summary_fwd_kernel<bf16>, dim3(grid), dim3(256), 0, lc.stream,
(const bf16*)Hm, spart, npart, n_tok,
                                                          alpha, S, T, D, L);
  return cudaGetLastError();
}

// -------------------------------------------------------------- Sec. 3.5
// Small products of the memory stage on CUDA cores (at most a few hundred rows
// of output, K <= a few thousand).  A CTA owns a 16 x 32 output tile and splits
// K over its 8 warps: lane l of warp w accumulates output column l for all 16
// rows over k = w, w+8, ...; the A values of a k are one 64-byte broadcast,
// the B value one conflict-free word.  K is staged in slices of kKS (all of a
// slice's loads are issued before the first use), and the 8 partial tiles are
// added in warp order at the end, so results are deterministic.
constexpr int kKS = 512;

// A slice: As[kk*16 + mm] = A(m0+mm, k0+kk) for kk < kKS (zero outside).
__device__ __forceinline__ void stage_a(float* As, const float* __restrict__ A, long sam, long sak,
                                        int m0, int Mr, int k0, int K) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    float v[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int e = threadIdx.x + (h * 16 + q) * 256;
      int mm, kk;
      if (sak == 1) { mm = e >> 9; kk = e & (kKS - 1); } else { kk = e >> 4; mm = e & 15; }
      const int m = m0 + mm, k = k0 + kk;
      v[q] = (m < Mr && k < K) ? A[(long)m * sam + (long)k * sak] : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int e = threadIdx.x + (h * 16 + q) * 256;
      int mm, kk;
      if (sak == 1) { mm = e >> 9; kk = e & (kKS - 1); } else { kk = e >> 4; mm = e & 15; }
      As[kk * 16 + mm] = v[q];
    }
  }
}

// B slice: Bs[kk*33 + nn] = B(k0+kk, n0+nn) (zero outside).
template <class TB>
__device__ __forceinline__ void stage_b(float* Bs, const TB* __restrict__ Bm, long sbk, long sbn,
                                        int k0, int K, int n0, int N) {
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    float v[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int e = threadIdx.x + (h * 16 + q) * 256;
      int kk, nn;
      if (sbn == 1) { kk = e >> 5; nn = e & 31; } else { nn = e >> 9; kk = e & (kKS - 1); }
      const int k = k0 + kk, n = n0 + nn;
      v[q] = (k < K && n < N) ? to_f(Bm[(long)k * sbk + (long)n * sbn]) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int e = threadIdx.x + (h * 16 + q) * 256;
      int kk, nn;
      if (sbn == 1) { kk = e >> 5; nn = e & 31; } else { nn = e >> 9; kk = e & (kKS - 1); }
      Bs[kk * 33 + nn] = v[q];
    }
  }
}

// acc[r] += sum over this warp's k of As[k][r] * Bs[k][lane]
__device__ __forceinline__ void mac_slice(const float* As, const float* Bs, int kn, int warp,
                                          int lane, float* acc) {
#pragma unroll 2
  for (int kk = warp; kk < kn; kk += 8) {
    const float4* a4 = reinterpret_cast<const float4*>(As + kk * 16);
    const float b = Bs[kk * 33 + lane];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 a = a4[q];
      acc[4 * q + 0] = fmaf(a.x, b, acc[4 * q + 0]);
      acc[4 * q + 1] = fmaf(a.y, b, acc[4 * q + 1]);
      acc[4 * q + 2] = fmaf(a.z, b, acc[4 * q + 2]);
      acc[4 * q + 3] = fmaf(a.w, b, acc[4 * q + 3]);
    }
  }
}

// The 8 warps' partial tiles added in warp order; thread t ends with output
// elements 2t and 2t+1 of the 16 x 32 tile (row (2t)/32, columns (2t)%32, +1).
__device__ __forceinline__ void reduce_tile(float* red, const float* acc, int warp, int lane,
                                            float& o0, float& o1) {
  __syncthreads();
#pragma unroll
  for (int r = 0; r < 16; ++r) red[warp * 512 + r * 32 + lane] = acc[r];
  __syncthreads();
  const int e = 2 * threadIdx.x;
  o0 = 0.f;
  o1 = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    o0 += red[w * 512 + e];
    o1 += red[w * 512 + e + 1];
  }
}

constexpr size_t kSmallSmem = (size_t)(kKS * 16 + kKS * 33) * sizeof(float);

// Memory rows for blocks i0 .. i0+15 of batch b, projected and shifted:
// C[b, i+1, n0 .. n0+31] = M_i W_m[:, n0 .. n0+31] (and C[b, 0] = 0).  The
// decayed scan
//   N_i = a N_{i-1} + S_i,  Z_i = a Z_{i-1} + 1,  M_i = N_i / Z_i
// (the recurrence form of M_i = sum_{j<=i} a^(i-j) S_j / sum_{j<=i} a^(i-j)) is
// recomputed per CTA from block 0 for each channel of the K slice straight
// into the A operand, so the projection needs no separate pass.  The CTAs of
// the first column tile also store M (for dW_m) and, for batch 0, Z (for the
// backward scan).  Grid (D/32, ceil(Nb/16), B).
template <class TW>
__global__ void __launch_bounds__(256)
    memory_fwd_kernel(const float* __restrict__ S, const float* __restrict__ decay,
                      const TW* __restrict__ w_m, float* __restrict__ M, float* __restrict__ Z,
                      float* __restrict__ Cmem, int Nb, int D) {
  pdl_enter();
  extern __shared__ __align__(16) float dyn[];
  float* As = dyn;
  float* Bs = dyn + kKS * 16;
  const int n0 = blockIdx.x * 32, i0 = blockIdx.y * 16, b = blockIdx.z;
  const int i1 = min(Nb, i0 + 16);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool keep = blockIdx.x == 0;
  float acc[16];
#pragma unroll
  for (int r = 0; r < 16; ++r) acc[r] = 0.f;
  for (int k0 = 0; k0 < D; k0 += kKS) {
    const int kn = min(kKS, D - k0);
    __syncthreads();
    stage_b<TW>(Bs, w_m, D, 1, k0, D, n0, D);  // W_m rows k0.., columns n0..n0+31
    for (int kk = threadIdx.x; kk < kKS; kk += blockDim.x) {
      const int k = k0 + kk;
      float mrow[16];
#pragma unroll
      for (int r = 0; r < 16; ++r) mrow[r] = 0.f;
      if (kk < kn) {
        const float a = decay[k];
        const float* Sk = S + (long)b * Nb * D + k;
        float Nn = 0.f, Zz = 0.f;
        for (int c0 = 0; c0 < i1; c0 += 16) {
          float sv[16];
#pragma unroll
          for (int u = 0; u < 16; ++u) sv[u] = (c0 + u < i1) ? Sk[(long)(c0 + u) * D] : 0.f;
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const int i = c0 + u;
            if (i < i1) {
              Nn = fmaf(a, Nn, sv[u]);
              Zz = fmaf(a, Zz, 1.0f);
              if (i >= i0) {
                const float m = Nn / Zz;
                mrow[u] = m;  // c0 == i0 whenever i >= i0 (i0 is a multiple of 16)
                if (keep) {
                  M[((long)b * Nb + i) * D + k] = m;
                  if (b == 0) Z[(long)i * D + k] = Zz;
                }
              }
            }
          }
        }
      }
      float4* dst = reinterpret_cast<float4*>(As + kk * 16);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        dst[q] = make_float4(mrow[4 * q], mrow[4 * q + 1], mrow[4 * q + 2], mrow[4 * q + 3]);
    }
    __syncthreads();
    mac_slice(As, Bs, kn, warp, lane, acc);
  }
  float o0, o1;
  reduce_tile(dyn, acc, warp, lane, o0, o1);
  const int r = (2 * threadIdx.x) >> 5, c = (2 * threadIdx.x) & 31;
  const int i = i0 + r;
  float* cb = Cmem + (long)b * Nb * D + n0 + c;
  if (i + 1 < Nb) {
    cb[(long)(i + 1) * D] = o0;
    cb[(long)(i + 1) * D + 1] = o1;
  }
  if (i0 == 0 && r == 0) {
    cb[0] = 0.f;
    cb[1] = 0.f;
  }
}

static cudaError_t opt_in_smem(const void* kern, size_t bytes, size_t* cached) {
  if (bytes <= *cached) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) *cached = bytes;
  return e;
}

cudaError_t memory_fwd(const Launch& lc, int dtype, const float* S, const float* decay,
                       const void* w_m, float* M, float* Z, float* Cmem, int B, int Nb, int D) {
  if (D % 64 != 0) return cudaErrorInvalidValue;
  dim3 grid(D / 32, (Nb + 15) / 16, B);
  static size_t attr_bytes[2] = {0, 0};
  cudaError_t e;
  if (dtype == 0) {
    e = opt_in_smem((const void*)memory_fwd_kernel<float>, kSmallSmem, &attr_bytes[0]);
    if (e == cudaSuccess)
      e = launch_k(memory_fwd_kernel<float>, grid, dim3(256), kSmallSmem, lc.stream, S, decay,
                   (const float*)w_m, M, Z, Cmem, Nb, D);
  } else {
    e = opt_in_smem((const void*)memory_fwd_kernel<bf16>, kSmallSmem, &attr_bytes[1]);
    if (e == cudaSuccess)
      e = launch_k(memory_fwd_kernel<bf16>, grid, dim3(256), kSmallSmem, lc.stream, S, decay,
                   (const bf16*)w_m, M, Z, Cmem, Nb, D);
  }
  return e != cudaSuccess ? e : cudaGetLastError();
}

// out[m, n] = sum_k A(m, k) B(k, n), A(m,k) = A[m*sam + k*sak] (fp32),
// B(k,n) = B[k*sbk + n*sbn] (fp32 or bf16), stored as TO.
template <class TB, class TO>
__global__ void __launch_bounds__(256)
    small_gemm_kernel(int Mr, int N, int K, const float* __restrict__ A, long sam, long sak,
                      const TB* __restrict__ Bm, long sbk, long sbn, TO* __restrict__ out,
                      long ldo) {
  pdl_enter();
  extern __shared__ __align__(16) float dyn[];
  float* As = dyn;
  float* Bs = dyn + kKS * 16;
  const int n0 = blockIdx.x * 32, m0 = blockIdx.y * 16;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float acc[16];
#pragma unroll
  for (int r = 0; r < 16; ++r) acc[r] = 0.f;
  for (int k0 = 0; k0 < K; k0 += kKS) {
    __syncthreads();
    stage_a(As, A, sam, sak, m0, Mr, k0, K);
    stage_b<TB>(Bs, Bm, sbk, sbn, k0, K, n0, N);
    __syncthreads();
    mac_slice(As, Bs, min(kKS, K - k0), warp, lane, acc);
  }
  float o0, o1;
  reduce_tile(dyn, acc, warp, lane, o0, o1);
  const int m = m0 + ((2 * threadIdx.x) >> 5), n = n0 + ((2 * threadIdx.x) & 31);
  if (m < Mr) {
    if (n < N) out[(long)m * ldo + n] = from_f<TO>(o0);
    if (n + 1 < N) out[(long)m * ldo + n + 1] = from_f<TO>(o1);
  }
}

cudaError_t small_gemm(const Launch& lc, int dtype_b, int dtype_out, int M, int N, int K,
                       const float* A, long sam, long sak, const void* B, long sbk, long sbn,
                       void* out, long ldo) {
  dim3 grid((N + 31) / 32, (M + 15) / 16);
  static size_t attr_bytes[4] = {0, 0, 0, 0};
  const size_t smem = kSmallSmem;
  cudaError_t e;
  if (dtype_b == 0 && dtype_out == 0) {
    e = opt_in_smem((const void*)small_gemm_kernel<float, float>, smem, &attr_bytes[0]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<float, float>, grid, dim3(256), smem, lc.stream, M, N, K, A,
                   sam, sak, (const float*)B, sbk, sbn, (float*)out, ldo);
  } else if (dtype_b == 0) {
    e = opt_in_smem((const void*)small_gemm_kernel<float, bf16>, smem, &attr_bytes[1]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<float, bf16>, grid, dim3(256), smem, lc.stream, M, N, K, A,
                   sam, sak, (const float*)B, sbk, sbn, (bf16*)out, ldo);
  } else if (dtype_out == 0) {
    e = opt_in_smem((const void*)small_gemm_kernel<bf16, float>, smem, &attr_bytes[2]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<bf16, float>, grid, dim3(256), smem, lc.stream, M, N, K, A,
                   sam, sak, (const bf16*)B, sbk, sbn, (float*)out, ldo);
  } else {
    e = opt_in_smem((const void*)small_gemm_kernel<bf16, bf16>, smem, &attr_bytes[3]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<bf16, bf16>, grid, dim3(256), smem, lc.stream, M, N, K, A,
                   sam, sak, (const bf16*)B, sbk, sbn, (bf16*)out, ldo);
  }
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ----------------------------------------------------- Sec. 3.8 backward
// One thread per 4 channels of one (block i, batch b): for the block's tokens,
//   dU = dY * C_i * G * (1 - G)      (through G = sigmoid(U))
//   dC_i = sum_t dY_t * G_t          (through Y = H + G * C_i)
// and dC_i becomes dP[b, i-1] (C_i = P_{i-1}); dP[b, Nb-1] = 0.
template <class T>
__global__ void __launch_bounds__(256)
    gate_bwd_kernel(const T* __restrict__ dY, const T* __restrict__ G,
                    const float* __restrict__ Cmem, T* __restrict__ dU, float* __restrict__ dP,
                    int Tlen, int D, int L) {
  pdl_enter();
  // 8 row groups x 32 threads of 4 channels: 128 channels per CTA.
  __shared__ float part[8][128 + 4];
  const int i = blockIdx.y, b = blockIdx.z, Nb = gridDim.y;
  const int rg = threadIdx.x >> 5, cq = threadIdx.x & 31;
  const int c = blockIdx.x * 128 + cq * 4;
  const int t0 = i * L, n = min(L, Tlen - t0);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  if (c < D) {
    float cm[4];
    load4(Cmem + ((long)b * Nb + i) * D + c, cm);
    for (int r = rg; r < n; r += 8) {
      const long o = ((long)b * Tlen + t0 + r) * D + c;
      float dy[4], g[4], du[4];
      load4(dY + o, dy);
      load4(G + o, g);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        du[e] = dy[e] * cm[e] * g[e] * (1.0f - g[e]);
        acc[e] = fmaf(dy[e], g[e], acc[e]);
      }
      store4(dU + o, du);
    }
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) part[rg][cq * 4 + e] = acc[e];
  __syncthreads();
  if (threadIdx.x < 128) {
    const int cc = blockIdx.x * 128 + threadIdx.x;
    if (cc < D) {
      float t = 0.f;
#pragma unroll
      for (int g = 0; g < 8; ++g) t += part[g][threadIdx.x];
      // dC_i becomes dP[b, i-1] (C_i = P_{i-1}); block 0 writes the zero row dP[b, Nb-1]
      const long o = (i > 0) ? ((long)b * Nb + i - 1) * D + cc : ((long)b * Nb + Nb - 1) * D + cc;
      if (i == 0) t = 0.f;
      dP[o] = t;
    }
  }
}

cudaError_t gate_bwd(const Launch& lc, int dtype, const void* dY, const void* G, const float* Cmem,
                     void* dU, float* dP, int B, int T, int D, int L) {
  const int Nb = (T + L - 1) / L;
  dim3 grid((D + 127) / 128, Nb, B);
  if (dtype == 0)
    launch_k(gate_bwd_kernel<float>, dim3(grid), dim3(256), 0, lc.stream,
(const float*)dY, (const float*)G, Cmem,
                                                        (float*)dU, dP, T, D, L);
  else
    launch_k(gate_bwd_kernel<bf16>, dim3(grid), dim3(256), 0, lc.stream,
(const bf16*)dY, (const bf16*)G, Cmem,
                                                       (bf16*)dU, dP, T, D, L);
  return cudaGetLastError();
}

// ----------------------------------------------------- Sec. 3.5 backward
// One thread per (batch b, channel c): with dM = dP W_m^T already computed,
// the reverse decayed scan of M_i = N_i / Z_i,
//   R_i = dM_i / Z_i + a R_{i+1},  dS_i = R_i  (= sum_{i'>=i} a^(i'-i) dM_i' / Z_i').
__global__ void __launch_bounds__(128)
    memory_scan_bwd_kernel(const float* __restrict__ dM, const float* __restrict__ decay,
                           const float* __restrict__ Z, float* __restrict__ dS, int Nb, int D) {
  pdl_enter();
  const int c = blockIdx.x * blockDim.x + threadIdx.x, b = blockIdx.y;
  if (c >= D) return;
  const float a = decay[c];
  const long base = (long)b * Nb * D + c;
  float R = 0.f;
  constexpr int U = 8;
  for (int i1 = Nb; i1 > 0; i1 -= U) {
    float mv[U], zv[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i1 - 1 - u;
      mv[u] = (i >= 0) ? dM[base + (long)i * D] : 0.f;
      zv[u] = (i >= 0) ? Z[(long)i * D + c] : 1.f;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i1 - 1 - u;
      if (i >= 0) {
        R = fmaf(a, R, mv[u] / zv[u]);
        dS[base + (long)i * D] = R;
      }
    }
  }
}

cudaError_t memory_scan_bwd(const Launch& lc, const float* dM, const float* decay, const float* Z,
                            float* dS, int B, int Nb, int D) {
  dim3 grid((D + 127) / 128, B);
  launch_k(memory_scan_bwd_kernel, dim3(grid), dim3(128), 0, lc.stream,
dM, decay, Z, dS, Nb, D);
  return cudaGetLastError();
}

// ----------------------------------------------------- Sec. 3.4 backward
// One CTA per (block i, batch b).  With S_i = sum_t alpha_t H_t and
// alpha = softmax(s): g_t = H_t . dS_i, ds_t = alpha_t (g_t - sum_u alpha_u g_u),
// and the block's share of dW_p = sum_t ds_t H_t.
template <class T>
__global__ void __launch_bounds__(256)
    summary_bwd_kernel(const T* __restrict__ Hm, const float* __restrict__ alpha,
                       const float* __restrict__ dS, float* __restrict__ ds_out,
                       float* __restrict__ dwp_part, int Tlen, int D, int L) {
  pdl_enter();
  __shared__ float g[kMaxL];
  __shared__ float cdot;
  __shared__ float part[8][256 + 4];
  const int i = blockIdx.x, b = blockIdx.y, Nb = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const T* Hb = Hm + ((long)b * Tlen + t0) * D;
  const float* dSi = dS + ((long)b * Nb + i) * D;
  const float* ab = alpha + (long)b * Tlen + t0;
  // g_t = H_t . dS_i, one warp per row, 8 channels per lane
  for (int r = warp; r < n; r += 8) {
    float d = 0.f;
    for (int c = lane * 8; c < D; c += 256) {
      float h[8], sv[8];
      load8(Hb + (long)r * D + c, h);
      load8(dSi + c, sv);
#pragma unroll
      for (int e = 0; e < 8; ++e) d = fmaf(h[e], sv[e], d);
    }
    d = warp_sum(d);
    if (lane == 0) g[r] = d;
  }
  __syncthreads();
  if (warp == 0) {
    float acc = 0.f;
    for (int r = lane; r < n; r += 32) acc = fmaf(ab[r], g[r], acc);
    acc = warp_sum(acc);
    if (lane == 0) cdot = acc;
  }
  __syncthreads();
  const float cd = cdot;
  for (int r = threadIdx.x; r < n; r += blockDim.x) {
    const float v = ab[r] * (g[r] - cd);
    ds_out[(long)b * Tlen + t0 + r] = v;
    g[r] = v;
  }
  __syncthreads();
  // the block's share of dW_p = sum_t ds_t H_t: 8 row groups x 32 lanes x 8 channels
  const int rg = warp, co = lane;
  for (int c0 = 0; c0 < D; c0 += 256) {
    const int c = c0 + co * 8;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (c < D) {
      for (int r = rg; r < n; r += 8) {
        float h[8];
        load8(Hb + (long)r * D + c, h);
        const float w = g[r];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = fmaf(w, h[e], acc[e]);
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) part[rg][co * 8 + e] = acc[e];
    __syncthreads();
    const int cc = c0 + threadIdx.x;
    if (cc < D) {
      float t = 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q) t += part[q][threadIdx.x];
      dwp_part[((long)b * Nb + i) * D + cc] = t;
    }
    __syncthreads();
  }
}

cudaError_t summary_bwd(const Launch& lc, int dtype, const void* Hm, const float* alpha,
                        const float* dS, float* ds, float* dwp_part, int B, int T, int D, int L) {
  if (L > kMaxL) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  dim3 grid(Nb, B);
  if (dtype == 0)
    launch_k(summary_bwd_kernel<float>, dim3(grid), dim3(256), 0, lc.stream,
(const float*)Hm, alpha, dS, ds,
                                                           dwp_part, T, D, L);
  else
    launch_k(summary_bwd_kernel<bf16>, dim3(grid), dim3(256), 0, lc.stream,
(const bf16*)Hm, alpha, dS, ds, dwp_part,
                                                          T, D, L);
  return cudaGetLastError();
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
  if (dtype_out == 0)
    launch_k(reduce_rows_kernel<float>, dim3(blocks), dim3(256), 0, lc.stream,
in, rows, cols, (float*)out);
  else
    launch_k(reduce_rows_kernel<bf16>, dim3(blocks), dim3(256), 0, lc.stream,
in, rows, cols, (bf16*)out);
  return cudaGetLastError();
}

cudaError_t fill_zero(const Launch& lc, void* p, size_t bytes) {
  return cudaMemsetAsync(p, 0, bytes, lc.stream);
}

}  // namespace bcmt
