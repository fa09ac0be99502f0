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
// One CTA per (block i, batch b): s_t = H_t . w_p; alpha = softmax(s) over the
// block's tokens; S_i = sum_t alpha_t H_t.
template <class T>
__global__ void __launch_bounds__(256)
    summary_fwd_kernel(const T* __restrict__ Hm, const T* __restrict__ w_p,
                       float* __restrict__ alpha, float* __restrict__ S, int Tlen, int D, int L) {
  __shared__ float sc[kMaxL];
  __shared__ float red[2];
  const int i = blockIdx.x, b = blockIdx.y, Nb = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const T* Hb = Hm + ((long)b * Tlen + t0) * D;
  for (int r = warp; r < n; r += 8) {
    float d = 0.f;
    for (int c = lane * 4; c < D; c += 128) {
      float h[4], w[4];
      load4(Hb + (long)r * D + c, h);
      load4(w_p + c, w);
      d += h[0] * w[0] + h[1] * w[1] + h[2] * w[2] + h[3] * w[3];
    }
    d = warp_sum(d);
    if (lane == 0) sc[r] = d;
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
    alpha[(long)b * Tlen + t0 + r] = a;
    sc[r] = a;
  }
  __syncthreads();
  for (int c = threadIdx.x * 4; c < D; c += blockDim.x * 4) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int r = 0; r < n; ++r) {
      float h[4];
      load4(Hb + (long)r * D + c, h);
      const float a = sc[r];
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[e] = fmaf(a, h[e], acc[e]);
    }
    store4(S + ((long)b * Nb + i) * D + c, acc);
  }
}

cudaError_t summary_fwd(const Launch& lc, int dtype, const void* Hm, const void* w_p, float* alpha,
                        float* S, int B, int T, int D, int L) {
  if (L > kMaxL) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  dim3 grid(Nb, B);
  if (dtype == 0)
    summary_fwd_kernel<float><<<grid, 256, 0, lc.stream>>>((const float*)Hm, (const float*)w_p,
                                                           alpha, S, T, D, L);
  else
    summary_fwd_kernel<bf16><<<grid, 256, 0, lc.stream>>>((const bf16*)Hm, (const bf16*)w_p, alpha,
                                                          S, T, D, L);
  return cudaGetLastError();
}

// -------------------------------------------------------------- Sec. 3.5
// One CTA per (64 output channels, batch b).  The decayed scan
//   N_i = a N_{i-1} + S_i,  Z_i = a Z_{i-1} + 1,  M_i = N_i / Z_i
// (the recurrence form of the normalised double sum) is recomputed per
// 64-channel slice of the K dimension straight into shared memory and
// multiplied by the matching W_m slice: C[b, i+1] = M_i W_m, C[b, 0] = 0.
template <class T>
__global__ void __launch_bounds__(256)
    memory_fwd_kernel(const float* __restrict__ S, const float* __restrict__ decay,
                      const T* __restrict__ w_m, float* __restrict__ M, float* __restrict__ Z,
                      float* __restrict__ Cmem, int Nb, int D) {
  __shared__ float Ms[64][64 + 4];
  __shared__ float Ws[64][64 + 4];
  const int n0 = blockIdx.x * 64, b = blockIdx.y;
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  const bool write_m = (blockIdx.x == 0), write_z = write_m && b == 0;
  for (int ic = 0; ic < Nb; ic += 64) {
    const int iend = min(Nb, ic + 64);
    float acc[4][4];
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
    for (int kc = 0; kc < D; kc += 64) {
      if (tid < 64) {
        const int k = kc + tid;
        const float a = decay[k];
        float Nn = 0.f, Zz = 0.f;
        for (int i = 0; i < iend; ++i) {
          Nn = fmaf(a, Nn, S[((long)b * Nb + i) * D + k]);
          Zz = fmaf(a, Zz, 1.0f);
          if (i >= ic) {
            const float m = Nn / Zz;
            Ms[i - ic][tid] = m;
            if (write_m) M[((long)b * Nb + i) * D + k] = m;
            if (write_z) Z[(long)i * D + k] = Zz;
          }
        }
        for (int i = iend; i < ic + 64; ++i) Ms[i - ic][tid] = 0.f;
      }
      for (int e = tid; e < 64 * 64; e += 256) {
        const int kk = e / 64, nn = e % 64;
        Ws[kk][nn] = to_f(w_m[(long)(kc + kk) * D + n0 + nn]);
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < 64; ++kk) {
        float a[4], w[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) a[r] = Ms[ty * 4 + r][kk];
#pragma unroll
        for (int c = 0; c < 4; ++c) w[c] = Ws[kk][tx * 4 + c];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(a[r], w[c], acc[r][c]);
      }
      __syncthreads();
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int i = ic + ty * 4 + r;
      if (i + 1 < Nb) store4(Cmem + ((long)b * Nb + i + 1) * D + n0 + tx * 4, acc[r]);
    }
  }
  if (tid < 16) {
    const float zero[4] = {0.f, 0.f, 0.f, 0.f};
    store4(Cmem + (long)b * Nb * D + n0 + tid * 4, zero);
  }
}

cudaError_t memory_fwd(const Launch& lc, int dtype, const float* S, const float* decay,
                       const void* w_m, float* M, float* Z, float* Cmem, int B, int Nb, int D) {
  if (D % 64 != 0) return cudaErrorInvalidValue;
  dim3 grid(D / 64, B);
  if (dtype == 0)
    memory_fwd_kernel<float><<<grid, 256, 0, lc.stream>>>(S, decay, (const float*)w_m, M, Z, Cmem,
                                                          Nb, D);
  else
    memory_fwd_kernel<bf16><<<grid, 256, 0, lc.stream>>>(S, decay, (const bf16*)w_m, M, Z, Cmem,
                                                         Nb, D);
  return cudaGetLastError();
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
  const int c = (blockIdx.x * blockDim.x + threadIdx.x) * 4;
  const int i = blockIdx.y, b = blockIdx.z, Nb = gridDim.y;
  if (c >= D) return;
  const int t0 = i * L, n = min(L, Tlen - t0);
  float cm[4];
  load4(Cmem + ((long)b * Nb + i) * D + c, cm);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int r = 0; r < n; ++r) {
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
  if (i > 0) store4(dP + ((long)b * Nb + i - 1) * D + c, acc);
  else {
    const float zero[4] = {0.f, 0.f, 0.f, 0.f};
    store4(dP + ((long)b * Nb + Nb - 1) * D + c, zero);
  }
}

cudaError_t gate_bwd(const Launch& lc, int dtype, const void* dY, const void* G, const float* Cmem,
                     void* dU, float* dP, int B, int T, int D, int L) {
  const int Nb = (T + L - 1) / L;
  dim3 grid((D / 4 + 255) / 256, Nb, B);
  if (dtype == 0)
    gate_bwd_kernel<float><<<grid, 256, 0, lc.stream>>>((const float*)dY, (const float*)G, Cmem,
                                                        (float*)dU, dP, T, D, L);
  else
    gate_bwd_kernel<bf16><<<grid, 256, 0, lc.stream>>>((const bf16*)dY, (const bf16*)G, Cmem,
                                                       (bf16*)dU, dP, T, D, L);
  return cudaGetLastError();
}

// ----------------------------------------------------- Sec. 3.5 backward
// One CTA per (64 channels c, batch b): dM_i[c] = sum_k dP_i[k] W_m[c][k]
// (P = M W_m), then the reverse decayed scan of M_i = N_i / Z_i:
//   R_i = dM_i / Z_i + a R_{i+1},  dS_i = R_i  (= sum_{i'>=i} a^(i'-i) dM_i' / Z_i').
template <class T>
__global__ void __launch_bounds__(256)
    memory_bwd_kernel(const float* __restrict__ dP, const float* __restrict__ decay,
                      const float* __restrict__ Z, const T* __restrict__ w_m,
                      float* __restrict__ dS, int Nb, int D) {
  __shared__ float Ps[64][64 + 4];
  __shared__ float Ws[64][64 + 4];
  const int c0 = blockIdx.x * 64, b = blockIdx.y;
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  float R = 0.f;
  const float a = (tid < 64) ? decay[c0 + tid] : 0.f;
  for (int iend = Nb; iend > 0; iend -= 64) {
    const int ic = max(0, iend - 64);
    float acc[4][4];
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
    for (int kc = 0; kc < D; kc += 64) {
      for (int e = tid; e < 64 * 64; e += 256) {
        const int ii = e / 64, kk = e % 64;
        const int i = ic + ii;
        Ps[ii][kk] = (i < iend) ? dP[((long)b * Nb + i) * D + kc + kk] : 0.f;
        const int cc = e / 64, k2 = e % 64;
        Ws[k2][cc] = to_f(w_m[(long)(c0 + cc) * D + kc + k2]);
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < 64; ++kk) {
        float p[4], w[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) p[r] = Ps[ty * 4 + r][kk];
#pragma unroll
        for (int c = 0; c < 4; ++c) w[c] = Ws[kk][tx * 4 + c];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(p[r], w[c], acc[r][c]);
      }
      __syncthreads();
    }
    // stash dM for the chunk in Ps, then scan it backwards per channel
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) Ps[ty * 4 + r][tx * 4 + c] = acc[r][c];
    __syncthreads();
    if (tid < 64) {
      const int c = c0 + tid;
      for (int i = iend - 1; i >= ic; --i) {
        R = fmaf(a, R, Ps[i - ic][tid] / Z[(long)i * D + c]);
        dS[((long)b * Nb + i) * D + c] = R;
      }
    }
    __syncthreads();
  }
}

cudaError_t memory_bwd(const Launch& lc, int dtype, const float* dP, const float* decay,
                       const float* Z, const void* w_m, float* dS, int B, int Nb, int D) {
  if (D % 64 != 0) return cudaErrorInvalidValue;
  dim3 grid(D / 64, B);
  if (dtype == 0)
    memory_bwd_kernel<float><<<grid, 256, 0, lc.stream>>>(dP, decay, Z, (const float*)w_m, dS, Nb, D);
  else
    memory_bwd_kernel<bf16><<<grid, 256, 0, lc.stream>>>(dP, decay, Z, (const bf16*)w_m, dS, Nb, D);
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
  __shared__ float g[kMaxL];
  __shared__ float cdot;
  const int i = blockIdx.x, b = blockIdx.y, Nb = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const T* Hb = Hm + ((long)b * Tlen + t0) * D;
  const float* dSi = dS + ((long)b * Nb + i) * D;
  const float* ab = alpha + (long)b * Tlen + t0;
  for (int r = warp; r < n; r += 8) {
    float d = 0.f;
    for (int c = lane * 4; c < D; c += 128) {
      float h[4], s[4];
      load4(Hb + (long)r * D + c, h);
      load4(dSi + c, s);
      d += h[0] * s[0] + h[1] * s[1] + h[2] * s[2] + h[3] * s[3];
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
  __syncthreads();
  for (int r = threadIdx.x; r < n; r += blockDim.x) {
    const float v = ab[r] * (g[r] - cd);
    ds_out[(long)b * Tlen + t0 + r] = v;
    g[r] = v;
  }
  __syncthreads();
  for (int c = threadIdx.x * 4; c < D; c += blockDim.x * 4) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int r = 0; r < n; ++r) {
      float h[4];
      load4(Hb + (long)r * D + c, h);
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[e] = fmaf(g[r], h[e], acc[e]);
    }
    store4(dwp_part + ((long)b * Nb + i) * D + c, acc);
  }
}

cudaError_t summary_bwd(const Launch& lc, int dtype, const void* Hm, const float* alpha,
                        const float* dS, float* ds, float* dwp_part, int B, int T, int D, int L) {
  if (L > kMaxL) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  dim3 grid(Nb, B);
  if (dtype == 0)
    summary_bwd_kernel<float><<<grid, 256, 0, lc.stream>>>((const float*)Hm, alpha, dS, ds,
                                                           dwp_part, T, D, L);
  else
    summary_bwd_kernel<bf16><<<grid, 256, 0, lc.stream>>>((const bf16*)Hm, alpha, dS, ds, dwp_part,
                                                          T, D, L);
  return cudaGetLastError();
}

// Column sums in row order.
template <class TO>
__global__ void reduce_rows_kernel(const float* __restrict__ in, int rows, int cols,
                                   TO* __restrict__ out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  float acc = 0.f;
  for (int r = 0; r < rows; ++r) acc += in[(long)r * cols + c];
  out[c] = from_f<TO>(acc);
}

cudaError_t reduce_rows(const Launch& lc, const float* in, int rows, int cols, int dtype_out,
                        void* out) {
  const int blocks = (cols + 255) / 256;
  if (dtype_out == 0)
    reduce_rows_kernel<float><<<blocks, 256, 0, lc.stream>>>(in, rows, cols, (float*)out);
  else
    reduce_rows_kernel<bf16><<<blocks, 256, 0, lc.stream>>>(in, rows, cols, (bf16*)out);
  return cudaGetLastError();
}

cudaError_t fill_zero(const Launch& lc, void* p, size_t bytes) {
  return cudaMemsetAsync(p, 0, bytes, lc.stream);
}

}  // namespace bcmt
