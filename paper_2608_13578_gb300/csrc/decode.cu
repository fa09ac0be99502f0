// Incremental decoding: one new token per sequence per call, with the state
// that the forward of Sec. 3 implies for a causal stream (the paper trains
// only; this follows from Sec. 3.3-3.8).  Token t = pos of block i = pos / L,
// slot j = pos % L:
//   * attention over the keys of block i up to slot j (the block's K/V cache);
//   * H_t, then G_t = sigmoid(H_t W_g) and Y_t = H_t + G_t * C_i, where C_i is
//     P_{i-1} = M_{i-1} W_m (zero in block 0);
//   * the block summary accumulated online: running max m, denominator
//     sum exp(s - m) and numerator sum exp(s - m) H of the scores s = H w_p;
//   * at the last slot of a block, S_i = num / den, the memory recurrence
//     N_i = a N_{i-1} + S_i, Z_i = a Z_{i-1} + 1, M_i = N_i / Z_i, and the next
//     block's memory row C_{i+1} = M_i W_m.
// Values the full forward stores in the storage dtype (Q/K/V, Concat(heads),
// H, M) are rounded to it here too, so that a decoded token reproduces the
// forward's output row.  Batches are small: the products are vector-matrix
// products that stream each weight once (HBM-bound), on CUDA cores.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace bcmt {

namespace {
constexpr int kMaxL = 1024;

template <class T>
__device__ __forceinline__ float round_to(float v) {
  return to_f<T>(from_f<T>(v));
}
}  // namespace

// out[m, n] = sum_k A[m, k] W[k, n] (fp32 accumulate), A fp32 [M, K], W [K, N]
// row-major.  CTA: 32 columns (lane = column) x R rows of A; its 32 warps
// split K (warp g takes rows g, g+32, ...), each thread issuing all eight
// weight loads of a 256-row chunk before using them, and the warps' sums are
// added in warp order.  With round_out the result is rounded to TW.
template <class TW, int R>
__global__ void __launch_bounds__(1024)
    decode_gemv_kernel(const float* __restrict__ A, int M, int K, const TW* __restrict__ W, int N,
                       float* __restrict__ out, int round_out) {
  pdl_enter();
  constexpr int KC = 256;  // K chunk staged in shared memory
  __shared__ float sA[R][KC];
  extern __shared__ float red[];  // [32 warps][R][33]
  const int tid = threadIdx.x, lane = tid & 31, g = tid >> 5;
  const int n = blockIdx.x * 32 + lane;
  const int m0 = blockIdx.y * R;
  const int mc = min(R, M - m0);
  float acc[R];
#pragma unroll
  for (int m = 0; m < R; ++m) acc[m] = 0.f;
  for (int k0 = 0; k0 < K; k0 += KC) {
    for (int i = tid; i < R * KC; i += 1024) {
      const int m = i / KC, k = i - m * KC;
      sA[m][k] = (m < mc && k0 + k < K) ? A[(long)(m0 + m) * K + k0 + k] : 0.f;
    }
    __syncthreads();
    if (n < N) {
      const int kend = min(KC, K - k0);
      float wv[KC / 32];
#pragma unroll
      for (int u = 0; u < KC / 32; ++u) {
        const int kk = g + 32 * u;
        wv[u] = kk < kend ? to_f(W[(long)(k0 + kk) * N + n]) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < KC / 32; ++u) {
        const int kk = g + 32 * u;  // < KC; zero weight past kend
#pragma unroll
        for (int m = 0; m < R; ++m) acc[m] = fmaf(sA[m][kk], wv[u], acc[m]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int m = 0; m < R; ++m) red[(g * R + m) * 33 + lane] = acc[m];
  __syncthreads();
  for (int i = tid; i < R * 32; i += 1024) {
    const int m = i / 32, c = i - m * 32;
    const int col = blockIdx.x * 32 + c;
    if (m < mc && col < N) {
      float t = 0.f;
      for (int q = 0; q < 32; ++q) t += red[(q * R + m) * 33 + c];
      out[(long)(m0 + m) * N + col] = round_out ? round_to<TW>(t) : t;
    }
  }
}

// One CTA per (head h, sequence b): stores k, v of the new token in the
// block's cache slot j, then attends the (rounded) query over slots 0..j.
template <class T>
__global__ void __launch_bounds__(128)
    decode_attn_kernel(const float* __restrict__ qkv, T* __restrict__ Kc, T* __restrict__ Vc,
                       float* __restrict__ hhat, int D, int dh, int L, int j, float scale) {
  pdl_enter();
  __shared__ float q[128];
  __shared__ float p[kMaxL];
  __shared__ float red[2][4];
  const int h = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const float* row = qkv + (long)b * 3 * D;
  const long cache = (long)b * L * D;
  if (tid >= dh) q[tid] = 0.f;  // channels past dh multiply zero-filled key values
  for (int c = tid; c < dh; c += 128) {
    const int col = h * dh + c;
    q[c] = round_to<T>(row[col]);
    Kc[cache + (long)j * D + col] = from_f<T>(row[D + col]);
    Vc[cache + (long)j * D + col] = from_f<T>(row[2 * D + col]);
  }
  __syncthreads();
  float mx = -INFINITY;
  for (int u = tid; u <= j; u += 128) {
    // key u's row, 32 channels at a time: the four 16-byte loads go out together
    const T* kr = Kc + cache + (long)u * D + h * dh;
    float s = 0.f;
    for (int c0 = 0; c0 < dh; c0 += 32) {
      float kv[32];
#pragma unroll
      for (int q8 = 0; q8 < 4; ++q8) {
        if (c0 + 8 * q8 < dh) {
          load8(kr + c0 + 8 * q8, kv + 8 * q8);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) kv[8 * q8 + e] = 0.f;
        }
      }
#pragma unroll
      for (int e = 0; e < 32; ++e) s = fmaf(q[min(c0 + e, 127)], kv[e], s);
    }
    s *= scale;
    p[u] = s;
    mx = fmaxf(mx, s);
  }
  mx = warp_max(mx);
  if (lane == 0) red[0][warp] = mx;
  __syncthreads();
  mx = fmaxf(fmaxf(red[0][0], red[0][1]), fmaxf(red[0][2], red[0][3]));
  float sum = 0.f;
  for (int u = tid; u <= j; u += 128) {
    const float e = expf(p[u] - mx);
    p[u] = e;
    sum += e;
  }
  sum = warp_sum(sum);
  if (lane == 0) red[1][warp] = sum;
  __syncthreads();
  sum = (red[1][0] + red[1][1]) + (red[1][2] + red[1][3]);
  const float inv = 1.0f / sum;
  for (int c = tid; c < dh; c += 128) {
    const T* vc = Vc + cache + h * dh + c;
    float o = 0.f;
#pragma unroll 8
    for (int u = 0; u <= j; ++u) o = fmaf(p[u], to_f(vc[(long)u * D]), o);
    hhat[(long)b * D + h * dh + c] = round_to<T>(o * inv);
  }
}

// One CTA per sequence b.  H (already rounded), U = H W_g (fp32) -> Y; the
// online block summary; at the block's last slot the summary, the memory
// recurrence and the rounded M for the next block's projection.
template <class T>
__global__ void __launch_bounds__(256)
    decode_post_kernel(const float* __restrict__ Hr, const float* __restrict__ U,
                       const T* __restrict__ w_p, const float* __restrict__ decay,
                       float* __restrict__ Cm, float* __restrict__ pm, float* __restrict__ pden,
                       float* __restrict__ pnum, float* __restrict__ Nn, float* __restrict__ Zz,
                       float* __restrict__ Mr, T* __restrict__ y, int D, int j, int last,
                       int honly) {
  pdl_enter();
  __shared__ float red[8];
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float* h = Hr + (long)b * D;
  if (honly) {
    for (int c = tid; c < D; c += 256) y[(long)b * D + c] = from_f<T>(h[c]);
    return;
  }
  float s = 0.f;
  for (int c = tid; c < D; c += 256) s = fmaf(h[c], to_f(w_p[c]), s);
  s = warp_sum(s);
  if (lane == 0) red[warp] = s;
  __syncthreads();
  s = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) s += red[w];
  // online softmax of the block's scores (slot 0 starts a new block)
  const float m_old = j == 0 ? s : pm[b];
  const float m_new = fmaxf(m_old, s);
  const float f_old = j == 0 ? 0.f : expf(m_old - m_new);
  const float e = expf(s - m_new);
  const float den = (j == 0 ? 0.f : pden[b]) * f_old + e;
  for (int c = tid; c < D; c += 256) {
    const long o = (long)b * D + c;
    y[o] = from_f<T>(fmaf(sigmoidf_(U[o]), Cm[o], h[c]));
    const float num = (j == 0 ? 0.f : pnum[o]) * f_old + e * h[c];
    if (last) {
      const float a = decay[c];
      const float n = fmaf(a, Nn[o], num / den);
      const float z = fmaf(a, Zz[o], 1.0f);
      Nn[o] = n;
      Zz[o] = z;
      Mr[o] = round_to<T>(n / z);
    } else {
      pnum[o] = num;
    }
  }
  __syncthreads();  // every thread has read pm[b] and pden[b]
  if (tid == 0 && !last) {
    pm[b] = m_new;
    pden[b] = den;
  }
}

// ---------------------------------------------------------------- host side
namespace {
template <class TW, int R>
cudaError_t gemv_r(const Launch& lc, const float* A, int M, int K, const void* W, int N, float* out,
                   bool round_out) {
  const int smem = 32 * R * 33 * (int)sizeof(float);
  static std::atomic<unsigned long long> opted{0};
  if (smem > 48 * 1024) {
    if (cudaError_t e = smem_opt_in(decode_gemv_kernel<TW, R>, smem, &opted); e != cudaSuccess)
      return e;
  }
  dim3 grid((N + 31) / 32, (M + R - 1) / R);
  cudaError_t e = launch_k(decode_gemv_kernel<TW, R>, grid, dim3(1024), smem, lc.stream, A, M, K,
                           (const TW*)W, N, out, round_out ? 1 : 0);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <class TW>
cudaError_t gemv(const Launch& lc, const float* A, int M, int K, const void* W, int N, float* out,
                 bool round_out) {
  if (M == 1) return gemv_r<TW, 1>(lc, A, M, K, W, N, out, round_out);
  if (M <= 4) return gemv_r<TW, 4>(lc, A, M, K, W, N, out, round_out);
  return gemv_r<TW, 16>(lc, A, M, K, W, N, out, round_out);
}

template <class T>
cudaError_t step_typed(const Launch& lc, const DecodeArgs& a) {
  const int B = a.B, D = a.D, j = a.j;
  cudaError_t e;
  const float* x = a.x;
  if ((e = gemv<T>(lc, x, B, D, a.w_qkv, 3 * D, a.s.qkv, false)) != cudaSuccess) return e;
  e = launch_k(decode_attn_kernel<T>, dim3(a.H, B), dim3(128), 0, lc.stream, (const float*)a.s.qkv,
               (T*)a.s.Kc, (T*)a.s.Vc, a.s.hhat, D, a.dh, a.L, j, 1.0f / sqrtf((float)a.dh));
  if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
  if ((e = gemv<T>(lc, a.s.hhat, B, D, a.w_o, D, a.s.H, true)) != cudaSuccess) return e;
  if (!a.honly && (e = gemv<T>(lc, a.s.H, B, D, a.w_g, D, a.s.U, false)) != cudaSuccess) return e;
  const int last = (j == a.L - 1) ? 1 : 0;
  e = launch_k(decode_post_kernel<T>, dim3(B), dim3(256), 0, lc.stream, (const float*)a.s.H,
               (const float*)a.s.U, (const T*)a.w_p, a.decay, a.s.C, a.s.pm, a.s.pden, a.s.pnum,
               a.s.N, a.s.Z, a.s.Mr, (T*)a.y, D, j, last, a.honly ? 1 : 0);
  if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
  // the next block's memory row C_{i+1} = M_i W_m
  if (last && !a.honly) return gemv<T>(lc, a.s.Mr, B, D, a.w_m, D, a.s.C, false);
  return cudaSuccess;
}
}  // namespace

cudaError_t decode_step(const Launch& lc, int dtype, const DecodeArgs& a) {
  if (a.L > kMaxL || a.dh > 128) return cudaErrorInvalidValue;
  return dtype == 0 ? step_typed<float>(lc, a) : step_typed<bf16>(lc, a);
}

// The token's input row is taken as fp32 by the first product; copy (and
// widen) x_t into the state's fp32 row.
template <class T>
__global__ void __launch_bounds__(256) decode_widen_kernel(const T* __restrict__ x, float* out,
                                                           long n) {
  pdl_enter();
  for (long i = blockIdx.x * 256L + threadIdx.x; i < n; i += (long)gridDim.x * 256)
    out[i] = to_f(x[i]);
}

cudaError_t decode_widen(const Launch& lc, int dtype, const void* x, float* out, long n) {
  const int blocks = (int)std::min<long>((n + 255) / 256, 1024);
  cudaError_t e = dtype == 0 ? launch_k(decode_widen_kernel<float>, dim3(blocks), dim3(256), 0,
                                        lc.stream, (const float*)x, out, n)
                             : launch_k(decode_widen_kernel<bf16>, dim3(blocks), dim3(256), 0,
                                        lc.stream, (const bf16*)x, out, n);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace bcmt
