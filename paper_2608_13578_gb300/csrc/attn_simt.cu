// Intra-block causal multi-head attention on CUDA cores (Sec. 3.3), forward
// and backward.  Used for fp32 tensors (true fp32 arithmetic) and for bf16
// shapes the tensor-core kernel does not cover.  One warp per query row
// (forward, dQ) or key row (dK, dV); each lane owns keys (scores) or channels
// (outputs).  Deterministic: every sum runs in a fixed order.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace bcmt {

namespace {
constexpr int kMaxL = 1024;   // longest block the SIMT kernels accept
constexpr int kMaxDh = 128;   // widest head
constexpr int kWarps = 4;
}  // namespace

// O[t] = sum_j softmax_j(q_t . k_j * scale) v_j over keys j in [blockstart(t), t].
template <class T>
__global__ void __launch_bounds__(kWarps * 32)
    attn_fwd_simt_kernel(const T* __restrict__ Q, const T* __restrict__ K, const T* __restrict__ V,
                         long ld, T* __restrict__ O, long ld_o, float* __restrict__ lse, int Tlen,
                         int H, int dh, int L, float scale) {
  pdl_enter();
  __shared__ float qs[kWarps][kMaxDh];
  __shared__ float ps[kWarps][kMaxL];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kWarps + warp, h = blockIdx.y, b = blockIdx.z;
  if (t >= Tlen) return;
  const int bs = (t / L) * L, nk = t - bs + 1;
  const long rowq = (long)b * Tlen + t;
  const int c0 = h * dh;
  for (int c = lane; c < dh; c += 32) qs[warp][c] = to_f(Q[rowq * ld + c0 + c]);
  __syncwarp();
  float mx = -INFINITY;
  for (int j = lane; j < nk; j += 32) {
    const T* kr = K + ((long)b * Tlen + bs + j) * ld + c0;
    float d = 0.f;
    for (int c = 0; c < dh; ++c) d = fmaf(qs[warp][c], to_f(kr[c]), d);
    d *= scale;
    ps[warp][j] = d;
    mx = fmaxf(mx, d);
  }
  mx = warp_max(mx);
  float sum = 0.f;
  for (int j = lane; j < nk; j += 32) {
    const float e = expf(ps[warp][j] - mx);
    ps[warp][j] = e;
    sum += e;
  }
  sum = warp_sum(sum);
  __syncwarp();
  const float inv = 1.0f / sum;
  for (int c = lane; c < dh; c += 32) {
    float acc = 0.f;
    for (int j = 0; j < nk; ++j)
      acc = fmaf(ps[warp][j], to_f(V[((long)b * Tlen + bs + j) * ld + c0 + c]), acc);
    O[rowq * ld_o + c0 + c] = from_f<T>(acc * inv);
  }
  if (lane == 0) lse[((long)b * H + h) * Tlen + t] = mx + logf(sum);
}

// Per query t: Drow_t = dO_t . O_t, and
// dQ_t = scale * sum_j P_tj (dO_t . v_j - Drow_t) k_j.
template <class T>
__global__ void __launch_bounds__(kWarps * 32)
    attn_bwd_q_simt_kernel(const T* __restrict__ Q, const T* __restrict__ K,
                           const T* __restrict__ V, long ld, const T* __restrict__ O,
                           const T* __restrict__ dO, long ld_o, const float* __restrict__ lse,
                           float* __restrict__ Drow, T* __restrict__ dQ, long ld_d, int Tlen, int H,
                           int dh, int L, float scale) {
  pdl_enter();
  __shared__ float qs[kWarps][kMaxDh];
  __shared__ float gs[kWarps][kMaxDh];
  __shared__ float ds[kWarps][kMaxL];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kWarps + warp, h = blockIdx.y, b = blockIdx.z;
  if (t >= Tlen) return;
  const int bs = (t / L) * L, nk = t - bs + 1;
  const long rowq = (long)b * Tlen + t;
  const int c0 = h * dh;
  float dd = 0.f;
  for (int c = lane; c < dh; c += 32) {
    qs[warp][c] = to_f(Q[rowq * ld + c0 + c]);
    const float g = to_f(dO[rowq * ld_o + c0 + c]);
    gs[warp][c] = g;
    dd = fmaf(g, to_f(O[rowq * ld_o + c0 + c]), dd);
  }
  dd = warp_sum(dd);
  __syncwarp();
  const float lt = lse[((long)b * H + h) * Tlen + t];
  for (int j = lane; j < nk; j += 32) {
    const long rk = ((long)b * Tlen + bs + j) * ld + c0;
    float s = 0.f, dp = 0.f;
    for (int c = 0; c < dh; ++c) {
      s = fmaf(qs[warp][c], to_f(K[rk + c]), s);
      dp = fmaf(gs[warp][c], to_f(V[rk + c]), dp);
    }
    const float p = expf(s * scale - lt);
    ds[warp][j] = p * (dp - dd);
  }
  __syncwarp();
  for (int c = lane; c < dh; c += 32) {
    float acc = 0.f;
    for (int j = 0; j < nk; ++j) acc = fmaf(ds[warp][j], to_f(K[((long)b * Tlen + bs + j) * ld + c0 + c]), acc);
    dQ[rowq * ld_d + c0 + c] = from_f<T>(acc * scale);
  }
  if (lane == 0) Drow[((long)b * H + h) * Tlen + t] = dd;
}

// Per key j: dV_j = sum_t P_tj dO_t, dK_j = scale * sum_t P_tj (dO_t . v_j - Drow_t) q_t
// over queries t in [j, blockend(j)).
template <class T>
__global__ void __launch_bounds__(kWarps * 32)
    attn_bwd_kv_simt_kernel(const T* __restrict__ Q, const T* __restrict__ K,
                            const T* __restrict__ V, long ld, const T* __restrict__ dO, long ld_o,
                            const float* __restrict__ lse, const float* __restrict__ Drow,
                            T* __restrict__ dK, T* __restrict__ dV, long ld_d, int Tlen, int H,
                            int dh, int L, float scale) {
  pdl_enter();
  __shared__ float ks[kWarps][kMaxDh];
  __shared__ float vs[kWarps][kMaxDh];
  __shared__ float ps[kWarps][kMaxL];
  __shared__ float ds[kWarps][kMaxL];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.x * kWarps + warp, h = blockIdx.y, b = blockIdx.z;
  if (j >= Tlen) return;
  const int be = min((j / L) * L + L, Tlen), nq = be - j;
  const long rowk = (long)b * Tlen + j;
  const int c0 = h * dh;
  for (int c = lane; c < dh; c += 32) {
    ks[warp][c] = to_f(K[rowk * ld + c0 + c]);
    vs[warp][c] = to_f(V[rowk * ld + c0 + c]);
  }
  __syncwarp();
  const long lb = ((long)b * H + h) * Tlen;
  for (int u = lane; u < nq; u += 32) {
    const int t = j + u;
    const long rq = ((long)b * Tlen + t);
    float s = 0.f, dp = 0.f;
    for (int c = 0; c < dh; ++c) {
      s = fmaf(to_f(Q[rq * ld + c0 + c]), ks[warp][c], s);
      dp = fmaf(to_f(dO[rq * ld_o + c0 + c]), vs[warp][c], dp);
    }
    const float p = expf(s * scale - lse[lb + t]);
    ps[warp][u] = p;
    ds[warp][u] = p * (dp - Drow[lb + t]);
  }
  __syncwarp();
  for (int c = lane; c < dh; c += 32) {
    float av = 0.f, ak = 0.f;
    for (int u = 0; u < nq; ++u) {
      const long rq = (long)b * Tlen + j + u;
      av = fmaf(ps[warp][u], to_f(dO[rq * ld_o + c0 + c]), av);
      ak = fmaf(ds[warp][u], to_f(Q[rq * ld + c0 + c]), ak);
    }
    dV[rowk * ld_d + c0 + c] = from_f<T>(av);
    dK[rowk * ld_d + c0 + c] = from_f<T>(ak * scale);
  }
}

template <class T>
static cudaError_t fwd_typed(const Launch& lc, const AttnArgs& a) {
  dim3 grid((a.T + kWarps - 1) / kWarps, a.H, a.B);
  launch_k(attn_fwd_simt_kernel<T>, dim3(grid), dim3(kWarps * 32), 0, lc.stream,

      (const T*)a.Q, (const T*)a.K, (const T*)a.V, a.ld_qkv, (T*)a.O, a.ld_o, a.lse, a.T, a.H,
      a.dh, a.L, 1.0f / sqrtf((float)a.dh));
  return cudaGetLastError();
}

template <class T>
static cudaError_t bwd_typed(const Launch& lc, const AttnBwdArgs& a) {
  const AttnArgs& f = a.f;
  dim3 grid((f.T + kWarps - 1) / kWarps, f.H, f.B);
  const float scale = 1.0f / sqrtf((float)f.dh);
  launch_k(attn_bwd_q_simt_kernel<T>, dim3(grid), dim3(kWarps * 32), 0, lc.stream,

      (const T*)f.Q, (const T*)f.K, (const T*)f.V, f.ld_qkv, (const T*)f.O, (const T*)a.dO, f.ld_o,
      f.lse, a.Drow, (T*)a.dQ, a.ld_dqkv, f.T, f.H, f.dh, f.L, scale);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_k(attn_bwd_kv_simt_kernel<T>, dim3(grid), dim3(kWarps * 32), 0, lc.stream,

      (const T*)f.Q, (const T*)f.K, (const T*)f.V, f.ld_qkv, (const T*)a.dO, f.ld_o, f.lse, a.Drow,
      (T*)a.dK, (T*)a.dV, a.ld_dqkv, f.T, f.H, f.dh, f.L, scale);
  return cudaGetLastError();
}

cudaError_t attn_fwd_simt(const Launch& lc, int dtype, const AttnArgs& a) {
  if (a.dh > kMaxDh || a.L > kMaxL) return cudaErrorInvalidValue;
  return dtype == 0 ? fwd_typed<float>(lc, a) : fwd_typed<bf16>(lc, a);
}

cudaError_t attn_bwd_simt(const Launch& lc, int dtype, const AttnBwdArgs& a) {
  if (a.f.dh > kMaxDh || a.f.L > kMaxL) return cudaErrorInvalidValue;
  return dtype == 0 ? bwd_typed<float>(lc, a) : bwd_typed<bf16>(lc, a);
}

// ------------------------------------------- allocation-free backward variant
// The backward above needs one fp32 scratch value per (batch, head, token):
// Drow = dO . O, written by the dQ kernel and read by the dK/dV kernel.  For
// callers that cannot allocate device memory, this variant keeps that scratch
// in a file-scope device array instead of caller memory.  It is allocated when
// the library is loaded, once on every GPU that loads it, and held until the
// process exits.  Every call shares it, so calls that overlap on the GPU (on
// different streams, or from different threads) race on it.  The dQ kernel
// writes every entry the dK/dV kernel reads, so nothing needs clearing between
// calls even though the array keeps the last call's contents.
static __device__ __align__(256) float g_noalloc_drow[kNoAllocDrowRows];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float* g_noalloc_ptr[kMaxDevices] = {};
}  // namespace

cudaError_t attn_bwd_simt_noalloc(const Launch& lc, int dtype, const AttnBwdArgs& a) {
  if ((long long)a.f.B * a.f.H * a.f.T > kNoAllocDrowRows) return cudaErrorInvalidValue;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  float* drow = nullptr;
  {
    // Set-up, once per device with that device current: the array's name is
    // only a host-side stand-in, so look up its device address.
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_drow);
      if (e != cudaSuccess) return e;
      g_noalloc_ptr[dev] = static_cast<float*>(p);
    }
    drow = g_noalloc_ptr[dev];
  }
  AttnBwdArgs b = a;
  b.Drow = drow;
  return attn_bwd_simt(lc, dtype, b);
}

}  // namespace bcmt
