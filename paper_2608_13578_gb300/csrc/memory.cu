// Adaptive block summaries (Sec. 3.4), the normalised exponential causal
// memory with its projection and one-block shift (Sec. 3.5), and the backward
// of these two stages and of the gated injection (Sec. 3.8).
//
// This work is O(T D) and O(N_b D^2) against O(T D^2) for the projections:
// small, and on the critical path of the layer.  So each direction runs as ONE
// persistent cooperative kernel whose CTAs walk the work items of a phase and
// meet at a grid barrier before the next phase -- instead of one launch (and
// one ramp-up) per phase:
//   forward:  summaries S  |  scan + projection + shift -> C = M_causal
//   backward: gate backward (dU, dP)  |  dM = dP W_m^T  |  reverse scan -> dS
//             |  pooling backward (ds, dW_p partials)
// All reductions run in a fixed order (deterministic); rows are read with
// 16-byte vector loads.
#include "common.cuh"
#include "internal.h"

namespace bcmt {

namespace {
constexpr int kMaxL = 1024;
constexpr int kThreads = 256;
// K slice of the small CUDA-core products (a power of two)
constexpr int kKS = 256;
constexpr int kKSLog = 8;
// shared memory: the largest phase (the small products: A [kKS][16], B [kKS][33])
constexpr size_t kCoopSmem = (size_t)(kKS * 16 + kKS * 33) * sizeof(float);
}  // namespace

// ----------------------------------------------------------- grid barrier
// Self-resetting barrier of a cooperative launch: the last CTA to arrive
// clears the count and bumps the generation the others wait on.  The wait is
// bounded: on expiry it sets kStatusTimeout and the kernel stops (every CTA
// then skips its remaining phases).  `gb` = {count, generation}, zeroed by the
// host before the launch.
__device__ __forceinline__ bool grid_sync(unsigned* gb, unsigned* status, int* sflag) {
  __syncthreads();
  if (threadIdx.x == 0) {
    volatile unsigned* vgen = gb + 1;
    const unsigned gen = *vgen;
    __threadfence();
    const unsigned arrived = atomicAdd(gb, 1u) + 1u;
    int ok = 1;
    if (arrived == gridDim.x * gridDim.y * gridDim.z) {
      atomicExch(gb, 0u);
      __threadfence();
      atomicAdd(gb + 1, 1u);
    } else {
      const long long t0 = clock64();
      while (*vgen == gen) {
        if (clock64() - t0 > (1ll << 31)) {
          atomicOr(status, kStatusTimeout);
          ok = 0;
          break;
        }
        __nanosleep(64);
      }
    }
    __threadfence();
    *sflag = ok;
  }
  __syncthreads();
  return *sflag != 0;
}

// ======================================================== work items (device)
// Sec. 3.4: item (i, b, z): pooling scores of block i of batch b summed from
// the npart partial dot products the W_O epilogue wrote, alpha = softmax over
// the block (stored by z == 0), S_i[256 z .. 256 z + 255] = sum_t alpha_t H_t.
template <class T>
__device__ void summary_item(float* sm, const T* __restrict__ Hm, const float* __restrict__ spart,
                             int npart, long n_tok, float* __restrict__ alpha,
                             float* S, int Tlen, int D, int L, int Nb, int i, int b,
                             int z) {
  float* sc = sm;                 // [kMaxL]
  float* red = sm + kMaxL;        // [2]
  float* part = sm + kMaxL + 4;   // [8][260]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const long row0 = (long)b * Tlen + t0;
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
  // 8 row groups x 32 threads of 8 channels, then a fixed-order sum of the groups
  const int rg = warp, co = lane;
  const int c = z * 256 + co * 8;
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
  for (int e = 0; e < 8; ++e) part[rg * 260 + co * 8 + e] = acc[e];
  __syncthreads();
  const int cc = z * 256 + threadIdx.x;
  if (cc < D) {
    float t = 0.f;
#pragma unroll
    for (int g = 0; g < 8; ++g) t += part[g * 260 + threadIdx.x];
    S[((long)b * Nb + i) * D + cc] = t;
  }
  __syncthreads();
}

// ---- small products on CUDA cores: a 16 x 32 output tile, K split over the
// 8 warps (lane l of warp w: column l, k = w, w+8, ...); the A values of a k
// are one 64-byte broadcast, the B value one conflict-free word.  All loads of
// a K slice are issued before the first is used.
__device__ __forceinline__ void stage_a(float* As, const float* A, long sam, long sak,
                                        int m0, int Mr, int k0, int K) {
  constexpr int PER = 16 * kKS / kThreads;  // 16
  float v[PER];
#pragma unroll
  for (int q = 0; q < PER; ++q) {
    const int e = threadIdx.x + q * kThreads;
    int mm, kk;
    if (sak == 1) { mm = e >> kKSLog; kk = e & (kKS - 1); } else { kk = e >> 4; mm = e & 15; }
    const int m = m0 + mm, k = k0 + kk;
    v[q] = (m < Mr && k < K) ? __ldcg(A + (long)m * sam + (long)k * sak) : 0.f;
  }
#pragma unroll
  for (int q = 0; q < PER; ++q) {
    const int e = threadIdx.x + q * kThreads;
    int mm, kk;
    if (sak == 1) { mm = e >> kKSLog; kk = e & (kKS - 1); } else { kk = e >> 4; mm = e & 15; }
    As[kk * 16 + mm] = v[q];
  }
}

template <class TB>
__device__ __forceinline__ void stage_b(float* Bs, const TB* __restrict__ Bm, long sbk, long sbn,
                                        int k0, int K, int n0, int N) {
  constexpr int PER = 32 * kKS / kThreads;  // 32, in two halves
#pragma unroll
  for (int h = 0; h < PER / 16; ++h) {
    float v[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int e = threadIdx.x + (h * 16 + q) * kThreads;
      int kk, nn;
      if (sbn == 1) { kk = e >> 5; nn = e & 31; } else { nn = e >> kKSLog; kk = e & (kKS - 1); }
      const int k = k0 + kk, n = n0 + nn;
      v[q] = (k < K && n < N) ? to_f(Bm[(long)k * sbk + (long)n * sbn]) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int e = threadIdx.x + (h * 16 + q) * kThreads;
      int kk, nn;
      if (sbn == 1) { kk = e >> 5; nn = e & 31; } else { nn = e >> kKSLog; kk = e & (kKS - 1); }
      Bs[kk * 33 + nn] = v[q];
    }
  }
}

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
// elements 2t and 2t+1 of the 16 x 32 tile (row 2t/32, columns 2t%32, +1).
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
  __syncthreads();
}

// out[m, n] = sum_k A(m, k) B(k, n) for the tile (m0.., n0..); A fp32.
template <class TB, class TO>
__device__ void small_gemm_item(float* sm, int Mr, int N, int K, const float* A,
                                long sam, long sak, const TB* __restrict__ Bm, long sbk, long sbn,
                                TO* out, long ldo, int m0, int n0) {
  float* As = sm;
  float* Bs = sm + kKS * 16;
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
  reduce_tile(sm, acc, warp, lane, o0, o1);
  const int m = m0 + ((2 * threadIdx.x) >> 5), n = n0 + ((2 * threadIdx.x) & 31);
  if (m < Mr) {
    if (n < N) out[(long)m * ldo + n] = from_f<TO>(o0);
    if (n + 1 < N) out[(long)m * ldo + n + 1] = from_f<TO>(o1);
  }
}

// Sec. 3.5: item (x, y, b): memory rows of blocks i0 = 16y .. i0+15 of batch b,
// projected and shifted: C[b, i+1, 32x .. 32x+31] = M_i W_m (and C[b, 0] = 0).
// The decayed scan
//   N_i = a N_{i-1} + S_i,  Z_i = a Z_{i-1} + 1,  M_i = N_i / Z_i
// (the recurrence form of M_i = sum_{j<=i} a^(i-j) S_j / sum_{j<=i} a^(i-j)) is
// recomputed per item from block 0 for each channel of the K slice, straight
// into the A operand of the projection.  Items with x == 0 also store M (for
// dW_m) and, for batch 0, Z (for the backward scan).
template <class TW>
__device__ void memory_item(float* sm, const float* S, const float* __restrict__ decay,
                            const TW* __restrict__ w_m, float* __restrict__ M,
                            float* __restrict__ Z, float* __restrict__ Cmem, int Nb, int D, int x,
                            int y, int b) {
  float* As = sm;
  float* Bs = sm + kKS * 16;
  const int n0 = x * 32, i0 = y * 16;
  const int i1 = min(Nb, i0 + 16);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool keep = x == 0;
  float acc[16];
#pragma unroll
  for (int r = 0; r < 16; ++r) acc[r] = 0.f;
  for (int k0 = 0; k0 < D; k0 += kKS) {
    const int kn = min(kKS, D - k0);
    __syncthreads();
    stage_b<TW>(Bs, w_m, D, 1, k0, D, n0, D);  // W_m rows k0.., columns n0..n0+31
    for (int kk = threadIdx.x; kk < kKS; kk += kThreads) {
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
          for (int u = 0; u < 16; ++u) sv[u] = (c0 + u < i1) ? __ldcg(Sk + (long)(c0 + u) * D) : 0.f;
#pragma unroll
          for (int u = 0; u < 16; ++u) {
            const int i = c0 + u;
            if (i < i1) {
              Nn = fmaf(a, Nn, sv[u]);
              Zz = fmaf(a, Zz, 1.0f);
              if (i >= i0) {  // then c0 == i0: i0 is a multiple of 16
                const float m = Nn / Zz;
                mrow[u] = m;
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
  reduce_tile(sm, acc, warp, lane, o0, o1);
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

// Sec. 3.8 reversed: item (x, i, b): 128 channels of block i of batch b.  For
// the block's tokens dU = dY * C_i * G * (1 - G) (through G = sigmoid(U)),
// and dC_i = sum_t dY_t * G_t (through Y = H + G * C_i) becomes dP[b, i-1]
// (C_i = P_{i-1}); block 0 writes the zero row dP[b, Nb-1].
template <class T>
__device__ void gate_bwd_item(float* sm, const T* __restrict__ dY, const T* __restrict__ G,
                              const float* __restrict__ Cmem, T* __restrict__ dU,
                              float* dP, int Tlen, int D, int L, int Nb, int x, int i,
                              int b) {
  float* part = sm;  // [8][132]
  const int rg = threadIdx.x >> 5, cq = threadIdx.x & 31;
  const int c = x * 128 + cq * 4;
  const int t0 = i * L, n = min(L, Tlen - t0);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  if (c < D) {
    float cm[4];
    load4(Cmem + ((long)b * Nb + i) * D + c, cm);
    // rows rg, rg+8, ... in batches of 8: every load of a batch is issued
    // before its first store
    for (int r0 = rg; r0 < n; r0 += 64) {
      float dy[8][4], g[8][4];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int r = r0 + 8 * u;
        if (r < n) {
          const long o = ((long)b * Tlen + t0 + r) * D + c;
          load4(dY + o, dy[u]);
          load4(G + o, g[u]);
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int r = r0 + 8 * u;
        if (r < n) {
          float du[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            du[e] = dy[u][e] * cm[e] * g[u][e] * (1.0f - g[u][e]);
            acc[e] = fmaf(dy[u][e], g[u][e], acc[e]);
          }
          store4(dU + ((long)b * Tlen + t0 + r) * D + c, du);
        }
      }
    }
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) part[rg * 132 + cq * 4 + e] = acc[e];
  __syncthreads();
  if (threadIdx.x < 128) {
    const int cc = x * 128 + threadIdx.x;
    if (cc < D) {
      float t = 0.f;
#pragma unroll
      for (int g = 0; g < 8; ++g) t += part[g * 132 + threadIdx.x];
      const long o = (i > 0) ? ((long)b * Nb + i - 1) * D + cc : ((long)b * Nb + Nb - 1) * D + cc;
      dP[o] = (i > 0) ? t : 0.f;
    }
  }
  __syncthreads();
}

// Sec. 3.5 reversed: item (x, b): channels 256x .. 256x+255.  With dM = dP W_m^T,
// the reverse decayed scan of M_i = N_i / Z_i,
//   R_i = dM_i / Z_i + a R_{i+1},  dS_i = R_i  (= sum_{i'>=i} a^(i'-i) dM_i' / Z_i').
__device__ void scan_bwd_item(const float* dM, const float* __restrict__ decay,
                              const float* __restrict__ Z, float* dS, int Nb, int D,
                              int x, int b) {
  const int c = x * kThreads + threadIdx.x;
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
      mv[u] = (i >= 0) ? __ldcg(dM + base + (long)i * D) : 0.f;
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

// Sec. 3.4 reversed: item (i, b).  With S_i = sum_t alpha_t H_t and
// alpha = softmax(s): g_t = H_t . dS_i, ds_t = alpha_t (g_t - sum_u alpha_u g_u),
// and the block's share of dW_p = sum_t ds_t H_t.
template <class T>
__device__ void summary_bwd_item(float* sm, const T* __restrict__ Hm,
                                 const float* __restrict__ alpha, const float* dS,
                                 float* __restrict__ ds_out, float* __restrict__ dwp_part,
                                 int Tlen, int D, int L, int Nb, int i, int b) {
  float* g = sm;                   // [kMaxL]
  float* cdot = sm + kMaxL;        // [1]
  float* part = sm + kMaxL + 4;    // [8][260]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = i * L, n = min(L, Tlen - t0);
  const T* Hb = Hm + ((long)b * Tlen + t0) * D;
  const float* dSi = dS + ((long)b * Nb + i) * D;
  const float* ab = alpha + (long)b * Tlen + t0;
  // g_t = H_t . dS_i: warp w takes rows w, w+8, ... four at a time; all the
  // loads of a 256-channel chunk for the four rows go out together
  for (int r0 = warp; r0 < n; r0 += 32) {
    float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
    for (int c = lane * 8; c < D; c += 256) {
      float sv[8], h[4][8];
      load8_cg(dSi + c, sv);
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (r0 + 8 * u < n) load8(Hb + (long)(r0 + 8 * u) * D + c, h[u]);
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (r0 + 8 * u < n) {
#pragma unroll
          for (int e = 0; e < 8; ++e) d[u] = fmaf(h[u][e], sv[e], d[u]);
        }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float t = warp_sum(d[u]);
      if (lane == 0 && r0 + 8 * u < n) g[r0 + 8 * u] = t;
    }
  }
  __syncthreads();
  if (warp == 0) {
    float acc = 0.f;
    for (int r = lane; r < n; r += 32) acc = fmaf(ab[r], g[r], acc);
    acc = warp_sum(acc);
    if (lane == 0) *cdot = acc;
  }
  __syncthreads();
  const float cd = *cdot;
  for (int r = threadIdx.x; r < n; r += kThreads) {
    const float v = ab[r] * (g[r] - cd);
    ds_out[(long)b * Tlen + t0 + r] = v;
    g[r] = v;
  }
  __syncthreads();
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
    for (int e = 0; e < 8; ++e) part[rg * 260 + co * 8 + e] = acc[e];
    __syncthreads();
    const int cc = c0 + threadIdx.x;
    if (cc < D) {
      float t = 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q) t += part[q * 260 + threadIdx.x];
      dwp_part[((long)b * Nb + i) * D + cc] = t;
    }
    __syncthreads();
  }
}

// =========================================================== cooperative kernels
template <class T>
__global__ void __launch_bounds__(kThreads)
    memory_fwd_kernel(const T* __restrict__ Hm, const float* __restrict__ spart, int npart,
                      float* __restrict__ alpha, float* S,
                      const float* __restrict__ decay, const T* __restrict__ w_m,
                      float* __restrict__ M, float* __restrict__ Z, float* __restrict__ Cmem,
                      int B, int Tlen, int D, int L, int Nb, unsigned* gbar, unsigned* status) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int sflag;
  const long n_tok = (long)B * Tlen;
  const int nz = (D + 255) / 256;
  const int items1 = Nb * B * nz;
  for (int it = blockIdx.x; it < items1; it += gridDim.x) {
    const int z = it % nz, rest = it / nz, i = rest % Nb, b = rest / Nb;
    summary_item<T>(sm, Hm, spart, npart, n_tok, alpha, S, Tlen, D, L, Nb, i, b, z);
  }
  if (!grid_sync(gbar, status, &sflag)) return;
  const int nx = D / 32, ny = (Nb + 15) / 16;
  const int items2 = nx * ny * B;
  for (int it = blockIdx.x; it < items2; it += gridDim.x) {
    const int x = it % nx, rest = it / nx, y = rest % ny, b = rest / ny;
    memory_item<T>(sm, S, decay, w_m, M, Z, Cmem, Nb, D, x, y, b);
  }
}

template <class T>
__global__ void __launch_bounds__(kThreads)
    memory_bwd_kernel(const T* __restrict__ dY, const T* __restrict__ G,
                      const float* __restrict__ Cmem, T* __restrict__ dU, float* dP,
                      const T* __restrict__ w_m, float* dM,
                      const float* __restrict__ decay, const float* __restrict__ Z,
                      float* dS, const T* __restrict__ Hm,
                      const float* __restrict__ alpha, float* __restrict__ ds,
                      float* __restrict__ dwp_part, int B, int Tlen, int D, int L, int Nb,
                      unsigned* gbar, unsigned* status) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int sflag;
  // phase 1: gate backward
  const int nx1 = (D + 127) / 128;
  for (int it = blockIdx.x; it < nx1 * Nb * B; it += gridDim.x) {
    const int x = it % nx1, rest = it / nx1, i = rest % Nb, b = rest / Nb;
    gate_bwd_item<T>(sm, dY, G, Cmem, dU, dP, Tlen, D, L, Nb, x, i, b);
  }
  if (!grid_sync(gbar, status, &sflag)) return;
  // phase 2: dM = dP W_m^T  ([B*Nb, D] x [D, D], B(k, n) = W_m[n][k])
  const int rows = B * Nb, nxt = D / 32, nyt = (rows + 15) / 16;
  for (int it = blockIdx.x; it < nxt * nyt; it += gridDim.x) {
    const int x = it % nxt, y = it / nxt;
    small_gemm_item<T, float>(sm, rows, D, D, dP, D, 1, w_m, 1, D, dM, D, y * 16, x * 32);
  }
  if (!grid_sync(gbar, status, &sflag)) return;
  // phase 3: reverse scan -> dS
  const int nx3 = (D + kThreads - 1) / kThreads;
  for (int it = blockIdx.x; it < nx3 * B; it += gridDim.x)
    scan_bwd_item(dM, decay, Z, dS, Nb, D, it % nx3, it / nx3);
  if (!grid_sync(gbar, status, &sflag)) return;
  // phase 4: pooling backward
  for (int it = blockIdx.x; it < Nb * B; it += gridDim.x)
    summary_bwd_item<T>(sm, Hm, alpha, dS, ds, dwp_part, Tlen, D, L, Nb, it % Nb, it / Nb);
}

// ============================================================== host side
namespace {
cudaError_t opt_in_smem(const void* kern, size_t bytes, size_t* cached) {
  if (bytes <= *cached) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) *cached = bytes;
  return e;
}

// Cooperative launch of `kern` with as many CTAs as fit on the GPU at once
// (never more than `items`): the grid barrier needs every CTA resident.
template <typename... KArgs, typename... Args>
cudaError_t launch_coop(void (*kern)(KArgs...), size_t* attr_cached, int* per_sm_cached, int items,
                        cudaStream_t st, Args&&... args) {
  cudaError_t e = opt_in_smem((const void*)kern, kCoopSmem, attr_cached);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if (*per_sm_cached < 1 &&
      (e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm_cached, kern, kThreads,
                                                         kCoopSmem)) != cudaSuccess)
    return e;
  if (*per_sm_cached < 1) return cudaErrorInvalidConfiguration;
  int grid = sms * *per_sm_cached;
  if (items < grid) grid = items < 1 ? 1 : items;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kCoopSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
  return e != cudaSuccess ? e : cudaGetLastError();
}
}  // namespace

cudaError_t memory_fwd_phase(const Launch& lc, int dtype, const void* Hm, const float* spart,
                             int npart, float* alpha, float* S, const float* decay,
                             const void* w_m, float* M, float* Z, float* Cmem, unsigned* gbar,
                             int B, int T, int D, int L) {
  if (L > kMaxL || D % 64 != 0) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  cudaError_t e = cudaMemsetAsync(gbar, 0, 2 * sizeof(unsigned), lc.stream);
  if (e != cudaSuccess) return e;
  const int items = max(Nb * B * ((D + 255) / 256), (D / 32) * ((Nb + 15) / 16) * B);
  static size_t attr[2] = {0, 0};
  static int per_sm[2] = {0, 0};
  if (dtype == 0)
    return launch_coop(memory_fwd_kernel<float>, &attr[0], &per_sm[0], items, lc.stream,
                       (const float*)Hm, spart, npart, alpha, S, decay, (const float*)w_m, M, Z,
                       Cmem, B, T, D, L, Nb, gbar, lc.status);
  return launch_coop(memory_fwd_kernel<bf16>, &attr[1], &per_sm[1], items, lc.stream,
                     (const bf16*)Hm, spart, npart, alpha, S, decay, (const bf16*)w_m, M, Z, Cmem,
                     B, T, D, L, Nb, gbar, lc.status);
}

cudaError_t memory_bwd_phase(const Launch& lc, int dtype, const void* dY, const void* G,
                             const float* Cmem, void* dU, float* dP, const void* w_m, float* dM,
                             const float* decay, const float* Z, float* dS, const void* Hm,
                             const float* alpha, float* ds, float* dwp_part, unsigned* gbar, int B,
                             int T, int D, int L) {
  if (L > kMaxL || D % 64 != 0) return cudaErrorInvalidValue;
  const int Nb = (T + L - 1) / L;
  cudaError_t e = cudaMemsetAsync(gbar, 0, 2 * sizeof(unsigned), lc.stream);
  if (e != cudaSuccess) return e;
  const int items = max(((D + 127) / 128) * Nb * B, (D / 32) * ((B * Nb + 15) / 16));
  static size_t attr[2] = {0, 0};
  static int per_sm[2] = {0, 0};
  if (dtype == 0)
    return launch_coop(memory_bwd_kernel<float>, &attr[0], &per_sm[0], items, lc.stream,
                       (const float*)dY, (const float*)G, Cmem, (float*)dU, dP, (const float*)w_m,
                       dM, decay, Z, dS, (const float*)Hm, alpha, ds, dwp_part, B, T, D, L, Nb,
                       gbar, lc.status);
  return launch_coop(memory_bwd_kernel<bf16>, &attr[1], &per_sm[1], items, lc.stream,
                     (const bf16*)dY, (const bf16*)G, Cmem, (bf16*)dU, dP, (const bf16*)w_m, dM,
                     decay, Z, dS, (const bf16*)Hm, alpha, ds, dwp_part, B, T, D, L, Nb, gbar,
                     lc.status);
}

// ----------------------------------------------------- standalone products
template <class TB, class TO>
__global__ void __launch_bounds__(kThreads)
    small_gemm_kernel(int Mr, int N, int K, const float* __restrict__ A, long sam, long sak,
                      const TB* __restrict__ Bm, long sbk, long sbn, TO* __restrict__ out,
                      long ldo) {
  pdl_enter();
  extern __shared__ __align__(16) float sm[];
  small_gemm_item<TB, TO>(sm, Mr, N, K, A, sam, sak, Bm, sbk, sbn, out, ldo, blockIdx.y * 16,
                          blockIdx.x * 32);
}

cudaError_t small_gemm(const Launch& lc, int dtype_b, int dtype_out, int M, int N, int K,
                       const float* A, long sam, long sak, const void* B, long sbk, long sbn,
                       void* out, long ldo) {
  dim3 grid((N + 31) / 32, (M + 15) / 16);
  static size_t attr[4] = {0, 0, 0, 0};
  cudaError_t e;
  if (dtype_b == 0 && dtype_out == 0) {
    e = opt_in_smem((const void*)small_gemm_kernel<float, float>, kCoopSmem, &attr[0]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<float, float>, grid, dim3(kThreads), kCoopSmem, lc.stream, M,
                   N, K, A, sam, sak, (const float*)B, sbk, sbn, (float*)out, ldo);
  } else if (dtype_b == 0) {
    e = opt_in_smem((const void*)small_gemm_kernel<float, bf16>, kCoopSmem, &attr[1]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<float, bf16>, grid, dim3(kThreads), kCoopSmem, lc.stream, M,
                   N, K, A, sam, sak, (const float*)B, sbk, sbn, (bf16*)out, ldo);
  } else if (dtype_out == 0) {
    e = opt_in_smem((const void*)small_gemm_kernel<bf16, float>, kCoopSmem, &attr[2]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<bf16, float>, grid, dim3(kThreads), kCoopSmem, lc.stream, M,
                   N, K, A, sam, sak, (const bf16*)B, sbk, sbn, (float*)out, ldo);
  } else {
    e = opt_in_smem((const void*)small_gemm_kernel<bf16, bf16>, kCoopSmem, &attr[3]);
    if (e == cudaSuccess)
      e = launch_k(small_gemm_kernel<bf16, bf16>, grid, dim3(kThreads), kCoopSmem, lc.stream, M,
                   N, K, A, sam, sak, (const bf16*)B, sbk, sbn, (bf16*)out, ldo);
  }
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
