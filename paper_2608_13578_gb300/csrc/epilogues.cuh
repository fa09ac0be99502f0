// GEMM epilogues shared by the SIMT and tcgen05 GEMMs.  A GEMM hands each
// epilogue a run of n consecutive accumulator values of one output row:
// (row, col .. col+n-1), n a multiple of 4 and col a multiple of 4, plus the
// K-split index z.  Row m is token (b, t) = (m / T, m % T) of block t / L.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace bcmt {

// Besides operator() (any n, used by the SIMT GEMM), every epilogue offers a
// two-phase form for the tcgen05 GEMM's 32-column TMEM chunks: load() fetches
// the chunk's extra inputs into registers (issued a chunk ahead, and for the
// first chunk before the accumulator is ready), apply() consumes them.
// Epilogues with kTma = true only transform the 32 values in place in
// apply(); the GEMM then stages them in shared memory and writes the output
// tile (out, ldo, split_stride, element type OutT) with TMA stores.
struct NoPre {};

template <class TO>
struct EpiStoreF {
  using Pre = NoPre;
  using OutT = TO;
  static constexpr bool kTma = true;
  static constexpr bool kDual = false;
  static constexpr bool kWarpWide = false;
  TO* out;
  long ldo;
  long split_stride;
  __device__ __forceinline__ void load(int, int, Pre&) const {}
  __device__ __forceinline__ void apply(int, int, float*, const Pre&, int) const {}
  __device__ __forceinline__ void operator()(int row, int col, const float* v, int n, int z) const {
    TO* p = out + (long)z * split_stride + (long)row * ldo + col;
    if (n % 8 == 0) {
      for (int j = 0; j < n; j += 8) store8(p + j, v + j);
    } else {
      for (int j = 0; j < n; j += 4) store4(p + j, v + j);
    }
  }
};

// Sec. 3.3 + 3.4: stores H = Concat(heads) W_O and, for the pooling scores
// s = H w_p, one partial dot product per output row and run of n columns
// (spart[(col / n) * n_rows + row]); the summary kernel adds them up.
// Every epilogue below reads all of its inputs before its first store: the
// pointers may alias as far as the compiler knows, so interleaving loads and
// stores would serialise one memory round trip per vector.
template <class TO>
struct EpiStoreScoreF {
  // tcgen05 path (bf16 only): w_p as raw bf16 pairs
  struct Pre {
    uint4 w[4];
  };
  using OutT = TO;
  static constexpr bool kTma = true;
  static constexpr bool kDual = false;
  static constexpr bool kWarpWide = false;
  static constexpr long split_stride = 0;
  TO* out;
  long ldo;
  const TO* w_p;
  float* spart;
  long n_rows;
  __device__ __forceinline__ void load(int, int col, Pre& pre) const {
    const bf16* wp = reinterpret_cast<const bf16*>(w_p) + col;
#pragma unroll
    for (int j = 0; j < 4; ++j) load8_raw(wp + 8 * j, pre.w[j]);
  }
  __device__ __forceinline__ void apply(int row, int col, float* v, const Pre& pre, int) const {
    float s = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float w[8];
      unpack8(pre.w[q], w);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        s = fmaf(__bfloat162float(__float2bfloat16_rn(v[8 * q + e])), w[e], s);
    }
    spart[(long)(col / 32) * n_rows + row] = s;
  }
  __device__ __forceinline__ void operator()(int row, int col, const float* v, int n, int) const {
    float w[32];
    for (int j = 0; j < n; j += 4) load4(w_p + col + j, w + j);
    TO* p = out + (long)row * ldo + col;
    float s = 0.f;
    for (int j = 0; j < n; ++j) s = fmaf(to_f(from_f<TO>(v[j])), w[j], s);  // the stored value
    if (n % 8 == 0) {
      for (int j = 0; j < n; j += 8) store8(p + j, v + j);
    } else {
      for (int j = 0; j < n; j += 4) store4(p + j, v + j);
    }
    spart[(long)(col / n) * n_rows + row] = s;
  }
};

// Sec. 3.8 gate: G = sigmoid(H W_g) in the storage dtype.  The injection
// Y = H + G * C_blk runs as its own pass once the memory rows C are ready, so
// that this GEMM does not wait for the memory stage.
template <class T>
struct EpiGateF {
  using Pre = NoPre;
  using OutT = T;
  static constexpr bool kTma = true;
  static constexpr bool kDual = false;
  static constexpr bool kWarpWide = false;
  static constexpr long split_stride = 0;
  T* out;
  long ldo;
  __device__ __forceinline__ void load(int, int, Pre&) const {}
  __device__ __forceinline__ void apply(int, int, float* v, const Pre&, int) const {
#pragma unroll
    for (int e = 0; e < 32; ++e) v[e] = sigmoid_bf16out(v[e]);
  }
  __device__ __forceinline__ void operator()(int row, int col, const float* v, int n, int) const {
    T* p = out + (long)row * ldo + col;
    float g[32];
    for (int j = 0; j < n; ++j) g[j] = sigmoidf_(v[j]);
    if (n % 8 == 0) {
      for (int j = 0; j < n; j += 8) store8(p + j, g + j);
    } else {
      for (int j = 0; j < n; j += 4) store4(p + j, g + j);
    }
  }
};

// Sec. 3.3, 3.4 and 3.8 in one product: Concat(heads) [W_O | W_O W_g] gives
// H (columns [0, n_split)) and the gate's pre-activation U = H W_g (columns
// [n_split, N)), because H W_g = Concat (W_O W_g).  The first part is stored
// as H together with the pooling-score partials (as EpiStoreScoreF), the
// second as G = sigmoid(U) through the second output (out2, row stride ldo2,
// its own tensor map: the GEMM stores column col of the second part at
// col - n_split).  tcgen05 path only; every tile lies in one part.
template <class TO>
struct EpiHGateF {
  struct Pre {
    uint4 w[4];
  };
  using OutT = TO;
  static constexpr bool kTma = true;
  static constexpr bool kDual = true;
  static constexpr bool kWarpWide = false;
  static constexpr long split_stride = 0;
  TO* out;
  long ldo;
  const TO* w_p;
  float* spart;
  long n_rows;
  TO* out2;
  long ldo2;
  int n_split;
  __device__ __forceinline__ void load(int, int col, Pre& pre) const {
    if (col >= n_split) return;
    const bf16* wp = reinterpret_cast<const bf16*>(w_p) + col;
#pragma unroll
    for (int j = 0; j < 4; ++j) load8_raw(wp + 8 * j, pre.w[j]);
  }
  __device__ __forceinline__ void apply(int row, int col, float* v, const Pre& pre, int) const {
    if (col >= n_split) {
#pragma unroll
      for (int e = 0; e < 32; ++e) v[e] = sigmoid_bf16out(v[e]);
      return;
    }
    float s = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float w[8];
      unpack8(pre.w[q], w);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        s = fmaf(__bfloat162float(__float2bfloat16_rn(v[8 * q + e])), w[e], s);
    }
    spart[(long)(col / 32) * n_rows + row] = s;
  }
  // the SIMT GEMM does not take this epilogue (fp32 runs W_O and W_g apart)
  __device__ __forceinline__ void operator()(int, int, const float*, int, int) const {}
};

// Sec. 3.5 reversed inside the memory-gradient product, computed transposed:
// dM^T = W_m dP^T, so that an output row is one channel c and its columns
// are the blocks (b, i) in order (column b*Nb + i).  The epilogue turns each
// batch's run of Nb columns into the summary gradients
//   dS_i = sum_{j>=i} a^(j-i) dM_j / Z_j,  i.e. R_i = dM_i / Z_i + a R_{i+1},
// the backward of M_i = N_i / Z_i, N_i = a N_{i-1} + S_i, with a the channel's
// decay: a thread's 32 columns hold 32 / Nb whole batches (Nb divides 32), so
// the recurrence runs in its registers, block Nb-1 down to 0.  It stores dS
// [B*Nb, ldo] row-major itself (lanes are consecutive channels: coalesced).
// Zinv [Nb, ldo] holds 1 / Z_i (written by the forward's scan).
struct EpiRevScanT {
  using Pre = NoPre;
  using OutT = float;
  static constexpr bool kTma = false;
  static constexpr bool kDual = false;
  static constexpr bool kWarpWide = false;
  static constexpr long split_stride = 0;
  float* out;           // dS [ncols, ldo]
  long ldo;             // D
  const float* Zinv;    // [Nb, ldo]
  const float* decay;   // [ldo]
  int Nb;
  int ncols;            // B * Nb
  __device__ __forceinline__ void load(int, int, Pre&) const {}
  __device__ __forceinline__ void apply(int row, int col, float* v, const Pre&, int) const {
    // Nb divides 32 (a power of two) and col is a multiple of 32, so column
    // col + e is block (e & (Nb - 1)) of its batch; all loads go out first
    const int msk = Nb - 1;
    float zi[32];
#pragma unroll
    for (int e = 0; e < 32; ++e) zi[e] = Zinv[(long)(e & msk) * ldo + row];
    const float a = decay[row];
    float R = 0.f;
#pragma unroll
    for (int e = 31; e >= 0; --e) {
      if ((e & msk) == msk) R = 0.f;  // a batch's last block starts its run
      R = fmaf(a, R, v[e] * zi[e]);
      v[e] = R;
    }
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (col + e < ncols) out[(long)(col + e) * ldo + row] = v[e];
  }
  // the SIMT GEMM does not take this epilogue
  __device__ __forceinline__ void operator()(int, int, const float*, int, int) const {}
};

}  // namespace bcmt
