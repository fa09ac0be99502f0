// Host-side interface between the C-ABI layer (bcmt_api.cu) and the kernel
// translation units.  Nothing here is exported from the shared library.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>

namespace bcmt {

// Where and how a kernel is launched.
struct Launch {
  cudaStream_t stream;
  unsigned* status;  // device status word (bounded waits OR bits into it)
};

// ----------------------------------------------------------------- GEMM
// C[M,N] = A[M,K] B[K,N] with fp32 accumulation, element (m,k) of A at
// A[m*sam + k*sak] and (k,n) of B at B[k*sbk + n*sbn].  The epilogue decides
// what is stored.  N must be a multiple of 64.
enum EpiKind {
  EPI_STORE = 0,        // out[m*ldo + n] = acc                       (out dtype = dtype_out)
  EPI_PARTIAL = 1,      // out(fp32)[z*split_stride + m*ldo + n] = acc of K-split z
  EPI_GATE = 2,         // out = G = sigmoid(acc) in the storage dtype        (Sec. 3.8)
  EPI_STORE_SCORE = 5,  // EPI_STORE, plus spart[col/n][m] = sum over the n columns of acc * w_p
  // the memory-gradient product dM^T = W_m dP^T [D, B*Nb] turned into its
  // reverse decayed scan dS [B*Nb, D] (fp32, row stride ldo) by the epilogue:
  // scan_nb divides 32, scan_zinv [scan_nb, D] = 1 / Z, scan_decay [D]
  EPI_REVSCAN = 7,
  // columns [0, n_split): EPI_STORE_SCORE into out; columns [n_split, N):
  // sigmoid(acc) into out2 (row stride ldo2) -- H and the gate G in one product
  // (tcgen05 path, bf16; n_split a multiple of 64)
  EPI_HGATE = 6,
};

struct EpiArgs {
  void* out = nullptr;
  long ldo = 0;
  long split_stride = 0;
  // EPI_STORE_SCORE: partial pooling scores, [D / n, M] fp32, and w_p
  float* spart = nullptr;
  const void* w_p = nullptr;
  // EPI_HGATE: the second output and the first column that goes to it, and
  // the B operand of those columns (same strides as B, columns from 0)
  void* out2 = nullptr;
  long ldo2 = 0;
  int n_split = 0;
  const void* b2 = nullptr;
  // EPI_REVSCAN
  const float* scan_zinv = nullptr;
  const float* scan_decay = nullptr;
  int scan_nb = 0;
  // EPI_GATE on the tensor cores: at most this many persistent CTAs (0: one
  // per SM), to leave SMs to a concurrent chain of small kernels
  int max_ctas = 0;
};

// A second product of a single-CTA tcgen05 launch: out[M, N] (bf16, row
// stride ldo) = A[M, K] B[K, N] with element strides as for gemm.
struct GemmProd {
  int M, N, K;
  const void* A;
  long sam, sak;
  const void* B;
  long sbk, sbn;
  void* out;
  long ldo;
};

// Number of non-empty K-splits when K (in 64-deep slices) is cut into
// `splits` equal ranges.
int effective_splits(int K, int splits);

// dtype: 0 fp32, 1 bf16 (inputs A and B); dtype_out applies to EPI_STORE.
// splits > 1 splits K into `splits` contiguous ranges (only with EPI_PARTIAL).
cudaError_t gemm(const Launch& lc, int dtype, int dtype_out, int M, int N, int K, const void* A,
                 long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                 const EpiArgs& ea, int splits, const char** kernel_name);

// SIMT GEMM (true fp32 FMA); used for fp32 tensors and for small problems.
cudaError_t gemm_simt(const Launch& lc, int dtype, int dtype_out, int M, int N, int K,
                      const void* A, long sam, long sak, const void* B, long sbk, long sbn,
                      EpiKind epi, const EpiArgs& ea, int splits);

// tcgen05 GEMM (bf16 inputs, fp32 TMEM accumulation).  A must be either
// K-major (sak == 1) or M-major (sam == 1), B either K-major (sbk == 1) or
// N-major (sbn == 1).  Returns cudaErrorNotSupported for other layouts.
// Test hook: forces the single-CTA tcgen05 GEMM's tile width (64, 128, 256;
// 0 = chosen per shape).
extern int g_force_bn;
// The CTA-pair tcgen05 GEMM (256 x 256 tiles), EPI_STORE / EPI_PARTIAL only.
cudaError_t gemm_tc_pair(const Launch& lc, int dtype_out, int M, int N, int K, const void* A,
                         long sam, long sak, const void* B, long sbk, long sbn, EpiKind epi,
                         const EpiArgs& ea, int splits);
// One product of a grouped CTA-pair GEMM: C[M,N] = A[M,K] B[K,N] (bf16
// inputs, element strides as for gemm), written to `out` with row stride ldo
// and, for K-split partials, split_stride elements between splits.
struct PairProduct {
  int M, N, K;
  const void* A;
  long sam, sak;
  const void* B;
  long sbk, sbn;
  void* out;
  long ldo, split_stride;
  int splits;
};
// Several products in one CTA-pair launch (256 x 256 tiles, N % 256 == 0 for
// each): p0 stored as bf16 with A and B K-major (dX = dQKV W_QKV^T), then
// w[0..nw-1] (1 <= nw <= 3) as fp32 K-split partials with A and B MN-major
// (the weight gradients dW = X^T dY).  The pairs take p0's tiles, then each
// w[i]'s in order, round-robin.  cudaErrorNotSupported for other layouts.
cudaError_t gemm_tc_pair_group(const Launch& lc, const PairProduct& p0, const PairProduct* w,
                               int nw);
// The largest pair load (in 64-deep slices of a 256 x 256 tile, plus a fixed
// overhead per item) of such a group under the longest-first schedule the
// launch uses: product 0 [M0, N0] over K0, weight products i [Mw, Nw] over Kw
// split in splits[i] (round-robin, as the launch deals them, when the group
// has too many items for a schedule).
long tc2_group_makespan(int M0, int N0, int K0, const int* Mw, const int* Nw, const int* Kw,
                        const int* splits, int nw, int max_pairs);
cudaError_t gemm_tc(const Launch& lc, int dtype_out, int M, int N, int K, const void* A, long sam,
                    long sak, const void* B, long sbk, long sbn, EpiKind epi, const EpiArgs& ea,
                    int splits);
bool gemm_tc_available();
// Two bf16 products in one single-CTA tcgen05 launch, both with A K-major and
// B MN-major and plain bf16 stores: out[M, N] = A B (row stride ldo), then
// p1's tiles in the idle slots of its last wave.  cudaErrorNotSupported when
// product 0 belongs on the CTA-pair kernel or the layouts differ.
cudaError_t gemm_tc_two(const Launch& lc, int M, int N, int K, const void* A, long sam, long sak,
                        const void* B, long sbk, long sbn, void* out, long ldo,
                        const GemmProd& p1);

// The same two products in one CTA-pair launch (both N multiples of 256).
cudaError_t gemm_tc_pair_two(const Launch& lc, int M, int N, int K, const void* A, long sam,
                             long sak, const void* B, long sbk, long sbn, void* out, long ldo,
                             const GemmProd& p1);

// Sum of `splits` fp32 partial buffers of `count` elements each, in split
// order, stored in dtype_out.
cudaError_t reduce_splits(const Launch& lc, const float* part, int splits, long count, int dtype_out,
                          void* out);
// Up to three such reductions in one launch (the same dtype_out).
struct SplitSum {
  const float* part;
  int splits;
  long count;
  void* out;
};
cudaError_t reduce_splits_n(const Launch& lc, const SplitSum* segs, int n, int dtype_out);

// ------------------------------------------------------------ attention
// Intra-block causal attention (Sec. 3.3).  Q, K, V rows of token (b,t) start
// at X + (b*T + t) * ld_qkv + head*dh.  O is [B*T, ld_o] (Concat of heads),
// lse [B, H, T] fp32 (natural-log sum-exp of the scaled scores per row).
struct AttnArgs {
  const void* Q;
  const void* K;
  const void* V;
  long ld_qkv;
  void* O;
  long ld_o;
  float* lse;
  int B, T, H, dh, L;
};
cudaError_t attn_fwd_simt(const Launch& lc, int dtype, const AttnArgs& a);
// Backward: dO = dL/dO [B*T, ld_o]; Drow scratch [B, H, T] fp32; writes dQ,
// dK, dV with the row stride ld_dqkv.
struct AttnBwdArgs {
  AttnArgs f;
  const void* dO;
  float* Drow;
  void* dQ;
  void* dK;
  void* dV;
  long ld_dqkv;
};
cudaError_t attn_bwd_simt(const Launch& lc, int dtype, const AttnBwdArgs& a);
// The same backward with its Drow scratch in a static device array of
// kNoAllocDrowRows floats instead of a.Drow; B*H*T must not exceed it.
constexpr long long kNoAllocDrowRows = 1ll << 20;
cudaError_t attn_bwd_simt_noalloc(const Launch& lc, int dtype, const AttnBwdArgs& a);

cudaError_t attn_fwd_tc(const Launch& lc, const AttnArgs& a);
cudaError_t attn_bwd_tc(const Launch& lc, const AttnBwdArgs& a);
bool attn_tc_supported(int dtype, int dh, int L);
// tcgen05 attention that walks key tiles (head widths 16/32/64, L dividing or
// a multiple of 128); the backward writes Drow itself (dQ kernel first).
bool attn_fl_supported(int dtype, int dh, int L);
cudaError_t attn_fwd_fl(const Launch& lc, const AttnArgs& a);
cudaError_t attn_bwd_fl(const Launch& lc, const AttnBwdArgs& a);

// ------------------------------------------------ summary, memory, gate
// Sec. 3.4: per block, s = H w_p (summed from npart partial dot products
// spart[j * B*T + token]), alpha = softmax(s), S = H^T alpha.
cudaError_t summary_fwd(const Launch& lc, int dtype, const void* Hm, const float* spart, int npart,
                        float* alpha, float* S, int B, int T, int D, int L);
// Sec. 3.5: M = normalised decayed scan of S over blocks (fp32, plus a bf16
// copy in Mb when non-null), Z its denominator [Nb, D] and Zinv = 1 / Z.  The projection
// P = M W_m is a K-split GEMM whose psplits fp32 partials [psplits][B*Nb][D]
// the injection and the gate backward sum, with the shift C_0 = 0,
// C_i = P_{i-1}, as they read them.
cudaError_t memory_scan_fwd(const Launch& lc, const float* S, const float* decay, float* M,
                            void* Mb, float* Z, float* Zinv, int B, int Nb, int D);
// Sec. 3.5 and the projection P = M W_m in one launch (bf16; P unshifted, one
// split [B*Nb, D]; also M, Mb, Z, Zinv), for shapes memory_proj_fits accepts
// (a batch's memory rows and a weight chunk in one CTA's shared memory, a
// small projection).
bool memory_proj_fits(int dtype, int B, int Nb, int D);
cudaError_t memory_proj_fwd(const Launch& lc, const float* S, const float* decay, const void* Wm,
                            float* P, float* M, void* Mb, float* Z, float* Zinv, int B, int Nb,
                            int D);
// Backward of the gate and injection: dU = dY*C*G*(1-G) (C from the partials
// Pm of P = M W_m); dP[b,i-1] = sum over block i of dY*G (also in bf16 in dPb
// when non-null); dP[b,Nb-1] = 0.
cudaError_t gate_bwd(const Launch& lc, int dtype, const void* dY, const void* G, const float* Pm,
                     int psplits, void* dU, float* dP, void* dPb, int B, int T, int D, int L);
// Backward of the memory scan: dS_j = sum_{i>=j} a^(i-j) dM_i / Z_i, given
// dM = dP W_m^T as msplits K-split fp32 partials [msplits][B*Nb][D]; when
// da_part is non-null also the decay gradient of each batch row, da_part
// [B, D] (M is the forward's fp32 memory, read only then).
cudaError_t memory_scan_bwd(const Launch& lc, const float* dM, int msplits, const float* decay,
                            const float* Z, const float* M, float* dS, float* da_part, int B,
                            int Nb, int D);
// Backward of the pooling, in chunks of a block's rows (grid
// summary_bwd_chunks(dtype, L, D) x Nb x B): g_t = H_t . dS_blk,
// ds_t = alpha_t (g_t - S_blk . dS_blk) (Sb: the forward's summaries),
// dwp_part[(b*Nb + i) * chunks + c] = sum over the chunk of ds_t H_t, and
// dH_t += dY_t + alpha_t dS_blk + ds_t w_p in place (dH holds dU W_g^T: the
// identity path's dY joins here).
int summary_bwd_chunks(int dtype, int L, int D);
cudaError_t summary_bwd(const Launch& lc, int dtype, const void* Hm, const float* alpha,
                        const float* Sb, const float* dS, const void* w_p, const void* dY,
                        void* dH, float* ds, float* dwp_part, int B, int T, int D, int L);
// Sec. 3.7-3.8 injection: Y = H + G * C[b, t / L], C from the psplits
// partials Pm of P = M W_m (shifted by one block, C_0 = 0).
cudaError_t inject(const Launch& lc, int dtype, const void* Hm, const void* G, const float* Pm,
                   int psplits, void* Y, int B, int T, int D, int L);
// Column sums of an fp32 [rows, cols] matrix in row order, stored in dtype_out.
cudaError_t reduce_rows(const Launch& lc, const float* in, int rows, int cols, int dtype_out,
                        void* out);
cudaError_t fill_zero(const Launch& lc, void* p, size_t bytes);

// ---------------------------------------------------------- decoding
// The per-layer decoding state (caller-owned device memory, zeroed by
// bcmt_decode_reset): the current block's K/V cache in the storage dtype, the
// online block summary, the memory recurrence and the current memory row, and
// the step's fp32 temporaries.
struct DecodeState {
  void *Kc, *Vc;                    // [B, L, D] storage dtype
  float *xf, *qkv, *hhat, *H, *U;   // step temporaries: [B, D], [B, 3D], [B, D] x3
  float *pm, *pden;                 // [B]: running max and denominator of the block's scores
  float *pnum;                      // [B, D]: running numerator sum exp(s - m) H
  float *N, *Z;                     // [B, D]: N_i, Z_i of the last completed block
  float *C;                         // [B, D]: memory row of the current block
  float *Mr;                        // [B, D]: M_i rounded to the storage dtype
};
struct DecodeArgs {
  int B, D, H, dh, L, j;  // j = slot of the token in its block
  bool honly;
  const float* x;         // the token's input rows, fp32 [B, D]
  const void *w_qkv, *w_o, *w_p, *w_m, *w_g;
  const float* decay;
  void* y;                // [B, D] storage dtype
  DecodeState s;
};
cudaError_t decode_widen(const Launch& lc, int dtype, const void* x, float* out, long n);
cudaError_t decode_step(const Launch& lc, int dtype, const DecodeArgs& a);

}  // namespace bcmt
