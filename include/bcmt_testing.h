/*
 * bcmt_testing.h -- entry points of the BCMT library meant for its tests.
 *
 * They expose single kernels of the layer (the GEMM and the intra-block
 * attention of Sec. 3.3) so each can be checked alone against the float64
 * oracle, and let a test run the layer with the tensor-core kernels switched
 * off.  Same conventions as bcmt.h: device pointers, caller-owned memory,
 * asynchronous on `stream`, nothing allocated.
 */
#ifndef BCMT_TESTING_H
#define BCMT_TESTING_H

#include "bcmt.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Selects the kernels bcmt_forward / bcmt_backward use from now on in this
 * process: gemm_on / attn_on = 1 for the tcgen05 tensor-core kernels (the
 * default), 0 for the SIMT kernels.  Returns a bit mask of what this GPU and
 * build support: bit 0 the tcgen05 GEMM, bit 1 the tcgen05 attention.  The
 * sizes bcmt_workspace_size and bcmt_scratch_size report depend on this
 * choice (the K-split layouts differ): query them after calling it. */
int bcmt_test_set_tensor_cores(int gemm_on, int attn_on);

/* C[M,N] = A[M,K] B[K,N] with fp32 accumulation, element (m,k) of A at
 * A[m*sam + k*sak] and (k,n) of B at B[k*sbk + n*sbn] (elements, not bytes);
 * C row-major with leading dimension ldc, of type dtype_out.  impl: 0 SIMT,
 * 1 tcgen05 (bf16 inputs; A and B each K-major or MN-major; tile chosen per
 * shape), 2 the CTA-pair tcgen05 kernel (N % 256 == 0), 3 / 4 / 5 the
 * single-CTA kernel with 128- / 256- / 64-wide tiles.  With
 * splits > 1, K is cut into ranges whose fp32 partial products go to
 * C + z*M*ldc (C must then be fp32 and hold every split).  N % 64 == 0.
 * Returns the number of K-splits written, or -1 on error. */
int bcmt_test_gemm(int impl, int dtype, int dtype_out, int M, int N, int K, const void* A,
                   long sam, long sak, const void* B, long sbk, long sbn, void* C, long ldc,
                   int splits, void* stream);

/* Two or three products in one launch of the CTA-pair tcgen05 GEMM (bf16
 * inputs), the grouping the backward pass uses for dX, dW_QKV and dW_g.
 * Product 0: C0[M0,N0] = A0[M0,K0] B0[K0,N0] stored as bf16 into C0
 * (row-major, leading dimension N0), with A0 row-major (leading dimension
 * lda0) and B0 given as its transpose B0t[N0,K0] (leading dimension ldb0t):
 * both operands K-major.  Products 1 and 2: the fp32 partial products of
 * Ci[Mi,Ni] = Ai[Mi,Ki] Bi[Ki,Ni] over splits_i ranges of K (as
 * bcmt_test_gemm), split z at part_i + z*Mi*Ni, with Ai given as its transpose
 * Ait[Ki,Mi] (leading dimension lda_it) and Bi row-major (leading dimension
 * ldb_i): both operands MN-major.  M2 = 0 leaves product 2 out.  N0, N1, N2
 * multiples of 256, leading dimensions multiples of 8.  Returns the number of
 * K-splits of product 1 written, or -1 on error (bcmt_last_error()). */
int bcmt_test_gemm_group(int M0, int N0, int K0, const void* A0, long lda0, const void* B0t,
                         long ldb0t, void* C0, int M1, int N1, int K1, const void* A1t, long lda1t,
                         const void* B1, long ldb1, float* part1, int splits1, int M2, int N2,
                         int K2, const void* A2t, long lda2t, const void* B2, long ldb2,
                         float* part2, int splits2, void* stream);

/* The intra-block causal attention of Sec. 3.3 alone, forward (backward = 0)
 * or backward (backward = 1), for the shape in *p (B, T, D, H, L, dtype).
 * q, k, v: rows of token (b,t) start at q + (b*T+t)*ld, head h at column
 * h*D/H.  o [B*T, D] Concat(heads), lse [B,H,T] fp32 (written by the forward,
 * read by the backward).  Backward: dO [B*T, D]; drow [B,H,T] fp32 scratch;
 * dq, dk, dv with row stride ld_d.  impl: 0 SIMT, 1 single-tile tcgen05 (head
 * width 16/32/64, L <= 128), 2 key-tile-walking tcgen05 (head width 16/32/64, L
 * dividing or a multiple of 128; its backward also writes drow).  Returns 0, or
 * -1 on error (bcmt_last_error()). */
int bcmt_test_attn(int impl, int backward, const bcmt_params* p, const void* q, const void* k,
                   const void* v, long ld, void* o, float* lse, const void* dO, float* drow,
                   void* dq, void* dk, void* dv, long ld_d, void* stream);

/* Failure detection without a fault: launches one single-thread CTA that
 * waits on an mbarrier nothing ever arrives at, with the library's bounded
 * wait cut to `cycles` SM clock cycles (1 <= cycles <= 2^31).  The wait
 * expires, the kernel sets the timeout bit of the device status word and
 * returns normally; bcmt_device_status() then reports BCMT_ERR_TIMEOUT (and
 * clears the word).  The kernel issues no TMA copy or tcgen05 operation and
 * holds no TMEM, so the context stays usable.  Returns 0, or -1 on a bad
 * argument or launch error (bcmt_last_error()). */
int bcmt_test_wait_expiry(long long cycles, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* BCMT_TESTING_H */
