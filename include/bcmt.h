/*
 * bcmt.h -- C ABI of the GB300 (sm_103a) BCMT token mixer.
 *
 * BCMT ("Blockwise Causal Memory Transformer") replaces dense causal
 * self-attention with four steps, all computed on the GPU by this library:
 *
 *   1. dense causal multi-head attention inside each length-L block, then the
 *      output projection W_O                                       (Sec. 3.2-3.3)
 *   2. an adaptive softmax-pooled summary S_i of each block          (Sec. 3.4)
 *   3. the normalised exponential causal memory
 *        M_i = sum_{j<=i} a^(i-j) S_j / sum_{j<=i} a^(i-j),
 *      projected by W_m and shifted by one block                     (Sec. 3.5)
 *   4. broadcast of the memory to the block's tokens and gated injection
 *        Y = H + sigmoid(H W_g) * M_tokens                           (Sec. 3.7-3.8)
 *
 * and the matching backward pass (the paper trains the layer with autograd,
 * Sec. 4.1; the gradients are derived from the forward definition).
 *
 * Conventions common to every entry point
 * ---------------------------------------
 *  - All tensor pointers are DEVICE pointers owned by the caller.  The library
 *    allocates no device memory per call; the caller provides a forward
 *    workspace (bcmt_workspace_size) that carries the activations saved for
 *    the backward pass, and a backward scratch buffer (bcmt_scratch_size).
 *  - Tensors are dense, row-major, without padding: x, y, q, k, v, dy, dx ...
 *    are [B, T, D]; token (b, t) is row b*T + t.
 *  - Weights follow the paper's row-vector convention (Q = X W_Q): a weight is
 *    [D_in, D_out] row-major.  W_qkv = [W_Q | W_K | W_V] is [D, 3D].  Head i
 *    owns columns i*dh .. (i+1)*dh - 1 of Q, K, V and of Concat(heads).
 *  - dtype: every tensor except `decay` has the storage type p->dtype (fp32 or
 *    bf16); arithmetic accumulates in fp32.  `decay` is always fp32 [D], each
 *    entry in [0, 1); pass 0.8 in every entry for the paper's setting.
 *  - Pointers must be 16-byte aligned.  Requirements on shapes: B, T >= 1;
 *    H >= 1 and D % H == 0; dh = D / H a multiple of 8 and <= 128; D a
 *    multiple of 64; 1 <= L <= 1024.  Any T is accepted: the last block may be
 *    ragged (Sec. 3.2).  bf16 shapes with dh in {16, 32, 64} run the tcgen05
 *    tensor-core attention: L in {16, 32, 64, 128} on the single-tile kernels
 *    (a 128-token tile holds whole blocks), L a multiple of 128 from 256 to
 *    1024 on the key-tile-walking kernels (an online softmax over the block's
 *    128-token key tiles).  fp32 shapes, other head widths and the remaining
 *    block sizes run a SIMT attention kernel in fp32.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls are
 *    asynchronous: they validate their arguments, enqueue kernels and return.
 *    On invalid arguments nothing is launched and an error code is returned;
 *    bcmt_last_error() then describes it.
 *  - Device-side waits are bounded.  A wait that expires sets a device status
 *    word instead of hanging; it is read by bcmt_device_status(), and
 *    automatically at the end of each call when p->flags has BCMT_FLAG_CHECK
 *    (which synchronises the stream).
 */
#ifndef BCMT_H
#define BCMT_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  BCMT_OK = 0,
  BCMT_ERR_ARG = 1,         /* null pointer or out-of-range parameter value        */
  BCMT_ERR_SHAPE = 2,       /* shape violates the requirements above               */
  BCMT_ERR_ALIGN = 3,       /* a pointer is not 16-byte aligned                    */
  BCMT_ERR_CUDA = 4,        /* a CUDA runtime call or kernel launch failed         */
  BCMT_ERR_TIMEOUT = 5,     /* a bounded device-side wait expired                  */
  BCMT_ERR_UNSUPPORTED = 6  /* valid for the method, not implemented by the library */
} bcmt_status;

typedef enum { BCMT_F32 = 0, BCMT_BF16 = 1 } bcmt_dtype;

/* p->flags bits */
#define BCMT_FLAG_HONLY 1u    /* the paper's HOnly ablation (Sec. 4.5): Y = H, no summary/memory/gate */
#define BCMT_FLAG_CHECK 2u    /* synchronise at the end of the call and report device status        */
#define BCMT_FLAG_PROFILE 4u  /* record CUDA events around every kernel (bcmt_profile_read)          */

typedef struct {
  int B;           /* batch                                      */
  int T;           /* sequence length                            */
  int D;           /* model width d_model                        */
  int H;           /* attention heads h (head width dh = D / H)  */
  int L;           /* block size (Sec. 3.2)                      */
  int dtype;       /* bcmt_dtype of every tensor except decay    */
  int input_is_x;  /* 1: layer starts at x and W_qkv (Sec. 3.3); 0: at Q, K, V */
  unsigned flags;  /* BCMT_FLAG_* bits                           */
} bcmt_params;

/* Bytes of forward workspace: the activations bcmt_forward saves for
 * bcmt_backward (Q/K/V when input_is_x, attention log-sum-exp, Concat(heads),
 * H, pooling weights, summaries, memory, its projection, the gate).  Returns 0
 * for invalid parameters. */
size_t bcmt_workspace_size(const bcmt_params* p);

/* Bytes of backward scratch (temporaries of one backward call; free to reuse
 * between calls).  Returns 0 for invalid parameters. */
size_t bcmt_scratch_size(const bcmt_params* p);

/* Forward pass, Sec. 3.2-3.8.
 *   x      [B,T,D]   used iff input_is_x (else may be NULL)
 *   q,k,v  [B,T,D]   used iff !input_is_x (else may be NULL)
 *   w_qkv  [D,3D]    used iff input_is_x
 *   w_o    [D,D]     output projection W_O (Sec. 3.3)
 *   w_p    [D]       pooling score vector W_p (Sec. 3.4)
 *   w_m    [D,D]     memory projection W_m (Sec. 3.5)
 *   w_g    [D,D]     gate W_g (Sec. 3.8)
 *   decay  [D] fp32  exponential decay a per channel, each in [0,1)
 *   y      [B,T,D]   output, written
 *   workspace        bcmt_workspace_size(p) bytes, written; keep it unchanged
 *                    until the matching bcmt_backward has run
 * With BCMT_FLAG_HONLY, w_p, w_m, w_g and decay are unused and Y = H. */
bcmt_status bcmt_forward(const bcmt_params* p, const void* x, const void* q, const void* k,
                         const void* v, const void* w_qkv, const void* w_o, const void* w_p,
                         const void* w_m, const void* w_g, const float* decay, void* y,
                         void* workspace, void* stream);

/* Backward pass: gradients of sum(dy * Y) with respect to the layer inputs
 * and weights, given the workspace of the matching bcmt_forward (same p and
 * same inputs).  The paper keeps the decay fixed (Sec. 3.5); its gradient,
 * for a learned per-channel decay (named as future work in Sec. 5), is
 * returned only when d_decay is non-NULL.
 *   dy       [B,T,D]
 *   x_or_q   the forward's x when input_is_x, else its q
 *   k, v     the forward's k and v iff !input_is_x (else may be NULL)
 *   w_qkv, w_o, w_p, w_m, w_g, decay: the forward's weights (w_qkv iff
 *            input_is_x)
 *   workspace  the forward's workspace (read only)
 *   scratch    bcmt_scratch_size(p) bytes
 *   dx_or_dq [B,T,D]  dx when input_is_x, else dq
 *   dk, dv   [B,T,D]  used iff !input_is_x
 *   dw_qkv   [D,3D]   used iff input_is_x
 *   dw_o [D,D], dw_p [D], dw_m [D,D], dw_g [D,D]
 *   d_decay  [D] fp32, optional (NULL: not computed)
 * Every output is overwritten (not accumulated).  With BCMT_FLAG_HONLY,
 * dw_p, dw_m, dw_g and d_decay are set to zero. */
bcmt_status bcmt_backward(const bcmt_params* p, const void* dy, const void* x_or_q,
                          const void* k, const void* v, const void* w_qkv, const void* w_o,
                          const void* w_p, const void* w_m, const void* w_g,
                          const float* decay, const void* workspace,
                          void* scratch, void* dx_or_dq, void* dk, void* dv, void* dw_qkv,
                          void* dw_o, void* dw_p, void* dw_m, void* dw_g, float* d_decay,
                          void* stream);

/* Incremental decoding (one new token per sequence per call).  The paper
 * trains only; decoding follows from the causal structure of Sec. 3.3-3.8:
 * token t of block i = t / L attends to the earlier tokens of its block, and
 * Y_t = H_t + sigmoid(H_t W_g) * C_i with C_i = M_{i-1} W_m (zero in block 0).
 * The state carries the current block's K/V cache, the block summary
 * accumulated online (Sec. 3.4), the memory recurrence N_i = a N_{i-1} + S_i,
 * Z_i = a Z_{i-1} + 1 (Sec. 3.5) and the current memory row.  Decoding the
 * tokens 0..T-1 of a sequence in order gives the rows of bcmt_forward's Y.
 *
 * p: B sequences decoded in lockstep, D, H, L, dtype and flags as for the
 * forward (BCMT_FLAG_HONLY: Y = H); input_is_x must be 1; p->T is ignored.
 *   state  bcmt_decode_state_size(p) bytes of device memory, caller-owned;
 *          bcmt_decode_reset zeroes it to start new sequences
 *   pos    position t of the token being decoded (0, 1, 2, ... in order; the
 *          state assumes the previous call decoded pos - 1)
 *   x_t    [B, D] the token's input row per sequence
 *   weights and decay as for bcmt_forward (x-entry: w_qkv [D, 3D])
 *   y_t    [B, D] output row, written
 * Calls are asynchronous on `stream`; consecutive steps of one state must be
 * issued in order on one stream. */
size_t bcmt_decode_state_size(const bcmt_params* p);
bcmt_status bcmt_decode_reset(const bcmt_params* p, void* state, void* stream);
bcmt_status bcmt_decode_step(const bcmt_params* p, void* state, long pos, const void* x_t,
                             const void* w_qkv, const void* w_o, const void* w_p,
                             const void* w_m, const void* w_g, const float* decay, void* y_t,
                             void* stream);

/* Allocation-free backward of the intra-block attention alone (the SIMT
 * kernels of the layer's backward; the paper has no counterpart -- it is an
 * interface for callers that cannot call cudaMalloc, such as a host framework
 * that owns all device memory and hands this library only input and output
 * buffers, or a latency-critical path where an allocation's implicit device
 * synchronisation is not acceptable).  It computes dq, dk, dv from the
 * forward's q, k, v (row stride ld, head h at column h*D/H), its output o
 * [B*T, D] and log-sum-exp lse [B,H,T] fp32, and the upstream gradient dO
 * [B*T, D]; dq, dk, dv are written with row stride ld_d.  Shapes as in *p
 * (B, T, D, H, L, dtype; input_is_x and flags other than BCMT_FLAG_CHECK are
 * ignored).
 *
 * Its one scratch buffer (one fp32 per batch, head and token) is a device
 * array inside the library: 4 MiB, allocated on every GPU that loads the
 * library and held until the process exits.  B*H*T must not exceed 1048576;
 * larger shapes are rejected with BCMT_ERR_SHAPE before anything is launched.
 * The first call on a device looks up that array's device address (once per
 * device, with that device current); make that first call before any stream
 * capture.  All calls share the array and it keeps the last call's contents:
 * calls that overlap on the GPU (other streams, other threads) race on it, so
 * serialise them.  Nothing is allocated: no cudaMalloc, cudaFree or
 * allocating library routine is called. */
bcmt_status bcmt_attention_backward_noalloc(const bcmt_params* p, const void* q, const void* k,
                                            const void* v, long ld, const void* o,
                                            const float* lse, const void* dO, void* dq, void* dk,
                                            void* dv, long ld_d, void* stream);

/* Reads and clears the device status word of the current device after
 * synchronising `stream`: BCMT_OK, or BCMT_ERR_TIMEOUT if any bounded
 * device-side wait has expired since the last read. */
bcmt_status bcmt_device_status(void* stream);

/* Message describing the last error of the calling thread ("" if none). */
const char* bcmt_last_error(void);

/* Profiling (BCMT_FLAG_PROFILE): per kernel name, the number of launches and
 * the summed CUDA-event time in milliseconds recorded since the last reset.
 * Synchronises the device.  Writes up to `cap` entries; returns the number of
 * distinct kernels recorded, or -1 on error.  names[i] point to static
 * strings. */
int bcmt_profile_read(const char** names, int* launches, double* ms, int cap);
void bcmt_profile_reset(void);

#ifdef __cplusplus
}
#endif

#endif /* BCMT_H */
