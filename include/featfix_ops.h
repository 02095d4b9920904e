/*
 * featfix_ops.h -- the individual kernels of the FeatFix hot path, exposed on
 * caller buffers so each can be tested and timed on its own.  The context
 * API in featfix.h composes exactly these kernels.
 *
 * Common rules: dev_* pointers are device memory on the current device and
 * stay owned by the caller; `stream` is a cudaStream_t (NULL = legacy
 * default stream); dtype is FEATFIX_DTYPE_F32 or FEATFIX_DTYPE_BF16; every
 * pointer must be 16-byte aligned and every element count that is read with
 * 16-byte vectors must keep that alignment (row strides in elements a
 * multiple of 8 for bf16, 4 for f32).  Work is enqueued asynchronously;
 * launch-configuration errors return FEATFIX_ERR_CUDA, argument errors
 * FEATFIX_ERR_INVALID_ARG, and nothing aborts or traps.
 */
#ifndef FEATFIX_OPS_H
#define FEATFIX_OPS_H

#include <stddef.h>
#include "featfix.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Draft of Eq. 2 in weight form: x[i] <- x[i] + sum_{j<n_terms} w[j]*hist[j][i]
 * for i < n.  hist[j] is the increment h^f - u stored at the j-th newest
 * refresh; w are the Taylor/Lagrange weights of featfix_plan_build
 * (n_terms = K_eff + 1 <= 4).  Arithmetic in fp32, result rounded to dtype.
 * In place on dev_x.                                                        */
FEATFIX_API featfix_status featfix_op_draft(int dtype, void* dev_x, const void* const* dev_hist, const double* w,
                                int n_terms, long long n, void* stream);

/* Scratch bytes featfix_op_verify needs for n elements.                    */
FEATFIX_API size_t featfix_op_verify_workspace(long long n);

/* Paid check at a site (Eqs. 3-5): forms h_d = u + sum_j w[j]*hist[j]
 * elementwise from the same incoming state dev_u, compares it with the exact
 * output dev_hf and writes the four sums
 *   dev_sums[0] = sum |h_d - h_f|,  dev_sums[1] = sum |h_f|,
 *   dev_sums[2] = sum (h_d - h_f)^2, dev_sums[3] = sum h_f^2
 * (double, device) with a fixed, run-to-run deterministic reduction order.
 * write_draft != 0 (Verify arm) also overwrites dev_u with h_d.  The per-CTA
 * partial sums live in dev_workspace (>= featfix_op_verify_workspace(n)
 * bytes, caller-owned).                                                     */
FEATFIX_API featfix_status featfix_op_verify(int dtype, void* dev_u, const void* const* dev_hist, const double* w,
                                 int n_terms, const void* dev_hf, long long n, int write_draft,
                                 double* dev_sums, void* dev_workspace, size_t ws_bytes, void* stream);

/* featfix_op_verify without any device allocation.  The paper has no
 * counterpart: this is a deployment convenience.
 *
 * Some callers cannot allocate device memory at all: a host application or
 * plugin framework that owns every byte of the GPU and forbids side
 * allocations, a memory-budgeted service that plans all device memory up
 * front, or a latency-critical loop where a cudaMalloc (with its implicit
 * synchronisation and possible failure) is not acceptable.  For them this
 * entry point computes exactly what featfix_op_verify computes (same sums,
 * same deterministic reduction order, same Verify-arm write of h_d) with the
 * per-cluster partial sums kept in a fixed scratch array of
 * FEATFIX_VERIFY_NOALLOC_SCRATCH_BYTES (16 KiB) compiled into the library.
 * The caller still provides dev_u, dev_hist, dev_hf and dev_sums.
 *
 *  - No cudaMalloc, cudaFree or other allocating routine is called.  Every
 *    GPU that loads the library holds the 16 KiB array until the process
 *    exits.
 *  - Every call looks up the array's device address with the calling
 *    thread's current device; the first call on a device may load the
 *    library's module there, so make that first call before any stream
 *    capture on the device.
 *  - A call needs featfix_op_verify_workspace(n) bytes of the array (one
 *    32-byte partial per 8-CTA cluster, at most 4 CTAs per SM); if that is
 *    more than 16 KiB (a GPU with more than 1024 SMs) the call returns
 *    FEATFIX_ERR_INVALID_ARG and launches nothing.
 *  - All calls, on every stream of a device, share the one array, which
 *    keeps the last call's contents.  Each launch writes every partial it
 *    reads back, so nothing needs clearing; but calls whose executions
 *    overlap on the GPU race on the array and may return wrong sums:
 *    serialise them (one stream, or events between streams).             */
#define FEATFIX_VERIFY_NOALLOC_SCRATCH_BYTES 16384
FEATFIX_API featfix_status featfix_op_verify_noalloc(int dtype, void* dev_u, const void* const* dev_hist,
                                                     const double* w, int n_terms, const void* dev_hf, long long n,
                                                     int write_draft, double* dev_sums, void* stream);

/* adaLN input of a branch: out[r,:] = LN(x[r,:]) * (1 + scale[b,:]) + shift[b,:]
 * with LN over C columns without affine (eps 1e-6), b = r / rows_per_batch,
 * shift/scale float32 rows of stride mod_stride.  x, out row-major [rows, C]. */
FEATFIX_API featfix_status featfix_op_ln_modulate(int dtype, const void* dev_x, void* dev_out, long long rows, int C,
                                      const float* dev_shift, const float* dev_scale, int mod_stride,
                                      int rows_per_batch, void* stream);

/* Linear layer with the block's fused epilogue:
 *   y = act(A W^T + bias);  out = resid + gate[b,:] * y  (or out = y)
 *   hist_out = out - hist_base                              (optional)
 * A [M,K] row-major (lda = K), W [N,K] (nn.Linear weight), bias [N] in
 * dtype; act 0 = identity, 1 = GELU (tanh); gate float32 rows of stride
 * gate_stride picked by b = row / rows_per_batch (NULL = no gate/resid);
 * resid, out, hist_base, hist_out [M,N] dtype with row stride N.  bf16 runs on
 * tcgen05 tensor cores with TMEM accumulators fed by TMA (K % 8 == 0);
 * f32 runs a CUDA-core kernel without TF32.                               */
FEATFIX_API featfix_status featfix_op_gemm(int dtype, int M, int N, int K, const void* dev_a, const void* dev_w,
                               const void* dev_bias, int act, const float* dev_gate, int gate_stride,
                               int rows_per_batch, const void* dev_resid, void* dev_out,
                               const void* dev_hist_base, void* dev_hist_out, void* stream);

/* Non-causal multi-head attention softmax(q k^T / sqrt(d)) v over the joint
 * [text ; image] sequence of each sample.  dev_qkv holds, for every token row
 * (featfix_token_row layout with batch samples, n_txt text and n_img image
 * tokens), q | k | v of H heads of width d at columns [0,C), [C,2C), [2C,3C),
 * row stride ld_qkv elements.  dev_out receives o [rows, C] with row stride
 * ld_out.  d % 8 == 0 and d <= 128.                                        */
FEATFIX_API featfix_status featfix_op_attention(int dtype, const void* dev_qkv, int ld_qkv, void* dev_out, int ld_out,
                                    int batch, int n_txt, int n_img, int heads, int head_dim,
                                    void* stream);

#ifdef __cplusplus
}
#endif
#endif /* FEATFIX_OPS_H */
