/*
 * vla_ops.h — kernel-level entry points of the GB300 LLM-prefix library.
 *
 * The same kernels vla_prefix_prefill runs, exposed one stage at a time so each can be
 * checked and timed in isolation. Conventions as in vla_prefix.h: bf16, row-major,
 * device pointers of the current device, asynchronous on `stream`, host-side argument
 * checks return before anything is enqueued.
 */
#ifndef VLA_OPS_H
#define VLA_OPS_H

#include "vla_prefix.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Projection stage of a block (QKV, output, gate/up, down projections; Sec. IV-B names
 * "projection" among a block's stages): C[M, N] = A[M, K] * B[N, K]^T with fp32 accumulation
 * on the tcgen05 tensor cores, C rounded to bf16. A, B, C are device bf16 row-major and
 * densely packed (row strides K, K, N); K must be a multiple of 8 and the base pointers
 * 16-byte aligned. M, N, K >= 1. Errors: INVALID_ARG, CUDA. */
vla_status vla_op_gemm_bf16(const void* A, const void* B, int M, int N, int K, void* C, vla_stream stream);

/* Attention stage of a block (Sec. IV-B): causal grouped-query attention of n_tokens queries
 * at positions pos0 .. pos0+n_tokens-1 over cache positions [0, pos0 + n_tokens).
 *   q        device [n_tokens, n_heads*head_dim] (post-rotary queries)
 *   k_plane, v_plane  device [n_kv_heads][max_ctx][head_dim] (one layer's cache planes)
 *   out      device [n_tokens, n_heads*head_dim]
 * Query head h reads KV head h / (n_heads / n_kv_heads); scale 1/sqrt(head_dim).
 * head_dim in {64, 128}; pos0 + n_tokens <= max_ctx. Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
vla_status vla_op_attention_prefill(const void* q, const void* k_plane, const void* v_plane, int n_tokens,
                                    int n_heads, int n_kv_heads, int head_dim, int max_ctx, int pos0, void* out,
                                    vla_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* VLA_OPS_H */
