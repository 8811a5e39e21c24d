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

/* Decode attention that allocates nothing. The paper has no counterpart: this entry point
 * serves callers that may not allocate device memory while they run, such as a vehicle's
 * real-time control loop that reserves all memory at start-up against a fixed budget (an
 * allocation there can block for an unbounded time or fail), or a host framework whose own
 * allocator owns the device memory.
 *
 * Computes, for one new token at position ctx-1, causal grouped-query attention over cache
 * positions [0, ctx): out[h] = sum_j softmax_j(q_h . k_gj / sqrt(head_dim)) v_gj with
 * g = h / (n_heads / n_kv_heads) — the same result vla_op_attention_prefill gives for
 * n_tokens = 1 and pos0 = ctx - 1.
 *   q        device bf16 [n_heads * head_dim] (post-rotary query)
 *   k_plane, v_plane  device bf16 [n_kv_heads][max_ctx][head_dim], 16-byte aligned
 *   out      device bf16 [n_heads * head_dim]
 * head_dim in {64, 128}; n_heads / n_kv_heads in {1, 2, 4, 8}; 1 <= ctx <= max_ctx.
 *
 * Memory: the per-split partial results go to one 2 MiB array compiled into the library
 * (present on every GPU that loads the library until the process exits); no call allocates
 * or frees memory. Limit: n_heads * (head_dim + 2) <= 524288 floats (one split must fit),
 * else VLA_ERR_SHAPE; the split count shrinks to fit the array. All calls share the array:
 * calls whose GPU work overlaps (e.g. on different streams) race on it and must be ordered
 * by the caller. The first call on a device resolves the array's device address (a
 * cudaGetSymbolAddress with that device current) and reads its SM count; make that first
 * call before any stream capture. The address belongs to the device's CUDA context: after
 * the context is destroyed and created again (cudaDeviceReset), the next call resolves it
 * anew, so that call too should come before any capture. With 152 SMs the split count never
 * needs to shrink for the array (splits * n_heads * (head_dim + 2) stays below 330,000
 * floats for every supported head grouping). Errors: INVALID_ARG, UNSUPPORTED, SHAPE, CUDA. */
vla_status vla_op_attention_decode_noalloc(const void* q, const void* k_plane, const void* v_plane, int ctx,
                                           int n_heads, int n_kv_heads, int head_dim, int max_ctx, void* out,
                                           vla_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* VLA_OPS_H */
