/*
 * vla_prefix.h — C ABI of the GB300 LLM-prefix library.
 *
 * The library runs a contiguous range [layer_begin, layer_end) of LLaMA-style decoder
 * blocks on one GPU: the "GPU-executed prefix" of block-layer partitioning (Sec. IV-B,
 * Eq. 4-6). Running [0, p) yields the boundary hidden state h^(p) of Eq. 5, which
 * vla_boundary_to_host hands to the host (the transfer T(.) of Eq. 6, sized by Eq. 11).
 * Because a block is the indivisible unit, ranges compose: [0, k) then [k, L) on the same
 * frame equals [0, L) (Eq. 6), and the split point may differ from frame to frame (the
 * scheduling zones of Sec. IV-D only move the boundary).
 *
 * Block (the paper names its stages, Sec. IV-B, not their formulas):
 *   u = RMSNorm(x) * g_attn;  q, k, v = u W_q^T, u W_k^T, u W_v^T;  rotate-half RoPE on q, k
 *   at positions pos0 + i; k, v appended to the KV cache; o = causal GQA attention;
 *   x = x + o W_o^T;  u = RMSNorm(x) * g_mlp;  x = x + (silu(u W_gate^T) * (u W_up^T)) W_down^T.
 *
 * Conventions for every call:
 *   - Tensors are bf16, row-major, contiguous. Weight matrices are [out, in].
 *   - Device pointers are CUDA device memory of the device that was current at
 *     vla_prefix_create; that device must be current for every later call.
 *   - Streams/events are cudaStream_t / cudaEvent_t (declared here as opaque pointers).
 *     NULL means the legacy default stream.
 *   - Compute calls are asynchronous on the given stream. Argument, shape and range errors
 *     are detected on the host and returned before anything is enqueued. A kernel whose
 *     bounded wait runs out records a device status read by vla_last_async_error.
 *   - No C++ exception crosses the ABI. No call takes ownership of caller memory.
 *   - Threads: drive the library from one host thread at a time (calls must not overlap;
 *     some launch paths cache kernel attributes per process without a lock). One device
 *     per process.
 */
#ifndef VLA_PREFIX_H
#define VLA_PREFIX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* vla_stream; /* == cudaStream_t */
typedef struct CUevent_st* vla_event;   /* == cudaEvent_t  */

typedef enum {
    VLA_OK = 0,
    VLA_ERR_INVALID_ARG = 1, /* null pointer, negative size, bad enum             */
    VLA_ERR_SHAPE = 2,       /* tokens or sizes outside what the object was made for */
    VLA_ERR_RANGE = 3,       /* layer range outside the model or the KV cache        */
    VLA_ERR_KV_FULL = 4,     /* the call would write past the KV cache's max_ctx     */
    VLA_ERR_NOT_PINNED = 5,  /* host destination is not page-locked                  */
    VLA_ERR_OOM = 6,         /* device or pinned allocation failed                   */
    VLA_ERR_CUDA = 7,        /* a CUDA runtime/driver call failed                    */
    VLA_ERR_TIMEOUT = 8,     /* a device-side bounded wait ran out                   */
    VLA_ERR_UNSUPPORTED = 9, /* model shape outside the supported set                */
    VLA_ERR_BUSY = 10        /* every pipeline slot is in flight (vla_cpu.h)         */
} vla_status;

/* Model shape. Supported: head_dim in {64, 128}; n_heads % n_kv_heads == 0 with
 * n_heads / n_kv_heads in {1, 2, 4, 8}; n_heads*head_dim and n_kv_heads*head_dim multiples
 * of 256; hidden a multiple of 256; ffn >= 1; rms_eps >= 0; rope_base > 1; max_ctx >= 1 is
 * the largest position count any KV cache or prefill of this object may use. */
typedef struct {
    int hidden;
    int n_heads;
    int n_kv_heads;
    int head_dim;
    int ffn;
    float rms_eps;
    float rope_base;
    int max_ctx;
} vla_config;

/* One block's weights: device bf16 pointers, [out, in] row-major.
 *   w_q [n_heads*head_dim, hidden]   w_k, w_v [n_kv_heads*head_dim, hidden]
 *   w_o [hidden, n_heads*head_dim]   w_gate, w_up [ffn, hidden]   w_down [hidden, ffn]
 *   g_attn, g_mlp [hidden] (RMSNorm gains) */
typedef struct {
    const void* w_q;
    const void* w_k;
    const void* w_v;
    const void* w_o;
    const void* w_gate;
    const void* w_up;
    const void* w_down;
    const void* g_attn;
    const void* g_mlp;
} vla_layer_weights;

typedef struct vla_prefix vla_prefix; /* model: repacked weights + workspace    */
typedef struct vla_kv vla_kv;         /* KV cache of a layer range              */

/* The ordered block list of Sec. IV-B (Eq. 4: every partition point p of the candidate set
 * splits this list). Copies `layer_count` blocks' weights into library-owned device memory
 * (fused QKV with g_attn folded in, gate/up interleaved with g_mlp folded in, W_down
 * zero-padded), allocates a workspace for up to cfg->max_ctx tokens per prefill call and the
 * rotary table. Synchronous: when it returns, the caller may free its weight buffers.
 * Errors: INVALID_ARG (null), UNSUPPORTED (shape), OOM, CUDA. *out is NULL on error. */
vla_status vla_prefix_create(const vla_config* cfg, const vla_layer_weights* weights, int layer_count,
                             vla_prefix** out);

/* Frees everything the object owns. Synchronises the device first. NULL is a no-op. */
vla_status vla_prefix_destroy(vla_prefix* p);

/* The shape `p` was created with and its block count. Either output may be NULL.
 * Errors: INVALID_ARG (p NULL). */
vla_status vla_prefix_info(const vla_prefix* p, vla_config* cfg, int* layer_count);

/* KV cache for blocks [layer_begin, layer_end) of `p`, up to max_ctx positions per layer
 * (max_ctx <= cfg.max_ctx). Layout per layer: K plane then V plane, each
 * [n_kv_heads][max_ctx][head_dim] bf16; keys are stored after the rotary embedding.
 * Library-allocated, caller-owned (vla_kv_destroy). Lengths start at 0. The decode-attention
 * launch plan for contexts up to max_ctx is fixed here (vla_kv_decode_plan).
 * Errors: INVALID_ARG, RANGE, SHAPE (max_ctx), UNSUPPORTED (no attention plan), OOM. */
vla_status vla_kv_create(vla_prefix* p, int layer_begin, int layer_end, int max_ctx, vla_kv** out);
/* The decode-attention plan of this cache: *tensor_cores = 1 for the tcgen05 kernel (head_dim
 * 128), 0 for the CUDA-core kernel; *cluster_size = CTAs per KV head (key splits, one thread-
 * block cluster); *keys_per_cta = keys one CTA holds in shared memory (tcgen05: its whole key
 * range; CUDA-core: one stage of its ring). Any output pointer may be NULL. Errors: INVALID_ARG. */
vla_status vla_kv_decode_plan(const vla_kv* kv, int* tensor_cores, int* cluster_size, int* keys_per_cta);
vla_status vla_kv_destroy(vla_kv* kv);
/* Sets every layer's length to 0 (contents are left as they are). Ordered on `stream`. */
vla_status vla_kv_reset(vla_kv* kv, vla_stream stream);
/* Minimum length over the cache's layers (host mirror); -1 if kv is NULL. */
int vla_kv_length(const vla_kv* kv);
/* Length of one layer (absolute layer index); -1 if out of range. */
int vla_kv_layer_length(const vla_kv* kv, int layer);
/* Device pointers to a layer's K and V planes (absolute layer index). */
vla_status vla_kv_data(const vla_kv* kv, int layer, void** k_plane, void** v_plane);
/* Declares positions [0, length) of every layer valid (for caches the caller filled through
 * vla_kv_data, e.g. a pre-filled context). Errors: INVALID_ARG, KV_FULL. */
vla_status vla_kv_set_length(vla_kv* kv, int length, vla_stream stream);

/* Multi-token prefill of blocks [layer_begin, layer_end) (Eq. 5 when layer_begin = 0).
 * hidden_in, hidden_out: device [n_tokens, hidden]; they may alias (in place). The frame's
 * tokens take positions p0 .. p0+n_tokens-1 where p0 is the common length of the range's
 * layers in `kv` (all must be equal, else RANGE); each layer's K/V are written there and its
 * length advances by n_tokens. hidden_out receives h^(layer_end), the residual stream after
 * the last block of the range (no final norm). An empty range copies in -> out.
 * n_tokens == 0 is a no-op. Errors: INVALID_ARG, RANGE, SHAPE (n_tokens > cfg.max_ctx),
 * KV_FULL, CUDA. */
vla_status vla_prefix_prefill(vla_prefix* p, const void* hidden_in, int n_tokens, int layer_begin, int layer_end,
                              vla_kv* kv, void* hidden_out, vla_stream stream);

/* vla_prefix_prefill that also delivers h^(layer_end) to the host without a separate copy:
 * the last block's down-projection epilogue stores each output tile both to hidden_out and,
 * through the coherent CPU-GPU link, into page-locked host memory `pinned_dst` [n_tokens,
 * hidden] bf16 (same layout). The boundary transfer T(.) of Eq. 6 then completes with the
 * kernel: once an event recorded on `stream` after this call has completed, pinned_dst
 * holds h^(layer_end). An empty range copies hidden_in to both. Errors: as prefill, plus
 * NOT_PINNED (pinned_dst not page-locked or not mapped into the device address space) and
 * INVALID_ARG (its device address not 16-byte aligned). */
vla_status vla_prefix_prefill_to_host(vla_prefix* p, const void* hidden_in, int n_tokens, int layer_begin,
                                      int layer_end, vla_kv* kv, void* hidden_out, void* pinned_dst,
                                      vla_stream stream);

/* One autoregressive step of blocks [layer_begin, layer_end) on hidden_in [1, hidden] at
 * position = the range's common KV length; appends one K/V position per layer. Same
 * aliasing, range and error rules as prefill. */
vla_status vla_prefix_decode(vla_prefix* p, const void* hidden_in, int layer_begin, int layer_end, vla_kv* kv,
                             void* hidden_out, vla_stream stream);

/* One decode step for `batch` (1..4) independent sequences at once: hidden_in / hidden_out
 * [batch, hidden] bf16 (row b = sequence b), kvs[b] = sequence b's cache (distinct caches of
 * one max_ctx, each covering the range; each sequence at its own cache's common length).
 * Every weight is streamed once for the whole batch. Each row equals what vla_prefix_decode
 * returns for that sequence alone, bit for bit. Errors: as decode, plus SHAPE (batch out of
 * range, caches of different max_ctx or first layer) and INVALID_ARG (a cache twice). */
vla_status vla_prefix_decode_batch(vla_prefix* p, const void* hidden_in, int batch, int layer_begin, int layer_end,
                                   vla_kv* const* kvs, void* hidden_out, vla_stream stream);

/* The boundary transfer T(h^(p)) of Eq. 6: copies n_tokens x hidden bf16 (Eq. 11 bytes,
 * B = 1, b = 2) from device `hidden_out` into page-locked host memory `pinned_dst` on
 * `side_stream`, after `ready` (if non-NULL) and before recording `done` (if non-NULL), so
 * the copy of frame t overlaps the prefix of frame t+1 (Sec. IV-C). The caller must not
 * overwrite hidden_out or read pinned_dst before `done`. Errors: INVALID_ARG, NOT_PINNED,
 * CUDA. */
vla_status vla_boundary_to_host(const void* hidden_out, int n_tokens, int hidden, void* pinned_dst,
                                vla_stream side_stream, vla_event ready, vla_event done);

/* Input hand-off of a frame: copies n_tokens x hidden bf16 hidden states from page-locked
 * host memory `pinned_src` into the device buffer `hidden_in` on `stream` (the tokens that
 * enter block 1 of the ordered block list, Eq. 4; in the paper's pipeline they come from the
 * vision encoder, Sec. IV-C). Asynchronous: the caller must not overwrite pinned_src before
 * work recorded on `stream` after this call has completed. Errors: INVALID_ARG, NOT_PINNED,
 * CUDA. */
vla_status vla_frame_to_device(const void* pinned_src, int n_tokens, int hidden, void* hidden_in, vla_stream stream);

/* Reads and clears the object's device status (blocking read; call after synchronising the
 * streams the object used). VLA_ERR_TIMEOUT if a kernel's bounded wait ran out. */
vla_status vla_last_async_error(vla_prefix* p);

/* Static string naming a status code. */
const char* vla_status_str(vla_status s);

/* Number of kernels the last prefill / decode call of `p` enqueued (for launch accounting). */
int vla_last_launch_count(const vla_prefix* p);

/* Measurement support (not part of the method): prefill and decode record a CUDA event pair
 * on the call's stream around every kernel of a stage whose bit (1 << stage id) is set in
 * the mask given to vla_prefix_set_timing (0 turns timing off).
 * vla_prefix_stage_times synchronises those events and returns, per stage id below, the
 * summed kernel time in milliseconds and the number of launches since the last read, then
 * clears them. Arrays have n_stages entries (VLA_STAGE_COUNT covers all). */
enum {
    VLA_STAGE_ROWSTAT = 0,      /* RMSNorm row statistics of a range's input     */
    VLA_STAGE_GEMM_QKV = 1,     /* QKV projection + RoPE + KV write (prefill)   */
    VLA_STAGE_ATTN = 2,         /* causal GQA attention (prefill)               */
    VLA_STAGE_GEMM_O = 3,       /* output projection + residual (prefill)       */
    VLA_STAGE_GEMM_GATEUP = 4,  /* gate/up projection + SwiGLU (prefill)        */
    VLA_STAGE_GEMM_DOWN = 5,    /* down projection + residual (prefill)         */
    VLA_STAGE_KV_LEN = 6,       /* KV length update (prefill: done by the QKV GEMM) */
    VLA_STAGE_DEC_QKV = 7,      /* decode: RMSNorm + QKV + RoPE + KV append      */
    VLA_STAGE_DEC_ATTN = 8,     /* decode: split-KV attention + merge            */
    VLA_STAGE_DEC_O = 9,        /* decode: output projection + residual          */
    VLA_STAGE_DEC_GATEUP = 10,  /* decode: RMSNorm + gate/up + SwiGLU            */
    VLA_STAGE_DEC_DOWN = 11,    /* decode: down projection + residual            */
    VLA_STAGE_COUNT = 12
};
vla_status vla_prefix_set_timing(vla_prefix* p, unsigned stage_mask);

/* Failure-detection test support (not part of the method): the next prefill launch of GEMM
 * stage `stage` (VLA_STAGE_GEMM_QKV, _O, _GATEUP or _DOWN) never loads the last k-block of
 * each CTA's first tile, so that kernel's bounded waits run out after wait_budget_cycles SM
 * cycles (1e5 .. 2e9; the default bound of every wait is 2e9, about 1 s). The kernel then
 * records VLA_ERR_TIMEOUT for vla_last_async_error, lets its copies in flight land, retires
 * its MMAs, releases its tensor memory and exits; the call's output is undefined, later calls
 * run normally. One launch consumes the request; stage = -1 cancels it. Errors: INVALID_ARG,
 * UNSUPPORTED (not a GEMM stage). */
vla_status vla_prefix_inject_stall(vla_prefix* p, int stage, long long wait_budget_cycles);
vla_status vla_prefix_stage_times(vla_prefix* p, float* ms_per_stage, int* launches_per_stage, int n_stages);

#ifdef __cplusplus
}
#endif

#endif /* VLA_PREFIX_H */
