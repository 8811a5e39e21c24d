/*
 * vla_cpu.h — the CPU-executed suffix and the cross-frame pipeline.
 *
 * Block-layer partitioning (Sec. IV-B, Eq. 6) runs blocks [0, p) on the GPU and hands the
 * boundary hidden state h^(p) to the CPU, which runs blocks [p, N). This header declares
 *   (1) the CPU side of that split: the same decoder block as vla_prefix.h, computed on the
 *       host cores from host memory (vla_cpu_model / vla_cpu_kv / vla_cpu_prefill), and
 *   (2) the cross-frame asynchronous pipeline of Sec. IV-C (Eq. 12-14): the GPU runs the
 *       prefix of frame t+1 while the CPU runs the suffix of frame t; frames are handed
 *       over through a producer-consumer queue that keeps their identities and order.
 *
 * CPU arithmetic: weights and activations are bf16 as on the GPU (the RMSNorm gains are
 * folded into the weights and rounded to bf16 the same way); products accumulate in fp32;
 * the stage outputs the GPU stores as bf16 (q, k, v, the attention output, the mid-block
 * residual, the SwiGLU product, the block output) are rounded to bf16 at the same points.
 * Results do not depend on the thread count. Softmax and SiLU use a portable four-lane exp
 * (Cody-Waite argument reduction and a degree-7 Taylor polynomial: within 2 ulp over the
 * normal fp32 range, results below it flushed to 0); the rotary angles use the C library's
 * sin / cos in double. CPU and GPU agree to rounding, not bit for bit.
 *
 * Conventions: tensors are bf16 (uint16 bit patterns), row-major, contiguous, in ordinary
 * host memory unless stated. Layer indices are absolute (block l of the model). No call
 * takes ownership of caller memory. No C++ exception crosses the ABI.
 */
#ifndef VLA_CPU_H
#define VLA_CPU_H

#include "vla_prefix.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct vla_cpu_model vla_cpu_model; /* packed host weights + thread pool + workspace */
typedef struct vla_cpu_kv vla_cpu_kv;       /* host KV cache of a layer range             */
typedef struct vla_pipeline vla_pipeline;   /* GPU prefix -> CPU suffix frame pipeline    */

/* CPU copy of blocks [layer_begin, layer_end) of a model with shape `cfg` (same rules as
 * vla_prefix_create). host_weights[i] holds block layer_begin + i, as HOST pointers, laid out
 * as in vla_layer_weights. The weights are folded and repacked into library-owned host
 * memory (2 bytes per parameter), so the caller may free its buffers when this returns.
 * n_threads >= 1 worker threads (the calling thread of a compute call takes part as one of
 * them); 0 picks the number of hardware threads. cfg->max_ctx bounds the tokens of one call
 * and every cache of the model.
 * Errors: INVALID_ARG (null, empty or negative range, n_threads < 0), UNSUPPORTED, OOM. */
vla_status vla_cpu_model_create(const vla_config* cfg, const vla_layer_weights* host_weights, int layer_begin,
                                int layer_end, int n_threads, vla_cpu_model** out);
/* Joins the threads and frees the model. NULL is a no-op. */
vla_status vla_cpu_model_destroy(vla_cpu_model* m);
/* Threads of the model's pool (including the calling thread); -1 if m is NULL. */
int vla_cpu_model_threads(const vla_cpu_model* m);
/* The model's shape and block range. Any output may be NULL. Errors: INVALID_ARG. */
vla_status vla_cpu_model_info(const vla_cpu_model* m, vla_config* cfg, int* layer_begin, int* layer_end);

/* Host KV cache for blocks [layer_begin, layer_end) (inside the model's range), up to
 * max_ctx <= cfg.max_ctx positions. Per layer a K plane then a V plane, each
 * [n_kv_heads][max_ctx][head_dim] bf16, keys after the rotary embedding (the GPU layout).
 * Lengths start at 0. Errors: INVALID_ARG, RANGE, SHAPE, OOM. */
vla_status vla_cpu_kv_create(vla_cpu_model* m, int layer_begin, int layer_end, int max_ctx, vla_cpu_kv** out);
vla_status vla_cpu_kv_destroy(vla_cpu_kv* kv);
/* Sets every layer's length to 0. */
vla_status vla_cpu_kv_reset(vla_cpu_kv* kv);
/* Minimum length over the cache's layers; -1 if kv is NULL. */
int vla_cpu_kv_length(const vla_cpu_kv* kv);
/* Host pointers to a layer's K and V planes (absolute layer index). Errors: INVALID_ARG. */
vla_status vla_cpu_kv_data(const vla_cpu_kv* kv, int layer, void** k_plane, void** v_plane);

/* Blocks [layer_begin, layer_end) on the host: the suffix B_{p+1..N}^cpu of Eq. 6 when
 * layer_begin = p and layer_end = N. hidden_in, hidden_out [n_tokens, hidden] (may alias).
 * The tokens take positions p0 .. p0+n_tokens-1, p0 = the range's common cache length (else
 * RANGE); each layer's K/V are written there. n_tokens = 1 is a decode step. An empty range
 * copies in -> out; n_tokens == 0 is a no-op. Synchronous; calls on one model are
 * serialised. Errors: INVALID_ARG, RANGE, SHAPE (n_tokens > cfg.max_ctx), KV_FULL. */
vla_status vla_cpu_prefill(vla_cpu_model* m, const void* hidden_in, int n_tokens, int layer_begin, int layer_end,
                           vla_cpu_kv* kv, void* hidden_out);

/* Per-frame stage times of the pipeline, the stage terms of Eq. 8-10:
 *   t_gpu_ms   T_G: prefix [0, p) on the GPU (CUDA events around it on the submit stream)
 *   t_xfer_ms  T_X: from the end of the prefix to the end of the boundary copy into pinned
 *              host memory (CUDA events; includes waiting for the side stream)
 *   t_cpu_ms   T_C: suffix [p, N) on the host cores (wall clock)
 *   t_submit_s, t_start_s, t_ready_s, t_done_s: host clock (seconds, steady clock of the
 *              process) when the frame was submitted, when the worker took it up (after the
 *              previous frame's suffix), when the worker saw its boundary copy complete, and
 *              when its suffix finished. t_ready_s - t_start_s is the time the CPU stage
 *              waited for the GPU stage: ~0 when the prefix and copy were hidden behind the
 *              previous frame's suffix. */
typedef struct {
    double t_gpu_ms;
    double t_xfer_ms;
    double t_cpu_ms;
    double t_submit_s;
    double t_start_s;
    double t_ready_s;
    double t_done_s;
    int split;
    int n_tokens;
} vla_frame_times;

/* A cross-frame pipeline over `gpu` (blocks [0, p) for every split p used) and `cpu`
 * (blocks [c0, N), N = the CPU model's layer_end; p >= c0). Up to `depth` (1..8) frames are
 * in flight. Owns, per slot, a device buffer and a page-locked host buffer of max_tokens x
 * hidden for h^(p) and a host output buffer; one GPU KV cache for [0, min(N, gpu layers))
 * and one host KV cache for [c0, N), both reset at every frame (each frame is a fresh
 * prefill); a side stream for the boundary copies and one host worker thread that runs the
 * suffixes in submission order on the CPU model's pool. The device current at this call
 * must be current for every later call, all frames must be submitted on one stream (the GPU
 * cache is reused frame after frame in that stream's order), and the models must outlive
 * the pipeline. Submit and collect may run on two different threads, but each from one
 * thread at a time (one producer, one consumer).
 * Errors: INVALID_ARG, SHAPE (configs differ, max_tokens), RANGE (layer ranges), OOM, CUDA. */
vla_status vla_pipeline_create(vla_prefix* gpu, vla_cpu_model* cpu, int max_tokens, int depth, vla_pipeline** out);

/* Enqueues frame `frame_id`: on `stream`, the GPU prefix [0, split) of hidden_in (device,
 * [n_tokens, hidden], read on `stream`; keep it unchanged until that work has run), then the
 * boundary copy of h^(split) to pinned memory on the side stream; the worker thread waits for
 * the copy and runs the CPU suffix [split, N). Returns once the GPU work is enqueued, so the
 * caller can submit frame t+1 while frame t is on the CPU. split = N runs everything on the
 * GPU (the suffix is a copy); split = 0 everything on the CPU.
 * Errors: INVALID_ARG, RANGE (split outside [c0, N] or beyond the GPU model), SHAPE
 * (n_tokens), BUSY (depth frames already in flight: collect one first), CUDA. */
vla_status vla_pipeline_submit(vla_pipeline* pl, int64_t frame_id, const void* hidden_in, int n_tokens, int split,
                               vla_stream stream);

/* Waits up to timeout_ms (< 0: no limit) for the OLDEST submitted frame to finish, copies its
 * final hidden state h^(N) [n_tokens, hidden] into hidden_out (host; may be NULL) and its id
 * and stage times into *frame_id / *times (may be NULL), and frees its slot. Frames come out
 * in submission order. Returns the frame's own status (TIMEOUT or CUDA if its boundary copy
 * never completed or failed). Errors: INVALID_ARG (nothing in flight), TIMEOUT (not finished
 * in time; the frame stays queued). */
vla_status vla_pipeline_collect(vla_pipeline* pl, int64_t* frame_id, void* hidden_out, int timeout_ms,
                                vla_frame_times* times);

/* Frames submitted and not yet collected; -1 if pl is NULL. */
int vla_pipeline_in_flight(const vla_pipeline* pl);

/* Waits for the worker to finish the queued frames, joins it and frees everything the
 * pipeline owns (not the models). NULL is a no-op. */
vla_status vla_pipeline_destroy(vla_pipeline* pl);

/* Flexible resource scheduling (Sec. IV-D, Eq. 15-17). The blocks form a GPU-fixed zone
 * [0, k_min), a dynamic zone and a CPU-fixed zone [k_max, N); the split p of each frame is one
 * of the candidate policies {k_min, ..., k_max} (Eq. 16), chosen by a controller Phi from the
 * runtime state z_t = [u_gpu, u_cpu, q_t] (Eq. 15, 17). The paper does not give Phi; this one:
 *   - keeps per-block cost estimates, g (GPU) and c (CPU) in ms per block, as exponential
 *     moving averages of T_G / p and T_C / (N - p) over observed frames, and the transfer
 *     time x likewise (vla_scheduler_observe; a side with no blocks in a frame is not updated);
 *   - scales them by the share of each processor other work leaves free: g / (1 - u_gpu),
 *     c / (1 - u_cpu), with the utilisations clamped to [0, 0.95];
 *   - predicts the steady interval of Eq. 13, max(p g', x + (N - p) c'), for every candidate
 *     and moves the split toward the best one (ties: the one nearest the current split) by at
 *     most max_step blocks per frame, so only boundary-adjacent blocks migrate;
 *   - when the backlog q_t reaches backlog_limit frames and the prediction asks for no move,
 *     moves one block away from the stage predicted to be slower;
 *   - keeps the split while either cost has never been observed. */
typedef struct {
    int n_layers;       /* N */
    int k_min, k_max;   /* 0 <= k_min <= k_max <= N */
    int k_init;         /* first split, in [k_min, k_max] */
    int max_step;       /* >= 1 */
    double alpha;       /* (0, 1]: weight of the newest frame in the moving averages */
    int backlog_limit;  /* >= 1 */
} vla_sched_config;

typedef struct {
    double u_gpu;  /* share of the GPU taken by other work, [0, 1] */
    double u_cpu;  /* share of the host cores taken by other work, [0, 1] */
    int backlog;   /* q_t: frames submitted and not yet finished */
} vla_sched_state;

typedef struct vla_scheduler vla_scheduler;

/* Errors: INVALID_ARG (null or inconsistent config), OOM. */
vla_status vla_scheduler_create(const vla_sched_config* cfg, vla_scheduler** out);
/* Folds one finished frame's stage times into the cost estimates. Errors: INVALID_ARG. */
vla_status vla_scheduler_observe(vla_scheduler* s, const vla_frame_times* t);
/* Phi(z_t): the split for the next frame (and the scheduler's new current split); -1 if an
 * argument is NULL. */
int vla_scheduler_next(vla_scheduler* s, const vla_sched_state* z);
/* Current estimates (ms per GPU block, ms per CPU block, ms per transfer); a never-observed
 * one reads -1. Any output may be NULL. Errors: INVALID_ARG. */
vla_status vla_scheduler_estimates(const vla_scheduler* s, double* g_ms, double* c_ms, double* x_ms);
vla_status vla_scheduler_destroy(vla_scheduler* s);

#ifdef __cplusplus
}
#endif

#endif /* VLA_CPU_H */
