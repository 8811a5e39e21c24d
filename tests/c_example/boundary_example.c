/* Using the boundary from C: one frame through the 16-block prefix of a 32-block 7B-class
 * stack, the boundary h^(16) handed to page-locked host memory on a side stream, then one
 * decode step. Error handling is elided: every call returns a vla_status.
 *
 * The function's parameters supply what a program would own: per-block device weights
 * (bf16 [out, in] pointers; the library repacks them and the caller may free them after
 * vla_prefix_create), the frame in page-locked host memory, device buffers for the frame and
 * h^(16), the host destination of the boundary, one decode token, and the streams and events.
 * tests/test_abi_cpu.py compiles this file as C11 against the public headers. */
#include <cuda_runtime.h>

#include "vla_ops.h"
#include "vla_prefix.h"

void example(const vla_layer_weights* layers, const void* frame_host, void* h_in, void* h_out, void* pinned,
             const void* x1, void* y1, cudaStream_t stream, cudaStream_t side_stream, cudaEvent_t ready,
             cudaEvent_t done) {
    vla_config cfg = {4096, 32, 8, 128, 11008, 1e-6f, 10000.f, /*max_ctx*/ 2368};
    vla_prefix* p;
    vla_prefix_create(&cfg, layers, 32, &p);
    vla_kv* kv;
    vla_kv_create(p, 0, 16, 2368, &kv); /* room for 64 decode steps after a 2304-token frame */

    /* frame: [2304, 4096] bf16 from the host -> h^(16) in h_out, KV written for blocks 0..15 */
    vla_frame_to_device(frame_host, 2304, 4096, h_in, stream);
    vla_kv_reset(kv, stream);
    vla_prefix_prefill(p, h_in, 2304, 0, 16, kv, h_out, stream);
    cudaEventRecord(ready, stream);
    vla_boundary_to_host(h_out, 2304, 4096, pinned, side_stream, ready, done); /* overlaps the next frame */

    vla_prefix_decode(p, x1, 0, 16, kv, y1, stream); /* one token at position 2304 */
    cudaStreamSynchronize(stream);
    cudaEventSynchronize(done);
    if (vla_last_async_error(p) != VLA_OK) { /* a kernel's bounded wait ran out */ }
    vla_kv_destroy(kv);
    vla_prefix_destroy(p);
}
