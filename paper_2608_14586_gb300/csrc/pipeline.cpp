// Cross-frame asynchronous pipeline (Sec. IV-C, Eq. 12-14): the GPU runs the prefix [0, p) of
// frame t+1 while the host cores run the suffix [p, N) of frame t.
//
// Producer: vla_pipeline_submit enqueues, on the caller's stream, the KV reset and the prefix
// of the frame into the device buffer of a free slot, bracketed by two timing events, and the
// boundary copy of h^(p) into the slot's page-locked buffer on the pipeline's side stream
// (vla_boundary_to_host, which records the slot's copy-done event). It returns at once.
// Consumer: one host thread takes the slots in submission order, waits (bounded) for the
// copy-done event, runs the CPU suffix into the slot's output buffer and marks the slot done.
// vla_pipeline_collect hands out the oldest frame once it is done, with its id, so the final
// output stays aligned with its input frame. Slots form a ring of `depth` entries; a full
// ring makes submit return BUSY instead of blocking, so a single thread can drive both ends.
#include <cuda_runtime.h>

#include <chrono>
#include <condition_variable>
#include <cstring>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "vla_cpu.h"

namespace {

constexpr int kMaxDepth = 8;
constexpr double kCopyWaitLimitS = 120.0;  // a boundary copy not complete by then fails the frame

double now_s() {
    return std::chrono::duration<double>(std::chrono::steady_clock::now().time_since_epoch()).count();
}

enum SlotState : int { kFree = 0, kReserved = 1, kQueued = 2, kDone = 3, kCollecting = 4 };

struct Slot {
    void* h_dev = nullptr;  // h^(p) on the device
    void* h_pin = nullptr;  // h^(p) in page-locked host memory
    std::vector<uint16_t> out;  // h^(N)
    cudaEvent_t g0 = nullptr, g1 = nullptr, x1 = nullptr;
    int state = kFree;
    int64_t frame = 0;
    int n = 0, split = 0;
    vla_status status = VLA_OK;
    vla_frame_times t{};
};

// Polls `e` until it completes, fails, or the limit passes.
vla_status wait_event(cudaEvent_t e, double limit_s) {
    const double t_end = now_s() + limit_s;
    for (;;) {
        const cudaError_t r = cudaEventQuery(e);
        if (r == cudaSuccess) return VLA_OK;
        if (r != cudaErrorNotReady) {
            cudaGetLastError();
            return VLA_ERR_CUDA;
        }
        if (now_s() > t_end) return VLA_ERR_TIMEOUT;
        std::this_thread::sleep_for(std::chrono::microseconds(50));
    }
}

}  // namespace

struct vla_pipeline {
    vla_prefix* gpu = nullptr;
    vla_cpu_model* cpu = nullptr;
    vla_config cfg{};
    int gpu_layers = 0, c0 = 0, N = 0, max_tokens = 0, depth = 0, device = 0;
    vla_kv* gkv = nullptr;
    vla_cpu_kv* ckv = nullptr;
    cudaStream_t side = nullptr;
    std::vector<Slot> slots;
    int head = 0;   // oldest frame in flight
    int count = 0;  // frames in flight
    int wpos = 0;   // next slot the worker takes
    bool stop = false;
    std::mutex mu;
    std::condition_variable cv_work, cv_done;
    std::thread worker;

    void run_worker() {
        cudaSetDevice(device);
        std::unique_lock<std::mutex> lk(mu);
        for (;;) {
            cv_work.wait(lk, [&] { return slots[wpos].state == kQueued || (stop && count_queued() == 0); });
            if (slots[wpos].state != kQueued) return;  // stopping and nothing left
            Slot& s = slots[wpos];
            lk.unlock();
            s.t.t_start_s = now_s();
            vla_status st = wait_event(s.x1, kCopyWaitLimitS);
            s.t.t_ready_s = now_s();
            if (st == VLA_OK) {
                float ms = 0.f;
                if (cudaEventElapsedTime(&ms, s.g0, s.g1) == cudaSuccess) s.t.t_gpu_ms = ms;
                if (cudaEventElapsedTime(&ms, s.g1, s.x1) == cudaSuccess) s.t.t_xfer_ms = ms;
                cudaGetLastError();
                vla_cpu_kv_reset(ckv);
                const double c0t = now_s();
                st = vla_cpu_prefill(cpu, s.h_pin, s.n, s.split, N, ckv, s.out.data());
                s.t.t_cpu_ms = (now_s() - c0t) * 1e3;
            }
            s.t.t_done_s = now_s();
            lk.lock();
            s.status = st;
            s.state = kDone;
            wpos = (wpos + 1) % depth;
            cv_done.notify_all();
        }
    }
    int count_queued() const {
        int q = 0;
        for (const Slot& s : slots) q += (s.state == kQueued || s.state == kReserved);
        return q;
    }
};

namespace {

void free_pipeline(vla_pipeline* pl) {
    if (!pl) return;
    if (pl->side) cudaStreamSynchronize(pl->side);
    for (Slot& s : pl->slots) {
        cudaFree(s.h_dev);
        cudaFreeHost(s.h_pin);
        if (s.g0) cudaEventDestroy(s.g0);
        if (s.g1) cudaEventDestroy(s.g1);
        if (s.x1) cudaEventDestroy(s.x1);
    }
    if (pl->side) cudaStreamDestroy(pl->side);
    vla_kv_destroy(pl->gkv);
    vla_cpu_kv_destroy(pl->ckv);
    cudaGetLastError();
    delete pl;
}

}  // namespace

extern "C" {

vla_status vla_pipeline_create(vla_prefix* gpu, vla_cpu_model* cpu, int max_tokens, int depth, vla_pipeline** out) {
    if (!out) return VLA_ERR_INVALID_ARG;
    *out = nullptr;
    if (!gpu || !cpu || depth < 1 || depth > kMaxDepth || max_tokens < 1) return VLA_ERR_INVALID_ARG;
    vla_config gc{}, cc{};
    int gl = 0, clb = 0, cle = 0;
    if (vla_prefix_info(gpu, &gc, &gl) != VLA_OK || vla_cpu_model_info(cpu, &cc, &clb, &cle) != VLA_OK)
        return VLA_ERR_INVALID_ARG;
    if (gc.hidden != cc.hidden || gc.n_heads != cc.n_heads || gc.n_kv_heads != cc.n_kv_heads ||
        gc.head_dim != cc.head_dim || gc.ffn != cc.ffn || gc.rms_eps != cc.rms_eps || gc.rope_base != cc.rope_base)
        return VLA_ERR_SHAPE;
    if (max_tokens > gc.max_ctx || max_tokens > cc.max_ctx) return VLA_ERR_SHAPE;
    if (clb > gl) return VLA_ERR_RANGE;  // some split must be reachable from both sides
    vla_pipeline* pl = new (std::nothrow) vla_pipeline();
    if (!pl) return VLA_ERR_OOM;
    pl->gpu = gpu;
    pl->cpu = cpu;
    pl->cfg = gc;
    pl->gpu_layers = gl;
    pl->c0 = clb;
    pl->N = cle;
    pl->max_tokens = max_tokens;
    pl->depth = depth;
    cudaGetDevice(&pl->device);
    const size_t bytes = (size_t)max_tokens * gc.hidden * 2;
    vla_status st = VLA_OK;
    const int g_end = cle < gl ? cle : gl;
    if (g_end > 0) st = vla_kv_create(gpu, 0, g_end, max_tokens, &pl->gkv);
    if (st == VLA_OK && clb < cle) st = vla_cpu_kv_create(cpu, clb, cle, max_tokens, &pl->ckv);
    if (st != VLA_OK) {
        free_pipeline(pl);
        return st;
    }
    bool ok = cudaStreamCreateWithFlags(&pl->side, cudaStreamNonBlocking) == cudaSuccess;
    try {
        pl->slots.resize(depth);
        for (Slot& s : pl->slots) {
            if (!ok) break;
            s.out.resize((size_t)max_tokens * gc.hidden);
            ok = cudaMalloc(&s.h_dev, bytes) == cudaSuccess && cudaMallocHost(&s.h_pin, bytes) == cudaSuccess &&
                 cudaEventCreate(&s.g0) == cudaSuccess && cudaEventCreate(&s.g1) == cudaSuccess &&
                 cudaEventCreate(&s.x1) == cudaSuccess;
        }
    } catch (...) {
        ok = false;
    }
    if (!ok) {
        cudaGetLastError();
        free_pipeline(pl);
        return VLA_ERR_OOM;
    }
    try {
        pl->worker = std::thread([pl] { pl->run_worker(); });
    } catch (...) {
        free_pipeline(pl);
        return VLA_ERR_OOM;
    }
    *out = pl;
    return VLA_OK;
}

vla_status vla_pipeline_submit(vla_pipeline* pl, int64_t frame_id, const void* hidden_in, int n_tokens, int split,
                               vla_stream stream) {
    if (!pl || !hidden_in) return VLA_ERR_INVALID_ARG;
    if (n_tokens < 1 || n_tokens > pl->max_tokens) return VLA_ERR_SHAPE;
    if (split < pl->c0 || split > pl->N || split > pl->gpu_layers) return VLA_ERR_RANGE;
    int idx;
    {
        std::lock_guard<std::mutex> lk(pl->mu);
        if (pl->count == pl->depth) return VLA_ERR_BUSY;
        idx = (pl->head + pl->count) % pl->depth;
        pl->slots[idx].state = kReserved;
        pl->count += 1;
    }
    Slot& s = pl->slots[idx];
    s.frame = frame_id;
    s.n = n_tokens;
    s.split = split;
    s.status = VLA_OK;
    s.t = vla_frame_times{};
    s.t.split = split;
    s.t.n_tokens = n_tokens;
    s.t.t_submit_s = now_s();
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    vla_status r = VLA_OK;
    if (pl->gkv) r = vla_kv_reset(pl->gkv, stream);
    if (r == VLA_OK && cudaEventRecord(s.g0, st) != cudaSuccess) r = VLA_ERR_CUDA;
    if (r == VLA_OK) r = vla_prefix_prefill(pl->gpu, hidden_in, n_tokens, 0, split, split > 0 ? pl->gkv : nullptr,
                                            s.h_dev, stream);
    if (r == VLA_OK && cudaEventRecord(s.g1, st) != cudaSuccess) r = VLA_ERR_CUDA;
    if (r == VLA_OK)
        r = vla_boundary_to_host(s.h_dev, n_tokens, pl->cfg.hidden, s.h_pin, reinterpret_cast<vla_stream>(pl->side),
                                 reinterpret_cast<vla_event>(s.g1), reinterpret_cast<vla_event>(s.x1));
    std::lock_guard<std::mutex> lk(pl->mu);
    if (r != VLA_OK) {
        // nothing of this frame reached the worker: give the slot back (it is the newest)
        cudaGetLastError();
        s.state = kFree;
        pl->count -= 1;
        return r;
    }
    s.state = kQueued;
    pl->cv_work.notify_one();
    return VLA_OK;
}

vla_status vla_pipeline_collect(vla_pipeline* pl, int64_t* frame_id, void* hidden_out, int timeout_ms,
                                vla_frame_times* times) {
    if (!pl) return VLA_ERR_INVALID_ARG;
    std::unique_lock<std::mutex> lk(pl->mu);
    if (pl->count == 0) return VLA_ERR_INVALID_ARG;
    Slot& s = pl->slots[pl->head];
    auto ready = [&] { return s.state == kDone; };
    if (timeout_ms < 0) {
        pl->cv_done.wait(lk, ready);
    } else if (!pl->cv_done.wait_for(lk, std::chrono::milliseconds(timeout_ms), ready)) {
        return VLA_ERR_TIMEOUT;
    }
    s.state = kCollecting;
    lk.unlock();
    if (hidden_out && s.status == VLA_OK) std::memcpy(hidden_out, s.out.data(), (size_t)s.n * pl->cfg.hidden * 2);
    if (frame_id) *frame_id = s.frame;
    if (times) *times = s.t;
    const vla_status st = s.status;
    lk.lock();
    s.state = kFree;
    pl->head = (pl->head + 1) % pl->depth;
    pl->count -= 1;
    return st;
}

int vla_pipeline_in_flight(const vla_pipeline* pl) {
    if (!pl) return -1;
    std::lock_guard<std::mutex> lk(const_cast<vla_pipeline*>(pl)->mu);
    return pl->count;
}

vla_status vla_pipeline_destroy(vla_pipeline* pl) {
    if (!pl) return VLA_OK;
    {
        std::lock_guard<std::mutex> lk(pl->mu);
        pl->stop = true;
    }
    pl->cv_work.notify_all();
    if (pl->worker.joinable()) pl->worker.join();
    free_pipeline(pl);
    return VLA_OK;
}

}  // extern "C"
