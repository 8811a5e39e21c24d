// Single-query decode attention that allocates nothing (vla_op_attention_decode_noalloc).
//
// Why it exists: some programs that embed this library must not allocate device memory once
// they are running. A vehicle's real-time control loop is the typical case: all memory is
// reserved at start-up against a fixed budget, and a cudaMalloc in the loop could block for
// an unbounded time or fail when the budget is spent. Other callers run inside a host
// framework whose own allocator owns the device memory and forbids side allocations. The
// split-KV decode attention needs scratch space for its per-split partial results; in the
// regular path that space comes from the vla_prefix object, which vla_prefix_create
// allocates. This variant takes its scratch from one fixed-size array compiled into the
// library instead, so a caller only hands in its own inputs and outputs.
//
// The array lives in device memory of every GPU that loads the library, for the life of the
// process (kNoAllocScratchFloats floats = 2 MiB). All calls share it: two calls whose GPU
// work overlaps (for example on two streams) race on it, so order such calls on one stream
// or serialise them. Each call writes every partial it later reads, so nothing in the array
// has to start at zero and no call depends on what an earlier call left there.
//
// The kernels below are the same split-KV algorithm as the decode step's attention, with the
// query taken as bf16 (the layout of the prefill attention's queries) and the key count
// passed as an argument.
#include <mutex>

#include "../../include/vla_ops.h"
#include "common.cuh"
#include "internal.h"

// 2 MiB of fp32 partials: splits * n_heads * (head_dim + 2) floats must fit.
static constexpr size_t kNoAllocScratchFloats = size_t(1) << 19;
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

namespace {

using vla::bf16;
using vla::bf16_hi;
using vla::bf16_lo;

constexpr int kThreads = 128;
constexpr int kMaxDevices = 64;

template <int DH, int G>
__global__ void __launch_bounds__(kThreads) noalloc_partial_kernel(const bf16* q, const bf16* kc, const bf16* vc,
                                                                   int ctx, int H, int max_ctx, int splits,
                                                                   float scale_log2, float* part_o, float* part_ml) {
    constexpr int DPL = DH / 8;
    constexpr int NW = kThreads / 32;
    __shared__ float sm_m[NW][G], sm_l[NW][G];
    __shared__ float sm_o[NW][G][DH];
    const int kvh = blockIdx.x, split = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane >> 3, l8 = lane & 7;
    const int chunk = (ctx + splits - 1) / splits;
    const int kb = split * chunk;
    const int ke = min(ctx, kb + chunk);

    float qv[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh)
#pragma unroll
        for (int d = 0; d < DPL; ++d)
            qv[hh][d] = __bfloat162float(q[(kvh * G + hh) * DH + l8 * DPL + d]) * scale_log2;
    float m[G], l[G], o[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        m[hh] = -INFINITY;
        l[hh] = 0.f;
#pragma unroll
        for (int d = 0; d < DPL; ++d) o[hh][d] = 0.f;
    }
    const bf16* kbase = kc + (size_t)kvh * max_ctx * DH + l8 * DPL;
    const bf16* vbase = vc + (size_t)kvh * max_ctx * DH + l8 * DPL;
    // warp-uniform loop; each 8-lane slot takes one key and skips the update past the range
    for (int k0 = kb + warp * 4; k0 < ke; k0 += NW * 4) {
        const int k = k0 + sub;
        const bool valid = k < ke;
        float kf[DPL], vf[DPL];
#pragma unroll
        for (int c = 0; c < DPL / 8; ++c) {
            uint4 kr = make_uint4(0u, 0u, 0u, 0u), vr = make_uint4(0u, 0u, 0u, 0u);
            if (valid) {
                kr = vla::ldg_stream(kbase + (size_t)k * DH + c * 8);
                vr = vla::ldg_stream(vbase + (size_t)k * DH + c * 8);
            }
            const uint32_t kw[4] = {kr.x, kr.y, kr.z, kr.w};
            const uint32_t vw[4] = {vr.x, vr.y, vr.z, vr.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                kf[c * 8 + 2 * i] = bf16_lo(kw[i]);
                kf[c * 8 + 2 * i + 1] = bf16_hi(kw[i]);
                vf[c * 8 + 2 * i] = bf16_lo(vw[i]);
                vf[c * 8 + 2 * i + 1] = bf16_hi(vw[i]);
            }
        }
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            float s = 0.f;
#pragma unroll
            for (int d = 0; d < DPL; ++d) s = fmaf(qv[hh][d], kf[d], s);
            s += __shfl_xor_sync(0xFFFFFFFFu, s, 1);
            s += __shfl_xor_sync(0xFFFFFFFFu, s, 2);
            s += __shfl_xor_sync(0xFFFFFFFFu, s, 4);
            if (!valid) continue;
            const float mn = fmaxf(m[hh], s);
            const float c = exp2f(m[hh] - mn);
            const float pe = exp2f(s - mn);
            l[hh] = l[hh] * c + pe;
#pragma unroll
            for (int d = 0; d < DPL; ++d) o[hh][d] = fmaf(o[hh][d], c, pe * vf[d]);
            m[hh] = mn;
        }
    }
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
#pragma unroll
        for (int off = 8; off <= 16; off <<= 1) {
            const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m[hh], off);
            const float l2 = __shfl_xor_sync(0xFFFFFFFFu, l[hh], off);
            const float mn = fmaxf(m[hh], m2);
            const float c1 = (mn == -INFINITY) ? 0.f : exp2f(m[hh] - mn);
            const float c2 = (mn == -INFINITY) ? 0.f : exp2f(m2 - mn);
            l[hh] = l[hh] * c1 + l2 * c2;
#pragma unroll
            for (int d = 0; d < DPL; ++d) {
                const float o2 = __shfl_xor_sync(0xFFFFFFFFu, o[hh][d], off);
                o[hh][d] = o[hh][d] * c1 + o2 * c2;
            }
            m[hh] = mn;
        }
    }
    if (sub == 0) {
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            if (l8 == 0) {
                sm_m[warp][hh] = m[hh];
                sm_l[warp][hh] = l[hh];
            }
#pragma unroll
            for (int d = 0; d < DPL; ++d) sm_o[warp][hh][l8 * DPL + d] = o[hh][d];
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < G * DH; e += kThreads) {
        const int hh = e / DH, d = e % DH;
        float mx = -INFINITY;
        for (int w = 0; w < NW; ++w) mx = fmaxf(mx, sm_m[w][hh]);
        float lt = 0.f, ot = 0.f;
        if (mx != -INFINITY) {
            for (int w = 0; w < NW; ++w) {
                const float c = exp2f(sm_m[w][hh] - mx);
                lt += sm_l[w][hh] * c;
                ot += sm_o[w][hh][d] * c;
            }
        }
        const int h = kvh * G + hh;
        part_o[((size_t)split * H + h) * DH + d] = ot;
        if (d == 0) {
            part_ml[((size_t)split * H + h) * 2 + 0] = mx;
            part_ml[((size_t)split * H + h) * 2 + 1] = lt;
        }
    }
}

__global__ void noalloc_combine_kernel(const float* part_o, const float* part_ml, int H, int dh, int splits,
                                       bf16* out) {
    const int h = blockIdx.x;
    for (int d = threadIdx.x; d < dh; d += blockDim.x) {
        float mx = -INFINITY;
        for (int s = 0; s < splits; ++s) mx = fmaxf(mx, part_ml[((size_t)s * H + h) * 2]);
        float lt = 0.f, ot = 0.f;
        for (int s = 0; s < splits; ++s) {
            const float ms = part_ml[((size_t)s * H + h) * 2];
            if (ms == -INFINITY) continue;
            const float c = exp2f(ms - mx);
            lt += part_ml[((size_t)s * H + h) * 2 + 1] * c;
            ot += part_o[((size_t)s * H + h) * dh + d] * c;
        }
        out[h * dh + d] = __float2bfloat16_rn(ot / lt);
    }
}

template <int DH, int G>
cudaError_t launch_partial(dim3 grid, cudaStream_t s, const bf16* q, const bf16* kc, const bf16* vc, int ctx, int H,
                           int max_ctx, int splits, float scale_log2, float* po, float* pml) {
    noalloc_partial_kernel<DH, G><<<grid, kThreads, 0, s>>>(q, kc, vc, ctx, H, max_ctx, splits, scale_log2, po, pml);
    return cudaGetLastError();
}

typedef CUresult (*PFN_ctxGetCurrent_t)(CUcontext*);
typedef CUresult (*PFN_ctxGetId_t)(CUcontext, unsigned long long*);

// Unique id of the calling thread's current CUDA context (0 when there is none yet). Ids are
// never reused within a process, so a context destroyed and created again (a device reset)
// gets a new one.
unsigned long long current_context_id() {
    static PFN_ctxGetCurrent_t get_current = nullptr;
    static PFN_ctxGetId_t get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<PFN_ctxGetCurrent_t>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<PFN_ctxGetId_t>(p);
    });
    if (!get_current || !get_id) return 0;
    CUcontext c = nullptr;
    unsigned long long id = 0;
    if (get_current(&c) != CUDA_SUCCESS || !c || get_id(c, &id) != CUDA_SUCCESS) return 0;
    return id;
}

struct DeviceSetup {
    unsigned long long ctx_id;  // context the address below belongs to
    float* scratch;
    int sms;
};

std::mutex g_setup_mu;
DeviceSetup g_setup[kMaxDevices] = {};

// Once per device and context, with that device current: resolve the array's device address
// (host code cannot use the symbol's name as a pointer) and read the SM count. The address
// belongs to the context it was resolved in, so a new context on the device (after a device
// reset) resolves it again.
vla_status setup_device(int dev, float** scratch, int* sms) {
    std::lock_guard<std::mutex> lock(g_setup_mu);
    DeviceSetup& d = g_setup[dev];
    const unsigned long long id = current_context_id();
    if (!d.scratch || id == 0 || id != d.ctx_id) {
        void* ptr = nullptr;  // this call also creates the device's context if there is none yet
        if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) {
            cudaGetLastError();
            return VLA_ERR_CUDA;
        }
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
            cudaGetLastError();
            return VLA_ERR_CUDA;
        }
        d.scratch = static_cast<float*>(ptr);
        d.sms = n;
        d.ctx_id = current_context_id();
    }
    *scratch = d.scratch;
    *sms = d.sms;
    return VLA_OK;
}

}  // namespace

extern "C" vla_status vla_op_attention_decode_noalloc(const void* q, const void* k_plane, const void* v_plane,
                                                      int ctx, int n_heads, int n_kv_heads, int head_dim,
                                                      int max_ctx, void* out, vla_stream stream) {
    if (!q || !k_plane || !v_plane || !out || ctx <= 0 || n_heads <= 0 || n_kv_heads <= 0 || max_ctx <= 0 ||
        ctx > max_ctx || n_heads % n_kv_heads)
        return VLA_ERR_INVALID_ARG;
    if (head_dim != 64 && head_dim != 128) return VLA_ERR_UNSUPPORTED;
    const int group = n_heads / n_kv_heads;
    if (group != 1 && group != 2 && group != 4 && group != 8) return VLA_ERR_UNSUPPORTED;
    if ((reinterpret_cast<uintptr_t>(k_plane) | reinterpret_cast<uintptr_t>(v_plane)) & 15u) return VLA_ERR_INVALID_ARG;
    // one split must fit the fixed scratch array: n_heads * (head_dim + 2) floats
    const size_t per_split = (size_t)n_heads * (head_dim + 2);
    if (per_split > kNoAllocScratchFloats) return VLA_ERR_SHAPE;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return VLA_ERR_CUDA;
    float* scratch = nullptr;
    int sms = 0;
    vla_status st = setup_device(dev, &scratch, &sms);
    if (st != VLA_OK) return st;
    int splits = (2 * sms + n_kv_heads - 1) / n_kv_heads;
    const int cap = (int)(kNoAllocScratchFloats / per_split);
    if (splits > cap) splits = cap;
    if (splits > ctx) splits = ctx;
    if (splits < 1) splits = 1;
    float* part_o = scratch;
    float* part_ml = scratch + (size_t)splits * n_heads * head_dim;
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
    const dim3 grid(n_kv_heads, splits);
    cudaStream_t s = (cudaStream_t)stream;
    const bf16* qb = (const bf16*)q;
    const bf16* kb = (const bf16*)k_plane;
    const bf16* vb = (const bf16*)v_plane;
    cudaError_t e = cudaErrorInvalidValue;
#define VLA_NOALLOC_CASE(DH_, G_)                                                                               \
    if (head_dim == DH_ && group == G_)                                                                         \
        e = launch_partial<DH_, G_>(grid, s, qb, kb, vb, ctx, n_heads, max_ctx, splits, scale_log2, part_o, part_ml);
    VLA_NOALLOC_CASE(64, 1)
    VLA_NOALLOC_CASE(64, 2)
    VLA_NOALLOC_CASE(64, 4)
    VLA_NOALLOC_CASE(64, 8)
    VLA_NOALLOC_CASE(128, 1)
    VLA_NOALLOC_CASE(128, 2)
    VLA_NOALLOC_CASE(128, 4)
    VLA_NOALLOC_CASE(128, 8)
#undef VLA_NOALLOC_CASE
    if (e != cudaSuccess) return VLA_ERR_CUDA;
    noalloc_combine_kernel<<<n_heads, head_dim, 0, s>>>(part_o, part_ml, n_heads, head_dim, splits, (bf16*)out);
    return cudaGetLastError() == cudaSuccess ? VLA_OK : VLA_ERR_CUDA;
}
