// Single-token decode of one block (the prefix range at M = 1, position = KV length).
//
// At M = 1 every projection is a matrix-vector product whose cost is streaming the weights
// once from HBM (354 MB per 7B-class block), so these kernels are built for bandwidth:
//   * one warp per pair of weight rows, 16-byte non-allocating loads, 8 chunks per row in
//     flight per lane, fp32 FMA, warp-shuffle reduction;
//   * the pair is chosen so the fused epilogue has both operands it needs: rows (j, j+dh/2)
//     of a head for the rotary embedding, the gate and up rows of one feed-forward unit for
//     SwiGLU, consecutive rows for the residual projections;
//   * the input vector is staged in shared memory; RMSNorm's 1/rms is computed per CTA
//     (the gains are folded into the weights);
//   * each kernel prefetches its first weight rows into L2 before reading its input vector,
//     so the weight stream starts while the input is still being staged.
// Attention is split over the context (fixed split count -> deterministic): each CTA owns
// one KV head (all query heads of its GQA group) and a contiguous key range, 8 lanes per key
// row, online softmax in fp32; the last CTA of each KV head merges the partials (max, sum,
// output) in fixed split order.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

enum GemvMode : int { kGemvQKV = 0, kGemvResid = 1, kGemvSwiGLU = 2 };

struct GemvParams {
    const bf16* W;  // [rows, K] row-major
    int K;          // multiple of 256
    int units;      // row pairs
    const bf16* xv;     // input vector [K]
    const bf16* resid;  // kGemvResid: residual [2*units]
    bf16* out;          // kGemvResid: [2*units]; kGemvSwiGLU: [units]
    float* q_out;       // kGemvQKV: post-RoPE query, fp32 [H*dh]
    bf16* kcache;
    bf16* vcache;
    const int* d_len;  // kGemvQKV: position of the new token
    const float2* rope;
    int dh, n_q_heads, n_kv_heads, max_ctx;
    float eps;
};

constexpr int kGemvThreads = 256;
constexpr int kGemvU = 8;  // 16-byte chunks per row in flight per lane

VLA_DEV float dot8(uint4 w, uint4 x) {
    float a = bf16_lo(w.x) * bf16_lo(x.x);
    a = fmaf(bf16_hi(w.x), bf16_hi(x.x), a);
    a = fmaf(bf16_lo(w.y), bf16_lo(x.y), a);
    a = fmaf(bf16_hi(w.y), bf16_hi(x.y), a);
    a = fmaf(bf16_lo(w.z), bf16_lo(x.z), a);
    a = fmaf(bf16_hi(w.z), bf16_hi(x.z), a);
    a = fmaf(bf16_lo(w.w), bf16_lo(x.w), a);
    a = fmaf(bf16_hi(w.w), bf16_hi(x.w), a);
    return a;
}

template <int MODE>
VLA_DEV void unit_rows(const GemvParams& p, int u, int& ra, int& rb) {
    if constexpr (MODE == kGemvQKV) {
        const int half = p.dh >> 1;
        const int head = u / half, j = u % half;
        ra = head * p.dh + j;
        rb = ra + half;
    } else if constexpr (MODE == kGemvSwiGLU) {
        const int grp = u >> 7, i = u & 127;
        ra = grp * 256 + i;
        rb = ra + 128;
    } else {
        ra = 2 * u;
        rb = 2 * u + 1;
    }
}

// Fused epilogue of one row pair (lane 0 of the warp that reduced it).
template <int MODE>
VLA_DEV void gemv_epilogue(const GemvParams& p, int u, int ra, int rb, float acc_a, float acc_b, float rinv, int pos) {
    if constexpr (MODE == kGemvResid) {
        const float ya = __bfloat162float(p.resid[ra]) + acc_a;
        const float yb = __bfloat162float(p.resid[rb]) + acc_b;
        *reinterpret_cast<uint32_t*>(p.out + ra) = pack_bf16x2(ya, yb);
    } else if constexpr (MODE == kGemvSwiGLU) {
        const float g = acc_a * rinv, up = acc_b * rinv;
        p.out[u] = __float2bfloat16_rn(g / (1.0f + __expf(-g)) * up);
    } else {
        const int half = p.dh >> 1;
        const int head = u / half, j = u % half;
        float a = acc_a * rinv, b = acc_b * rinv;
        if (head < p.n_q_heads + p.n_kv_heads) {
            const float2 cs = p.rope[(size_t)pos * half + j];
            const float a2 = a * cs.x - b * cs.y;
            const float b2 = b * cs.x + a * cs.y;
            a = a2;
            b = b2;
        }
        if (head < p.n_q_heads) {
            p.q_out[head * p.dh + j] = a;
            p.q_out[head * p.dh + j + half] = b;
        } else if (head < p.n_q_heads + p.n_kv_heads) {
            bf16* kp = p.kcache + ((size_t)(head - p.n_q_heads) * p.max_ctx + pos) * p.dh;
            kp[j] = __float2bfloat16_rn(a);
            kp[j + half] = __float2bfloat16_rn(b);
        } else {
            bf16* vp = p.vcache + ((size_t)(head - p.n_q_heads - p.n_kv_heads) * p.max_ctx + pos) * p.dh;
            vp[j] = __float2bfloat16_rn(a);
            vp[j + half] = __float2bfloat16_rn(b);
        }
    }
}

template <int MODE>
__global__ void __launch_bounds__(kGemvThreads, 2) gemv_kernel(GemvParams p) {
    extern __shared__ uint4 xs[];
    __shared__ float red[kGemvThreads / 32];
    __shared__ float s_rinv;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gw = blockIdx.x * (kGemvThreads / 32) + warp;
    const int nw = gridDim.x * (kGemvThreads / 32);
    const int nchunk = p.K >> 3;        // 16-byte chunks per row
    const int nstep = nchunk >> 5;      // chunk steps of the whole warp

    // weights do not depend on the previous kernel: warm L2 with this warp's first rows
    if (gw < p.units) {
        int ra, rb;
        unit_rows<MODE>(p, gw, ra, rb);
        const char* pa = reinterpret_cast<const char*>(p.W + (size_t)ra * p.K);
        const char* pb = reinterpret_cast<const char*>(p.W + (size_t)rb * p.K);
        for (int l = lane; l < (p.K * 2) / 128; l += 32) {
            asm volatile("prefetch.global.L2 [%0];" ::"l"(pa + l * 128));
            asm volatile("prefetch.global.L2 [%0];" ::"l"(pb + l * 128));
        }
    }
    const uint4* xg = reinterpret_cast<const uint4*>(p.xv);
    for (int i = threadIdx.x; i < nchunk; i += kGemvThreads) xs[i] = xg[i];
    __syncthreads();
    float rinv = 1.f;
    if constexpr (MODE != kGemvResid) {
        float ss = 0.f;
        for (int i = threadIdx.x; i < nchunk; i += kGemvThreads) {
            const uint4 v = xs[i];
            ss += dot8(v, v);
        }
        ss = warp_sum(ss);
        if (lane == 0) red[warp] = ss;
        __syncthreads();
        if (threadIdx.x == 0) {
            float t = 0.f;
            for (int w = 0; w < kGemvThreads / 32; ++w) t += red[w];
            s_rinv = 1.0f / sqrtf(t / (float)p.K + p.eps);
        }
        __syncthreads();
        rinv = s_rinv;
    }

    int pos = 0;
    if constexpr (MODE == kGemvQKV) pos = *p.d_len;

    for (int u = gw; u < p.units; u += nw) {
        int ra, rb;
        unit_rows<MODE>(p, u, ra, rb);
        const uint4* wa = reinterpret_cast<const uint4*>(p.W + (size_t)ra * p.K);
        const uint4* wb = reinterpret_cast<const uint4*>(p.W + (size_t)rb * p.K);
        float acc_a = 0.f, acc_b = 0.f;
        for (int s = 0; s < nstep; s += kGemvU) {
            uint4 va[kGemvU], vb[kGemvU];
#pragma unroll
            for (int i = 0; i < kGemvU; ++i) {
                if (s + i < nstep) {
                    const int c = (s + i) * 32 + lane;
                    va[i] = ldg_stream(wa + c);
                    vb[i] = ldg_stream(wb + c);
                }
            }
#pragma unroll
            for (int i = 0; i < kGemvU; ++i) {
                if (s + i < nstep) {
                    const uint4 x = xs[(s + i) * 32 + lane];
                    acc_a += dot8(va[i], x);
                    acc_b += dot8(vb[i], x);
                }
            }
        }
        acc_a = warp_sum(acc_a);
        acc_b = warp_sum(acc_b);
        if (lane == 0) gemv_epilogue<MODE>(p, u, ra, rb, acc_a, acc_b, rinv, pos);
    }
}

// ---------------------------------------------------------------------------------------
// split-KV attention
// ---------------------------------------------------------------------------------------
struct AttnDecParams {
    const float* q;  // [H*dh]
    const bf16* kc;  // layer base [Hkv][max_ctx][dh]
    const bf16* vc;
    const int* d_len;  // position of the new token; context = d_len + 1
    int H, Hkv, max_ctx, splits;
    float scale_log2;
    float* part_o;   // [splits][H][dh]
    float* part_ml;  // [splits][H][2]
    unsigned* tickets;  // [Hkv] arrival counters (0 between launches)
    bf16* out;          // [H*dh] merged attention output
    int cap;            // keys of one split held in shared memory (>= ceil(max_ctx / splits))
    unsigned* status;
};

constexpr int kAttnThreads = 256;
constexpr int kAttnWarps = kAttnThreads / 32;

// CTA = (KV head g, split): keys [kb, ke) of the context. One thread bulk-copies the split's K
// and V rows (contiguous in the cache) into shared memory in one round trip; the 8 warps then
// take 2 keys per pass (16 lanes per key row, d_h/16 dims per lane) for all G query heads of
// the group with an fp32 online softmax; warp states merge in shared memory into the split's
// partial (max, sum, unnormalised output). The last CTA of the KV head to finish (atomic
// ticket) merges the splits in fixed order and writes the attention output.
template <int DH, int G>
__global__ void __launch_bounds__(kAttnThreads) attn_decode_kernel(AttnDecParams p) {
    constexpr int DPL = DH / 16;
    extern __shared__ __align__(128) uint8_t smem[];
    bf16* sK = reinterpret_cast<bf16*>(smem);
    bf16* sV = sK + (size_t)p.cap * DH;
    float* scratch = reinterpret_cast<float*>(sV + (size_t)p.cap * DH);
    __shared__ uint64_t bar;
    __shared__ float sm_m[kAttnWarps][G], sm_l[kAttnWarps][G];
    __shared__ float sm_o[kAttnWarps][G][DH];
    __shared__ unsigned s_ticket;
    __shared__ int s_ok;
    const int kvh = blockIdx.x, split = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane >> 4, l16 = lane & 15;
    const int ctx = *p.d_len + 1;
    const int chunk = (ctx + p.splits - 1) / p.splits;
    const int kb = split * chunk;
    const int ke = min(ctx, kb + chunk);
    const int nk = max(0, min(ke - kb, p.cap));
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
        s_ok = 1;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const uint32_t bytes = (uint32_t)nk * DH * 2u;
        mbar_arrive_expect_tx(&bar, 2u * bytes);
        if (bytes) {
            const size_t off = ((size_t)kvh * p.max_ctx + kb) * DH;
            bulk_load(sK, p.kc + off, bytes, &bar);
            bulk_load(sV, p.vc + off, bytes, &bar);
        }
    }
    float qv[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh)
#pragma unroll
        for (int d = 0; d < DPL; ++d) qv[hh][d] = p.q[(kvh * G + hh) * DH + l16 * DPL + d] * p.scale_log2;
    if (!mbar_wait(&bar, 0)) s_ok = 0;  // bounded; the copy itself always completes
    __syncthreads();
    float m[G], l[G], o[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        m[hh] = -INFINITY;
        l[hh] = 0.f;
#pragma unroll
        for (int d = 0; d < DPL; ++d) o[hh][d] = 0.f;
    }
    if (s_ok) {
        for (int k0 = warp * 2; k0 < nk; k0 += kAttnWarps * 2) {  // warp-uniform bound
            const int k = k0 + sub;
            const bool valid = k < nk;
            float kf[DPL], vf[DPL];
            const bf16* kr = sK + (size_t)(valid ? k : 0) * DH + l16 * DPL;
            const bf16* vr = sV + (size_t)(valid ? k : 0) * DH + l16 * DPL;
#pragma unroll
            for (int c = 0; c < DPL / 4; ++c) {
                const uint2 kw = *reinterpret_cast<const uint2*>(kr + 4 * c);
                const uint2 vw = *reinterpret_cast<const uint2*>(vr + 4 * c);
                kf[4 * c] = bf16_lo(kw.x);
                kf[4 * c + 1] = bf16_hi(kw.x);
                kf[4 * c + 2] = bf16_lo(kw.y);
                kf[4 * c + 3] = bf16_hi(kw.y);
                vf[4 * c] = bf16_lo(vw.x);
                vf[4 * c + 1] = bf16_hi(vw.x);
                vf[4 * c + 2] = bf16_lo(vw.y);
                vf[4 * c + 3] = bf16_hi(vw.y);
            }
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                float sc = 0.f;
#pragma unroll
                for (int d = 0; d < DPL; ++d) sc = fmaf(qv[hh][d], kf[d], sc);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 1);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 2);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 4);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 8);
                if (!valid) continue;
                const float mn = fmaxf(m[hh], sc);
                const float c = exp2f(m[hh] - mn);
                const float pe = exp2f(sc - mn);
                l[hh] = l[hh] * c + pe;
#pragma unroll
                for (int d = 0; d < DPL; ++d) o[hh][d] = fmaf(o[hh][d], c, pe * vf[d]);
                m[hh] = mn;
            }
        }
    }
    // merge the two key slots of the warp (lanes l16 and l16 + 16), then the warps
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m[hh], 16);
        const float l2 = __shfl_xor_sync(0xFFFFFFFFu, l[hh], 16);
        const float mn = fmaxf(m[hh], m2);
        const float c1 = (mn == -INFINITY) ? 0.f : exp2f(m[hh] - mn);
        const float c2 = (mn == -INFINITY) ? 0.f : exp2f(m2 - mn);
        l[hh] = l[hh] * c1 + l2 * c2;
#pragma unroll
        for (int d = 0; d < DPL; ++d) {
            const float o2 = __shfl_xor_sync(0xFFFFFFFFu, o[hh][d], 16);
            o[hh][d] = o[hh][d] * c1 + o2 * c2;
        }
        m[hh] = mn;
    }
    if (sub == 0) {
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            if (l16 == 0) {
                sm_m[warp][hh] = m[hh];
                sm_l[warp][hh] = l[hh];
            }
#pragma unroll
            for (int d = 0; d < DPL; ++d) sm_o[warp][hh][l16 * DPL + d] = o[hh][d];
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < G * DH; e += kAttnThreads) {
        const int hh = e / DH, d = e % DH;
        float mx = -INFINITY;
        for (int w = 0; w < kAttnWarps; ++w) mx = fmaxf(mx, sm_m[w][hh]);
        float lt = 0.f, ot = 0.f;
        if (mx != -INFINITY) {
            for (int w = 0; w < kAttnWarps; ++w) {
                const float c = exp2f(sm_m[w][hh] - mx);
                lt += sm_l[w][hh] * c;
                ot += sm_o[w][hh][d] * c;
            }
        }
        const int h = kvh * G + hh;
        p.part_o[((size_t)split * p.H + h) * DH + d] = ot;
        if (d == 0) {
            p.part_ml[((size_t)split * p.H + h) * 2 + 0] = mx;
            p.part_ml[((size_t)split * p.H + h) * 2 + 1] = lt;
        }
    }
    if (!s_ok && threadIdx.x == 0) set_status(p.status, kDevTimeout);
    // the last CTA of this KV head merges its splits (fixed order), then re-arms the counter
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_ticket = atomicAdd(&p.tickets[kvh], 1u);
    __syncthreads();
    if (s_ticket != (unsigned)(p.splits - 1)) return;
    __threadfence();
    float* wgt = scratch;                   // [G][splits] max -> weights
    float* wl = scratch + G * p.splits;     // [G][splits] sums
    float* tot = wl + G * p.splits;         // [G]
    for (int e = threadIdx.x; e < G * p.splits; e += kAttnThreads) {
        const int hh = e / p.splits, s2 = e % p.splits;
        const float2 ml = __ldcg(reinterpret_cast<const float2*>(p.part_ml + ((size_t)s2 * p.H + kvh * G + hh) * 2));
        wgt[e] = ml.x;
        wl[e] = ml.y;
    }
    __syncthreads();
    if (threadIdx.x < G) {
        const int hh = threadIdx.x;
        float mx = -INFINITY;
        for (int s2 = 0; s2 < p.splits; ++s2) mx = fmaxf(mx, wgt[hh * p.splits + s2]);
        float lt = 0.f;
        for (int s2 = 0; s2 < p.splits; ++s2) {
            const float ms = wgt[hh * p.splits + s2];
            const float c = (ms == -INFINITY) ? 0.f : exp2f(ms - mx);
            wgt[hh * p.splits + s2] = c;
            lt += wl[hh * p.splits + s2] * c;
        }
        tot[hh] = lt;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < G * DH; e += kAttnThreads) {
        const int hh = e / DH, d = e % DH;
        const int h = kvh * G + hh;
        float ot = 0.f;
#pragma unroll 16
        for (int s2 = 0; s2 < p.splits; ++s2)
            ot += __ldcg(p.part_o + ((size_t)s2 * p.H + h) * DH + d) * wgt[hh * p.splits + s2];
        p.out[h * DH + d] = __float2bfloat16_rn(ot / tot[hh]);
    }
    if (threadIdx.x == 0) p.tickets[kvh] = 0u;
}

__global__ void advance_lengths_kernel(int* d_len, int count) {
    const int i = threadIdx.x;
    if (i < count) d_len[i] += 1;
}

template <int MODE>
cudaError_t launch_gemv(const GemvParams& p, int num_sms, cudaStream_t s) {
    const size_t smem = (size_t)p.K * 2;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemv_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, 64 * 1024);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int warps_needed = p.units;
    int grid = 2 * num_sms;
    const int gmax = (warps_needed + 7) / 8;
    if (grid > gmax) grid = gmax;
    gemv_kernel<MODE><<<grid, kGemvThreads, smem, s>>>(p);
    return cudaGetLastError();
}

template <int DH, int G>
cudaError_t launch_attn_dec(const AttnDecParams& p, cudaStream_t s) {
    const size_t smem = (size_t)2 * p.cap * DH * 2 + (size_t)(2 * G * p.splits + G) * sizeof(float);
    static size_t attr = 0;
    if (smem > attr) {
        cudaError_t e = cudaFuncSetAttribute(attn_decode_kernel<DH, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        attr = smem;
    }
    attn_decode_kernel<DH, G><<<dim3(p.Hkv, p.splits), kAttnThreads, smem, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_attn_dec_any(int dh, int group, const AttnDecParams& p, cudaStream_t s) {
    if (dh == 128) {
        switch (group) {
            case 1: return launch_attn_dec<128, 1>(p, s);
            case 2: return launch_attn_dec<128, 2>(p, s);
            case 4: return launch_attn_dec<128, 4>(p, s);
            case 8: return launch_attn_dec<128, 8>(p, s);
        }
    } else if (dh == 64) {
        switch (group) {
            case 1: return launch_attn_dec<64, 1>(p, s);
            case 2: return launch_attn_dec<64, 2>(p, s);
            case 4: return launch_attn_dec<64, 4>(p, s);
            case 8: return launch_attn_dec<64, 8>(p, s);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_decode_layer(const DecodeLayer& L, const DecodeDims& d, const DecodeWork& w, const bf16* x_in,
                                bf16* x_out, int num_sms, cudaStream_t stream, const StageHook& hook) {
    cudaError_t e;
    const int qc = d.H * d.dh, kvc = d.Hkv * d.dh;
    // 1. RMSNorm + QKV + RoPE + KV append
    GemvParams g = {};
    g.W = L.w_qkv;
    g.K = d.D;
    g.units = (qc + 2 * kvc) / 2;
    g.xv = x_in;
    g.q_out = w.q;
    g.kcache = L.kcache;
    g.vcache = L.vcache;
    g.d_len = L.d_len;
    g.rope = w.rope;
    g.dh = d.dh;
    g.n_q_heads = d.H;
    g.n_kv_heads = d.Hkv;
    g.max_ctx = d.max_ctx;
    g.eps = d.eps;
    hook(kStageDecQKV, true);
    e = launch_gemv<kGemvQKV>(g, num_sms, stream);
    hook(kStageDecQKV, false);
    if (e != cudaSuccess) return e;
    // 2. split-KV attention + combine
    AttnDecParams a = {};
    a.q = w.q;
    a.kc = L.kcache;
    a.vc = L.vcache;
    a.d_len = L.d_len;
    a.H = d.H;
    a.Hkv = d.Hkv;
    a.max_ctx = d.max_ctx;
    a.splits = w.splits;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)d.dh);
    a.part_o = w.part_o;
    a.part_ml = w.part_ml;
    a.tickets = w.tickets;
    a.out = w.attn;
    a.cap = (d.max_ctx + w.splits - 1) / w.splits;
    a.status = w.status;
    hook(kStageDecAttn, true);
    e = launch_attn_dec_any(d.dh, d.H / d.Hkv, a, stream);
    hook(kStageDecAttn, false);
    if (e != cudaSuccess) return e;
    // 3. O projection + residual
    GemvParams o = {};
    o.W = L.w_o;
    o.K = qc;
    o.units = d.D / 2;
    o.xv = w.attn;
    o.resid = x_in;
    o.out = w.x_mid;
    hook(kStageDecO, true);
    e = launch_gemv<kGemvResid>(o, num_sms, stream);
    hook(kStageDecO, false);
    if (e != cudaSuccess) return e;
    // 4. RMSNorm + gate/up + SwiGLU
    GemvParams gu = {};
    gu.W = L.w_gu;
    gu.K = d.D;
    gu.units = d.F_pad;
    gu.xv = w.x_mid;
    gu.out = w.m;
    gu.eps = d.eps;
    hook(kStageDecGateUp, true);
    e = launch_gemv<kGemvSwiGLU>(gu, num_sms, stream);
    hook(kStageDecGateUp, false);
    if (e != cudaSuccess) return e;
    // 5. down projection + residual
    GemvParams dn = {};
    dn.W = L.w_d;
    dn.K = d.F_pad;
    dn.units = d.D / 2;
    dn.xv = w.m;
    dn.resid = w.x_mid;
    dn.out = x_out;
    hook(kStageDecDown, true);
    e = launch_gemv<kGemvResid>(dn, num_sms, stream);
    hook(kStageDecDown, false);
    return e;
}

cudaError_t launch_advance_lengths(int* d_len, int count, cudaStream_t stream) {
    if (count <= 0) return cudaSuccess;
    advance_lengths_kernel<<<1, ((count + 31) / 32) * 32, 0, stream>>>(d_len, count);
    return cudaGetLastError();
}

}  // namespace vla
