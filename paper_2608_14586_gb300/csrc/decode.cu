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
// row, online softmax in fp32; a combine kernel merges the partial (max, sum, output).
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
};

constexpr int kAttnThreads = 128;

template <int DH, int G>
__global__ void __launch_bounds__(kAttnThreads) attn_decode_partial_kernel(AttnDecParams p) {
    constexpr int DPL = DH / 8;  // dims per lane (8 lanes per key row)
    constexpr int NW = kAttnThreads / 32;
    __shared__ float sm_m[NW][G], sm_l[NW][G];
    __shared__ float sm_o[NW][G][DH];
    const int kvh = blockIdx.x, split = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane >> 3, l8 = lane & 7;
    const int ctx = *p.d_len + 1;
    const int chunk = (ctx + p.splits - 1) / p.splits;
    const int kb = split * chunk;
    const int ke = min(ctx, kb + chunk);

    float qv[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh)
#pragma unroll
        for (int d = 0; d < DPL; ++d) qv[hh][d] = p.q[(kvh * G + hh) * DH + l8 * DPL + d] * p.scale_log2;
    float m[G], l[G], o[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        m[hh] = -INFINITY;
        l[hh] = 0.f;
#pragma unroll
        for (int d = 0; d < DPL; ++d) o[hh][d] = 0.f;
    }
    const bf16* kbase = p.kc + (size_t)kvh * p.max_ctx * DH + l8 * DPL;
    const bf16* vbase = p.vc + (size_t)kvh * p.max_ctx * DH + l8 * DPL;
    // The loop bound is warp-uniform (k0 steps by warp); each 8-lane slot takes key k0 + sub
    // and skips the update when that key is past the range, so every lane reaches every
    // full-warp shuffle below.
    for (int k0 = kb + warp * 4; k0 < ke; k0 += NW * 4) {
        const int k = k0 + sub;
        const bool valid = k < ke;
        uint4 kr[DPL / 8], vr[DPL / 8];
#pragma unroll
        for (int c = 0; c < DPL / 8; ++c) {
            if (valid) {
                kr[c] = ldg_stream(kbase + (size_t)k * DH + c * 8);
                vr[c] = ldg_stream(vbase + (size_t)k * DH + c * 8);
            } else {
                kr[c] = make_uint4(0u, 0u, 0u, 0u);
                vr[c] = make_uint4(0u, 0u, 0u, 0u);
            }
        }
        float kf[DPL], vf[DPL];
#pragma unroll
        for (int c = 0; c < DPL / 8; ++c) {
            const uint32_t kw[4] = {kr[c].x, kr[c].y, kr[c].z, kr[c].w};
            const uint32_t vw[4] = {vr[c].x, vr[c].y, vr[c].z, vr[c].w};
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
            const float c = exp2f(m[hh] - mn);  // m = -inf -> 0
            const float pe = exp2f(s - mn);
            l[hh] = l[hh] * c + pe;
#pragma unroll
            for (int d = 0; d < DPL; ++d) o[hh][d] = fmaf(o[hh][d], c, pe * vf[d]);
            m[hh] = mn;
        }
    }
    // merge the 4 key slots of the warp (lanes l8, l8+8, l8+16, l8+24)
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
    // merge warps: thread t handles (head hh, dim d) entries
    for (int e = threadIdx.x; e < G * DH; e += kAttnThreads) {
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
        p.part_o[((size_t)split * p.H + h) * DH + d] = ot;
        if (d == 0) {
            p.part_ml[((size_t)split * p.H + h) * 2 + 0] = mx;
            p.part_ml[((size_t)split * p.H + h) * 2 + 1] = lt;
        }
    }
}

// out[h*dh + d] = sum_s o_s e^(m_s - M) / sum_s l_s e^(m_s - M)   (fixed split order)
__global__ void attn_decode_combine_kernel(const float* part_o, const float* part_ml, int H, int dh, int splits,
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
    attn_decode_partial_kernel<DH, G><<<dim3(p.Hkv, p.splits), kAttnThreads, 0, s>>>(p);
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
    hook(kStageDecAttn, true);
    e = launch_attn_dec_any(d.dh, d.H / d.Hkv, a, stream);
    hook(kStageDecAttn, false);
    if (e != cudaSuccess) return e;
    hook(kStageDecCombine, true);
    attn_decode_combine_kernel<<<d.H, d.dh, 0, stream>>>(w.part_o, w.part_ml, d.H, d.dh, w.splits, w.attn);
    e = cudaGetLastError();
    hook(kStageDecCombine, false);
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
