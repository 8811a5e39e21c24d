// Single-token decode of one block (the prefix range at M = 1, position = KV length).
//
// At M = 1 every projection is a matrix-vector product whose cost is streaming the weights
// once from HBM (354 MB per 7B-class block), so these kernels are built for bandwidth:
//   * each warp takes a contiguous range of row pairs (the same count for every warp) and
//     streams their rows through a ring of shared-memory slots with 1-D bulk copies
//     (cp.async.bulk, completion on per-slot mbarriers), up to 24 KB per warp and 192 KB per
//     SM in flight; fp32 FMA over 16-byte chunks, warp-shuffle reduction;
//   * the pair is chosen so the fused epilogue has both operands it needs: dims (j, j+dh/2)
//     of a head for the rotary embedding (adjacent rows of the repacked q/k weights), the
//     gate and up rows of one feed-forward unit for SwiGLU, consecutive rows for the
//     residual projections;
//   * the input vector is staged in shared memory; RMSNorm's 1/rms is computed per CTA
//     (the gains are folded into the weights);
//   * under programmatic dependent launch each kernel starts while its predecessor drains:
//     it requests the first ring slots of its weight rows, and reads nothing that an earlier
//     kernel of the step wrote before griddepcontrol.wait.
// Attention is split over the context inside one thread-block cluster per KV head (16 CTAs
// where the device schedules such clusters, else 8; fixed split count -> deterministic): each
// CTA bulk-copies its contiguous key range of K and V into shared memory (the rows that
// predate the step before the wait, so the copy overlaps the QKV kernel), scores it for all
// query heads of the GQA group with an online softmax, and the cluster merges the partial
// (max, sum, output) states through distributed shared memory in fixed rank order.
#include <algorithm>
#include <cstring>

#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

enum GemvMode : int { kGemvQKV = 0, kGemvResid = 1, kGemvSwiGLU = 2 };

// A batch of NB token vectors (NB <= kMaxDecodeBatch), each of its own sequence: the
// weights stream once for all of them. Per-sequence arrays are [NB][...] with the stride of
// one vector.
struct GemvParams {
    const bf16* W;  // [rows, K] row-major
    int K;          // multiple of 256
    int units;      // row pairs
    const bf16* xv;     // input vectors [NB][K]
    const bf16* resid;  // kGemvResid: residual [NB][2*units]
    bf16* out;          // kGemvResid: [NB][2*units]; kGemvSwiGLU: [NB][units]
    float* q_out;       // kGemvQKV: post-RoPE queries, fp32 [NB][H*dh]
    bf16* kcache[kMaxDecodeBatch];  // kGemvQKV: each sequence's layer K / V planes
    bf16* vcache[kMaxDecodeBatch];
    const int* d_len[kMaxDecodeBatch];  // kGemvQKV: position of each sequence's new token
    const float2* rope;
    int dh, n_q_heads, n_kv_heads, max_ctx;
    float eps;
    unsigned* status;  // timeout report (a weight copy that never lands)
    int per_warp;      // row pairs per warp (set at launch)
    int stages;        // ring slots per warp (set at launch)
};

constexpr int kGemvThreads = 256;
constexpr int kGemvWarps = kGemvThreads / 32;
constexpr int kGemvSegBytes = 4096;  // bytes of each row per ring slot
constexpr int kGemvMaxStages = 3;
constexpr size_t kGemvSmemBudget = 226 * 1024;  // dynamic shared memory of one CTA (of 227 KB)

// a * b + c on the low (HI false) or high bf16 halves of two packed words, rounded once to
// fp32 by the mixed-precision fma: a bf16 product is exact in fp32, so this is fmaf on the
// widened values, without the widening instructions
template <bool HI>
VLA_DEV float fma_bf16(uint32_t a, uint32_t b, float c) {
    float d;
    if constexpr (HI)
        asm("{\n\t.reg .b16 al, ah, bl, bh;\n\tmov.b32 {al, ah}, %1;\n\tmov.b32 {bl, bh}, %2;\n\t"
            "fma.rn.f32.bf16 %0, ah, bh, %3;\n\t}"
            : "=f"(d)
            : "r"(a), "r"(b), "f"(c));
    else
        asm("{\n\t.reg .b16 al, ah, bl, bh;\n\tmov.b32 {al, ah}, %1;\n\tmov.b32 {bl, bh}, %2;\n\t"
            "fma.rn.f32.bf16 %0, al, bl, %3;\n\t}"
            : "=f"(d)
            : "r"(a), "r"(b), "f"(c));
    return d;
}

// sum of the eight products of two packed bf16 vectors, in order (the first product alone:
// adding -0 keeps the sign of a zero product, as a plain multiply would)
VLA_DEV float dot8(uint4 w, uint4 x) {
    float a = fma_bf16<false>(w.x, x.x, -0.0f);
    a = fma_bf16<true>(w.x, x.x, a);
    a = fma_bf16<false>(w.y, x.y, a);
    a = fma_bf16<true>(w.y, x.y, a);
    a = fma_bf16<false>(w.z, x.z, a);
    a = fma_bf16<true>(w.z, x.z, a);
    a = fma_bf16<false>(w.w, x.w, a);
    a = fma_bf16<true>(w.w, x.w, a);
    return a;
}

template <int MODE>
VLA_DEV void unit_rows(const GemvParams& p, int u, int& ra, int& rb) {
    if constexpr (MODE == kGemvQKV) {
        const int half = p.dh >> 1;
        const int head = u / half, j = u % half;
        if (head < p.n_q_heads + p.n_kv_heads) {  // q, k: the pair's rows are adjacent
            ra = head * p.dh + 2 * j;
            rb = ra + 1;
        } else {
            ra = head * p.dh + j;
            rb = ra + half;
        }
    } else if constexpr (MODE == kGemvSwiGLU) {
        const int grp = u >> 7, i = u & 127;
        ra = grp * 256 + i;
        rb = ra + 128;
    } else {
        ra = 2 * u;
        rb = 2 * u + 1;
    }
}

// Fused epilogue of one row pair for sequence b (lane 0 of the warp that reduced it).
template <int MODE>
VLA_DEV void gemv_epilogue(const GemvParams& p, int b, int u, int ra, int rb, float acc_a, float acc_b, float rinv,
                           int pos) {
    if constexpr (MODE == kGemvResid) {
        const size_t n = (size_t)2 * p.units * b;
        const float ya = __bfloat162float(p.resid[n + ra]) + acc_a;
        const float yb = __bfloat162float(p.resid[n + rb]) + acc_b;
        *reinterpret_cast<uint32_t*>(p.out + n + ra) = pack_bf16x2(ya, yb);
    } else if constexpr (MODE == kGemvSwiGLU) {
        const float g = acc_a * rinv, up = acc_b * rinv;
        p.out[(size_t)p.units * b + u] = __float2bfloat16_rn(g / (1.0f + __expf(-g)) * up);
    } else {
        const int half = p.dh >> 1;
        const int head = u / half, j = u % half;
        float a = acc_a * rinv, bb = acc_b * rinv;
        if (head < p.n_q_heads + p.n_kv_heads) {
            const float2 cs = p.rope[(size_t)pos * half + j];
            const float a2 = a * cs.x - bb * cs.y;
            const float b2 = bb * cs.x + a * cs.y;
            a = a2;
            bb = b2;
        }
        if (head < p.n_q_heads) {
            float* q = p.q_out + (size_t)b * p.n_q_heads * p.dh;
            q[head * p.dh + j] = a;
            q[head * p.dh + j + half] = bb;
        } else if (head < p.n_q_heads + p.n_kv_heads) {
            bf16* kp = p.kcache[b] + ((size_t)(head - p.n_q_heads) * p.max_ctx + pos) * p.dh;
            kp[j] = __float2bfloat16_rn(a);
            kp[j + half] = __float2bfloat16_rn(bb);
        } else {
            bf16* vp = p.vcache[b] + ((size_t)(head - p.n_q_heads - p.n_kv_heads) * p.max_ctx + pos) * p.dh;
            vp[j] = __float2bfloat16_rn(a);
            vp[j + half] = __float2bfloat16_rn(bb);
        }
    }
}

// One warp per contiguous range of `per_warp` row pairs (balanced: every warp but the last
// takes the same count, and the grid has as many CTAs as that needs, at most one per SM).
// Lane 0 of each warp streams its pairs' rows through the warp's ring of `stages` slots, each
// slot a 4 KB segment of both rows of a pair, with 1-D bulk copies completing on the slot's
// mbarrier; the first slots are requested before griddepcontrol.wait, since the weights do
// not depend on the previous kernel. Lane l accumulates the 16-byte chunks l, l + 32, ... of
// the row in order (fp32), then the warp reduces and lane 0 applies the fused epilogue.
template <int MODE, int NB>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_kernel(const __grid_constant__ GemvParams p) {
    extern __shared__ __align__(16) uint8_t gsm[];
    uint4* xs = reinterpret_cast<uint4*>(gsm);  // [NB][K/8] input vectors
    __shared__ uint64_t full[kGemvWarps][kGemvMaxStages];
    __shared__ float red[NB][kGemvWarps];
    __shared__ float s_rinv[NB];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gw = blockIdx.x * kGemvWarps + warp;
    const int nchunk = p.K >> 3;  // 16-byte chunks per row
    const int row_bytes = p.K * 2;
    const int nseg = (row_bytes + kGemvSegBytes - 1) / kGemvSegBytes;
    const int u0 = gw * p.per_warp;
    const int T = max(0, min(p.units, u0 + p.per_warp) - u0) * nseg;  // ring stages of this warp
    const int S = p.stages;
    uint8_t* ring = gsm + (size_t)NB * row_bytes + (size_t)warp * S * 2 * kGemvSegBytes;

    // lane 0: segment t % nseg of row pair u0 + t / nseg into slot t % S
    auto issue = [&](int t) {
        const int u = u0 + t / nseg, sg = t % nseg;
        int ra, rb;
        unit_rows<MODE>(p, u, ra, rb);
        const int off = sg * kGemvSegBytes;
        const uint32_t bytes = (uint32_t)min(kGemvSegBytes, row_bytes - off);
        uint64_t* bar = &full[warp][t % S];
        uint8_t* dst = ring + (size_t)(t % S) * 2 * kGemvSegBytes;
        mbar_arrive_expect_tx(bar, 2 * bytes);
        bulk_load(dst, reinterpret_cast<const uint8_t*>(p.W + (size_t)ra * p.K) + off, bytes, bar);
        bulk_load(dst + kGemvSegBytes, reinterpret_cast<const uint8_t*>(p.W + (size_t)rb * p.K) + off, bytes, bar);
    };
    if (lane == 0) {
        for (int j = 0; j < S; ++j) mbar_init(&full[warp][j], 1);
        fence_barrier_init();
        for (int t = 0; t < min(T, S); ++t) issue(t);
    }
    pdl_wait();
    pdl_trigger();
    const uint4* xg = reinterpret_cast<const uint4*>(p.xv);
    for (int i = threadIdx.x; i < NB * nchunk; i += kGemvThreads) xs[i] = __ldcg(xg + i);
    __syncthreads();  // also publishes the barrier initialisation to the whole warp
    float rinv[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) rinv[b] = 1.f;
    if constexpr (MODE != kGemvResid) {
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            float ss = 0.f;
            for (int i = threadIdx.x; i < nchunk; i += kGemvThreads) {
                const uint4 v = xs[b * nchunk + i];
                ss += dot8(v, v);
            }
            ss = warp_sum(ss);
            if (lane == 0) red[b][warp] = ss;
        }
        __syncthreads();
        if (threadIdx.x < NB) {
            float t = 0.f;
            for (int w = 0; w < kGemvWarps; ++w) t += red[threadIdx.x][w];
            s_rinv[threadIdx.x] = 1.0f / sqrtf(t / (float)p.K + p.eps);
        }
        __syncthreads();
#pragma unroll
        for (int b = 0; b < NB; ++b) rinv[b] = s_rinv[b];
    }

    int pos[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) pos[b] = 0;
    if constexpr (MODE == kGemvQKV) {
#pragma unroll
        for (int b = 0; b < NB; ++b) pos[b] = *p.d_len[b];
    }

    float acc_a[NB], acc_b[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) acc_a[b] = acc_b[b] = 0.f;
    int t = 0;
    for (; t < T; ++t) {
        const int slot = t % S, sg = t % nseg;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait(&full[warp][slot], (uint32_t)(t / S) & 1u))) break;
        const uint4* wa = reinterpret_cast<const uint4*>(ring + (size_t)slot * 2 * kGemvSegBytes);
        const uint4* wb = wa + kGemvSegBytes / 16;
        const int c0 = sg * (kGemvSegBytes / 16);                       // first chunk of the segment
        const int nch = min(kGemvSegBytes, row_bytes - sg * kGemvSegBytes) >> 4;  // a multiple of 32
#pragma unroll 4
        for (int c = lane; c < nch; c += 32) {
            const uint4 va = wa[c], vb = wb[c];
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                const uint4 x = xs[b * nchunk + c0 + c];
                acc_a[b] += dot8(va, x);
                acc_b[b] += dot8(vb, x);
            }
        }
        __syncwarp();  // every lane has read the slot
        if (lane == 0 && t + S < T) {
            fence_proxy_async_smem();
            issue(t + S);
        }
        if (sg == nseg - 1) {
            const int u = u0 + t / nseg;
            int ra, rb;
            unit_rows<MODE>(p, u, ra, rb);
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                const float sa = warp_sum(acc_a[b]);
                const float sb = warp_sum(acc_b[b]);
                if (lane == 0) gemv_epilogue<MODE>(p, b, u, ra, rb, sa, sb, rinv[b], pos[b]);
                acc_a[b] = acc_b[b] = 0.f;
            }
        }
    }
    if (t < T) {
        // a copy did not land within the wait budget: report it and let the copies already
        // requested into this warp's ring finish (again bounded) before the CTA exits
        if (lane == 0) {
            set_status(p.status, kDevTimeout);
            for (int r = t; r < min(T, t + S); ++r) mbar_wait(&full[warp][r % S], (uint32_t)(r / S) & 1u);
        }
        __syncwarp();
    }
}

// ---------------------------------------------------------------------------------------
// split-KV attention: one thread-block cluster per KV head
// ---------------------------------------------------------------------------------------
struct AttnDecParams {
    const float* q;  // [nb][H*dh] post-RoPE queries, fp32
    const bf16* kc[kMaxDecodeBatch];  // each sequence's layer base [Hkv][max_ctx][dh]
    const bf16* vc[kMaxDecodeBatch];
    const int* d_len[kMaxDecodeBatch];  // positions of the new tokens; context = d_len + 1
    int nb, H, Hkv, max_ctx;
    int cs;      // CTAs per cluster = key splits per KV head
    int cap;     // keys per shared-memory stage
    int stages;  // 1 or 2
    float scale_log2;
    bf16* out;  // [nb][H*dh] attention outputs
    unsigned* status;
};

constexpr int kAttnThreads = 256;
constexpr int kAttnWarps = kAttnThreads / 32;
constexpr int kMaxCluster = 16;

template <int DPL>
VLA_DEV void load_row_part(const bf16* src, float (&f)[DPL]) {
    if constexpr (DPL == 8) {
        const uint4 w = *reinterpret_cast<const uint4*>(src);
        f[0] = bf16_lo(w.x), f[1] = bf16_hi(w.x), f[2] = bf16_lo(w.y), f[3] = bf16_hi(w.y);
        f[4] = bf16_lo(w.z), f[5] = bf16_hi(w.z), f[6] = bf16_lo(w.w), f[7] = bf16_hi(w.w);
    } else {
        const uint2 w = *reinterpret_cast<const uint2*>(src);
        f[0] = bf16_lo(w.x), f[1] = bf16_hi(w.x), f[2] = bf16_lo(w.y), f[3] = bf16_hi(w.y);
    }
}

// Cluster (cs CTAs) = KV head g; CTA rank r owns keys [r*ceil(ctx/cs), ...) of the context.
// Thread 0 bulk-copies the rows of each chunk (cap keys) of K and V into a shared-memory stage;
// 8 warps take 2 keys per pass (16 lanes per key row, d_h/16 dims per lane) for all G query
// heads of the group with an fp32 online softmax (scores in the log2 domain). Warp states merge
// in shared memory into the CTA's (max, sum, unnormalised output); after a cluster barrier, CTA
// r merges output elements [r*G*dh/cs, (r+1)*G*dh/cs) over the cs CTAs through distributed
// shared memory, in fixed rank order, and writes them. No partials leave the chip.
template <int DH, int G>
__global__ void __launch_bounds__(kAttnThreads) attn_decode_kernel(const __grid_constant__ AttnDecParams p) {
    constexpr int DPL = DH / 16;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ uint64_t full[2];
    __shared__ float sm_m[kAttnWarps][G], sm_l[kAttnWarps][G];
    __shared__ float sm_o[kAttnWarps][G][DH];
    __shared__ float c_m[G], c_l[G];
    __shared__ __align__(16) float c_o[G * DH];
    __shared__ int s_ok;
    const int rank = blockIdx.x, kvh = blockIdx.y, seq = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bf16* kc = p.kc[seq];
    const bf16* vc = p.vc[seq];
    const int sub = lane >> 4, l16 = lane & 15;
    const size_t stage_elems = (size_t)2 * p.cap * DH;  // K rows then V rows
    bf16* const sbase = reinterpret_cast<bf16*>(smem);
    // d_len was last written by an earlier step (complete before this one started)
    const int ctx = *p.d_len[seq] + 1;
    const int per = (ctx + p.cs - 1) / p.cs;
    const int kb = rank * per;
    const int ke = min(ctx, kb + per);
    const int nk = max(0, ke - kb);
    const int nchunks = (nk + p.cap - 1) / p.cap;
    const int new_row = ctx - 1;  // written by the QKV kernel this one depends on
    // bulk copy of chunk c's rows that existed before this step (rows < new_row)
    auto issue = [&](int c) {
        const int r0 = kb + c * p.cap;
        const int rows = min(p.cap, ke - r0);
        const int old_rows = max(0, min(rows, new_row - r0));
        const uint32_t bytes = (uint32_t)old_rows * DH * 2u;
        bf16* sk = sbase + (size_t)(c % p.stages) * stage_elems;
        uint64_t* bar = &full[c % p.stages];
        mbar_arrive_expect_tx(bar, 2u * bytes);
        if (bytes) {
            const size_t off = ((size_t)kvh * p.max_ctx + r0) * DH;
            bulk_load(sk, kc + off, bytes, bar);
            bulk_load(sk + (size_t)p.cap * DH, vc + off, bytes, bar);
        }
    };
    if (tid == 0) {
        mbar_init(&full[0], 1);
        mbar_init(&full[1], 1);
        fence_barrier_init();
        s_ok = 1;
        for (int c = 0; c < min(nchunks, p.stages); ++c) issue(c);
    }
    pdl_wait();
    pdl_trigger();
    float qv[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh)
#pragma unroll
        for (int d = 0; d < DPL; ++d)
            qv[hh][d] = __ldcg(p.q + ((size_t)seq * p.H + kvh * G + hh) * DH + l16 * DPL + d) * p.scale_log2;
    float m[G], l[G], o[G][DPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        m[hh] = -INFINITY;
        l[hh] = 0.f;
#pragma unroll
        for (int d = 0; d < DPL; ++d) o[hh][d] = 0.f;
    }
    __syncthreads();  // barrier init visible before any wait
    for (int c = 0; c < nchunks; ++c) {
        const int r0 = kb + c * p.cap;
        const int rows = min(p.cap, ke - r0);
        const bf16* sk = sbase + (size_t)(c % p.stages) * stage_elems;
        const bf16* sv = sk + (size_t)p.cap * DH;
        const int nr = new_row - r0;
        if (nr >= 0 && nr < rows && tid < DH / 8) {
            const size_t off = ((size_t)kvh * p.max_ctx + new_row) * DH;
            reinterpret_cast<uint4*>(const_cast<bf16*>(sk) + (size_t)nr * DH)[tid] =
                __ldcg(reinterpret_cast<const uint4*>(kc + off) + tid);
            reinterpret_cast<uint4*>(const_cast<bf16*>(sv) + (size_t)nr * DH)[tid] =
                __ldcg(reinterpret_cast<const uint4*>(vc + off) + tid);
        }
        if (!mbar_wait(&full[c % p.stages], (uint32_t)(c / p.stages) & 1u)) s_ok = 0;
        __syncthreads();
        if (!s_ok) break;  // CTA-uniform
        for (int k0 = warp * 2; k0 < rows; k0 += kAttnWarps * 2) {  // warp-uniform bound
            const int k = k0 + sub;
            const bool valid = k < rows;
            float kf[DPL], vf[DPL];
            load_row_part<DPL>(sk + (size_t)(valid ? k : 0) * DH + l16 * DPL, kf);
            load_row_part<DPL>(sv + (size_t)(valid ? k : 0) * DH + l16 * DPL, vf);
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                float sc = 0.f;
#pragma unroll
                for (int d = 0; d < DPL; ++d) sc = fmaf(qv[hh][d], kf[d], sc);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 1);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 2);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 4);
                sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 8);
                if (valid) {
                    const float mn = fmaxf(m[hh], sc);
                    const float cr = ex2_approx(m[hh] - mn);
                    const float pe = ex2_approx(sc - mn);
                    l[hh] = fmaf(l[hh], cr, pe);
#pragma unroll
                    for (int d = 0; d < DPL; ++d) o[hh][d] = fmaf(o[hh][d], cr, pe * vf[d]);
                    m[hh] = mn;
                }
            }
        }
        __syncthreads();  // stage free
        if (tid == 0 && c + p.stages < nchunks) issue(c + p.stages);
    }
    // merge the two key slots of each warp (lanes l16 and l16 + 16), then the warps
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m[hh], 16);
        const float l2 = __shfl_xor_sync(0xFFFFFFFFu, l[hh], 16);
        const float mn = fmaxf(m[hh], m2);
        const float c1 = (mn == -INFINITY) ? 0.f : ex2_approx(m[hh] - mn);
        const float c2 = (mn == -INFINITY) ? 0.f : ex2_approx(m2 - mn);
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
    for (int e = tid; e < G * DH; e += kAttnThreads) {
        const int hh = e / DH, d = e % DH;
        float mx = -INFINITY;
#pragma unroll
        for (int w = 0; w < kAttnWarps; ++w) mx = fmaxf(mx, sm_m[w][hh]);
        float lt = 0.f, ot = 0.f;
        if (mx != -INFINITY) {
#pragma unroll
            for (int w = 0; w < kAttnWarps; ++w) {
                const float cw = ex2_approx(sm_m[w][hh] - mx);
                lt = fmaf(sm_l[w][hh], cw, lt);
                ot = fmaf(sm_o[w][hh][d], cw, ot);
            }
        }
        c_o[e] = ot;
        if (d == 0) {
            c_m[hh] = mx;
            c_l[hh] = lt;
        }
    }
    if (!s_ok && tid == 0) set_status(p.status, kDevTimeout);
    cluster_sync_all();  // every CTA's (c_m, c_l, c_o) is complete and visible to the cluster
    const int per_cta = G * DH / p.cs;
    if (tid < per_cta) {
        const int e = rank * per_cta + tid;
        const int hh = e / DH;
        float mr[kMaxCluster], lr[kMaxCluster], orr[kMaxCluster];
#pragma unroll
        for (int r = 0; r < kMaxCluster; ++r) {
            if (r < p.cs) {
                mr[r] = ld_dsmem_f32(&c_m[hh], (uint32_t)r);
                lr[r] = ld_dsmem_f32(&c_l[hh], (uint32_t)r);
                orr[r] = ld_dsmem_f32(&c_o[e], (uint32_t)r);
            }
        }
        float mx = -INFINITY;
#pragma unroll
        for (int r = 0; r < kMaxCluster; ++r)
            if (r < p.cs) mx = fmaxf(mx, mr[r]);
        float lt = 0.f, ot = 0.f;
#pragma unroll
        for (int r = 0; r < kMaxCluster; ++r) {
            if (r < p.cs && mr[r] != -INFINITY) {
                const float cw = ex2_approx(mr[r] - mx);
                lt = fmaf(lr[r], cw, lt);
                ot = fmaf(orr[r], cw, ot);
            }
        }
        p.out[((size_t)seq * p.H + kvh * G) * DH + e] = __float2bfloat16_rn(ot / lt);
    }
    cluster_sync_all();  // keep this CTA's shared memory alive until the cluster has read it
}

struct LenPtrs {
    int* p[kMaxDecodeBatch];
};

// block b: the sequence's layer lengths += 1
__global__ void advance_lengths_kernel(const __grid_constant__ LenPtrs lp, int count) {
    const int i = threadIdx.x;
    if (i < count) lp.p[blockIdx.x][i] += 1;
}

template <int MODE, int NB>
cudaError_t launch_gemv_nb(const GemvParams& p_in, int num_sms, cudaStream_t s, bool pdl) {
    GemvParams p = p_in;
    if (p.K % 256 != 0 || p.units <= 0) return cudaErrorInvalidValue;
    // as many ring slots per warp (up to three) as the shared memory of one CTA per SM holds
    // beside the NB input vectors
    const size_t xbytes = (size_t)NB * p.K * 2;
    const size_t slot_bytes = (size_t)kGemvWarps * 2 * kGemvSegBytes;
    if (xbytes + slot_bytes > kGemvSmemBudget) return cudaErrorInvalidValue;
    p.stages = (int)std::min<size_t>(kGemvMaxStages, (kGemvSmemBudget - xbytes) / slot_bytes);
    const size_t smem = xbytes + (size_t)p.stages * slot_bytes;
    auto kern = gemv_kernel<MODE, NB>;
    static size_t attr = 0;
    if (smem > attr) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr = smem;
    }
    // as few row pairs per warp as one CTA per SM allows, then as few warps as that count needs
    const int max_warps = num_sms * kGemvWarps;
    p.per_warp = (p.units + max_warps - 1) / max_warps;
    const int warps = (p.units + p.per_warp - 1) / p.per_warp;
    const int grid = (warps + kGemvWarps - 1) / kGemvWarps;
    return launch_ex(kern, dim3(grid), dim3(kGemvThreads), smem, s, pdl, p);
}

template <int MODE>
cudaError_t launch_gemv(const GemvParams& p, int nb, int num_sms, cudaStream_t s, bool pdl) {
    switch (nb) {
        case 1: return launch_gemv_nb<MODE, 1>(p, num_sms, s, pdl);
        case 2: return launch_gemv_nb<MODE, 2>(p, num_sms, s, pdl);
        case 3: return launch_gemv_nb<MODE, 3>(p, num_sms, s, pdl);
        case 4: return launch_gemv_nb<MODE, 4>(p, num_sms, s, pdl);
    }
    return cudaErrorInvalidValue;
}

template <int DH, int G>
size_t attn_dec_smem(const AttnDecParams& p) {
    return (size_t)p.stages * 2 * p.cap * DH * sizeof(bf16);
}

template <int DH, int G>
cudaError_t attn_dec_prepare(int cs, size_t smem) {
    cudaError_t e = cudaFuncSetAttribute(attn_decode_kernel<DH, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e == cudaSuccess && cs > 8)
        e = cudaFuncSetAttribute(attn_decode_kernel<DH, G>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

template <int DH, int G>
cudaError_t launch_attn_dec(const AttnDecParams& p, cudaStream_t s, bool pdl) {
    const size_t smem = attn_dec_smem<DH, G>(p);
    static size_t attr_smem = 0;
    static int attr_cs = 0;
    if (smem > attr_smem || p.cs > attr_cs) {
        cudaError_t e = attn_dec_prepare<DH, G>(p.cs, smem);
        if (e != cudaSuccess) return e;
        attr_smem = smem > attr_smem ? smem : attr_smem;
        attr_cs = p.cs > attr_cs ? p.cs : attr_cs;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.cs, p.Hkv, p.nb);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = p.cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, attn_decode_kernel<DH, G>, p);
}

// Cluster size and shared-memory staging for a context of up to max_ctx keys: 16 CTAs per KV
// head when the device can co-schedule such clusters, else 8; one stage holding all of a
// CTA's keys when that fits in 160 KB, else two stages of a fixed chunk.
template <int DH, int G>
cudaError_t attn_dec_plan(int Hkv, int max_ctx, int* cs, int* cap, int* stages) {
    constexpr size_t kBudget = 160 * 1024;
    const size_t row_pair = (size_t)2 * DH * sizeof(bf16);
    for (int c : {16, 8}) {
        const int keys = (max_ctx + c - 1) / c;
        int st = 1, cp = keys;
        if ((size_t)keys * row_pair > kBudget) {
            st = 2;
            cp = (int)(kBudget / (2 * row_pair));
        }
        const size_t smem = (size_t)st * cp * row_pair;
        if (attn_dec_prepare<DH, G>(c, smem) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(c, Hkv);
        cfg.blockDim = dim3(kAttnThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = c;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, attn_decode_kernel<DH, G>, &cfg) != cudaSuccess) {
            cudaGetLastError();
            n = 0;
        }
        if (n >= 1) {
            *cs = c;
            *cap = cp;
            *stages = st;
            return cudaSuccess;
        }
    }
    return cudaErrorInvalidConfiguration;
}

#define VLA_ATTN_DISPATCH(dh, group, CALL)          \
    if (dh == 128) {                                 \
        switch (group) {                             \
            case 1: return CALL(128, 1);             \
            case 2: return CALL(128, 2);             \
            case 4: return CALL(128, 4);             \
            case 8: return CALL(128, 8);             \
        }                                            \
    } else if (dh == 64) {                           \
        switch (group) {                             \
            case 1: return CALL(64, 1);              \
            case 2: return CALL(64, 2);              \
            case 4: return CALL(64, 4);              \
            case 8: return CALL(64, 8);              \
        }                                            \
    }                                                \
    return cudaErrorInvalidValue;

cudaError_t launch_attn_dec_any(int dh, int group, const AttnDecParams& p, cudaStream_t s, bool pdl) {
#define VLA_CALL(D, GG) launch_attn_dec<D, GG>(p, s, pdl)
    VLA_ATTN_DISPATCH(dh, group, VLA_CALL)
#undef VLA_CALL
}

}  // namespace

cudaError_t plan_decode_attention(int dh, int group, int Hkv, int max_ctx, int* cs, int* cap, int* stages) {
#define VLA_CALL(D, GG) attn_dec_plan<D, GG>(Hkv, max_ctx, cs, cap, stages)
    VLA_ATTN_DISPATCH(dh, group, VLA_CALL)
#undef VLA_CALL
}

cudaError_t launch_decode_layer(const DecodeLayer& L, const DecodeDims& d, const DecodeWork& w, const bf16* x_in,
                                bf16* x_out, int num_sms, cudaStream_t stream, const StageHook& hook, bool pdl_first) {
    cudaError_t e;
    if (L.nb < 1 || L.nb > kMaxDecodeBatch) return cudaErrorInvalidValue;
    // stage timing records events between the launches: launch those fully serialized
    const bool pdl = hook.fn == nullptr && pdl_enabled();
    pdl_first = pdl_first && pdl;
    const int qc = d.H * d.dh, kvc = d.Hkv * d.dh;
    // 1. RMSNorm + QKV + RoPE + KV append
    GemvParams g = {};
    g.W = L.w_qkv;
    g.K = d.D;
    g.units = (qc + 2 * kvc) / 2;
    g.xv = x_in;
    g.q_out = w.q;
    for (int b = 0; b < L.nb; ++b) {
        g.kcache[b] = L.kcache[b];
        g.vcache[b] = L.vcache[b];
        g.d_len[b] = L.d_len[b];
    }
    g.rope = w.rope;
    g.dh = d.dh;
    g.n_q_heads = d.H;
    g.n_kv_heads = d.Hkv;
    g.max_ctx = d.max_ctx;
    g.eps = d.eps;
    g.status = w.status;
    hook(kStageDecQKV, true);
    e = launch_gemv<kGemvQKV>(g, L.nb, num_sms, stream, pdl_first);
    hook(kStageDecQKV, false);
    if (e != cudaSuccess) return e;
    // 2. split-KV attention, one cluster per (sequence, KV head)
    const float scale_log2 = 1.4426950408889634f / sqrtf((float)d.dh);
    hook(kStageDecAttn, true);
    if (w.attn_tc) {
        DecKVMaps maps;
        memset(&maps, 0, sizeof(maps));
        AttnDecTcParams t = {};
        for (int b = 0; b < L.nb; ++b) {
            if (!make_tmap_bf16_3d(&maps.k[b], L.kcache[b], d.dh, d.max_ctx, d.Hkv, (uint64_t)d.max_ctx * d.dh, 32) ||
                !make_tmap_bf16_3d(&maps.v[b], L.vcache[b], d.dh, d.max_ctx, d.Hkv, (uint64_t)d.max_ctx * d.dh, 32))
                return cudaErrorInvalidValue;
            t.kc[b] = L.kcache[b];
            t.vc[b] = L.vcache[b];
            t.d_len[b] = L.d_len[b];
        }
        t.q = w.q;
        t.nb = L.nb;
        t.H = d.H;
        t.Hkv = d.Hkv;
        t.max_ctx = d.max_ctx;
        t.cs = w.attn_cs;
        t.rows = w.attn_cap;
        t.scale_log2 = scale_log2;
        t.out = w.attn;
        t.status = w.status;
        e = launch_attn_decode_tc(maps, d.H / d.Hkv, t, stream, pdl);
    } else {
        AttnDecParams a = {};
        for (int b = 0; b < L.nb; ++b) {
            a.kc[b] = L.kcache[b];
            a.vc[b] = L.vcache[b];
            a.d_len[b] = L.d_len[b];
        }
        a.q = w.q;
        a.nb = L.nb;
        a.H = d.H;
        a.Hkv = d.Hkv;
        a.max_ctx = d.max_ctx;
        a.cs = w.attn_cs;
        a.cap = w.attn_cap;
        a.stages = w.attn_stages;
        a.scale_log2 = scale_log2;
        a.out = w.attn;
        a.status = w.status;
        e = launch_attn_dec_any(d.dh, d.H / d.Hkv, a, stream, pdl);
    }
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
    o.status = w.status;
    hook(kStageDecO, true);
    e = launch_gemv<kGemvResid>(o, L.nb, num_sms, stream, pdl);
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
    gu.status = w.status;
    hook(kStageDecGateUp, true);
    e = launch_gemv<kGemvSwiGLU>(gu, L.nb, num_sms, stream, pdl);
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
    dn.status = w.status;
    hook(kStageDecDown, true);
    e = launch_gemv<kGemvResid>(dn, L.nb, num_sms, stream, pdl);
    hook(kStageDecDown, false);
    return e;
}

cudaError_t launch_advance_lengths(int* const* d_len, int nb, int count, cudaStream_t stream) {
    if (count <= 0 || nb <= 0) return cudaSuccess;
    if (nb > kMaxDecodeBatch) return cudaErrorInvalidValue;
    LenPtrs lp = {};
    for (int b = 0; b < nb; ++b) lp.p[b] = d_len[b];
    advance_lengths_kernel<<<nb, ((count + 31) / 32) * 32, 0, stream>>>(lp, count);
    return cudaGetLastError();
}

}  // namespace vla
