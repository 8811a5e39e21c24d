// Causal grouped-query attention for multi-token prefill on the tcgen05 tensor cores.
//
// o[i, h] = sum_{j <= pos0 + i} softmax_j(q_ih . k_gj / sqrt(d_h)) v_gj,  g = h / (H / H_kv)
//
// One CTA = 128 query rows of one head (one CTA per SM: 192 threads, up to 225 KB smem):
//   warp 0      TMA: the Q tile once, then K and V blocks of 128 keys into two separate
//               2-stage rings (a K stage is released as soon as S has consumed it, a V stage
//               after PV); one thread polls both rings and issues whichever load is free.
//               K/V come from the layer's cache through a 3-D tensor map whose key extent
//               ends at the context length, so keys past it arrive as zeros.
//   warp 1      TMEM allocation; one thread issues S = Q K^T (M=128, N=128 keys, K=d_h) into
//               one of two TMEM S buffers, and O += P V (M=128, N=d_h, K=128 keys) with P from
//               shared memory (K-major) and V as an MN-major operand.
//   warps 2..5  softmax, one thread per query row (TMEM lane): reads its S row once with
//               tcgen05.ld, masks, takes the row max, writes P = exp2(s - m) as bf16 into a
//               128-byte-swizzled shared tile, keeps the row sum; rescales its O row in TMEM
//               only when the running max grows by more than 2^8 (otherwise the stale max is
//               exact arithmetic with values up to 2^8); final O / l to global memory.
// S and P are double-buffered so the tensor core computes S(j+1) and PV(j) while the
// softmax warps work on block j+1. Every wait is bounded.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kThreads = 192;
constexpr float kRescaleLog2 = 8.0f;

template <int DH>
struct AttnCfg {
    static constexpr int KCH = DH / 64;                 // 64-wide head-dim chunks
    static constexpr uint32_t CHUNK = 128 * 64 * 2;     // one [128 rows][64] bf16 chunk
    static constexpr uint32_t Q_BYTES = KCH * CHUNK;
    static constexpr uint32_t KV_BYTES = KCH * CHUNK;
    static constexpr uint32_t P_BYTES = 2 * CHUNK;       // 128 keys = 2 chunks of 64
    // K is needed one block before V (S = QK^T precedes PV), so K gets the deeper ring; one P
    // tile suffices because PV(j) is issued as soon as P(j) is written
    static constexpr int K_STAGES = 3;
    static constexpr int V_STAGES = 2;
    static constexpr uint32_t OFF_K = Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + K_STAGES * KV_BYTES;
    static constexpr uint32_t OFF_P = OFF_V + V_STAGES * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_P + P_BYTES;
    static constexpr uint32_t SMEM = OFF_BAR + 256 + 1024;
    static constexpr uint32_t TMEM_COLS = 512;           // S0 [0,128) S1 [128,256) O [256, 256+DH)
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(kBM, kBN);
    static constexpr uint32_t IDESC_O = idesc_bf16_f32_bmn(kBM, DH);
};

struct Bars {
    uint64_t q_full, k_full[3], k_empty[3], v_full[2], v_empty[2], s_full[2], s_free[2], p_full, p_free, o_final,
        mma_done;
    uint32_t tmem_slot;
};

VLA_DEV bool wait_ab(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (*abort_flag) return false;
        if (clock64() - t0 > kWaitBudgetCycles) return false;
    }
    return true;
}

struct TcAttnArgs {
    int M, H, Hkv, pos0, ctx, ld_out;
    float scale_log2;
    bf16* out;
    unsigned* status;
};

template <int DH>
__global__ void __launch_bounds__(kThreads, 1)
    attn_prefill_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                           const __grid_constant__ CUtensorMap tmV, TcAttnArgs a) {
    using C = AttnCfg<DH>;
    extern __shared__ uint8_t smem_raw[];
    __shared__ volatile int s_abort;
    const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    Bars* bars = reinterpret_cast<Bars*>(smem + C::OFF_BAR);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_m = (a.M + kBM - 1) / kBM;
    // CTAs launch x-fastest: every head of the heaviest (latest) query tile first, then the
    // next, so the long causal tiles start early and the short ones fill in (longest first)
    const int mt = num_m - 1 - (int)blockIdx.y;
    const int h = blockIdx.x;
    const int g = h / (a.H / a.Hkv);
    const int m0 = mt * kBM;
    const int key_end = a.pos0 + min(m0 + kBM, a.M);
    const int nblk = (key_end + kBN - 1) / kBN;

    if (threadIdx.x == 0) {
        mbar_init(&bars->q_full, 1);
        for (int b = 0; b < C::K_STAGES; ++b) {
            mbar_init(&bars->k_full[b], 1);
            mbar_init(&bars->k_empty[b], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->v_full[b], 1);
            mbar_init(&bars->v_empty[b], 1);
            mbar_init(&bars->s_full[b], 1);
            mbar_init(&bars->s_free[b], 128);
        }
        mbar_init(&bars->p_full, 128);
        mbar_init(&bars->p_free, 1);
        mbar_init(&bars->o_final, 1);
        mbar_init(&bars->mma_done, 1);
        s_abort = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmQ);
        tma_prefetch_desc(&tmK);
        tma_prefetch_desc(&tmV);
    }
    if (warp == 1) {
        tmem_alloc(&bars->tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem_slot;
    pdl_wait();  // Q, K and V are the previous kernel's output
    pdl_trigger();

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer ----------------
            bool ok = true;
            uint32_t issued_k = 0, issued_v = 0, ph_k = 0, ph_v = 0;
            mbar_arrive_expect_tx(&bars->q_full, C::Q_BYTES);
            for (int c = 0; c < C::KCH; ++c)
                tma_load_2d(smem + c * C::CHUNK, &tmQ, &bars->q_full, h * DH + c * 64, m0);
            int jk = 0, jv = 0;
            long long t0 = clock64();
            while (jk < nblk || jv < nblk) {
                bool progressed = false;
                if (jk < nblk) {
                    const int b = jk % C::K_STAGES;
                    const uint32_t n = (uint32_t)(jk / C::K_STAGES);
                    if (mbar_try_wait(&bars->k_empty[b], (n & 1u) ^ 1u)) {
                        mbar_arrive_expect_tx(&bars->k_full[b], C::KV_BYTES);
                        for (int c = 0; c < C::KCH; ++c)
                            tma_load_3d(smem + C::OFF_K + b * C::KV_BYTES + c * C::CHUNK, &tmK, &bars->k_full[b],
                                        c * 64, jk * kBN, g);
                        issued_k |= 1u << b;
                        ph_k = (ph_k & ~(1u << b)) | ((n & 1u) << b);
                        ++jk;
                        progressed = true;
                    }
                }
                if (jv < nblk && jv < jk) {
                    const int b = jv & 1;
                    const uint32_t n = (uint32_t)(jv >> 1);
                    if (mbar_try_wait(&bars->v_empty[b], (n & 1u) ^ 1u)) {
                        mbar_arrive_expect_tx(&bars->v_full[b], C::KV_BYTES);
                        for (int c = 0; c < C::KCH; ++c)
                            tma_load_3d(smem + C::OFF_V + b * C::KV_BYTES + c * C::CHUNK, &tmV, &bars->v_full[b],
                                        c * 64, jv * kBN, g);
                        issued_v |= 1u << b;
                        ph_v = (ph_v & ~(1u << b)) | ((n & 1u) << b);
                        ++jv;
                        progressed = true;
                    }
                }
                if (progressed) {
                    t0 = clock64();
                } else if (s_abort || clock64() - t0 > kWaitBudgetCycles) {
                    ok = false;
                    break;
                }
            }
            mbar_wait(&bars->q_full, 0);  // the Q copy has landed whatever happens below
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
                for (int b = 0; b < C::K_STAGES; ++b)
                    if (issued_k & (1u << b)) mbar_wait(&bars->k_full[b], (ph_k >> b) & 1u);
                for (int b = 0; b < 2; ++b)
                    if (issued_v & (1u << b)) mbar_wait(&bars->v_full[b], (ph_v >> b) & 1u);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            bool ok = wait_ab(&bars->q_full, 0, &s_abort);
            const uint32_t sQ = smem_u32(smem);
            auto issue_pv = [&](int i) -> bool {
                const int bi = i & 1;
                const uint32_t ni = (uint32_t)(i >> 1);
                if (!wait_ab(&bars->p_full, (uint32_t)i & 1u, &s_abort)) return false;
                if (!wait_ab(&bars->v_full[bi], ni & 1u, &s_abort)) return false;
                tc_fence_after();
                const uint32_t sP = smem_u32(smem + C::OFF_P);
                const uint32_t sV = smem_u32(smem + C::OFF_V + bi * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk) {
                    const uint64_t ad = sw128_kmajor_desc(sP + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    const uint64_t bd = sw128_mnmajor_desc(sV + kk * 16 * 128, C::CHUNK);
                    umma_bf16_ss(tmem + 256, ad, bd, C::IDESC_O, (i > 0 || kk > 0) ? 1u : 0u);
                }
                umma_commit(&bars->p_free);
                umma_commit(&bars->v_empty[bi]);
                return true;
            };
            for (int j = 0; j < nblk && ok; ++j) {
                const int b = j & 1;
                const uint32_t n = (uint32_t)(j >> 1);
                const int kb = j % C::K_STAGES;
                if (!wait_ab(&bars->k_full[kb], (uint32_t)(j / C::K_STAGES) & 1u, &s_abort) ||
                    !wait_ab(&bars->s_free[b], (n & 1u) ^ 1u, &s_abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sK = smem_u32(smem + C::OFF_K + kb * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const uint64_t ad = sw128_kmajor_desc(sQ + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    const uint64_t bd = sw128_kmajor_desc(sK + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    umma_bf16_ss(tmem + b * kBN, ad, bd, C::IDESC_S, kk > 0 ? 1u : 0u);
                }
                umma_commit(&bars->s_full[b]);
                umma_commit(&bars->k_empty[kb]);
                if (j >= 1 && !issue_pv(j - 1)) ok = false;
            }
            if (ok && !issue_pv(nblk - 1)) ok = false;
            if (ok) umma_commit(&bars->o_final);
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
            }
            umma_commit(&bars->mma_done);
            mbar_wait(&bars->mma_done, 0);
        }
    } else {
        // ---------------- softmax / correction / epilogue (warps 2..5) ----------------
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const int qpos = a.pos0 + m0 + row;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const int min_qpos = a.pos0 + m0;
        float m_run = -INFINITY, l_run = 0.f;
        bool ok = true;
        for (int j = 0; j < nblk; ++j) {
            const int b = j & 1;
            const uint32_t n = (uint32_t)(j >> 1);
            const int kb = j * kBN;
            const bool need_mask = (kb + kBN - 1 > min_qpos) || (kb + kBN > a.ctx);
            ok = wait_ab(&bars->s_full[b], n & 1u, &s_abort);
            __syncwarp();
            if (!__all_sync(0xFFFFFFFFu, ok)) break;
            tc_fence_after();
            // the whole S row (128 keys) in registers; row max of the raw masked scores
            uint32_t sr[kBN];
            tmem_ld128(trow + b * kBN, sr);
            if (need_mask) {
#pragma unroll
                for (int i = 0; i < kBN; ++i) {
                    const int key = kb + i;
                    if (key > qpos || key >= a.ctx) sr[i] = 0xFF800000u;  // -inf
                }
            }
            // row max in 8 independent chains (the single softmax warp of each sub-partition has
            // nothing else to issue meanwhile), then combined
            float mc[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) mc[j] = __uint_as_float(sr[j]);
#pragma unroll
            for (int i = 8; i < kBN; ++i) mc[i & 7] = fmaxf(mc[i & 7], __uint_as_float(sr[i]));
            const float mraw = fmaxf(fmaxf(fmaxf(mc[0], mc[1]), fmaxf(mc[2], mc[3])),
                                     fmaxf(fmaxf(mc[4], mc[5]), fmaxf(mc[6], mc[7])));
            const float mx = mraw * a.scale_log2;  // scale > 0
            float m_new = m_run;
            bool need = false;
            if (m_run == -INFINITY) {
                m_new = mx;
            } else if (mx > m_run + kRescaleLog2) {
                need = true;
                m_new = mx;
            }
            const float corr = need ? ex2_approx(m_run - m_new) : 1.f;
            l_run *= corr;
            const bool warp_need = __any_sync(0xFFFFFFFFu, need);
            // the P buffer of block j was last read by PV(j-2)
            // the P tile was last read by PV(j-1)
            if (j >= 1) ok = wait_ab(&bars->p_free, (uint32_t)(j - 1) & 1u, &s_abort);
            if (!__all_sync(0xFFFFFFFFu, ok)) break;
            // P = exp2(s * scale - m) -> bf16 in the 128-byte-swizzled K-major tile
            uint8_t* prow = smem + C::OFF_P + row * 128;
            const float neg_m = -m_new;
            float ls[4] = {0.f, 0.f, 0.f, 0.f};  // independent partial sums of the row
#pragma unroll
            for (int c = 0; c < kBN / 8; ++c) {  // 16-byte chunks of 8 keys
                uint32_t pk[4];
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    const float p0 = ex2_approx(fmaf(__uint_as_float(sr[8 * c + 2 * t]), a.scale_log2, neg_m));
                    const float p1 = ex2_approx(fmaf(__uint_as_float(sr[8 * c + 2 * t + 1]), a.scale_log2, neg_m));
                    ls[t] += p0 + p1;
                    pk[t] = pack_bf16x2(p0, p1);
                }
                // keys [8c, 8c+8): 64-key half c/8, 16-byte chunk c%8, swizzled by the row
                uint8_t* half = prow + (c >> 3) * C::CHUNK;
                *reinterpret_cast<uint4*>(half + (((c & 7) ^ (row & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
            l_run += (ls[0] + ls[1]) + (ls[2] + ls[3]);
            tc_fence_before();
            mbar_arrive(&bars->s_free[b]);
            if (warp_need) {
                // O must hold PV(j-1) before it is rescaled
                ok = wait_ab(&bars->p_free, (uint32_t)(j - 1) & 1u, &s_abort);
                if (!__all_sync(0xFFFFFFFFu, ok)) break;
                tc_fence_after();
#pragma unroll 1
                for (int c = 0; c < DH / 32; ++c) {
                    uint32_t r[32];
                    tmem_ld32(trow + 256 + c * 32, r);
#pragma unroll
                    for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * corr);
                    tmem_st32(trow + 256 + c * 32, r);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&bars->p_full);
            m_run = m_new;
        }
        if (ok) ok = wait_ab(&bars->o_final, 0, &s_abort);
        __syncwarp();
        if (__all_sync(0xFFFFFFFFu, ok)) {
            tc_fence_after();
            const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
            const bool row_ok = (m0 + row) < a.M;
            bf16* orow = a.out + (size_t)(m0 + row) * a.ld_out + h * DH;
#pragma unroll 1
            for (int c = 0; c < DH / 32; ++c) {
                uint32_t r[32];
                tmem_ld32(trow + 256 + c * 32, r);
                if (!row_ok) continue;
                uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    dst[t] = make_uint4(pack_bf16x2(__uint_as_float(r[8 * t]) * inv, __uint_as_float(r[8 * t + 1]) * inv),
                                        pack_bf16x2(__uint_as_float(r[8 * t + 2]) * inv, __uint_as_float(r[8 * t + 3]) * inv),
                                        pack_bf16x2(__uint_as_float(r[8 * t + 4]) * inv, __uint_as_float(r[8 * t + 5]) * inv),
                                        pack_bf16x2(__uint_as_float(r[8 * t + 6]) * inv, __uint_as_float(r[8 * t + 7]) * inv));
                }
            }
        } else {
            s_abort = 1;
            set_status(a.status, kDevTimeout);
        }
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

template <int DH>
cudaError_t launch_dh(const AttnPrefillParams& p, unsigned* status, cudaStream_t stream, bool pdl) {
    using C = AttnCfg<DH>;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e =
            cudaFuncSetAttribute(attn_prefill_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int ctx = p.pos0 + p.M;
    CUtensorMap tq, tk, tv;
    if (!make_tmap_bf16(&tq, p.q, p.M, (uint64_t)p.H * DH, p.ld_q, 128) ||
        !make_tmap_bf16_3d(&tk, p.kc, DH, ctx, p.Hkv, (uint64_t)p.max_ctx * DH, 128) ||
        !make_tmap_bf16_3d(&tv, p.vc, DH, ctx, p.Hkv, (uint64_t)p.max_ctx * DH, 128))
        return cudaErrorInvalidValue;
    TcAttnArgs a;
    a.M = p.M;
    a.H = p.H;
    a.Hkv = p.Hkv;
    a.pos0 = p.pos0;
    a.ctx = ctx;
    a.ld_out = p.ld_out;
    a.scale_log2 = p.scale_log2;
    a.out = p.out;
    a.status = status;
    dim3 grid(p.H, (p.M + kBM - 1) / kBM);
    return launch_ex(attn_prefill_tc_kernel<DH>, grid, dim3(kThreads), C::SMEM, stream, pdl, tq, tk, tv, a);
}

}  // namespace

cudaError_t launch_attn_prefill_tc(const AttnPrefillParams& p, unsigned* status, cudaStream_t stream, bool pdl) {
    if (p.M <= 0) return cudaSuccess;
    if (p.head_dim == 128) return launch_dh<128>(p, status, stream, pdl);
    if (p.head_dim == 64) return launch_dh<64>(p, status, stream, pdl);
    return cudaErrorInvalidValue;
}

}  // namespace vla
