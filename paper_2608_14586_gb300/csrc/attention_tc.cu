// Causal grouped-query attention for multi-token prefill on the tcgen05 tensor cores.
//
// o[i, h] = sum_{j <= pos0 + i} softmax_j(q_ih . k_gj / sqrt(d_h)) v_gj,  g = h / (H / H_kv)
//
// Persistent: one CTA per SM (192 threads, 225 KB smem, all 512 TMEM columns) walks a list of
// tiles (128 query rows of one head), numbered longest causal tile first and dealt to the CTAs
// in a snake so that every CTA gets a similar number of key blocks.
//   warp 0      TMA: each tile's Q into one of two Q buffers, then its K and V blocks of 128
//               keys into two 2-stage rings (a K stage is released as soon as S has consumed
//               it, a V stage after PV); one thread polls both rings and issues whichever load
//               is free. K/V come from the layer's cache through a 3-D tensor map whose key
//               extent ends at the context length, so keys past it arrive as zeros.
//   warp 1      TMEM allocation; one thread issues S = Q K^T (M=128, N=128 keys, K=d_h) into
//               one of two TMEM S buffers, and O += P V (M=128, N=d_h, K=128 keys) with P from
//               shared memory (K-major) and V as an MN-major operand, into one of two TMEM O
//               accumulators (alternating by tile, so a tile's epilogue overlaps the next).
//   warps 2..5  softmax, one thread per query row (TMEM lane): reads its S row once with
//               tcgen05.ld, masks, takes the row max, writes P = exp2(s - m) as bf16 into a
//               128-byte-swizzled shared tile, keeps the row sum; rescales its O row in TMEM
//               only when the running max grows by more than 2^8 (otherwise the stale max is
//               exact arithmetic with values up to 2^8); then the tile's O / l to global memory.
// The ring and buffer phases run on per-CTA block and tile counters across tiles. Every wait
// is bounded.
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
    static constexpr int K_STAGES = 2;
    static constexpr int V_STAGES = 2;
    // Q is double-buffered across the CTA's tiles; one P tile suffices because PV(j) is
    // issued as soon as P(j) is written
    static constexpr uint32_t OFF_K = 2 * Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + K_STAGES * KV_BYTES;
    static constexpr uint32_t OFF_P = OFF_V + V_STAGES * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_P + P_BYTES;
    static constexpr uint32_t SMEM = OFF_BAR + 256 + 1024;
    // S0 [0,128) S1 [128,256), then two O accumulators of DH columns (one per tile in flight)
    static constexpr uint32_t TMEM_COLS = 512;
    static constexpr uint32_t O_COL = 256;
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(kBM, kBN);
    static constexpr uint32_t IDESC_O = idesc_bf16_f32_bmn(kBM, DH);
};

struct Bars {
    uint64_t q_full[2], q_free[2], k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], s_free[2], p_full,
        p_free, o_full[2], o_free[2], mma_done;
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

// One causal tile: 128 query rows of one head, and the key blocks it needs.
struct Tile {
    int mt, h, g, m0, nblk;
};

// The CTA's k-th tile, or false. Tiles are numbered longest first (every head of the latest
// query tile, then the next query tile, ...) and dealt to the persistent CTAs in a snake
// (round r: CTA c takes tile r*G + c on even rounds, (r+1)*G - 1 - c on odd ones), so each CTA
// gets a mix of long and short causal tiles.
VLA_DEV bool cta_tile(int k, int num_m, const TcAttnArgs& a, Tile& t) {
    const int G = gridDim.x, c = blockIdx.x;
    const int idx = (k & 1) ? (k + 1) * G - 1 - c : k * G + c;
    if (idx >= num_m * a.H) return false;
    t.mt = num_m - 1 - idx / a.H;
    t.h = idx % a.H;
    t.g = t.h / (a.H / a.Hkv);
    t.m0 = t.mt * kBM;
    const int key_end = a.pos0 + min(t.m0 + kBM, a.M);
    t.nblk = (key_end + kBN - 1) / kBN;
    return true;
}

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

    if (threadIdx.x == 0) {
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->q_full[b], 1);
            mbar_init(&bars->q_free[b], 1);
            mbar_init(&bars->k_full[b], 1);
            mbar_init(&bars->k_empty[b], 1);
            mbar_init(&bars->v_full[b], 1);
            mbar_init(&bars->v_empty[b], 1);
            mbar_init(&bars->s_full[b], 1);
            mbar_init(&bars->s_free[b], 128);
            mbar_init(&bars->o_full[b], 1);
            mbar_init(&bars->o_free[b], 128);
        }
        mbar_init(&bars->p_full, 128);
        mbar_init(&bars->p_free, 1);
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
            // ring slot of global block n: n % 2, phase (n / 2) & 1 (K and V alike; Q by tile)
            bool ok = true;
            uint32_t issued_k = 0, issued_v = 0, issued_q = 0, ph_k = 0, ph_v = 0, ph_q = 0;
            uint32_t nk = 0, nv = 0;  // K / V blocks issued so far (all tiles)
            Tile t;
            long long t0 = clock64();
            for (int k = 0; ok && cta_tile(k, num_m, a, t); ++k) {
                const int qb = k & 1;
                const uint32_t qn = (uint32_t)(k >> 1);
                if (!wait_ab(&bars->q_free[qb], (qn & 1u) ^ 1u, &s_abort)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(&bars->q_full[qb], C::Q_BYTES);
                for (int c = 0; c < C::KCH; ++c)
                    tma_load_2d(smem + qb * C::Q_BYTES + c * C::CHUNK, &tmQ, &bars->q_full[qb], t.h * DH + c * 64,
                                t.m0);
                issued_q |= 1u << qb;
                ph_q = (ph_q & ~(1u << qb)) | ((qn & 1u) << qb);
                int jk = 0, jv = 0;
                t0 = clock64();
                while (jk < t.nblk || jv < t.nblk) {
                    bool progressed = false;
                    if (jk < t.nblk) {
                        const int b = nk & 1;
                        const uint32_t n = nk >> 1;
                        if (mbar_try_wait(&bars->k_empty[b], (n & 1u) ^ 1u)) {
                            mbar_arrive_expect_tx(&bars->k_full[b], C::KV_BYTES);
                            for (int c = 0; c < C::KCH; ++c)
                                tma_load_3d(smem + C::OFF_K + b * C::KV_BYTES + c * C::CHUNK, &tmK, &bars->k_full[b],
                                            c * 64, jk * kBN, t.g);
                            issued_k |= 1u << b;
                            ph_k = (ph_k & ~(1u << b)) | ((n & 1u) << b);
                            ++jk;
                            ++nk;
                            progressed = true;
                        }
                    }
                    if (jv < t.nblk && jv < jk) {
                        const int b = nv & 1;
                        const uint32_t n = nv >> 1;
                        if (mbar_try_wait(&bars->v_empty[b], (n & 1u) ^ 1u)) {
                            mbar_arrive_expect_tx(&bars->v_full[b], C::KV_BYTES);
                            for (int c = 0; c < C::KCH; ++c)
                                tma_load_3d(smem + C::OFF_V + b * C::KV_BYTES + c * C::CHUNK, &tmV, &bars->v_full[b],
                                            c * 64, jv * kBN, t.g);
                            issued_v |= 1u << b;
                            ph_v = (ph_v & ~(1u << b)) | ((n & 1u) << b);
                            ++jv;
                            ++nv;
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
            }
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
            }
            // every copy this thread issued lands before the CTA can exit
            for (int b = 0; b < 2; ++b) {
                if (issued_q & (1u << b)) mbar_wait(&bars->q_full[b], (ph_q >> b) & 1u);
                if (issued_k & (1u << b)) mbar_wait(&bars->k_full[b], (ph_k >> b) & 1u);
                if (issued_v & (1u << b)) mbar_wait(&bars->v_full[b], (ph_v >> b) & 1u);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            bool ok = true;
            uint32_t gb = 0;  // global block counter (S buffers, K/V rings, P)
            // PV of global block n for a tile whose O accumulator is ob (first: no accumulate)
            auto issue_pv = [&](uint32_t n, int ob, bool first) -> bool {
                const int vb = n & 1;
                if (!wait_ab(&bars->p_full, n & 1u, &s_abort)) return false;
                if (!wait_ab(&bars->v_full[vb], (n >> 1) & 1u, &s_abort)) return false;
                tc_fence_after();
                const uint32_t sP = smem_u32(smem + C::OFF_P);
                const uint32_t sV = smem_u32(smem + C::OFF_V + vb * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk) {
                    const uint64_t ad = sw128_kmajor_desc(sP + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    const uint64_t bd = sw128_mnmajor_desc(sV + kk * 16 * 128, C::CHUNK);
                    umma_bf16_ss(tmem + C::O_COL + ob * DH, ad, bd, C::IDESC_O, (!first || kk > 0) ? 1u : 0u);
                }
                umma_commit(&bars->p_free);
                umma_commit(&bars->v_empty[vb]);
                return true;
            };
            Tile t;
            for (int k = 0; ok && cta_tile(k, num_m, a, t); ++k) {
                const int qb = k & 1, ob = k & 1;
                const uint32_t qn = (uint32_t)(k >> 1);
                // Q of this tile landed, and the O accumulator's previous tile (k-2) was read out
                if (!wait_ab(&bars->q_full[qb], qn & 1u, &s_abort) ||
                    !wait_ab(&bars->o_free[ob], (qn & 1u) ^ 1u, &s_abort)) {
                    ok = false;
                    break;
                }
                const uint32_t sQ = smem_u32(smem + qb * C::Q_BYTES);
                for (int j = 0; j < t.nblk && ok; ++j) {
                    const uint32_t n = gb + j;
                    const int b = n & 1;
                    if (!wait_ab(&bars->k_full[b], (n >> 1) & 1u, &s_abort) ||
                        !wait_ab(&bars->s_free[b], ((n >> 1) & 1u) ^ 1u, &s_abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sK = smem_u32(smem + C::OFF_K + b * C::KV_BYTES);
#pragma unroll
                    for (int kk = 0; kk < DH / 16; ++kk) {
                        const uint64_t ad = sw128_kmajor_desc(sQ + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                        const uint64_t bd = sw128_kmajor_desc(sK + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                        umma_bf16_ss(tmem + b * kBN, ad, bd, C::IDESC_S, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(&bars->s_full[b]);
                    umma_commit(&bars->k_empty[b]);
                    if (j == t.nblk - 1) umma_commit(&bars->q_free[qb]);  // the tile's last read of Q
                    if (j >= 1 && !issue_pv(n - 1, ob, j == 1)) ok = false;
                }
                if (ok && !issue_pv(gb + t.nblk - 1, ob, t.nblk == 1)) ok = false;
                if (ok) umma_commit(&bars->o_full[ob]);
                gb += t.nblk;
            }
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
            }
            // all MMAs issued by this thread retire before TMEM can be released
            umma_commit(&bars->mma_done);
            mbar_wait(&bars->mma_done, 0);
        }
    } else {
        // ---------------- softmax / correction / epilogue (warps 2..5) ----------------
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        bool ok = true;
        uint32_t gb = 0;
        Tile t;
        for (int k = 0; ok && cta_tile(k, num_m, a, t); ++k) {
            const int ob = k & 1;
            const uint32_t ocol = C::O_COL + ob * DH;
            const int qpos = a.pos0 + t.m0 + row;
            const int min_qpos = a.pos0 + t.m0;
            float m_run = -INFINITY, l_run = 0.f;
            for (int j = 0; j < t.nblk; ++j) {
                const uint32_t n = gb + j;
                const int b = n & 1;
                const int kb = j * kBN;
                const bool need_mask = (kb + kBN - 1 > min_qpos) || (kb + kBN > a.ctx);
                ok = wait_ab(&bars->s_full[b], (n >> 1) & 1u, &s_abort);
                __syncwarp();
                if (!__all_sync(0xFFFFFFFFu, ok)) {
                    ok = false;
                    break;
                }
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
                // row max in 8 independent chains, then combined
                float mc[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) mc[q] = __uint_as_float(sr[q]);
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
                // the P tile was last read by PV of the previous global block
                if (n >= 1) ok = wait_ab(&bars->p_free, (n - 1) & 1u, &s_abort);
                if (!__all_sync(0xFFFFFFFFu, ok)) {
                    ok = false;
                    break;
                }
                // P = exp2(s * scale - m) -> bf16 in the 128-byte-swizzled K-major tile
                uint8_t* prow = smem + C::OFF_P + row * 128;
                const float neg_m = -m_new;
                float ls[4] = {0.f, 0.f, 0.f, 0.f};  // independent partial sums of the row
#pragma unroll
                for (int c = 0; c < kBN / 8; ++c) {  // 16-byte chunks of 8 keys
                    uint32_t pk[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float p0 = ex2_approx(fmaf(__uint_as_float(sr[8 * c + 2 * q]), a.scale_log2, neg_m));
                        const float p1 = ex2_approx(fmaf(__uint_as_float(sr[8 * c + 2 * q + 1]), a.scale_log2, neg_m));
                        ls[q] += p0 + p1;
                        pk[q] = pack_bf16x2(p0, p1);
                    }
                    // keys [8c, 8c+8): 64-key half c/8, 16-byte chunk c%8, swizzled by the row
                    uint8_t* half = prow + (c >> 3) * C::CHUNK;
                    *reinterpret_cast<uint4*>(half + (((c & 7) ^ (row & 7)) << 4)) =
                        make_uint4(pk[0], pk[1], pk[2], pk[3]);
                }
                l_run += (ls[0] + ls[1]) + (ls[2] + ls[3]);
                tc_fence_before();
                mbar_arrive(&bars->s_free[b]);
                if (warp_need) {
                    // O must hold PV of the previous block before it is rescaled (j >= 1 here)
                    ok = wait_ab(&bars->p_free, (n - 1) & 1u, &s_abort);
                    if (!__all_sync(0xFFFFFFFFu, ok)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll 1
                    for (int c = 0; c < DH / 32; ++c) {
                        uint32_t r[32];
                        tmem_ld32(trow + ocol + c * 32, r);
#pragma unroll
                        for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * corr);
                        tmem_st32(trow + ocol + c * 32, r);
                    }
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(&bars->p_full);
                m_run = m_new;
            }
            if (!ok) break;
            // epilogue of this tile (overlaps the first S blocks of the next one)
            ok = wait_ab(&bars->o_full[ob], (uint32_t)(k >> 1) & 1u, &s_abort);
            __syncwarp();
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
            const bool row_ok = (t.m0 + row) < a.M;
            bf16* orow = a.out + (size_t)(t.m0 + row) * a.ld_out + t.h * DH;
#pragma unroll 1
            for (int c = 0; c < DH / 32; ++c) {
                uint32_t r[32];
                tmem_ld32(trow + ocol + c * 32, r);
                if (!row_ok) continue;
                uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    dst[q] = make_uint4(pack_bf16x2(__uint_as_float(r[8 * q]) * inv, __uint_as_float(r[8 * q + 1]) * inv),
                                        pack_bf16x2(__uint_as_float(r[8 * q + 2]) * inv, __uint_as_float(r[8 * q + 3]) * inv),
                                        pack_bf16x2(__uint_as_float(r[8 * q + 4]) * inv, __uint_as_float(r[8 * q + 5]) * inv),
                                        pack_bf16x2(__uint_as_float(r[8 * q + 6]) * inv, __uint_as_float(r[8 * q + 7]) * inv));
                }
            }
            tc_fence_before();
            mbar_arrive(&bars->o_free[ob]);
            gb += t.nblk;
        }
        if (!ok) {
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
    // persistent: one CTA per SM (tensor-memory kernels get one per SM), each walking its tiles
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    const int tiles = ((p.M + kBM - 1) / kBM) * p.H;
    const dim3 grid(tiles < sms ? tiles : sms);
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
