// Causal grouped-query attention for multi-token prefill on the tcgen05 tensor cores.
//
// o[i, h] = sum_{j <= pos0 + i} softmax_j(q_ih . k_gj / sqrt(d_h)) v_gj,  g = h / (H / H_kv)
//
// Persistent: one CTA per SM (352 threads, all 512 TMEM columns) walks a list of work units,
// each one query tile (128 rows) of one head, numbered longest first and dealt to the CTAs in
// a snake so that every CTA gets a similar number of 128-key blocks (with 18 tiles of 32 heads
// on 152 SMs exactly 36 each). A CTA's key blocks form one sequence g = 0, 1, ... over its
// units. Tensor memory: three S buffers (columns [0, 128), [128, 256), [256, 384)) and O
// (d_h columns from 384).
//   warp 0      TMA: the units' Q tiles into two shared-memory buffers, and K and V blocks of
//               128 keys through 3- and 2-stage rings, from the layer's cache through 3-D tensor
//               maps whose key extent ends at the context length (keys past it arrive as zeros,
//               so stale cache contents never reach P V).
//   warp 1      TMEM allocation; one thread issues O += P(g) V_g with P(g) (packed bf16 over the
//               first 64 columns of S buffer g % 3) read from tensor memory and V_g as an
//               MN-major shared-memory operand, and commits the PV's completion on the barrier
//               of that buffer.
//   warp 10     one thread issues S(g) = Q K_g^T into S buffer g % 3 once PV(g - 3), the last
//               reader of that buffer, has completed. The S of a block is requested three blocks
//               ahead of its softmax, and with two issuing threads one's waits overlap the
//               other's issue, so the tensor core is fed from both.
//   warps 2..5  softmax, one thread per query row (TMEM lane): reads its S row once
//               (tcgen05.ld), masks, takes the row max, writes P = exp2(s - m) as bf16 into tensor
//               memory (tcgen05.st) and keeps the row sum. Only when the running max grows by
//               more than 2^8 (a stale max below that is exact arithmetic with values up to 2^8)
//               does it rescale its O row, once PV(g - 1) has completed. At the end of a tile it
//               hands the row sum to warps 6..9 through shared memory.
//   warps 6..9  after a tile's last PV: read O, divide by the row sum and store the output rows.
// Phases of every barrier follow per-CTA block and unit counters; no waiter can fall two
// phases behind its barrier (each producer of a phase needs the waiter's previous step, or, for
// the PV barriers the softmax waits on only before a rescale, see there). Every wait is bounded.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kThreads = 352;  // + warp 10: the S issuer
constexpr int kSBufs = 3;
constexpr int kKStages = 3;
constexpr int kVStages = 2;
constexpr float kRescaleLog2 = 8.0f;

template <int DH>
struct AttnCfg {
    static constexpr int KCH = DH / 64;              // 64-wide head-dim chunks
    static constexpr uint32_t CHUNK = 128 * 64 * 2;  // one [128 rows][64] bf16 chunk
    static constexpr uint32_t Q_BYTES = KCH * CHUNK;
    static constexpr uint32_t KV_BYTES = KCH * CHUNK;
    static constexpr uint32_t OFF_K = 2 * Q_BYTES;  // two Q buffers
    static constexpr uint32_t OFF_V = OFF_K + kKStages * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_V + kVStages * KV_BYTES;
    static constexpr uint32_t OFF_L = OFF_BAR + 512;  // row sums handed to the epilogue: [2][128] fp32
    static constexpr uint32_t SMEM = OFF_L + 2 * kBM * 4 + 1024;
    static constexpr uint32_t TMEM_COLS = 512;
    static constexpr uint32_t O_COL = kSBufs * kBN;
    static_assert(O_COL + DH <= TMEM_COLS, "tensor memory columns");
    static_assert(SMEM <= 232448, "shared memory");
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(kBM, kBN);
    static constexpr uint32_t IDESC_O = idesc_bf16_f32_bmn(kBM, DH);
};

struct Bars {
    uint64_t k_full[kKStages], k_empty[kKStages], v_full[kVStages], v_empty[kVStages];
    uint64_t s_full[kSBufs], p_full[kSBufs];  // per S buffer
    uint64_t q_full[2], q_free[2];            // per Q buffer
    uint64_t l_full[2], l_free[2];            // per row-sum buffer
    uint64_t pv_done[kSBufs];                 // PV(g) by g % 3 (the S buffer it read)
    uint64_t o_full, o_free, mma_done, s_done;
    uint32_t tmem_slot;
};
static_assert(sizeof(Bars) <= 512, "barrier block");

VLA_DEV bool wait_ab(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (*abort_flag) return false;
        if (clock64() - t0 > kWaitBudgetCycles) return false;
    }
    return true;
}

// the same wait in every lane of a warp, true only if every lane's wait succeeded
VLA_DEV bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    const bool ok = wait_ab(bar, parity, abort_flag);
    __syncwarp();
    return __all_sync(0xFFFFFFFFu, ok);
}

struct TcAttnArgs {
    int M, H, Hkv, pos0, ctx, ld_out;
    float scale_log2;
    bf16* out;
    unsigned* status;
};

// A query tile of one head: rows [m0, m0 + 128) (clipped to M) of head h, KV head g, and the
// n key blocks of 128 it attends to.
struct Unit {
    int h, g, m0, n;
};

// The CTA's k-th unit, or false. Units are numbered longest first (every head of the last
// query tile, then of the one before, ...) and dealt to the persistent CTAs in a snake
// (round r: CTA c takes unit r*G + c on even rounds, (r+1)*G - 1 - c on odd ones).
VLA_DEV bool cta_unit(int k, int num_t, const TcAttnArgs& a, Unit& u) {
    const int G = gridDim.x, c = blockIdx.x;
    const int idx = (k & 1) ? (k + 1) * G - 1 - c : k * G + c;
    if (idx >= num_t * a.H) return false;
    const int tm = num_t - 1 - idx / a.H;
    u.h = idx % a.H;
    u.g = u.h / (a.H / a.Hkv);
    u.m0 = tm * kBM;
    u.n = (a.pos0 + min(u.m0 + kBM, a.M) + kBN - 1) / kBN;
    return true;
}

// A position (unit k, block j of it) in the CTA's block sequence.
struct Cursor {
    int k, j;
    Unit u;
    bool valid;
    VLA_DEV void start(int num_t, const TcAttnArgs& a) {
        k = 0;
        j = 0;
        valid = cta_unit(0, num_t, a, u);
    }
    VLA_DEV void next(int num_t, const TcAttnArgs& a) {
        if (++j == u.n) {
            j = 0;
            ++k;
            valid = cta_unit(k, num_t, a, u);
        }
    }
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
    float* lbuf = reinterpret_cast<float*>(smem + C::OFF_L);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_t = (a.M + kBM - 1) / kBM;

    if (threadIdx.x == 0) {
        for (int b = 0; b < kKStages; ++b) {
            mbar_init(&bars->k_full[b], 1);
            mbar_init(&bars->k_empty[b], 1);
        }
        for (int b = 0; b < kVStages; ++b) {
            mbar_init(&bars->v_full[b], 1);
            mbar_init(&bars->v_empty[b], 1);
        }
        for (int b = 0; b < kSBufs; ++b) {
            mbar_init(&bars->s_full[b], 1);
            mbar_init(&bars->p_full[b], 128);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->q_full[b], 1);
            mbar_init(&bars->q_free[b], 1);
            mbar_init(&bars->l_full[b], 128);
            mbar_init(&bars->l_free[b], 128);
        }
        for (int b = 0; b < kSBufs; ++b) mbar_init(&bars->pv_done[b], 1);
        mbar_init(&bars->o_full, 1);
        mbar_init(&bars->o_free, 128);
        mbar_init(&bars->mma_done, 1);
        mbar_init(&bars->s_done, 1);
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
            // Q of unit k into Q buffer k % 2, K(g) into K slot g % 3 and V(g) into V slot g % 2,
            // each in order; whichever has a free slot goes next
            bool ok = true;
            Cursor ck, cv;
            ck.start(num_t, a);
            cv.start(num_t, a);
            int kq = 0;
            Unit uq;
            bool q_left = cta_unit(0, num_t, a, uq);
            uint32_t nk = 0, nv = 0;
            uint32_t issued_k = 0, ph_k = 0, issued_v = 0, ph_v = 0, issued_q = 0, ph_q = 0;
            long long t0 = clock64();
            while (ck.valid || cv.valid || q_left) {
                bool progressed = false;
                if (q_left) {
                    const uint32_t b = (uint32_t)kq & 1u, n = (uint32_t)kq >> 1;
                    if (mbar_try_wait(&bars->q_free[b], (n & 1u) ^ 1u)) {
                        mbar_arrive_expect_tx(&bars->q_full[b], C::Q_BYTES);
                        for (int c = 0; c < C::KCH; ++c)
                            tma_load_2d(smem + b * C::Q_BYTES + c * C::CHUNK, &tmQ, &bars->q_full[b],
                                        uq.h * DH + c * 64, uq.m0);
                        issued_q |= 1u << b;
                        ph_q = (ph_q & ~(1u << b)) | ((n & 1u) << b);
                        ++kq;
                        q_left = cta_unit(kq, num_t, a, uq);
                        progressed = true;
                    }
                }
                if (ck.valid) {
                    const uint32_t b = nk % kKStages, n = nk / kKStages;
                    if (mbar_try_wait(&bars->k_empty[b], (n & 1u) ^ 1u)) {
                        mbar_arrive_expect_tx(&bars->k_full[b], C::KV_BYTES);
                        for (int c = 0; c < C::KCH; ++c)
                            tma_load_3d(smem + C::OFF_K + b * C::KV_BYTES + c * C::CHUNK, &tmK, &bars->k_full[b],
                                        c * 64, ck.j * kBN, ck.u.g);
                        issued_k |= 1u << b;
                        ph_k = (ph_k & ~(1u << b)) | ((n & 1u) << b);
                        ++nk;
                        ck.next(num_t, a);
                        progressed = true;
                    }
                }
                if (cv.valid) {
                    const uint32_t b = nv % kVStages, n = nv / kVStages;
                    if (mbar_try_wait(&bars->v_empty[b], (n & 1u) ^ 1u)) {
                        mbar_arrive_expect_tx(&bars->v_full[b], C::KV_BYTES);
                        for (int c = 0; c < C::KCH; ++c)
                            tma_load_3d(smem + C::OFF_V + b * C::KV_BYTES + c * C::CHUNK, &tmV, &bars->v_full[b],
                                        c * 64, cv.j * kBN, cv.u.g);
                        issued_v |= 1u << b;
                        ph_v = (ph_v & ~(1u << b)) | ((n & 1u) << b);
                        ++nv;
                        cv.next(num_t, a);
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
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
            }
            // every copy this thread issued lands before the CTA can exit
            for (int b = 0; b < 2; ++b)
                if (issued_q & (1u << b)) mbar_wait(&bars->q_full[b], (ph_q >> b) & 1u);
            for (int b = 0; b < kKStages; ++b)
                if (issued_k & (1u << b)) mbar_wait(&bars->k_full[b], (ph_k >> b) & 1u);
            for (int b = 0; b < kVStages; ++b)
                if (issued_v & (1u << b)) mbar_wait(&bars->v_full[b], (ph_v >> b) & 1u);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- PV issuer ----------------
            bool ok = true;
            uint32_t g = 0;  // PV issued so far
            Unit u;
            for (int k = 0; ok && cta_unit(k, num_t, a, u); ++k) {
                for (int j = 0; j < u.n; ++j, ++g) {
                    const uint32_t sb = g % kSBufs, vb = g % kVStages;
                    if (!wait_ab(&bars->p_full[sb], (g / kSBufs) & 1u, &s_abort) ||
                        (j == 0 && !wait_ab(&bars->o_free, ((uint32_t)k & 1u) ^ 1u, &s_abort)) ||
                        !wait_ab(&bars->v_full[vb], (g / kVStages) & 1u, &s_abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sV = smem_u32(smem + C::OFF_V + vb * C::KV_BYTES);
#pragma unroll
                    for (int kk = 0; kk < kBN / 16; ++kk) {
                        const uint64_t bd = sw128_mnmajor_desc(sV + kk * 16 * 128, C::CHUNK);
                        umma_bf16_ts(tmem + C::O_COL, tmem + sb * kBN + kk * 8, bd, C::IDESC_O,
                                     (j > 0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(&bars->v_empty[vb]);
                    umma_commit(&bars->pv_done[sb]);  // the S issuer reuses buffer sb after it
                    if (j == u.n - 1) umma_commit(&bars->o_full);  // O of the unit is final
                }
            }
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
            }
            // all MMAs issued by this thread retire before TMEM can be released
            umma_commit(&bars->mma_done);
            mbar_wait(&bars->mma_done, 0);
        }
    } else if (warp == 10) {
        if (lane == 0) {
            // ---------------- S issuer ----------------
            // S(g) into buffer g % 3 once PV(g - 3), the last reader of that buffer, has
            // completed (its commit on pv_done[g % 3]; every phase waited in order, and the next
            // phase needs S(g) itself, so the wait is exact), and the unit's Q and K_g are in
            bool ok = true;
            Cursor cs;
            cs.start(num_t, a);
            for (uint32_t gs = 0; ok && cs.valid; ++gs) {
                const uint32_t qb = (uint32_t)cs.k & 1u;
                const uint32_t kb = gs % kKStages;
                if ((gs >= (uint32_t)kSBufs &&
                     !wait_ab(&bars->pv_done[gs % kSBufs], ((gs / kSBufs) - 1u) & 1u, &s_abort)) ||
                    (cs.j == 0 && !wait_ab(&bars->q_full[qb], ((uint32_t)cs.k >> 1) & 1u, &s_abort)) ||
                    !wait_ab(&bars->k_full[kb], (gs / kKStages) & 1u, &s_abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sQ = smem_u32(smem + qb * C::Q_BYTES);
                const uint32_t sK = smem_u32(smem + C::OFF_K + kb * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const uint64_t ad = sw128_kmajor_desc(sQ + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    const uint64_t bd = sw128_kmajor_desc(sK + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    umma_bf16_ss(tmem + (gs % kSBufs) * kBN, ad, bd, C::IDESC_S, kk > 0 ? 1u : 0u);
                }
                umma_commit(&bars->s_full[gs % kSBufs]);
                umma_commit(&bars->k_empty[kb]);
                if (cs.j == cs.u.n - 1) umma_commit(&bars->q_free[qb]);  // the unit's last S
                cs.next(num_t, a);
            }
            if (!ok) {
                s_abort = 1;
                set_status(a.status, kDevTimeout);
            }
            umma_commit(&bars->s_done);
            mbar_wait(&bars->s_done, 0);
        }
    } else if (warp < 6) {
        // ---------------- softmax (warps 2..5) ----------------
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        bool ok = true;
        uint32_t g = 0;  // blocks so far (S buffer phases)
        Unit u;
        for (int k = 0; ok && cta_unit(k, num_t, a, u); ++k) {
            const int qpos = a.pos0 + u.m0 + row;
            const int min_qpos = a.pos0 + u.m0;
            float m_run = -INFINITY, l_run = 0.f;
            for (int j = 0; j < u.n; ++j, ++g) {
                const uint32_t scol = (g % kSBufs) * kBN;
                uint32_t sr[kBN];
                float m_new = m_run;
                bool need = false;
                {
                    const int kb = j * kBN;
                    const bool need_mask = (kb + kBN - 1 > min_qpos) || (kb + kBN > a.ctx);
                    if (!warp_wait(&bars->s_full[g % kSBufs], (g / kSBufs) & 1u, &s_abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    tmem_ld128(trow + scol, sr);
                    if (need_mask) {
#pragma unroll
                        for (int i = 0; i < kBN; ++i) {
                            const int key = kb + i;
                            if (key > qpos || key >= a.ctx) sr[i] = 0xFF800000u;  // -inf
                        }
                    }
                    // row max with three-input max instructions, eight independent chains
                    float mc[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) mc[q] = __uint_as_float(sr[q]);
#pragma unroll
                    for (int i = 8; i < kBN; i += 16) {
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            mc[q] = fmax3(mc[q], __uint_as_float(sr[i + q]),
                                          i + 8 + q < kBN ? __uint_as_float(sr[i + 8 + q]) : mc[q]);
                    }
                    const float mraw = fmax3(fmax3(mc[0], mc[1], mc[2]), fmax3(mc[3], mc[4], mc[5]), fmaxf(mc[6], mc[7]));
                    const float mx = mraw * a.scale_log2;  // scale > 0
                    if (m_run == -INFINITY) {
                        m_new = mx;
                    } else if (mx > m_run + kRescaleLog2) {
                        need = true;
                        m_new = mx;
                    }
                }
                {
                    const float corr = need ? ex2_approx(m_run - m_new) : 1.f;
                    l_run *= corr;
                    const bool warp_need = __any_sync(0xFFFFFFFFu, need);
                    // P = exp2(s * scale - m) as packed bf16 over the first 64 columns of S,
                    // two columns per instruction for the scaling and the row sum (packed fp32)
                    const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
                    const float2 nm2 = make_float2(-m_new, -m_new);
                    float2 ls[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};  // partial row sums
                    // packed P in four 16-column stores, waited on once: the packed words take
                    // the place of the S values they replace, so fewer registers are live
                    uint32_t pk[64];
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int c = 32 * h + 2 * i;
                            const float2 x = __ffma2_rn(make_float2(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])),
                                                        sc2, nm2);
                            const float2 pp = make_float2(ex2_approx(x.x), ex2_approx(x.y));
                            ls[i & 1] = __fadd2_rn(ls[i & 1], pp);
                            pk[16 * h + i] = pack_bf16x2(pp.x, pp.y);
                        }
                        tmem_st16_async(trow + scol + 16 * h, &pk[16 * h]);
                    }
                    tmem_wait_st();
                    l_run += (ls[0].x + ls[1].x) + (ls[0].y + ls[1].y);
                    if (warp_need) {
                        // O is rescaled once PV(g - 1) has completed (it commits to the barrier
                        // of its S buffer). PV(g - 3) has completed (S(g), seen above, was issued
                        // after it, so PV(g - 4) too) and PV(g + 2) cannot start before P(g + 2)
                        // exists, so among the PVs of that buffer only PV(g - 1) may be
                        // outstanding: the barrier is exactly one phase short or complete,
                        // though this wait is skipped whenever no rescale is needed.
                        if (!warp_wait(&bars->pv_done[(g - 1) % kSBufs], ((g - 1) / kSBufs) & 1u, &s_abort)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
#pragma unroll 1
                        for (int c = 0; c < DH / 32; ++c) {
                            uint32_t r[32];
                            tmem_ld32(trow + C::O_COL + c * 32, r);
#pragma unroll
                            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * corr);
                            tmem_st32(trow + C::O_COL + c * 32, r);
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(&bars->p_full[g % kSBufs]);
                    m_run = m_new;
                }
            }
            if (!ok) break;
            // the row sum to the epilogue thread of the same row
            const uint32_t lb = (uint32_t)k & 1u;
            if (!warp_wait(&bars->l_free[lb], (((uint32_t)k >> 1) & 1u) ^ 1u, &s_abort)) {
                ok = false;
                break;
            }
            lbuf[lb * kBM + row] = l_run;
            mbar_arrive(&bars->l_full[lb]);
        }
        if (!ok) {
            s_abort = 1;
            set_status(a.status, kDevTimeout);
        }
    } else if (warp < 10) {
        // ---------------- output epilogue (warps 6..9) ----------------
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        bool ok = true;
        Unit u;
        for (int k = 0; ok && cta_unit(k, num_t, a, u); ++k) {
            const uint32_t lb = (uint32_t)k & 1u;
            if (!warp_wait(&bars->o_full, (uint32_t)k & 1u, &s_abort) ||
                !warp_wait(&bars->l_full[lb], ((uint32_t)k >> 1) & 1u, &s_abort)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const float l = lbuf[lb * kBM + row];
            uint32_t o[DH];
            if constexpr (DH == 128) {
                tmem_ld128(trow + C::O_COL, o);
            } else {
#pragma unroll
                for (int c = 0; c < DH / 32; ++c)
                    tmem_ld32(trow + C::O_COL + c * 32, *reinterpret_cast<uint32_t(*)[32]>(o + 32 * c));
            }
            tc_fence_before();
            mbar_arrive(&bars->o_free);
            mbar_arrive(&bars->l_free[lb]);
            const float inv = l > 0.f ? 1.f / l : 0.f;
            if (u.m0 + row < a.M) {
                uint4* dst = reinterpret_cast<uint4*>(a.out + (size_t)(u.m0 + row) * a.ld_out + u.h * DH);
#pragma unroll
                for (int q = 0; q < DH / 8; ++q)
                    dst[q] = make_uint4(pack_bf16x2(__uint_as_float(o[8 * q]) * inv, __uint_as_float(o[8 * q + 1]) * inv),
                                        pack_bf16x2(__uint_as_float(o[8 * q + 2]) * inv, __uint_as_float(o[8 * q + 3]) * inv),
                                        pack_bf16x2(__uint_as_float(o[8 * q + 4]) * inv, __uint_as_float(o[8 * q + 5]) * inv),
                                        pack_bf16x2(__uint_as_float(o[8 * q + 6]) * inv, __uint_as_float(o[8 * q + 7]) * inv));
            }
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
    // once per process (thread-safe initialisation of local statics)
    static const cudaError_t attr =
        cudaFuncSetAttribute(attn_prefill_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (attr != cudaSuccess) return attr;
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
    // persistent: one CTA per SM (tensor-memory kernels get one per SM), each walking its units
    static const int sms = [] {
        int dev = 0, n = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        return n > 0 ? n : 1;
    }();
    const int units = ((p.M + kBM - 1) / kBM) * p.H;
    const dim3 grid(units < sms ? units : sms);
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
