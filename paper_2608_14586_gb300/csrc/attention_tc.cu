// Causal grouped-query attention for multi-token prefill on the tcgen05 tensor cores.
//
// o[i, h] = sum_{j <= pos0 + i} softmax_j(q_ih . k_gj / sqrt(d_h)) v_gj,  g = h / (H / H_kv)
//
// Persistent: one CTA per SM (320 threads, all 512 TMEM columns) walks a list of work units,
// each a PAIR of query tiles of one head (tile A = 128 query rows, tile B = the next 128),
// numbered longest first and dealt to the CTAs in a snake so every CTA gets a similar number
// of key blocks. Both tiles read the same key/value blocks, which are loaded once for the pair.
//   warp 0      TMA: the pair's two Q tiles, then K and V blocks of 128 keys through a 2-stage K
//               ring and a 3-stage V ring shared by the two tiles. K/V come from the layer's cache through a 3-D
//               tensor map whose key extent ends at the context length, so keys past it arrive
//               as zeros.
//   warp 1      TMEM allocation; one thread issues, per tile t, S_t = Q_t K^T (M=128, N=128
//               keys, K=d_h) into TMEM columns [128t, 128t+128) and O_t += P_t V (M=128, N=d_h,
//               K=128 keys) into TMEM columns [256 + t*d_h, ...), with P_t read from tensor
//               memory (the softmax writes it as packed bf16 over the first 64 columns of S_t)
//               and V from shared memory as an MN-major operand. The next S_t is issued right
//               behind PV_t: one thread's MMAs execute in issue order, so PV_t has read P_t
//               before S_t is overwritten, and the thread never waits on an MMA.
//   warps 2..5  softmax of tile A, warps 6..9 of tile B; one thread per query row (TMEM lane):
//               reads its S row once (tcgen05.ld), masks, takes the row max, writes
//               P = exp2(s - m) as bf16 into tensor memory (tcgen05.st), keeps the row sum, and
//               rescales its O row only when the running max grows by more than 2^8 (a stale max
//               below that is exact arithmetic with values up to 2^8). Each tile is a chain
//               S -> softmax -> PV -> next S; the two chains of a pair run side by side, so
//               the tensor core works on one tile while the other's softmax runs. At the end of
//               a pair each group writes its tile's O / l.
// Phases of every barrier follow per-CTA block and pair counters. Every wait is bounded.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kThreads = 320;
constexpr float kRescaleLog2 = 8.0f;

template <int DH>
struct AttnCfg {
    static constexpr int KCH = DH / 64;              // 64-wide head-dim chunks
    static constexpr uint32_t CHUNK = 128 * 64 * 2;  // one [128 rows][64] bf16 chunk
    static constexpr uint32_t Q_BYTES = KCH * CHUNK;
    static constexpr uint32_t KV_BYTES = KCH * CHUNK;
    static constexpr int K_STAGES = 2;
    static constexpr int V_STAGES = 3;
    static constexpr uint32_t OFF_K = 2 * Q_BYTES;  // Q of tile A, then of tile B
    static constexpr uint32_t OFF_V = OFF_K + K_STAGES * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_V + V_STAGES * KV_BYTES;
    static constexpr uint32_t SMEM = OFF_BAR + 256 + 1024;
    static constexpr uint32_t TMEM_COLS = 512;
    static constexpr uint32_t O_COL = 256;  // O of tile t at O_COL + t * DH
    static constexpr uint32_t IDESC_S = idesc_bf16_f32(kBM, kBN);
    static constexpr uint32_t IDESC_O = idesc_bf16_f32_bmn(kBM, DH);
};

struct Bars {
    uint64_t q_full, q_free, k_full[2], k_empty[2], v_full[3], v_empty[3];
    uint64_t s_full[2], p_full[2], pv_done[2], o_free[2];  // per tile
    uint64_t mma_done;
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

// A pair of query tiles of one head: tile A at rows [m0, m0+128), tile B at [m0+128, m0+256)
// (absent when m0 + 128 >= M), and the key blocks each needs.
struct Pair {
    int h, g, m0, n[2];  // n[1] == 0: no tile B
};

// The CTA's k-th pair, or false. Pairs are numbered longest first (every head of the latest
// pair of query tiles, then the next, ...) and dealt to the persistent CTAs in a snake
// (round r: CTA c takes unit r*G + c on even rounds, (r+1)*G - 1 - c on odd ones).
VLA_DEV bool cta_pair(int k, int num_p, const TcAttnArgs& a, Pair& p) {
    const int G = gridDim.x, c = blockIdx.x;
    const int idx = (k & 1) ? (k + 1) * G - 1 - c : k * G + c;
    if (idx >= num_p * a.H) return false;
    const int pm = num_p - 1 - idx / a.H;
    p.h = idx % a.H;
    p.g = p.h / (a.H / a.Hkv);
    p.m0 = pm * 2 * kBM;
    for (int t = 0; t < 2; ++t) {
        const int r0 = p.m0 + t * kBM;
        p.n[t] = r0 < a.M ? (a.pos0 + min(r0 + kBM, a.M) + kBN - 1) / kBN : 0;
    }
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
    const int num_p = (a.M + 2 * kBM - 1) / (2 * kBM);

    if (threadIdx.x == 0) {
        mbar_init(&bars->q_full, 1);
        mbar_init(&bars->q_free, 1);
        for (int b = 0; b < 3; ++b) {
            mbar_init(&bars->v_full[b], 1);
            mbar_init(&bars->v_empty[b], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->k_full[b], 1);
            mbar_init(&bars->k_empty[b], 1);
            mbar_init(&bars->s_full[b], 1);
            mbar_init(&bars->p_full[b], 128);
            mbar_init(&bars->pv_done[b], 1);
            mbar_init(&bars->o_free[b], 128);
        }
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
            // ring slot of global block n: n % 2, phase (n / 2) & 1 (K and V alike)
            bool ok = true;
            uint32_t issued_k = 0, issued_v = 0, ph_k = 0, ph_v = 0;
            bool issued_q = false;
            uint32_t ph_q = 0;
            uint32_t nk = 0, nv = 0;  // K / V blocks issued so far (all pairs)
            Pair p;
            long long t0 = clock64();
            for (int k = 0; ok && cta_pair(k, num_p, a, p); ++k) {
                if (!wait_ab(&bars->q_free, ((uint32_t)k & 1u) ^ 1u, &s_abort)) {
                    ok = false;
                    break;
                }
                const int ntiles = p.n[1] > 0 ? 2 : 1;
                mbar_arrive_expect_tx(&bars->q_full, C::Q_BYTES * ntiles);
                for (int t = 0; t < ntiles; ++t)
                    for (int c = 0; c < C::KCH; ++c)
                        tma_load_2d(smem + t * C::Q_BYTES + c * C::CHUNK, &tmQ, &bars->q_full, p.h * DH + c * 64,
                                    p.m0 + t * kBM);
                issued_q = true;
                ph_q = (uint32_t)k & 1u;
                const int nmax = max(p.n[0], p.n[1]);
                int jk = 0, jv = 0;
                t0 = clock64();
                while (jk < nmax || jv < nmax) {
                    bool progressed = false;
                    if (jk < nmax) {
                        const int b = nk & 1;
                        const uint32_t n = nk >> 1;
                        if (mbar_try_wait(&bars->k_empty[b], (n & 1u) ^ 1u)) {
                            mbar_arrive_expect_tx(&bars->k_full[b], C::KV_BYTES);
                            for (int c = 0; c < C::KCH; ++c)
                                tma_load_3d(smem + C::OFF_K + b * C::KV_BYTES + c * C::CHUNK, &tmK, &bars->k_full[b],
                                            c * 64, jk * kBN, p.g);
                            issued_k |= 1u << b;
                            ph_k = (ph_k & ~(1u << b)) | ((n & 1u) << b);
                            ++jk;
                            ++nk;
                            progressed = true;
                        }
                    }
                    if (jv < nmax) {  // V runs ahead of K as far as its ring allows
                        const int b = (int)(nv % 3u);
                        const uint32_t n = nv / 3u;
                        if (mbar_try_wait(&bars->v_empty[b], (n & 1u) ^ 1u)) {
                            mbar_arrive_expect_tx(&bars->v_full[b], C::KV_BYTES);
                            for (int c = 0; c < C::KCH; ++c)
                                tma_load_3d(smem + C::OFF_V + b * C::KV_BYTES + c * C::CHUNK, &tmV, &bars->v_full[b],
                                            c * 64, jv * kBN, p.g);
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
            if (issued_q) mbar_wait(&bars->q_full, ph_q);
            for (int b = 0; b < 3; ++b) {
                if (b < 2 && (issued_k & (1u << b))) mbar_wait(&bars->k_full[b], (ph_k >> b) & 1u);
                if (issued_v & (1u << b)) mbar_wait(&bars->v_full[b], (ph_v >> b) & 1u);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            bool ok = true;
            uint32_t gt[2] = {0, 0};  // blocks of tile slot t so far (S, P, PV phases)
            uint32_t et[2] = {0, 0};  // pairs in which tile slot t existed (O phases)
            uint32_t nkv = 0;         // K/V blocks so far (ring phases)
            auto issue_s = [&](int t, uint32_t n, uint32_t sQ) {
                const uint32_t sK = smem_u32(smem + C::OFF_K + (n & 1) * C::KV_BYTES);
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const uint64_t ad = sw128_kmajor_desc(sQ + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    const uint64_t bd = sw128_kmajor_desc(sK + (kk >> 2) * C::CHUNK) + 2 * (kk & 3);
                    umma_bf16_ss(tmem + t * kBN, ad, bd, C::IDESC_S, kk > 0 ? 1u : 0u);
                }
                umma_commit(&bars->s_full[t]);
            };
            Pair p;
            for (int k = 0; ok && cta_pair(k, num_p, a, p); ++k) {
                const int nmax = max(p.n[0], p.n[1]);
                if (!wait_ab(&bars->q_full, (uint32_t)k & 1u, &s_abort) ||
                    !wait_ab(&bars->k_full[nkv & 1], (nkv >> 1) & 1u, &s_abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // S of block 0 for both tiles: their columns hold the previous pair's last P,
                // read by a PV issued before (issue order, as below)
                for (int t = 0; t < 2; ++t)
                    if (p.n[t] > 0) issue_s(t, nkv, smem_u32(smem + t * C::Q_BYTES));
                umma_commit(&bars->k_empty[nkv & 1]);
                if (nmax == 1) umma_commit(&bars->q_free);
                for (int j = 0; j < nmax && ok; ++j) {
                    const uint32_t n = nkv + j;
                    const uint32_t vs = n % 3u;  // V ring slot of block n, phase (n / 3) & 1
                    if (!wait_ab(&bars->v_full[vs], (n / 3u) & 1u, &s_abort) ||
                        (j + 1 < nmax && !wait_ab(&bars->k_full[(n + 1) & 1], ((n + 1) >> 1) & 1u, &s_abort))) {
                        ok = false;
                        break;
                    }
                    for (int t = 0; t < 2 && ok; ++t) {
                        if (j >= p.n[t]) continue;
                        if (!wait_ab(&bars->p_full[t], gt[t] & 1u, &s_abort) ||
                            (j == 0 && !wait_ab(&bars->o_free[t], (et[t] & 1u) ^ 1u, &s_abort))) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t sV = smem_u32(smem + C::OFF_V + vs * C::KV_BYTES);
#pragma unroll
                        for (int kk = 0; kk < kBN / 16; ++kk) {
                            const uint64_t bd = sw128_mnmajor_desc(sV + kk * 16 * 128, C::CHUNK);
                            umma_bf16_ts(tmem + C::O_COL + t * DH, tmem + t * kBN + kk * 8, bd, C::IDESC_O,
                                         (j > 0 || kk > 0) ? 1u : 0u);
                        }
                        // the block's last PV: V_j's slot is free once it completes (committed
                        // before the next S, so the producer can refill it while that S runs)
                        if (t == 1 || j >= p.n[1]) umma_commit(&bars->v_empty[vs]);
                        // The next S of this tile overwrites P_t in the same columns. It is issued
                        // right behind the PV that reads P_t: the tensor core executes one thread's
                        // MMAs in issue order, so the PV's operand reads precede the S's writes.
                        // Its commit also tells the softmax that PV_t has completed (O_t may be
                        // rescaled).
                        if (j + 1 < p.n[t]) issue_s(t, n + 1, smem_u32(smem + t * C::Q_BYTES));
                        else umma_commit(&bars->pv_done[t]);  // the tile's last PV: O_t is final
                        ++gt[t];
                    }
                    if (!ok) break;
                    if (j + 1 < nmax) {
                        umma_commit(&bars->k_empty[(n + 1) & 1]);
                        if (j + 2 == nmax) umma_commit(&bars->q_free);  // the pair's last S was just issued
                    }
                }
                if (!ok) break;
                for (int t = 0; t < 2; ++t)
                    if (p.n[t] > 0) ++et[t];
                nkv += nmax;
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
        // ---------------- softmax / correction / epilogue: tile A (warps 2..5), B (6..9) ----------------
        const int t = (warp - 2) >> 2;
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t scol = (uint32_t)t * kBN;
        const uint32_t ocol = C::O_COL + (uint32_t)t * DH;
        bool ok = true;
        uint32_t g = 0;   // blocks of this tile slot so far (S and P phases)
        uint32_t np = 0;  // pairs in which this tile slot existed (final-PV phases)
        Pair p;
        for (int k = 0; ok && cta_pair(k, num_p, a, p); ++k) {
            if (p.n[t] == 0) continue;  // no tile B in this pair
            const int m0 = p.m0 + t * kBM;
            const int qpos = a.pos0 + m0 + row;
            const int min_qpos = a.pos0 + m0;
            float m_run = -INFINITY, l_run = 0.f;
            for (int j = 0; j < p.n[t]; ++j) {
                uint32_t sr[kBN];
                float m_new = m_run;
                bool need = false;
                {
                    const int kb = j * kBN;
                    const bool need_mask = (kb + kBN - 1 > min_qpos) || (kb + kBN > a.ctx);
                    ok = wait_ab(&bars->s_full[t], g & 1u, &s_abort);
                    __syncwarp();
                    if (!__all_sync(0xFFFFFFFFu, ok)) {
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
                    // P = exp2(s * scale - m) as packed bf16 over the first 64 columns of S
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
                        // PV of the previous block has completed: this block's S was issued after it
#pragma unroll 1
                        for (int c = 0; c < DH / 32; ++c) {
                            uint32_t r[32];
                            tmem_ld32(trow + ocol + c * 32, r);
#pragma unroll
                            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * corr);
                            tmem_st32(trow + ocol + c * 32, r);
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(&bars->p_full[t]);
                    m_run = m_new;
                    ++g;
                }
            }
            if (!ok) break;
            // epilogue of this tile: after its last PV
            ok = wait_ab(&bars->pv_done[t], np & 1u, &s_abort);
            ++np;
            __syncwarp();
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
            const bool row_ok = (m0 + row) < a.M;
            bf16* orow = a.out + (size_t)(m0 + row) * a.ld_out + p.h * DH;
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
            mbar_arrive(&bars->o_free[t]);
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
    // persistent: one CTA per SM (tensor-memory kernels get one per SM), each walking its pairs
    static const int sms = [] {
        int dev = 0, n = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        return n > 0 ? n : 1;
    }();
    const int units = ((p.M + 2 * kBM - 1) / (2 * kBM)) * p.H;
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
