// CPU-executed decoder blocks: the suffix B_{p+1..N}^cpu of block-layer partitioning (Eq. 6),
// run on the host cores from host memory.
//
// The block is the one the GPU prefix runs (RMSNorm with its gain folded into the next
// projection, QKV + rotary embedding + KV write, causal GQA attention, output projection +
// residual, RMSNorm, gate/up + SwiGLU, down projection + residual), with bf16 weights and
// activations, fp32 accumulation and bf16 rounding at the points where the GPU stores bf16:
//   * projections C = A W^T: W is repacked at create time into panels of 8 output rows,
//     [panel][k][8] bf16, gains folded in and rounded to bf16 as on the GPU. The register
//     tile is 12 rows x 8 columns: three 4-row vectors of A times each of the 8 weight values
//     of a k step (24 fp32 vector accumulators; GCC vector extensions over 128-bit lanes: NEON
//     on an Arm host, SSE on x86). A task tile is 144 rows x 128 columns over 512-deep k
//     blocks; each k block's weight slice is widened to fp32 once and reused by the tile's
//     twelve 12-row panels, and a task takes two column tiles so that each packed A block
//     serves both. Every output element's k order is fixed, so results do not depend on how
//     tiles fall to threads. The epilogues mirror the GPU's: 1/rms scaling, RoPE and
//     the KV write for QKV; the residual add for O and down; SwiGLU for gate/up, whose rows
//     are grouped as 64 gate rows then the 64 matching up rows so one tile holds both halves;
//   * attention: one task per (KV head, block of 16 queries), longest first; per 64-key block
//     the scores and the output update run on the same register tile (S^T = K Q^T, O^T +=
//     V^T P^T) around an fp32 online softmax; a key past a query's position gets probability
//     0 and a key block wholly past it leaves that query's state unchanged, so each query's
//     result does not depend on which other queries share its call (causal invariance);
//   * a fixed pool of worker threads that draw tasks from an atomic counter; the thread that
//     makes a compute call works too.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <condition_variable>
#include <cstdint>
#include <cstring>
#include <functional>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "cpu_math.h"
#include "vla_cpu.h"

namespace {

typedef float v4f __attribute__((vector_size(16)));
typedef uint16_t v4h __attribute__((vector_size(8)));
typedef uint32_t v4u __attribute__((vector_size(16)));

constexpr int kMR = 12;   // rows of one register tile (three 4-lane vectors)
constexpr int kNR = 8;    // columns of one register tile = weight rows of one panel
constexpr int kKC = 512;  // k block
constexpr int kTM = 144;  // rows of one task tile
constexpr int kTN = 128;  // columns of one task tile
constexpr int kTG = 2;    // column tiles per task at most (they share one packed A block)
constexpr int kGU = 64;   // feed-forward units per gate/up tile (64 gate + 64 up columns)
constexpr int kQB = 16;   // queries per attention task
constexpr int kKB = 64;   // keys per attention block
constexpr int kKPan = (kKB + kMR - 1) / kMR;  // register-tile panels of one key block
static_assert(kKB % 4 == 0 && kGU % 4 == 0, "the softmax and SiLU loops take four lanes at a time");

inline float bf2f(uint16_t b) {
    const uint32_t u = (uint32_t)b << 16;
    float f;
    std::memcpy(&f, &u, 4);
    return f;
}

// Round to the nearest bf16, ties to even (NaN stays NaN).
inline uint16_t f2bf(float f) {
    uint32_t u;
    std::memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((u >> 16) | ((u & 0xFFFFu) ? 0x40u : 0u));
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

inline v4f ld_bf4(const uint16_t* p) {
    v4h h;
    std::memcpy(&h, p, sizeof h);
    const v4u u = __builtin_convertvector(h, v4u) << 16;
    return (v4f)u;
}

inline float hsum(v4f v) { return (v[0] + v[1]) + (v[2] + v[3]); }

// ---------------------------------------------------------------------------------------
// thread pool
// ---------------------------------------------------------------------------------------
class Pool {
  public:
    explicit Pool(int n) : n_(n < 1 ? 1 : n) {
        try {
            for (int i = 1; i < n_; ++i) th_.emplace_back([this, i] { worker(i); });
        } catch (...) {
            shutdown();  // join the threads already started before the failure propagates
            throw;
        }
    }
    ~Pool() { shutdown(); }
    int size() const { return n_; }
    // fn(task, thread) for every task in [0, n_tasks); returns when all have finished.
    void run(int n_tasks, const std::function<void(int, int)>& fn) {
        if (n_tasks <= 0) return;
        if (n_ == 1 || n_tasks == 1) {
            for (int t = 0; t < n_tasks; ++t) fn(t, 0);
            return;
        }
        std::unique_lock<std::mutex> lk(m_);
        fn_ = &fn;
        tasks_ = n_tasks;
        next_.store(0);
        active_ = n_ - 1;
        ++gen_;
        lk.unlock();
        cv_.notify_all();
        drain(0);
        lk.lock();
        done_.wait(lk, [&] { return active_ == 0; });
        fn_ = nullptr;
    }

  private:
    void shutdown() {
        {
            std::lock_guard<std::mutex> lk(m_);
            stop_ = true;
            ++gen_;
        }
        cv_.notify_all();
        for (auto& t : th_)
            if (t.joinable()) t.join();
        th_.clear();
    }
    void drain(int tid) {
        for (int t = next_.fetch_add(1); t < tasks_; t = next_.fetch_add(1)) (*fn_)(t, tid);
    }
    void worker(int tid) {
        uint64_t seen = 0;
        std::unique_lock<std::mutex> lk(m_);
        for (;;) {
            cv_.wait(lk, [&] { return gen_ != seen; });
            seen = gen_;
            if (stop_) return;
            lk.unlock();
            drain(tid);
            lk.lock();
            if (--active_ == 0) done_.notify_one();
        }
    }
    int n_;
    std::vector<std::thread> th_;
    std::mutex m_;
    std::condition_variable cv_, done_;
    const std::function<void(int, int)>* fn_ = nullptr;
    std::atomic<int> next_{0};
    int tasks_ = 0, active_ = 0;
    uint64_t gen_ = 0;
    bool stop_ = false;
};

// ---------------------------------------------------------------------------------------
// packed weights and the micro-kernel
// ---------------------------------------------------------------------------------------
struct Packed {
    int N = 0, K = 0;           // N: a multiple of kTN
    std::vector<uint16_t> w;    // [N / kNR][K][kNR]
};

struct Scratch {
    std::vector<float> apack;   // [kTM / kMR][kKC][kMR]
    std::vector<float> bf;      // [kKC][kNR]: one panel's k block widened to fp32
    std::vector<float> ctile;   // kTG tiles of [kTN][kTM], column-major
    std::vector<float> qpk, ppk, st, ot;  // attention operands (see attention())
    std::vector<float> mx, l;                        // [G * kQB]
};

// c[8 columns][4*MV rows] (column stride ldc) = (init ? 0 : c) + a-panel x b-panel over kc
// steps; a-panel [k][kMR] fp32 (rows), b-panel [k][kNR] fp32 (columns).
template <int MV>
inline void micro(const float* a, const float* b, int kc, float* c, int ldc, bool init) {
    v4f acc[kNR][MV];
    for (int j = 0; j < kNR; ++j)
        for (int i = 0; i < MV; ++i) {
            if (init) {
                acc[j][i] = v4f{0.f, 0.f, 0.f, 0.f};
            } else {
                std::memcpy(&acc[j][i], c + (size_t)j * ldc + 4 * i, sizeof(v4f));
            }
        }
    for (int k = 0; k < kc; ++k) {
        v4f av[MV];
        for (int i = 0; i < MV; ++i) std::memcpy(&av[i], a + 4 * i, sizeof(v4f));
        a += kMR;
        for (int j = 0; j < kNR; ++j) {
            const float bj = b[j];
            for (int i = 0; i < MV; ++i) acc[j][i] += av[i] * bj;
        }
        b += kNR;
    }
    for (int j = 0; j < kNR; ++j)
        for (int i = 0; i < MV; ++i) std::memcpy(c + (size_t)j * ldc + 4 * i, &acc[j][i], sizeof(v4f));
}

inline void micro_any(int rows, const float* a, const float* b, int kc, float* c, int ldc, bool init) {
    if (rows > 8) micro<3>(a, b, kc, c, ldc, init);
    else if (rows > 4) micro<2>(a, b, kc, c, ldc, init);
    else micro<1>(a, b, kc, c, ldc, init);
}

}  // namespace

struct vla_cpu_model {
    vla_config cfg;
    int lb = 0, le = 0;
    int qc = 0, kvc = 0, qkv_n = 0, F_pad = 0;
    struct Layer {
        Packed qkv, o, gu, down;
    };
    std::vector<Layer> layers;
    std::vector<float> rope;  // [max_ctx][dh/2] (cos, sin) pairs
    Pool* pool = nullptr;
    std::vector<Scratch> scratch;
    std::mutex mu;
    // workspace for cfg.max_ctx tokens
    std::vector<uint16_t> h[2], q, att, xmid, mbuf;
    std::vector<float> rinv;
    std::vector<float> xrows;  // [4][max K]: the rows of a short (decode) projection in fp32
    std::vector<float> kvpk;   // one call's keys and values as register-tile panels (attention())
    ~vla_cpu_model() { delete pool; }
};

struct vla_cpu_kv {
    vla_cpu_model* m = nullptr;
    int lb = 0, le = 0, max_ctx = 0;
    size_t plane = 0;
    std::vector<uint16_t> data;
    std::vector<int> len;
    uint16_t* k_plane(int l) { return data.data() + (size_t)(l - lb) * 2 * plane; }
    uint16_t* v_plane(int l) { return data.data() + ((size_t)(l - lb) * 2 + 1) * plane; }
};

namespace {

using Model = vla_cpu_model;

// Packs rows [0, N) of a [N, K] operand given row by row (row(n) = K bf16, or nullptr for a
// zero row), each element times gain[k] (fp32 product rounded to bf16) when gain is set.
template <class RowFn>
void pack(Pool& pool, Packed& P, int N, int K, RowFn row, const uint16_t* gain) {
    P.N = N;
    P.K = K;
    P.w.assign((size_t)N * K, 0);
    std::vector<float> g;
    if (gain) {
        g.resize(K);
        for (int k = 0; k < K; ++k) g[k] = bf2f(gain[k]);
    }
    pool.run(N / kNR, [&](int panel, int) {
        uint16_t* dst = P.w.data() + (size_t)panel * K * kNR;
        for (int c = 0; c < kNR; ++c) {
            const uint16_t* src = row(panel * kNR + c);
            if (!src) continue;
            if (gain) {
                for (int k = 0; k < K; ++k) dst[(size_t)k * kNR + c] = f2bf(bf2f(src[k]) * g[k]);
            } else {
                for (int k = 0; k < K; ++k) dst[(size_t)k * kNR + c] = src[k];
            }
        }
    });
}

// Up to kGemvRows rows (decode): each weight panel streams once, straight from its bf16
// words, into 2 x R vector accumulators. Every element sees the same sequence of fused
// multiply-adds as in the tiled path (k ascending from 0), so both give the same bits.
constexpr int kGemvRows = 4;

template <int R>
void gemv_panel(const float* x, int K, const uint16_t* bp, float* c, int ldc) {
    v4f acc[R][2];
    for (int r = 0; r < R; ++r) acc[r][0] = acc[r][1] = v4f{0.f, 0.f, 0.f, 0.f};
    for (int k = 0; k < K; ++k) {
        const v4f w0 = ld_bf4(bp + (size_t)k * kNR), w1 = ld_bf4(bp + (size_t)k * kNR + 4);
        for (int r = 0; r < R; ++r) {
            const float xr = x[(size_t)r * K + k];
            acc[r][0] += w0 * xr;
            acc[r][1] += w1 * xr;
        }
    }
    for (int r = 0; r < R; ++r)
        for (int j = 0; j < 4; ++j) {
            c[(size_t)j * ldc + r] = acc[r][0][j];
            c[(size_t)(j + 4) * ldc + r] = acc[r][1][j];
        }
}

// C = A W^T over task tiles; epi(m0, rows, n0, C, ldc) consumes each finished tile, whose
// element (row m0 + r, column n0 + n) is C[n * ldc + r].
template <class Epi>
void gemm(Model* m, const uint16_t* A, int M, const Packed& B, const Epi& epi) {
    const int K = B.K;
    if (M <= kGemvRows) {
        float* x = m->xrows.data();
        for (size_t i = 0; i < (size_t)M * K; ++i) x[i] = bf2f(A[i]);
        m->pool->run(B.N / kTN, [&](int t, int tid) {
            float* C = m->scratch[tid].ctile.data();
            const int n0 = t * kTN;
            for (int j = 0; j < kTN / kNR; ++j) {
                const uint16_t* bp = B.w.data() + (size_t)(n0 / kNR + j) * K * kNR;
                float* c = C + (size_t)j * kNR * kTM;
                switch (M) {
                    case 4: gemv_panel<4>(x, K, bp, c, kTM); break;
                    case 3: gemv_panel<3>(x, K, bp, c, kTM); break;
                    case 2: gemv_panel<2>(x, K, bp, c, kTM); break;
                    default: gemv_panel<1>(x, K, bp, c, kTM); break;
                }
            }
            epi(0, M, n0, C, kTM);
        });
        return;
    }
    // A task is one block of kTM rows times up to kTG column tiles, which reuse each packed
    // A block; fewer column tiles per task where that would leave under 4 tasks per thread.
    const int tm = (M + kTM - 1) / kTM, tn = B.N / kTN;
    int grp = kTG;
    while (grp > 1 && tm * ((tn + grp - 1) / grp) < 4 * m->pool->size()) grp >>= 1;
    const int tg = (tn + grp - 1) / grp;
    m->pool->run(tm * tg, [&](int t, int tid) {
        Scratch& s = m->scratch[tid];
        const int im = t % tm, j0 = (t / tm) * grp, j1 = std::min(tn, j0 + grp);
        const int m0 = im * kTM, rows = std::min(kTM, M - m0);
        const int np = (rows + kMR - 1) / kMR;
        float* bf = s.bf.data();
        for (int k0 = 0; k0 < K; k0 += kKC) {
            const int kc = std::min(kKC, K - k0);
            for (int p = 0; p < np; ++p) {
                float* ap = s.apack.data() + (size_t)p * kKC * kMR;
                for (int i = 0; i < kMR; ++i) {
                    const int r = p * kMR + i;
                    if (r < rows) {
                        const uint16_t* src = A + (size_t)(m0 + r) * K + k0;
                        for (int k = 0; k < kc; ++k) ap[k * kMR + i] = bf2f(src[k]);
                    } else {
                        for (int k = 0; k < kc; ++k) ap[k * kMR + i] = 0.f;
                    }
                }
            }
            for (int jt = j0; jt < j1; ++jt) {
                float* C = s.ctile.data() + (size_t)(jt - j0) * kTN * kTM;
                for (int j = 0; j < kTN / kNR; ++j) {
                    const uint16_t* bp = B.w.data() + ((size_t)(jt * kTN / kNR + j) * K + k0) * kNR;
                    for (int e = 0; e < kc * kNR; e += 4) {
                        const v4f v = ld_bf4(bp + e);
                        std::memcpy(bf + e, &v, sizeof v);
                    }
                    for (int p = 0; p < np; ++p)
                        micro_any(rows - p * kMR, s.apack.data() + (size_t)p * kKC * kMR, bf, kc,
                                  C + (size_t)j * kNR * kTM + p * kMR, kTM, k0 == 0);
                }
            }
        }
        for (int jt = j0; jt < j1; ++jt) epi(m0, rows, jt * kTN, s.ctile.data() + (size_t)(jt - j0) * kTN * kTM, kTM);
    });
}

// 1/rms of each row: 1 / sqrt(mean(x^2) + eps), fp32 sum in column order.
void row_rinv(Model* m, const uint16_t* x, int M, float* out) {
    const int D = m->cfg.hidden;
    const int chunk = 64;
    m->pool->run((M + chunk - 1) / chunk, [&](int t, int) {
        for (int r = t * chunk; r < std::min(M, (t + 1) * chunk); ++r) {
            const uint16_t* xr = x + (size_t)r * D;
            v4f acc = {0.f, 0.f, 0.f, 0.f};
            for (int k = 0; k < D; k += 4) {
                const v4f v = ld_bf4(xr + k);
                acc += v * v;
            }
            out[r] = 1.0f / std::sqrt(hsum(acc) / (float)D + m->cfg.rms_eps);
        }
    });
}

// Causal GQA attention of M queries at positions p0.. over cache positions [0, p0 + M).
// Every 64-key block of every KV head is first widened to fp32 register-tile panels, once
// per call. Per task (KV head g, block of kQB queries): the G query heads' vectors of the
// block form nq = G * rows columns. Per 64-key block: S^T = K Q^T and O^T += V^T P^T on the
// register tile (keys resp. head dims as rows, queries as columns), with the online-softmax
// update (running max, rescale of the running sum and output) in between. Keys past a
// query's position get probability 0 and a block wholly past it leaves its state unchanged.
void attention(Model* m, const uint16_t* q, const uint16_t* kp, const uint16_t* vp, int max_ctx, int p0, int M,
               uint16_t* out) {
    const int H = m->cfg.n_heads, Hkv = m->cfg.n_kv_heads, dh = m->cfg.head_dim, G = H / Hkv;
    const float scale = 1.0f / std::sqrt((float)dh);
    const int nqb = (M + kQB - 1) / kQB;
    const int dpan = (dh + kMR - 1) / kMR;  // head-dim panels of the O tile
    // per (g, key block): keys [kKPan][dh][kMR] (zero rows past the context), then values
    // [dpan][kKB][kMR]
    const int nkb = (p0 + M + kKB - 1) / kKB;
    const size_t kstride = (size_t)kKPan * dh * kMR, bstride = kstride + (size_t)dpan * kKB * kMR;
    float* kvpk = m->kvpk.data();
    m->pool->run(Hkv * nkb, [&](int t, int) {
        const int g = t % Hkv, kb = t / Hkv, kb0 = kb * kKB, kn = std::min(kKB, p0 + M - kb0);
        float* kpk = kvpk + ((size_t)g * nkb + kb) * bstride;
        float* vpk = kpk + kstride;
        const uint16_t* kg = kp + (size_t)g * max_ctx * dh;
        const uint16_t* vg = vp + (size_t)g * max_ctx * dh;
        for (int j = 0; j < (kn + kMR - 1) / kMR * kMR; ++j) {
            float* dst = kpk + (size_t)(j / kMR) * dh * kMR + (j % kMR);
            if (j < kn) {
                const uint16_t* src = kg + (size_t)(kb0 + j) * dh;
                for (int d = 0; d < dh; ++d) dst[(size_t)d * kMR] = bf2f(src[d]);
            } else {
                for (int d = 0; d < dh; ++d) dst[(size_t)d * kMR] = 0.f;
            }
        }
        for (int j = 0; j < kn; ++j) {
            const uint16_t* src = vg + (size_t)(kb0 + j) * dh;
            for (int d = 0; d < dh; ++d) vpk[((size_t)(d / kMR) * kKB + j) * kMR + (d % kMR)] = bf2f(src[d]);
        }
    });
    m->pool->run(Hkv * nqb, [&](int t, int tid) {
        Scratch& s = m->scratch[tid];
        const int g = t % Hkv, qb = nqb - 1 - t / Hkv;  // longest query blocks first
        const int r0 = qb * kQB, r1 = std::min(M, r0 + kQB), nr = r1 - r0;
        const int nq = G * nr, nqp = (nq + kNR - 1) / kNR;  // query columns, column panels
        float* qpk = s.qpk.data();  // [nqp][dh][kNR]   queries (scaled), B operand of S
        float* ppk = s.ppk.data();  // [nqp][kKB][kNR]  probabilities, B operand of O
        float* st = s.st.data();    // [nqp * kNR][kKB] scores, query-major
        float* ot = s.ot.data();    // [nqp * kNR][dh]  unnormalised outputs, query-major
        std::fill(qpk, qpk + (size_t)nqp * dh * kNR, 0.f);
        for (int c = 0; c < nq; ++c) {
            const int hh = c / nr, i = c % nr;
            const uint16_t* src = q + (size_t)(r0 + i) * H * dh + (size_t)(g * G + hh) * dh;
            float* dst = qpk + (size_t)(c / kNR) * dh * kNR + (c % kNR);
            for (int d = 0; d < dh; ++d) dst[(size_t)d * kNR] = bf2f(src[d]) * scale;
        }
        std::fill(ot, ot + (size_t)nqp * kNR * dh, 0.f);
        std::fill(s.mx.begin(), s.mx.begin() + nq, -INFINITY);
        std::fill(s.l.begin(), s.l.begin() + nq, 0.f);
        const int nkeys = p0 + r1;  // keys visible to the block's last query
        for (int kb0 = 0; kb0 < nkeys; kb0 += kKB) {
            const int kn = std::min(kKB, nkeys - kb0);
            const int kpan = (kn + kMR - 1) / kMR;
            const float* kpk = kvpk + ((size_t)g * nkb + kb0 / kKB) * bstride;
            const float* vpk = kpk + kstride;
            for (int cp = 0; cp < nqp; ++cp)
                for (int kq = 0; kq < kpan; ++kq)
                    micro_any(kn - kq * kMR, kpk + (size_t)kq * dh * kMR, qpk + (size_t)cp * dh * kNR, dh,
                              st + (size_t)cp * kNR * kKB + kq * kMR, kKB, true);
            std::fill(ppk, ppk + (size_t)nqp * kKB * kNR, 0.f);
            for (int c = 0; c < nq; ++c) {
                const int i = c % nr;
                const int jn = std::min(kn, p0 + r0 + i - kb0 + 1);  // keys at or before the query
                if (jn <= 0) continue;
                const float* sc = st + (size_t)c * kKB;
                float smax = -INFINITY;
                for (int j = 0; j < jn; ++j) smax = std::max(smax, sc[j]);
                const float mold = s.mx[c], mnew = std::max(mold, smax);
                const float corr = vla_cpu::exp1(mold - mnew);  // 0 when mold = -inf
                float lsum = s.l[c] * corr;
                float* pc = ppk + (size_t)(c / kNR) * kKB * kNR + (c % kNR);
                // four scores at a time (the lanes past jn read scores of this block's
                // zero-padded key rows and are dropped), then summed in key order
                float pv[kKB];
                for (int j = 0; j < jn; j += 4) {
                    v4f a;
                    std::memcpy(&a, sc + j, sizeof a);
                    const v4f e = vla_cpu::exp4(a - mnew);
                    std::memcpy(pv + j, &e, sizeof e);
                }
                for (int j = 0; j < jn; ++j) {
                    lsum += pv[j];
                    pc[(size_t)j * kNR] = pv[j];
                }
                float* oc = ot + (size_t)c * dh;
                for (int d = 0; d < dh; ++d) oc[d] *= corr;
                s.mx[c] = mnew;
                s.l[c] = lsum;
            }
            for (int cp = 0; cp < nqp; ++cp)
                for (int dp = 0; dp < dpan; ++dp)
                    micro_any(dh - dp * kMR, vpk + (size_t)dp * kKB * kMR, ppk + (size_t)cp * kKB * kNR, kn,
                              ot + (size_t)cp * kNR * dh + dp * kMR, dh, false);
        }
        for (int c = 0; c < nq; ++c) {
            const int hh = c / nr, i = c % nr;
            const float inv = 1.0f / s.l[c];
            uint16_t* dst = out + (size_t)(r0 + i) * H * dh + (size_t)(g * G + hh) * dh;
            const float* oc = ot + (size_t)c * dh;
            for (int d = 0; d < dh; ++d) dst[d] = f2bf(oc[d] * inv);
        }
    });
}

// One block l on x [M, D] at positions p0.. -> y (may alias x).
void block(Model* m, int l, const uint16_t* x, int M, int p0, vla_cpu_kv* kv, uint16_t* y) {
    const vla_config& c = m->cfg;
    const int D = c.hidden, H = c.n_heads, Hkv = c.n_kv_heads, dh = c.head_dim, half = dh / 2;
    const int qc = m->qc, F_pad = m->F_pad;
    const vla_cpu_model::Layer& W = m->layers[l - m->lb];
    float* rinv = m->rinv.data();
    uint16_t* q = m->q.data();
    uint16_t* att = m->att.data();
    uint16_t* xmid = m->xmid.data();
    uint16_t* mb = m->mbuf.data();
    uint16_t* kp = kv->k_plane(l);
    uint16_t* vp = kv->v_plane(l);
    const int max_ctx = kv->max_ctx;
    const float* rope = m->rope.data();

    // RMSNorm statistics; QKV projection + 1/rms + RoPE + KV write
    row_rinv(m, x, M, rinv);
    gemm(m, x, M, W.qkv, [&](int m0, int rows, int n0, const float* C, int ldc) {
        for (int h0 = n0; h0 < n0 + kTN; h0 += dh) {
            const int head = h0 / dh;
            for (int r = 0; r < rows; ++r) {
                const int pos = p0 + m0 + r;
                const float ri = rinv[m0 + r];
                const float* cr = C + (size_t)(h0 - n0) * ldc + r;  // column j at cr[j * ldc]
                uint16_t* dst;
                if (head < H) dst = q + (size_t)(m0 + r) * qc + (size_t)head * dh;
                else if (head < H + Hkv) dst = kp + ((size_t)(head - H) * max_ctx + pos) * dh;
                else dst = vp + ((size_t)(head - H - Hkv) * max_ctx + pos) * dh;
                if (head < H + Hkv) {
                    const float* cs = rope + (size_t)pos * dh;  // (cos, sin) of the pairs j < dh/2
                    for (int j = 0; j < half; ++j) {
                        const float a = cr[(size_t)j * ldc] * ri, b = cr[(size_t)(j + half) * ldc] * ri;
                        dst[j] = f2bf(a * cs[2 * j] - b * cs[2 * j + 1]);
                        dst[j + half] = f2bf(b * cs[2 * j] + a * cs[2 * j + 1]);
                    }
                } else {
                    for (int d = 0; d < dh; ++d) dst[d] = f2bf(cr[(size_t)d * ldc] * ri);
                }
            }
        }
    });
    attention(m, q, kp, vp, max_ctx, p0, M, att);
    // output projection + residual
    gemm(m, att, M, W.o, [&](int m0, int rows, int n0, const float* C, int ldc) {
        for (int r = 0; r < rows; ++r) {
            const uint16_t* xr = x + (size_t)(m0 + r) * D + n0;
            uint16_t* dst = xmid + (size_t)(m0 + r) * D + n0;
            for (int n = 0; n < kTN; ++n) dst[n] = f2bf(bf2f(xr[n]) + C[(size_t)n * ldc + r]);
        }
    });
    // RMSNorm statistics; gate/up + SwiGLU
    row_rinv(m, xmid, M, rinv);
    gemm(m, xmid, M, W.gu, [&](int m0, int rows, int n0, const float* C, int ldc) {
        const int u0 = n0 / 2;
        for (int r = 0; r < rows; ++r) {
            const float ri = rinv[m0 + r];
            uint16_t* dst = mb + (size_t)(m0 + r) * F_pad + u0;
            for (int i = 0; i < kGU; i += 4) {
                v4f gt, up;
                for (int e = 0; e < 4; ++e) {
                    gt[e] = C[(size_t)(i + e) * ldc + r] * ri;
                    up[e] = C[(size_t)(kGU + i + e) * ldc + r] * ri;
                }
                const v4f sw = gt / (1.0f + vla_cpu::exp4(-gt)) * up;
                for (int e = 0; e < 4; ++e) dst[i + e] = f2bf(sw[e]);
            }
        }
    });
    // down projection + residual
    gemm(m, mb, M, W.down, [&](int m0, int rows, int n0, const float* C, int ldc) {
        for (int r = 0; r < rows; ++r) {
            const uint16_t* xr = xmid + (size_t)(m0 + r) * D + n0;
            uint16_t* dst = y + (size_t)(m0 + r) * D + n0;
            for (int n = 0; n < kTN; ++n) dst[n] = f2bf(bf2f(xr[n]) + C[(size_t)n * ldc + r]);
        }
    });
}

vla_status check_cfg(const vla_config* c) {
    if (c->hidden <= 0 || c->n_heads <= 0 || c->n_kv_heads <= 0 || c->head_dim <= 0 || c->ffn <= 0 ||
        c->max_ctx <= 0 || !(c->rms_eps >= 0.f) || !(c->rope_base > 1.f))
        return VLA_ERR_INVALID_ARG;
    if (c->head_dim != 64 && c->head_dim != 128) return VLA_ERR_UNSUPPORTED;
    if (c->n_heads % c->n_kv_heads) return VLA_ERR_UNSUPPORTED;
    const int grp = c->n_heads / c->n_kv_heads;
    if (grp != 1 && grp != 2 && grp != 4 && grp != 8) return VLA_ERR_UNSUPPORTED;
    if ((c->n_heads * c->head_dim) % 256 || (c->n_kv_heads * c->head_dim) % 256) return VLA_ERR_UNSUPPORTED;
    if (c->hidden % 256) return VLA_ERR_UNSUPPORTED;
    return VLA_OK;
}

}  // namespace

extern "C" {

vla_status vla_cpu_model_create(const vla_config* cfg, const vla_layer_weights* host_weights, int layer_begin,
                                int layer_end, int n_threads, vla_cpu_model** out) {
    if (!out) return VLA_ERR_INVALID_ARG;
    *out = nullptr;
    if (!cfg || !host_weights || layer_begin < 0 || layer_end <= layer_begin || n_threads < 0)
        return VLA_ERR_INVALID_ARG;
    vla_status st = check_cfg(cfg);
    if (st != VLA_OK) return st;
    const int nl = layer_end - layer_begin;
    for (int i = 0; i < nl; ++i) {
        const vla_layer_weights& w = host_weights[i];
        if (!w.w_q || !w.w_k || !w.w_v || !w.w_o || !w.w_gate || !w.w_up || !w.w_down || !w.g_attn || !w.g_mlp)
            return VLA_ERR_INVALID_ARG;
    }
    Model* m = new (std::nothrow) Model();
    if (!m) return VLA_ERR_OOM;
    try {
        m->cfg = *cfg;
        m->lb = layer_begin;
        m->le = layer_end;
        const int D = cfg->hidden, H = cfg->n_heads, Hkv = cfg->n_kv_heads, dh = cfg->head_dim, F = cfg->ffn;
        const int T = cfg->max_ctx, G = H / Hkv;
        m->qc = H * dh;
        m->kvc = Hkv * dh;
        m->qkv_n = m->qc + 2 * m->kvc;
        m->F_pad = (F + kGU - 1) / kGU * kGU;
        int nt = n_threads;
        if (nt == 0) nt = (int)std::max(1u, std::thread::hardware_concurrency());
        m->pool = new Pool(nt);
        m->scratch.resize(m->pool->size());
        for (Scratch& s : m->scratch) {
            s.apack.assign((size_t)kTM * kKC, 0.f);
            s.bf.assign((size_t)kKC * kNR, 0.f);
            s.ctile.assign((size_t)kTG * kTM * kTN, 0.f);
            const int qcols = (G * kQB + kNR - 1) / kNR * kNR;
            s.qpk.assign((size_t)qcols * dh, 0.f);
            s.ppk.assign((size_t)qcols * kKB, 0.f);
            s.st.assign((size_t)qcols * kKB, 0.f);
            s.ot.assign((size_t)qcols * dh, 0.f);
            s.mx.assign((size_t)G * kQB, 0.f);
            s.l.assign((size_t)G * kQB, 0.f);
        }
        // rotary table in double: angle pos * base^(-2j/dh)
        m->rope.resize((size_t)T * dh);
        for (int pos = 0; pos < T; ++pos)
            for (int j = 0; j < dh / 2; ++j) {
                const double ang = (double)pos * std::pow((double)cfg->rope_base, -2.0 * j / dh);
                m->rope[(size_t)pos * dh + 2 * j] = (float)std::cos(ang);
                m->rope[(size_t)pos * dh + 2 * j + 1] = (float)std::sin(ang);
            }
        m->layers.resize(nl);
        for (int i = 0; i < nl; ++i) {
            const vla_layer_weights& w = host_weights[i];
            auto* wq = static_cast<const uint16_t*>(w.w_q);
            auto* wk = static_cast<const uint16_t*>(w.w_k);
            auto* wv = static_cast<const uint16_t*>(w.w_v);
            auto* wo = static_cast<const uint16_t*>(w.w_o);
            auto* wg = static_cast<const uint16_t*>(w.w_gate);
            auto* wu = static_cast<const uint16_t*>(w.w_up);
            auto* wd = static_cast<const uint16_t*>(w.w_down);
            vla_cpu_model::Layer& L = m->layers[i];
            const int qc = m->qc, kvc = m->kvc;
            pack(*m->pool, L.qkv, m->qkv_n, D,
                 [&](int n) -> const uint16_t* {
                     if (n < qc) return wq + (size_t)n * D;
                     if (n < qc + kvc) return wk + (size_t)(n - qc) * D;
                     return wv + (size_t)(n - qc - kvc) * D;
                 },
                 static_cast<const uint16_t*>(w.g_attn));
            pack(*m->pool, L.o, D, qc, [&](int n) -> const uint16_t* { return wo + (size_t)n * qc; }, nullptr);
            pack(*m->pool, L.gu, 2 * m->F_pad, D,
                 [&](int n) -> const uint16_t* {
                     const int grp = n / (2 * kGU), i2 = n % (2 * kGU);
                     const int unit = grp * kGU + (i2 % kGU);
                     if (unit >= F) return nullptr;
                     return (i2 < kGU ? wg : wu) + (size_t)unit * D;
                 },
                 static_cast<const uint16_t*>(w.g_mlp));
            // down: K padded with zero columns from F to F_pad
            L.down.N = D;
            L.down.K = m->F_pad;
            L.down.w.assign((size_t)D * m->F_pad, 0);
            m->pool->run(D / kNR, [&](int panel, int) {
                uint16_t* dst = L.down.w.data() + (size_t)panel * m->F_pad * kNR;
                for (int c = 0; c < kNR; ++c) {
                    const uint16_t* src = wd + (size_t)(panel * kNR + c) * F;
                    for (int k = 0; k < F; ++k) dst[(size_t)k * kNR + c] = src[k];
                }
            });
        }
        m->h[0].resize((size_t)T * D);
        m->h[1].resize((size_t)T * D);
        m->q.resize((size_t)T * m->qc);
        m->att.resize((size_t)T * m->qc);
        m->xmid.resize((size_t)T * D);
        m->mbuf.resize((size_t)T * m->F_pad);
        m->rinv.resize(T);
        m->xrows.resize((size_t)kGemvRows * std::max(std::max(D, m->qc), m->F_pad));
        const size_t kv_blocks = (size_t)Hkv * ((T + kKB - 1) / kKB);
        m->kvpk.assign(kv_blocks * ((size_t)kKPan * dh * kMR + (size_t)((dh + kMR - 1) / kMR) * kKB * kMR), 0.f);
    } catch (const std::bad_alloc&) {
        delete m;
        return VLA_ERR_OOM;
    } catch (...) {
        delete m;
        return VLA_ERR_OOM;
    }
    *out = m;
    return VLA_OK;
}

vla_status vla_cpu_model_destroy(vla_cpu_model* m) {
    delete m;
    return VLA_OK;
}

int vla_cpu_model_threads(const vla_cpu_model* m) { return m ? m->pool->size() : -1; }

vla_status vla_cpu_model_info(const vla_cpu_model* m, vla_config* cfg, int* layer_begin, int* layer_end) {
    if (!m) return VLA_ERR_INVALID_ARG;
    if (cfg) *cfg = m->cfg;
    if (layer_begin) *layer_begin = m->lb;
    if (layer_end) *layer_end = m->le;
    return VLA_OK;
}

vla_status vla_cpu_kv_create(vla_cpu_model* m, int layer_begin, int layer_end, int max_ctx, vla_cpu_kv** out) {
    if (!out) return VLA_ERR_INVALID_ARG;
    *out = nullptr;
    if (!m) return VLA_ERR_INVALID_ARG;
    if (layer_begin < m->lb || layer_end > m->le || layer_end <= layer_begin) return VLA_ERR_RANGE;
    if (max_ctx < 1 || max_ctx > m->cfg.max_ctx) return VLA_ERR_SHAPE;
    vla_cpu_kv* kv = new (std::nothrow) vla_cpu_kv();
    if (!kv) return VLA_ERR_OOM;
    try {
        kv->m = m;
        kv->lb = layer_begin;
        kv->le = layer_end;
        kv->max_ctx = max_ctx;
        kv->plane = (size_t)m->cfg.n_kv_heads * max_ctx * m->cfg.head_dim;
        kv->data.assign(kv->plane * 2 * (layer_end - layer_begin), 0);
        kv->len.assign(layer_end - layer_begin, 0);
    } catch (...) {
        delete kv;
        return VLA_ERR_OOM;
    }
    *out = kv;
    return VLA_OK;
}

vla_status vla_cpu_kv_destroy(vla_cpu_kv* kv) {
    delete kv;
    return VLA_OK;
}

vla_status vla_cpu_kv_reset(vla_cpu_kv* kv) {
    if (!kv) return VLA_ERR_INVALID_ARG;
    std::fill(kv->len.begin(), kv->len.end(), 0);
    return VLA_OK;
}

int vla_cpu_kv_length(const vla_cpu_kv* kv) {
    if (!kv) return -1;
    return *std::min_element(kv->len.begin(), kv->len.end());
}

vla_status vla_cpu_kv_data(const vla_cpu_kv* kv, int layer, void** k_plane, void** v_plane) {
    if (!kv || layer < kv->lb || layer >= kv->le) return VLA_ERR_INVALID_ARG;
    vla_cpu_kv* k = const_cast<vla_cpu_kv*>(kv);
    if (k_plane) *k_plane = k->k_plane(layer);
    if (v_plane) *v_plane = k->v_plane(layer);
    return VLA_OK;
}

vla_status vla_cpu_prefill(vla_cpu_model* m, const void* hidden_in, int n_tokens, int layer_begin, int layer_end,
                           vla_cpu_kv* kv, void* hidden_out) {
    if (!m || !hidden_in || !hidden_out || n_tokens < 0) return VLA_ERR_INVALID_ARG;
    if (layer_begin < m->lb || layer_end > m->le || layer_end < layer_begin) return VLA_ERR_RANGE;
    if (n_tokens > m->cfg.max_ctx) return VLA_ERR_SHAPE;
    if (n_tokens == 0) return VLA_OK;
    const int D = m->cfg.hidden;
    if (layer_begin == layer_end) {
        if (hidden_in != hidden_out) std::memmove(hidden_out, hidden_in, (size_t)n_tokens * D * 2);
        return VLA_OK;
    }
    if (!kv || kv->m != m) return VLA_ERR_INVALID_ARG;
    if (layer_begin < kv->lb || layer_end > kv->le) return VLA_ERR_RANGE;
    std::lock_guard<std::mutex> lk(m->mu);
    const int p0 = kv->len[layer_begin - kv->lb];
    for (int l = layer_begin; l < layer_end; ++l)
        if (kv->len[l - kv->lb] != p0) return VLA_ERR_RANGE;
    if (p0 + n_tokens > kv->max_ctx) return VLA_ERR_KV_FULL;
    const uint16_t* x = static_cast<const uint16_t*>(hidden_in);
    for (int l = layer_begin; l < layer_end; ++l) {
        uint16_t* y = (l == layer_end - 1) ? static_cast<uint16_t*>(hidden_out) : m->h[(l - layer_begin) & 1].data();
        block(m, l, x, n_tokens, p0, kv, y);
        kv->len[l - kv->lb] = p0 + n_tokens;
        x = y;
    }
    return VLA_OK;
}

}  // extern "C"
