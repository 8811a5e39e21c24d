// Persistent warp-specialised bf16 GEMM on the 5th-generation tensor cores (tcgen05).
//
//   C[M, N] = A[M, K] * B[N, K]^T, fp32 accumulation in tensor memory (TMEM).
//
// Roles per CTA (192 threads, one CTA per SM):
//   warp 0      one thread issues TMA tile loads (A: 128 x 64, B: BN x 64, 128-byte swizzle)
//               into a STAGES-deep shared-memory ring guarded by full/empty mbarriers;
//   warp 1      allocates 2*BN TMEM columns; one thread issues tcgen05.mma (M=128, N=BN,
//               K=16) and commits each stage back to the producer and each finished tile to
//               the epilogue;
//   warps 2..5  epilogue: each warp reads its 32-lane quarter of the accumulator with
//               tcgen05.ld, applies the fused step and stores bf16 results.
// Two accumulator buffers let the epilogue of tile i overlap the mainloop of tile i+1.
// Tiles are walked M-fastest so CTAs running together share the weight (B) tiles in L2.
//
// Fused epilogues (the block stages of the decoder, see the header of runtime.cu):
//   kEpiQKV     RMSNorm row scale, rotate-half RoPE of q and k (the weights hold each rotation
//               pair in adjacent rows, so any 32-column chunk is whole pairs and tiles of 192
//               columns are possible), q to the query buffer, post-RoPE k and v to the layer's
//               KV cache at positions pos0 + row
//   kEpiResid   residual add (attention output projection, MLP down projection)
//   kEpiSwiGLU  RMSNorm row scale and silu(gate) * up on 128-column interleaved tiles
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;

template <int BN, int EPI>
struct GemmCfg {
    static constexpr uint32_t A_BYTES = kBM * kBK * 2;
    static constexpr uint32_t B_BYTES = BN * kBK * 2;
    static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    // residual epilogue at 256-column tiles: per epilogue warp two 32 x 32 bf16 staging boxes
    // for its TMA stores (224-column tiles keep their fifth stage and store directly)
    static constexpr uint32_t OUT_BYTES = (EPI == kEpiResid && BN == 256) ? 4 * 2 * 2048 : 0;
    static constexpr uint32_t FIXED = 1024 /*align*/ + 1024 /*barriers, staging alignment*/ + OUT_BYTES;
    // as many stages as fit in 227 KB next to the fixed part, at most 6
    static constexpr int STAGES = (232448 - FIXED) / STAGE_BYTES < 6 ? (232448 - FIXED) / STAGE_BYTES : 6;
    static constexpr uint32_t TMEM_COLS = 2 * BN <= 256 ? 256 : 512;  // two accumulators, a power of two
    static constexpr uint32_t OFF_OUT = STAGES * STAGE_BYTES + 1024;  // 1024-aligned
    static constexpr uint32_t SMEM_BYTES = STAGES * STAGE_BYTES + FIXED;
    static constexpr uint32_t IDESC = idesc_bf16_f32(kBM, BN);
};

VLA_DEV float f32(uint32_t u) { return __uint_as_float(u); }

VLA_DEV void store_bf16x32(bf16* dst, const float (&v)[32]) {
    uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        uint4 o;
        o.x = pack_bf16x2(v[i * 8 + 0], v[i * 8 + 1]);
        o.y = pack_bf16x2(v[i * 8 + 2], v[i * 8 + 3]);
        o.z = pack_bf16x2(v[i * 8 + 4], v[i * 8 + 5]);
        o.w = pack_bf16x2(v[i * 8 + 6], v[i * 8 + 7]);
        d[i] = o;
    }
}

// ---------------------------------------------------------------------------------------
// Epilogues. Each thread owns one output row (TMEM lane); all 32 lanes of a warp execute
// every tcgen05.ld; stores are masked per row / column.
// ---------------------------------------------------------------------------------------
// 32 lanes x 32 fp32 columns at each of two TMEM addresses, one wait for both loads
VLA_DEV void tmem_ld32x2(uint32_t ta, uint32_t tb, uint32_t (&a)[32], uint32_t (&b)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%64];\n\t"
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%65];\n\t"
        "tcgen05.wait::ld.sync.aligned;\n"
        : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3]), "=r"(a[4]), "=r"(a[5]), "=r"(a[6]), "=r"(a[7]), "=r"(a[8]), "=r"(a[9]), "=r"(a[10]), "=r"(a[11]), "=r"(a[12]), "=r"(a[13]), "=r"(a[14]), "=r"(a[15]), "=r"(a[16]), "=r"(a[17]), "=r"(a[18]), "=r"(a[19]), "=r"(a[20]), "=r"(a[21]), "=r"(a[22]), "=r"(a[23]), "=r"(a[24]), "=r"(a[25]), "=r"(a[26]), "=r"(a[27]), "=r"(a[28]), "=r"(a[29]), "=r"(a[30]), "=r"(a[31]), "=r"(b[0]), "=r"(b[1]), "=r"(b[2]), "=r"(b[3]), "=r"(b[4]), "=r"(b[5]), "=r"(b[6]), "=r"(b[7]), "=r"(b[8]), "=r"(b[9]), "=r"(b[10]), "=r"(b[11]), "=r"(b[12]), "=r"(b[13]), "=r"(b[14]), "=r"(b[15]), "=r"(b[16]), "=r"(b[17]), "=r"(b[18]), "=r"(b[19]), "=r"(b[20]), "=r"(b[21]), "=r"(b[22]), "=r"(b[23]), "=r"(b[24]), "=r"(b[25]), "=r"(b[26]), "=r"(b[27]), "=r"(b[28]), "=r"(b[29]), "=r"(b[30]), "=r"(b[31])
        : "r"(ta), "r"(tb)
        : "memory");
}

// Per 32-column chunk (each inside one of the q, k, v regions, whose widths are multiples of
// 32): q and k columns hold rotation pairs side by side (columns 2j, 2j+1 of a head = dims j,
// j + dh/2), so a chunk is 16 whole pairs; their rotated values go to dims [i0, i0+16) and
// [i0 + dh/2, i0 + dh/2 + 16). Value columns are in natural order.
// 1/rms of an input row from its 32-column partial sums of squares, added in group order
VLA_DEV float row_rinv(const EpiParams& ep, int row) {
    const float* ps = ep.ss_in + (size_t)row * ep.ss_groups;
    float t = 0.f;
    if ((ep.ss_groups & 3) == 0) {  // batches of eight 16-byte loads, each summed in order
        const float4* p4 = reinterpret_cast<const float4*>(ps);
        const int n4 = ep.ss_groups >> 2;
#pragma unroll 1
        for (int b = 0; b < n4; b += 8) {
            float4 q[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) q[i] = b + i < n4 ? __ldcg(p4 + b + i) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (b + i < n4) {
                    t += q[i].x;
                    t += q[i].y;
                    t += q[i].z;
                    t += q[i].w;
                }
            }
        }
    } else {
        for (int c = 0; c < ep.ss_groups; ++c) t += ps[c];
    }
    return 1.0f / sqrtf(t / (float)ep.norm_dim + ep.eps);
}

template <int BN>
VLA_DEV void epi_plain_resid(uint32_t taddr, int row, int n0, const EpiParams& ep) {
    const bool row_ok = row < ep.M;
    float ss = 0.f;  // ss_width 256: the tile's 256-column partial, its 8 group sums in order
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
        uint32_t r[32];
        tmem_ld32(taddr + c, r);
        const int col = n0 + c;
        if (!row_ok || col >= ep.N) continue;
        float v[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = f32(r[i]);
        bf16* op = ep.out + (size_t)row * ep.ld_out + col;
        if (col + 32 <= ep.N) {
            if (ep.resid) {
                const uint4* rp = reinterpret_cast<const uint4*>(ep.resid + (size_t)row * ep.ld_resid + col);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    uint4 q = rp[i];
                    v[i * 8 + 0] += bf16_lo(q.x);
                    v[i * 8 + 1] += bf16_hi(q.x);
                    v[i * 8 + 2] += bf16_lo(q.y);
                    v[i * 8 + 3] += bf16_hi(q.y);
                    v[i * 8 + 4] += bf16_lo(q.z);
                    v[i * 8 + 5] += bf16_hi(q.z);
                    v[i * 8 + 6] += bf16_lo(q.w);
                    v[i * 8 + 7] += bf16_hi(q.w);
                }
            }
            store_bf16x32(op, v);
            if (ep.out_host) store_bf16x32(ep.out_host + (size_t)row * ep.ld_out + col, v);
            if (ep.ss_out) {  // the group's sum of squares of the stored values, a chain from zero
                float g = 0.f;
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float r = __bfloat162float(__float2bfloat16_rn(v[i]));
                    g = fmaf(r, r, g);
                }
                if (ep.ss_width == 32) ep.ss_out[(size_t)row * ep.ss_groups + (col >> 5)] = g;
                else ss += g;
            }
        } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                if (col + i < ep.N) {
                    float x = v[i];
                    if (ep.resid) x += __bfloat162float(ep.resid[(size_t)row * ep.ld_resid + col + i]);
                    op[i] = __float2bfloat16_rn(x);
                    if (ep.out_host) ep.out_host[(size_t)row * ep.ld_out + col + i] = op[i];
                }
            }
        }
    }
    if (ep.ss_out && ep.ss_width == 256 && row_ok && n0 < ep.N) ep.ss_out[(size_t)row * ep.ss_groups + n0 / 256] = ss;
}

// The same residual epilogue with the stores made by TMA: each 32-column chunk of the warp's
// 32 rows is packed into a 32 x 32 bf16 box in shared memory (64-byte swizzle, so the 16-byte
// writes of the 32 lanes spread over all banks) and one lane stores the box with
// cp.async.bulk.tensor; the box rows past M and columns past N are clipped by the tensor map.
// Chunks go in pairs: one tensor-memory wait for both, both boxes of the warp filled, one
// proxy fence, two stores in one bulk group (the previous pair's group has read its boxes
// before they are refilled). Needs N a multiple of 32, an even chunk count and no host copy
// (out_host). Row statistics as epi_plain_resid.
template <int BN>
VLA_DEV void epi_resid_tma(uint32_t taddr, int row, int row0, int n0, const EpiParams& ep, const CUtensorMap* tm_out,
                           uint8_t* stage, uint32_t& nstore, int lane) {
    constexpr int NC = BN / 32;
    static_assert(NC % 2 == 0, "chunk pairs");
    const bool row_ok = row < ep.M;
    const bool has_res = row_ok && ep.resid != nullptr;
    const uint4* rrow = has_res ? reinterpret_cast<const uint4*>(ep.resid + (size_t)row * ep.ld_resid + n0) : nullptr;
    // the residual chunks are requested one pair ahead of their use, so their latency overlaps
    // the tensor-memory reads and the stores of the pair before
    uint4 res[4][4];
    auto fetch = [&](int c) {
        if (has_res && n0 + 32 * c < ep.N) {
#pragma unroll
            for (int i = 0; i < 4; ++i) res[c % 4][i] = rrow[4 * c + i];
        }
    };
    fetch(0);
    fetch(1);
    float ss = 0.f;
#pragma unroll
    for (int c = 0; c < NC; c += 2) {
        if (c + 2 < NC) {
            fetch(c + 2);
            fetch(c + 3);
        }
        uint32_t r2[2][32];
        tmem_ld32x2(taddr + 32 * c, taddr + 32 * (c + 1), r2[0], r2[1]);
        if (n0 + 32 * c >= ep.N) continue;  // uniform over the warp (then so is the second chunk)
        if (lane == 0) bulk_wait_group_read<0>();  // the previous pair's stores have read both boxes
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const int col = n0 + 32 * (c + j);
            if (col >= ep.N) continue;
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = f32(r2[j][i]);
            if (has_res) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint4 q = res[(c + j) % 4][i];
                    v[i * 8 + 0] += bf16_lo(q.x);
                    v[i * 8 + 1] += bf16_hi(q.x);
                    v[i * 8 + 2] += bf16_lo(q.y);
                    v[i * 8 + 3] += bf16_hi(q.y);
                    v[i * 8 + 4] += bf16_lo(q.z);
                    v[i * 8 + 5] += bf16_hi(q.z);
                    v[i * 8 + 6] += bf16_lo(q.w);
                    v[i * 8 + 7] += bf16_hi(q.w);
                }
            }
            if (ep.ss_out && row_ok) {  // the group's sum of squares of the stored values, a chain from zero
                float g = 0.f;
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float rr = __bfloat162float(__float2bfloat16_rn(v[i]));
                    g = fmaf(rr, rr, g);
                }
                if (ep.ss_width == 32) ep.ss_out[(size_t)row * ep.ss_groups + (col >> 5)] = g;
                else ss += g;
            }
            uint8_t* box = stage + (uint32_t)j * 2048u;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 o = make_uint4(pack_bf16x2(v[8 * q + 0], v[8 * q + 1]), pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                                           pack_bf16x2(v[8 * q + 4], v[8 * q + 5]), pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
                *reinterpret_cast<uint4*>(box + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4)) = o;
            }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            tma_store_2d(tm_out, stage, n0 + 32 * c, row0);
            if (n0 + 32 * (c + 1) < ep.N) tma_store_2d(tm_out, stage + 2048u, n0 + 32 * (c + 1), row0);
            bulk_commit_group();
        }
        nstore += 2;
    }
    if (ep.ss_out && ep.ss_width == 256 && row_ok && n0 < ep.N) ep.ss_out[(size_t)row * ep.ss_groups + n0 / 256] = ss;
}

VLA_DEV void store_bf16x16(bf16* dst, const float* v) {
    uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        uint4 o;
        o.x = pack_bf16x2(v[i * 8 + 0], v[i * 8 + 1]);
        o.y = pack_bf16x2(v[i * 8 + 2], v[i * 8 + 3]);
        o.z = pack_bf16x2(v[i * 8 + 4], v[i * 8 + 5]);
        o.w = pack_bf16x2(v[i * 8 + 6], v[i * 8 + 7]);
        d[i] = o;
    }
}

// One 32-column chunk at output column `col` of the QKV epilogue; cs: the chunk's 16 (cos, sin)
// pairs, two per float4 (q and k chunks only).
VLA_DEV void qkv_chunk(const uint32_t (&r)[32], int col, const float4 (&cs)[8], float s, int row, int pos,
                       const EpiParams& ep) {
    const int dh = ep.head_dim;
    if (col >= ep.q_cols + ep.kv_cols) {
        const int n = col - ep.q_cols - ep.kv_cols;
        const int g = n / dh, d = n % dh;
        float v[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = f32(r[i]) * s;
        store_bf16x32(ep.vcache + ((size_t)g * ep.max_ctx + pos) * dh + d, v);
        return;
    }
    const bool is_q = col < ep.q_cols;
    const int n = is_q ? col : col - ep.q_cols;
    const int head = n / dh, i0 = (n % dh) >> 1;
    float va[16], vb[16];
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
        const float4 c4 = cs[i >> 1];
        const float a0 = f32(r[2 * i]) * s, b0 = f32(r[2 * i + 1]) * s;
        const float a1 = f32(r[2 * i + 2]) * s, b1 = f32(r[2 * i + 3]) * s;
        va[i] = a0 * c4.x - b0 * c4.y;
        vb[i] = b0 * c4.x + a0 * c4.y;
        va[i + 1] = a1 * c4.z - b1 * c4.w;
        vb[i + 1] = b1 * c4.z + a1 * c4.w;
    }
    bf16* dst = is_q ? ep.out + (size_t)row * ep.ld_out + (size_t)head * dh
                     : ep.kcache + ((size_t)head * ep.max_ctx + pos) * dh;
    store_bf16x16(dst + i0, va);
    store_bf16x16(dst + i0 + (dh >> 1), vb);
}

// Per 32-column chunk (each inside one of the q, k, v regions, whose widths are multiples of
// 32): q and k columns hold rotation pairs side by side (columns 2j, 2j+1 of a head = dims j,
// j + dh/2), so a chunk is 16 whole pairs; their rotated values go to dims [i0, i0+16) and
// [i0 + dh/2, i0 + dh/2 + 16). Value columns are in natural order. With 256-column tiles and
// d_h = 128 the chunks c and c + 4 are the same dims of two heads: they are read from tensor
// memory with one wait and share one load of the row's (cos, sin) pairs.
template <int BN>
VLA_DEV void epi_qkv(uint32_t taddr, int row, int n0, const EpiParams& ep) {
    const bool row_ok = row < ep.M;
    const float s = row_ok ? row_rinv(ep, row) : 0.f;
    const int pos = ep.pos0 + row;
    const int dh = ep.head_dim;
    const int half = dh >> 1;
    const int rope_cols = ep.q_cols + ep.kv_cols;  // columns [0, rope_cols) are rotated
    const float2* rope = ep.rope + (size_t)(row_ok ? pos : 0) * half;
    if (BN == 256 && dh == 128) {
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
            const int col = n0 + 32 * c;  // and col + 128: the same dims of the next head
            const int i0 = (col % dh) >> 1;
            float4 cs[8];
            if (row_ok && (col < rope_cols || col + 128 < rope_cols)) {
#pragma unroll
                for (int i = 0; i < 8; ++i) cs[i] = __ldg(reinterpret_cast<const float4*>(rope + i0 + 2 * i));
            }
            uint32_t ra[32], rb[32];
            tmem_ld32x2(taddr + 32 * c, taddr + 32 * c + 128, ra, rb);
            if (!row_ok) continue;
            if (col < ep.N) qkv_chunk(ra, col, cs, s, row, pos, ep);
            if (col + 128 < ep.N) qkv_chunk(rb, col + 128, cs, s, row, pos, ep);
        }
        return;
    }
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
        const int col = n0 + c;
        float4 cs[8];
        if (row_ok && col < rope_cols) {
            const int i0 = (col % dh) >> 1;
#pragma unroll
            for (int i = 0; i < 8; ++i) cs[i] = __ldg(reinterpret_cast<const float4*>(rope + i0 + 2 * i));
        }
        uint32_t r[32];
        tmem_ld32(taddr + c, r);
        if (!row_ok || col >= ep.N) continue;
        qkv_chunk(r, col, cs, s, row, pos, ep);
    }
}

// SiLU(g) * u with g, u the gate and up accumulators scaled by 1/rms. The division is the
// fast reciprocal form (__fdividef: within 2 ulp of fp32, far below the bf16 rounding of the
// stored value; for g below about -87 the denominator overflows and the product is 0, the
// function's limit).
template <int BN>
VLA_DEV void epi_swiglu(uint32_t taddr, int row, int n0, const EpiParams& ep) {
    constexpr int HALF = BN / 2;
    const bool row_ok = row < ep.M;
    const float s = row_ok ? row_rinv(ep, row) : 0.f;
    const int f0 = (n0 / BN) * HALF;
#pragma unroll 1
    for (int c = 0; c < HALF; c += 32) {
        uint32_t rg[32], ru[32];
        tmem_ld32x2(taddr + c, taddr + HALF + c, rg, ru);
        if (!row_ok) continue;
        float v[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            const float g = f32(rg[i]) * s;
            const float u = f32(ru[i]) * s;
            v[i] = __fdividef(g, 1.0f + __expf(-g)) * u;
        }
        store_bf16x32(ep.out + (size_t)row * ep.ld_out + f0 + c, v);
    }
}

// Bounded wait that also gives up when another role has aborted.
VLA_DEV bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort_flag, long long budget) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (*abort_flag) return false;
        if (clock64() - t0 > budget) return false;
    }
    return true;
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_bf16_tcgen05(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmOut, int M, int N, int K, EpiParams ep) {
    using C = GemmCfg<BN, EPI>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    __shared__ volatile int s_abort;

    const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * C::A_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
    uint64_t* full = bars;
    uint64_t* empty = bars + STAGES;
    uint64_t* tfull = bars + 2 * STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int num_m = (M + kBM - 1) / kBM;
    const int num_n = (N + BN - 1) / BN;
    const int num_tiles = num_m * num_n;
    const int num_kb = (K + kBK - 1) / kBK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 128);
        }
        mbar_init(mma_done, 1);
        s_abort = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer ----------------
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0, issued_phase = 0;  // per-stage bit masks of loads in flight
            bool ok = true;
            // The weight tiles (B) do not depend on the previous kernel: under programmatic
            // dependent launch the first ring's worth of them is requested before the wait,
            // while the previous kernel drains. Activations (A) only after it.
            const int pre = (blockIdx.x < num_tiles) ? min(STAGES, num_kb) : 0;
            for (int kb = 0; kb < pre; ++kb) {
                if (kb == ep.stall_kb) continue;  // failure-detection test: never armed (below)
                mbar_arrive_expect_tx(&full[kb], C::STAGE_BYTES);
                tma_load_2d(sB + kb * C::B_BYTES, &tmB, &full[kb], kb * kBK, (blockIdx.x / num_m) * BN);
                issued |= 1u << kb;
            }
            pdl_wait();
            pdl_trigger();
            bool first = true;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
                const int m0 = (tile % num_m) * kBM;
                const int n0 = (tile / num_m) * BN;
                for (int kb = 0; kb < num_kb; ++kb) {
                    if (!wait_or_abort(&empty[stage], phase ^ 1u, &s_abort, ep.wait_budget)) {
                        ok = false;
                        break;
                    }
                    const bool withhold = first && kb == ep.stall_kb;
                    if (withhold) {
                        // failure-detection test: this stage is never armed or loaded, so the
                        // MMA's wait on it runs out and the launch winds down
                    } else if (first && kb < pre) {  // B of this stage is already in flight
                        tma_load_2d(sA + stage * C::A_BYTES, &tmA, &full[stage], kb * kBK, m0);
                    } else {
                        mbar_arrive_expect_tx(&full[stage], C::STAGE_BYTES);
                        tma_load_2d(sA + stage * C::A_BYTES, &tmA, &full[stage], kb * kBK, m0);
                        tma_load_2d(sB + stage * C::B_BYTES, &tmB, &full[stage], kb * kBK, n0);
                    }
                    if (!withhold) {
                        issued |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                    }
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                first = false;
            }
            if (!ok) {
                s_abort = 1;
                set_status(ep.status, kDevTimeout);
            }
            if (!ok || ep.stall_kb >= 0) {
                // let every copy already issued land before the CTA can exit (with a withheld
                // stage the MMA stops early and may leave later copies unconsumed)
                for (int s = 0; s < STAGES; ++s)
                    if (issued & (1u << s)) mbar_wait(&full[s], (issued_phase >> s) & 1u, ep.wait_budget);
            }
        }
    } else if (warp == 1) {
        pdl_wait();
        pdl_trigger();
        // the layer's KV length advances with the keys this kernel writes (read only by later
        // launches: decode takes the new token's position from it)
        if (EPI == kEpiQKV && ep.len_out && blockIdx.x == 0 && lane == 0) *ep.len_out = ep.len_value;
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int it = 0;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++it) {
                const int acc = it & 1;
                const uint32_t acc_phase = (it >> 1) & 1;
                if (!wait_or_abort(&tempty[acc], acc_phase ^ 1u, &s_abort, ep.wait_budget)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + acc * BN;
                for (int kb = 0; kb < num_kb; ++kb) {
                    if (!wait_or_abort(&full[stage], phase, &s_abort, ep.wait_budget)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t a_desc = sw128_kmajor_desc(smem_u32(sA + stage * C::A_BYTES));
                    const uint64_t b_desc = sw128_kmajor_desc(smem_u32(sB + stage * C::B_BYTES));
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        // advance 16 bf16 (32 B) along K inside the 128-byte swizzle row
                        umma_bf16_ss(d_tmem, a_desc + 2 * k, b_desc + 2 * k, C::IDESC, (kb | k) != 0);
                    }
                    umma_commit(&empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (ok) umma_commit(&tfull[acc]);
            }
            if (!ok) {
                s_abort = 1;
                set_status(ep.status, kDevTimeout);
            }
            // all MMAs issued by this thread retire before TMEM can be released
            umma_commit(mma_done);
            mbar_wait(mma_done, 0, ep.wait_budget);
        }
    } else {
        // ---------------- epilogue (warps 2..5) ----------------
        pdl_wait();  // the epilogue reads 1/rms and the residual written by earlier kernels
        pdl_trigger();
        const int quarter = warp & 3;  // TMEM lanes [32*quarter, 32*quarter + 32)
        int it = 0;
        uint32_t nstore = 0;  // TMA stores of this warp (residual epilogue through TMA)
        uint8_t* stage_out = smem + C::OFF_OUT + (uint32_t)(warp - 2) * 4096u;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++it) {
            const int acc = it & 1;
            const uint32_t acc_phase = (it >> 1) & 1;
            const bool ok = wait_or_abort(&tfull[acc], acc_phase, &s_abort, ep.wait_budget);
            __syncwarp();
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                s_abort = 1;
                set_status(ep.status, kDevTimeout);
                break;
            }
            tc_fence_after();
            const int m0 = (tile % num_m) * kBM;
            const int n0 = (tile / num_m) * BN;
            const int row = m0 + quarter * 32 + lane;
            const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
            if constexpr (EPI == kEpiQKV) {
                epi_qkv<BN>(taddr, row, n0, ep);
            } else if constexpr (EPI == kEpiSwiGLU) {
                epi_swiglu<BN>(taddr, row, n0, ep);
            } else {
                if constexpr (C::OUT_BYTES != 0) {  // 256-column tiles: a staging box pair per warp
                    if (ep.tma_out)
                        epi_resid_tma<BN>(taddr, row, m0 + quarter * 32, n0, ep, &tmOut, stage_out, nstore, lane);
                    else
                        epi_plain_resid<BN>(taddr, row, n0, ep);
                } else {
                    epi_plain_resid<BN>(taddr, row, n0, ep);
                }
            }
            tc_fence_before();
            mbar_arrive(&tempty[acc]);
        }
        // the TMA stores of this warp are complete (their writes performed) before the CTA exits
        if (C::OUT_BYTES && ep.tma_out && lane == 0) bulk_wait_group_all();
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

template <int BN, int EPI>
cudaError_t launch_one(const CUtensorMap& A, const CUtensorMap& B, const CUtensorMap& Out, int M, int N, int K,
                       const EpiParams& ep, int num_sms, cudaStream_t stream, bool pdl) {
    using C = GemmCfg<BN, EPI>;
    static bool attr_set = false;
    auto kern = gemm_bf16_tcgen05<BN, EPI>;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int tiles = ((M + kBM - 1) / kBM) * ((N + BN - 1) / BN);
    const int grid = tiles < num_sms ? tiles : num_sms;
    return launch_ex(kern, dim3(grid), dim3(kThreads), C::SMEM_BYTES, stream, pdl, A, B, Out, M, N, K, ep);
}

}  // namespace

cudaError_t launch_gemm(int mode, int bn, const CUtensorMap& A, const CUtensorMap& B, int M, int N, int K,
                        const EpiParams& ep_in, int num_sms, cudaStream_t stream, bool pdl, const CUtensorMap* out_map) {
    if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
    EpiParams ep = ep_in;
    // residual / plain epilogue through TMA stores when an output map is given (no host copy)
    ep.tma_out =
        (out_map && bn == 256 && (mode == kEpiResid || mode == kEpiPlain) && !ep.out_host && N % 32 == 0) ? 1 : 0;
    const CUtensorMap& O = ep.tma_out ? *out_map : A;  // unused unless tma_out
    if (bn == 256) {
        switch (mode) {
            case kEpiPlain:
            case kEpiResid: return launch_one<256, kEpiResid>(A, B, O, M, N, K, ep, num_sms, stream, pdl);
            case kEpiQKV: return launch_one<256, kEpiQKV>(A, B, O, M, N, K, ep, num_sms, stream, pdl);
            case kEpiSwiGLU: return launch_one<256, kEpiSwiGLU>(A, B, O, M, N, K, ep, num_sms, stream, pdl);
        }
    } else if (bn == 224) {
        if (ep.ss_out && ep.ss_width != 32) return cudaErrorInvalidValue;  // partials would straddle tiles
        if (mode == kEpiResid || mode == kEpiPlain)
            return launch_one<224, kEpiResid>(A, B, O, M, N, K, ep, num_sms, stream, pdl);
    } else if (bn == 192) {
        if (mode == kEpiQKV) return launch_one<192, kEpiQKV>(A, B, O, M, N, K, ep, num_sms, stream, pdl);
    }
    return cudaErrorInvalidValue;
}

}  // namespace vla
