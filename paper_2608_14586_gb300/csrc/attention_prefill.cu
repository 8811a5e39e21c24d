// Causal grouped-query attention for multi-token prefill (flash-style, online softmax).
//
// o[i, h] = sum_{j <= pos0 + i} softmax_j(q_ih . k_gj / sqrt(d_h)) v_gj,  g = h / (H / H_kv)
//
// Keys/values are read from the layer's KV cache (positions [0, pos0 + M)), which the QKV
// epilogue has just written for this call, so a prefill can continue an existing context.
//
// CTA = 128 query rows of one head (8 warps x 16 rows); key blocks of 64 are streamed through
// a double-buffered, XOR-swizzled shared-memory ring with cp.async. S = Q K^T and O += P V
// run on bf16 mma.sync.m16n8k16 with fp32 accumulation; the probabilities P stay in registers
// (the S accumulator fragment is re-packed as the A operand of P V). Row max and row sum are
// kept per thread and reduced across the 4-lane quad. Key blocks above the diagonal are
// skipped; only blocks that straddle it are masked. Heavier (later) query tiles start first.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

constexpr int kBM = 128;
constexpr int kBN = 64;
constexpr int kWarps = 8;

// byte offset of element (row, col) in a [rows][DH] bf16 tile whose 16-byte chunks are
// XOR-swizzled with (row & 7)
template <int DH>
VLA_DEV uint32_t swz(int row, int col) {
    return (uint32_t)(row * DH * 2 + ((((col >> 3) ^ (row & 7))) << 4) + ((col & 7) << 1));
}

VLA_DEV void cp_async16(uint32_t smem_addr, const void* gptr, bool valid) {
    const int src_bytes = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr), "l"(gptr), "r"(src_bytes)
                 : "memory");
}
VLA_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
VLA_DEV void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

VLA_DEV void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
VLA_DEV void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

VLA_DEV void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int DH>
__global__ void __launch_bounds__(kWarps * 32) attn_prefill_kernel(AttnPrefillParams p) {
    constexpr int KCH = DH / 16;  // 16-wide k chunks of the head dim
    constexpr int DT = DH / 8;    // 8-wide dim tiles of the output
    constexpr uint32_t TILE_Q = kBM * DH * 2;
    constexpr uint32_t TILE_KV = kBN * DH * 2;
    extern __shared__ __align__(128) uint8_t smem[];
    const uint32_t sQ = smem_u32(smem);
    const uint32_t sK0 = sQ + TILE_Q;            // K buffers: sK0, sK0 + TILE_KV
    const uint32_t sV0 = sK0 + 2 * TILE_KV;      // V buffers

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t4 = lane & 3;
    const int num_m = (p.M + kBM - 1) / kBM;
    const int mt = num_m - 1 - (int)blockIdx.x;  // heavy tiles first
    const int h = blockIdx.y;
    const int kvh = h / (p.H / p.Hkv);
    const int m0 = mt * kBM;
    const int ctx = p.pos0 + p.M;                          // valid cache positions
    const int key_end = p.pos0 + min(m0 + kBM, p.M);       // keys needed by this tile
    const int nblocks = (key_end + kBN - 1) / kBN;
    const bf16* kbase = p.kc + (size_t)kvh * p.max_ctx * DH;
    const bf16* vbase = p.vc + (size_t)kvh * p.max_ctx * DH;

    // ---- load Q tile (rows >= M zero-filled) and the first K/V block
    for (int c = tid; c < kBM * DH / 8; c += kWarps * 32) {
        const int r = c / (DH / 8), col = (c % (DH / 8)) * 8;
        const bool ok = (m0 + r) < p.M;
        const bf16* src = p.q + (size_t)(ok ? (m0 + r) : 0) * p.ld_q + h * DH + col;
        cp_async16(sQ + swz<DH>(r, col), src, ok);
    }
    auto load_kv = [&](int blk, int buf) {
        const int k0 = blk * kBN;
        for (int c = tid; c < kBN * DH / 8; c += kWarps * 32) {
            const int r = c / (DH / 8), col = (c % (DH / 8)) * 8;
            const int kp = k0 + r;
            const bool ok = kp < ctx;
            const size_t off = (size_t)(ok ? kp : 0) * DH + col;
            cp_async16(sK0 + buf * TILE_KV + swz<DH>(r, col), kbase + off, ok);
            cp_async16(sV0 + buf * TILE_KV + swz<DH>(r, col), vbase + off, ok);
        }
    };
    load_kv(0, 0);
    cp_async_commit();

    uint32_t qf[KCH][4];
    float o[DT][4];
#pragma unroll
    for (int i = 0; i < DT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY};
    float lrow[2] = {0.f, 0.f};
    const int qrow0 = m0 + warp * 16 + g;                 // this thread's rows: qrow0, qrow0 + 8
    const int qpos0 = p.pos0 + qrow0, qpos1 = qpos0 + 8;
    const int warp_min_pos = p.pos0 + m0 + warp * 16;

    for (int blk = 0; blk < nblocks; ++blk) {
        const int buf = blk & 1;
        cp_async_wait<0>();
        __syncthreads();
        if (blk + 1 < nblocks) load_kv(blk + 1, buf ^ 1);
        cp_async_commit();
        if (blk == 0) {
#pragma unroll
            for (int kc = 0; kc < KCH; ++kc) {
                const int r = warp * 16 + (lane & 15);
                const int col = kc * 16 + (lane >> 4) * 8;
                ldsm_x4(sQ + swz<DH>(r, col), qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3]);
            }
        }
        const int k0 = blk * kBN;
        if (k0 > warp_min_pos + 15) continue;  // whole block above this warp's diagonal

        // ---- S = Q K^T (16 x 64 per warp)
        float s[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
        const uint32_t kt = sK0 + buf * TILE_KV;
#pragma unroll
        for (int kc = 0; kc < KCH; ++kc) {
#pragma unroll
            for (int np = 0; np < 4; ++np) {  // pairs of 8-key tiles
                const int r = np * 16 + (lane & 7) + ((lane >> 4) << 3);
                const int col = kc * 16 + ((lane >> 3) & 1) * 8;
                uint32_t b0, b1, b2, b3;
                ldsm_x4(kt + swz<DH>(r, col), b0, b1, b2, b3);
                mma_bf16(s[2 * np], qf[kc], b0, b1);
                mma_bf16(s[2 * np + 1], qf[kc], b2, b3);
            }
        }
        // ---- scale, causal mask, online softmax
        const bool need_mask = (k0 + kBN - 1 > warp_min_pos) || (k0 + kBN > ctx);
        float bmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                float v = s[nt][e] * p.scale_log2;
                if (need_mask) {
                    const int kp = k0 + nt * 8 + 2 * t4 + (e & 1);
                    const int qp = (e < 2) ? qpos0 : qpos1;
                    if (kp > qp) v = -INFINITY;
                }
                s[nt][e] = v;
                bmax[e >> 1] = fmaxf(bmax[e >> 1], v);
            }
        }
        float corr[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            bmax[r] = fmaxf(bmax[r], __shfl_xor_sync(0xFFFFFFFFu, bmax[r], 1));
            bmax[r] = fmaxf(bmax[r], __shfl_xor_sync(0xFFFFFFFFu, bmax[r], 2));
            const float mnew = fmaxf(mrow[r], bmax[r]);
            corr[r] = (mrow[r] == -INFINITY) ? 0.f : exp2f(mrow[r] - mnew);
            mrow[r] = mnew;
            lrow[r] *= corr[r];
        }
#pragma unroll
        for (int i = 0; i < DT; ++i) {
            o[i][0] *= corr[0];
            o[i][1] *= corr[0];
            o[i][2] *= corr[1];
            o[i][3] *= corr[1];
        }
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float pv = exp2f(s[nt][e] - mrow[e >> 1]);
                s[nt][e] = pv;
                lrow[e >> 1] += pv;
            }
        }
        // ---- O += P V
        const uint32_t vt = sV0 + buf * TILE_KV;
#pragma unroll
        for (int kc = 0; kc < kBN / 16; ++kc) {
            uint32_t pa[4];
            pa[0] = pack_bf16x2(s[2 * kc][0], s[2 * kc][1]);
            pa[1] = pack_bf16x2(s[2 * kc][2], s[2 * kc][3]);
            pa[2] = pack_bf16x2(s[2 * kc + 1][0], s[2 * kc + 1][1]);
            pa[3] = pack_bf16x2(s[2 * kc + 1][2], s[2 * kc + 1][3]);
#pragma unroll
            for (int dp = 0; dp < DT / 2; ++dp) {
                const int r = kc * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
                const int col = dp * 16 + (lane >> 4) * 8;
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vt + swz<DH>(r, col), b0, b1, b2, b3);
                mma_bf16(o[2 * dp], pa, b0, b1);
                mma_bf16(o[2 * dp + 1], pa, b2, b3);
            }
        }
    }
    cp_async_wait<0>();

    // ---- normalise and store
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        lrow[r] += __shfl_xor_sync(0xFFFFFFFFu, lrow[r], 1);
        lrow[r] += __shfl_xor_sync(0xFFFFFFFFu, lrow[r], 2);
    }
    const float inv0 = lrow[0] > 0.f ? 1.f / lrow[0] : 0.f;
    const float inv1 = lrow[1] > 0.f ? 1.f / lrow[1] : 0.f;
#pragma unroll
    for (int i = 0; i < DT; ++i) {
        const int col = h * DH + i * 8 + 2 * t4;
        if (qrow0 < p.M)
            *reinterpret_cast<uint32_t*>(p.out + (size_t)qrow0 * p.ld_out + col) =
                pack_bf16x2(o[i][0] * inv0, o[i][1] * inv0);
        if (qrow0 + 8 < p.M)
            *reinterpret_cast<uint32_t*>(p.out + (size_t)(qrow0 + 8) * p.ld_out + col) =
                pack_bf16x2(o[i][2] * inv1, o[i][3] * inv1);
    }
}

template <int DH>
cudaError_t launch_dh(const AttnPrefillParams& p, cudaStream_t stream) {
    constexpr uint32_t smem = kBM * DH * 2 + 4 * kBN * DH * 2;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(attn_prefill_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    dim3 grid((p.M + kBM - 1) / kBM, p.H);
    attn_prefill_kernel<DH><<<grid, kWarps * 32, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attn_prefill(const AttnPrefillParams& p, cudaStream_t stream) {
    if (p.M <= 0) return cudaSuccess;
    if (p.head_dim == 128) return launch_dh<128>(p, stream);
    if (p.head_dim == 64) return launch_dh<64>(p, stream);
    return cudaErrorInvalidValue;
}

}  // namespace vla
