// Single-token (decode) attention on the 5th-generation tensor cores, head_dim 128.
//
// One thread-block cluster of `cs` CTAs per (sequence, KV head g); CTA rank r owns the contiguous key range
// [r*ceil(ctx/cs), ...) of the context (the attention stage of a block, Sec. IV-B, at one query
// position, split over keys). Per CTA, for the G query heads of the GQA group:
//   1. First thing, the lanes of warp 0 issue TMA copies of the range's K and V rows that
//      predate this step (32-row boxes, 128-byte swizzle) into shared memory sized to the
//      range; after griddepcontrol.wait, Q and the new token's K and V rows are read while
//      tensor memory is allocated, then written into shared memory (the new rows over their
//      slots).
//   2. S^T = K Q^T on tcgen05 per 128-key tile (M = 128 keys, N = 16 >= G heads, K = d_h),
//      fp32 in TMEM; lane 0 of warp t issues tile t, so the tiles' MMAs go out in parallel.
//   3. One thread per key row reads its G scores, the CTA takes the per-head max and sum of
//      exp2(s * log2(e)/sqrt(d_h) - max), and writes P^T (bf16, 128-byte-swizzled K-major).
//   4. O^T partial of tile t = V_t^T P_t^T on tcgen05 (M = d_h, N = 16, K = the tile's keys;
//      V^T read MN-major in place), again one issuing thread per tile; the partials are added
//      in tile order when they are read.
//   5. Each CTA stores its (max, sum, unnormalised O) through distributed shared memory into
//      the inbox of the rank that merges each element slice; after one cluster barrier CTA r
//      merges output elements [r*G*d_h/cs, (r+1)*G*d_h/cs) from its inbox in fixed rank order
//      and writes them as bf16.
// Every mbarrier wait is bounded; a timeout sets the status word and the kernel winds down.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

constexpr int kDH = 128;
constexpr int kThreads = 128;
constexpr int kBoxRows = 32;
constexpr uint32_t kChunk = 128u * 128u;            // [128 rows][64 bf16] per d_h half
constexpr uint32_t kTileBytes = 2u * kChunk;        // 128 keys x 128 d_h
constexpr int kMaxRows = 384;                       // keys per CTA (3 tiles)
constexpr uint32_t kQBytes = 2u * 16u * 128u;       // [16 rows][128] as two halves of 64
constexpr uint32_t kPTileBytes = 2u * 16u * 128u;   // [16 heads][128 keys] as two halves of 64
constexpr uint32_t kBoxBytes = kBoxRows * 128u;     // one [32 rows][64] box
constexpr uint32_t kTmemCols = 128;  // S^T of tile t at [16t, 16t+16), its O^T partial at [64+16t, ...)
constexpr uint32_t kOCol = 64;
constexpr int kMaxCs = 16;

// byte offset of (row, 16-byte chunk j) inside a 128-byte-swizzled tile of 128-byte rows
VLA_DEV uint32_t sw128_off(int row, int j) { return (uint32_t)row * 128u + ((uint32_t)(j ^ (row & 7)) << 4); }

// Shared memory for `rows` keys per CTA (a multiple of 32): K and V as tiles of 128 keys, the
// last tile holding only the remaining rows; tile t's two d_h halves are rows_t * 128 bytes
// apart. The S MMA of a partial tile reads all 128 rows of each half window, past the tile's
// own rows into the buffers that follow (never past the allocation, since rows_t >= 32);
// those keys are masked, and the O MMA reads only the 16-key steps that hold keys.
struct Smem {
    uint32_t off_k, off_v, off_q, off_p, total;
};

__host__ __device__ inline Smem smem_layout(int rows) {
    Smem s;
    s.off_k = 0;
    s.off_v = (uint32_t)rows * 256u;
    s.off_q = 2u * s.off_v;
    s.off_p = s.off_q + kQBytes;
    s.total = s.off_p + (uint32_t)((rows + 127) / 128) * kPTileBytes + 1024;  // + alignment slack
    return s;
}

// byte offset of d_h half `half` of tile t for `rows` allocated keys
__host__ __device__ inline uint32_t half_off(int rows, int t, int half) {
    const int rt = min(128, rows - 128 * t);
    return (uint32_t)t * kTileBytes + (uint32_t)half * (uint32_t)rt * 128u;
}

template <int G>
__global__ void __launch_bounds__(kThreads, 1)
    attn_decode_tc_kernel(const __grid_constant__ DecKVMaps maps, const __grid_constant__ AttnDecTcParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t bar_kv, bar_s[3], bar_o[3];  // K/V landed; per 128-key tile: S^T, O^T done
    __shared__ uint32_t tmem_slot;
    __shared__ float red_m[4][G], red_l[4][G];
    // merge inbox: from each rank of the cluster, its (max, sum) per head and its unnormalised
    // output over this CTA's element slice
    __shared__ float rx_m[kMaxCs][G], rx_l[kMaxCs][G];
    __shared__ float rx_o[kMaxCs][G * kDH / 8];
    __shared__ int s_ok;
    const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    const Smem L = smem_layout(p.rows);
    uint8_t* sK = smem + L.off_k;
    uint8_t* sV = smem + L.off_v;
    uint8_t* sQ = smem + L.off_q;
    uint8_t* sP = smem + L.off_p;
    const int rank = blockIdx.x, kvh = blockIdx.y, seq = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const CUtensorMap* tmK = &maps.k[seq];
    const CUtensorMap* tmV = &maps.v[seq];
    const bf16* kc = p.kc[seq];
    const bf16* vc = p.vc[seq];
    const float* q = p.q + (size_t)seq * p.H * kDH;

    // d_len was last written by an earlier step (complete before this one started)
    const int ctx = *p.d_len[seq] + 1;
    const int per = (ctx + p.cs - 1) / p.cs;
    const int kb = rank * per;
    const int nk = max(0, min(min(ctx, kb + per) - kb, p.rows));
    const int nbox = (nk + kBoxRows - 1) / kBoxRows;
    const int new_row = ctx - 1 - kb;  // slot of the token written by the QKV kernel

    // warp 0 requests the range's K and V rows that predate this step first: the copy is the
    // longest part of the kernel when its CTAs start only as the QKV kernel's CTAs leave
    if (warp == 0) {
        if (lane == 0) {
            mbar_init(&bar_kv, 1);
            for (int t = 0; t < 3; ++t) {
                mbar_init(&bar_s[t], 1);
                mbar_init(&bar_o[t], 1);
            }
            fence_barrier_init();
            s_ok = 1;
            mbar_arrive_expect_tx(&bar_kv, (uint32_t)nbox * 4u * kBoxBytes);
        }
        __syncwarp();
        // lane l issues the copies (box b, d_h half c) = l, l + 32, ...
        for (int i = lane; i < nbox * 2; i += 32) {
            const int b = i >> 1, c = i & 1;
            const int y = kb + b * kBoxRows;
            const uint32_t dst = half_off(p.rows, b >> 2, c) + (uint32_t)(b & 3) * kBoxBytes;
            tma_load_3d(sK + dst, tmK, &bar_kv, c * 64, y, kvh);
            tma_load_3d(sV + dst, tmV, &bar_kv, c * 64, y, kvh);
        }
    }
    pdl_wait();
    pdl_trigger();

    // global reads of what the QKV kernel wrote (Q and the new token's K and V rows) go out
    // first; tensor memory and the zeroing of the Q and P tiles overlap their latency
    const bool has_new = new_row >= 0 && new_row < nk && tid < 32;
    const int nh = tid >> 4, nj = (tid >> 1) & 7, nwhich = tid & 1;  // 2 halves x 8 chunks x {K, V}
    uint4 new_chunk = make_uint4(0u, 0u, 0u, 0u);
    if (has_new)
        new_chunk = __ldcg(reinterpret_cast<const uint4*>((nwhich ? vc : kc) +
                                                          ((size_t)kvh * p.max_ctx + (ctx - 1)) * kDH + nh * 64 + nj * 8));
    const int qh = tid >> 4, qj = tid & 15;  // Q: head, 16-byte chunk of 8 dims (G * 16 <= kThreads)
    float4 qa = make_float4(0.f, 0.f, 0.f, 0.f), qb = qa;
    if (tid < G * 16) {
        const float4* src = reinterpret_cast<const float4*>(q + (size_t)(kvh * G + qh) * kDH + qj * 8);
        qa = __ldcg(src);
        qb = __ldcg(src + 1);
    }
    if (warp == 0) {  // allocates and (at exit) frees the tensor memory
        tmem_alloc(&tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    // zero Q rows >= G and the P^T tiles (rows >= G stay zero; rows < G are rewritten)
    for (uint32_t i = tid; i < (L.total - 1024 - L.off_q) / 16; i += kThreads)
        reinterpret_cast<uint4*>(sQ)[i] = make_uint4(0u, 0u, 0u, 0u);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    cluster_arrive_relaxed();  // waited on before the first push into another CTA's inbox
    const uint32_t tmem = tmem_slot;
    // Q (post-RoPE, fp32) -> bf16 rows [0, G) of the swizzled K-major tile
    if (tid < G * 16)
        *reinterpret_cast<uint4*>(sQ + (qj >> 3) * (16 * 128) + sw128_off(qh, qj & 7)) =
            make_uint4(pack_bf16x2(qa.x, qa.y), pack_bf16x2(qa.z, qa.w), pack_bf16x2(qb.x, qb.y),
                       pack_bf16x2(qb.z, qb.w));
    if (!mbar_wait(&bar_kv, 0)) s_ok = 0;
    // the new token's K and V rows over their (stale) slots; V rows past the range -> 0 so that
    // zero probabilities never meet non-finite values
    if (has_new)
        *reinterpret_cast<uint4*>((nwhich ? sV : sK) + half_off(p.rows, new_row >> 7, nh) +
                                  sw128_off(new_row & 127, nj)) = new_chunk;
    const int nt = (nk + 127) >> 7;
    const int zero_end = min(p.rows, (nk + 31) & ~31);  // rows the O MMA may read
    for (int i = nk * 16 + tid; i < zero_end * 16; i += kThreads) {  // (row, half, chunk) triples
        const int row = i >> 4, half = (i >> 3) & 1, j = i & 7;
        *reinterpret_cast<uint4*>(sV + half_off(p.rows, row >> 7, half) + sw128_off(row & 127, j)) =
            make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();
    __syncthreads();
    const bool run = s_ok && nk > 0;  // CTA-uniform

    // S^T = K Q^T of 128-key tile t into TMEM columns [16t, 16t + 16), issued by lane 0 of
    // warp t (the tiles' MMAs go out in parallel)
    if (run && lane == 0 && warp < nt) {
        const int t = warp;
        tc_fence_after();
        constexpr uint32_t idesc = idesc_bf16_f32(128, 16);
        const uint32_t qt = smem_u32(sQ);
#pragma unroll
        for (int kk = 0; kk < kDH / 16; ++kk) {
            const uint64_t ad = sw128_kmajor_desc(smem_u32(sK + half_off(p.rows, t, kk >> 2))) + 2 * (kk & 3);
            const uint64_t bd = sw128_kmajor_desc(qt + (kk >> 2) * (16 * 128)) + 2 * (kk & 3);
            umma_bf16_ss(tmem + t * 16, ad, bd, idesc, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bar_s[t]);
    }
    float s[3][G];
    float m_loc[G], l_loc[G];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) m_loc[hh] = -INFINITY, l_loc[hh] = 0.f;
    if (run) {
        for (int t = 0; t < nt; ++t)
            if (!mbar_wait(&bar_s[t], 0)) s_ok = 0;
        tc_fence_after();
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
        for (int t = 0; t < 3; ++t) {
            if (t < nt) {
                uint32_t r[16];
                tmem_ld16(trow + t * 16, r);
                const bool valid = t * 128 + warp * 32 + lane < nk;
#pragma unroll
                for (int hh = 0; hh < G; ++hh) {
                    s[t][hh] = valid ? __uint_as_float(r[hh]) * p.scale_log2 : -INFINITY;
                    m_loc[hh] = fmaxf(m_loc[hh], s[t][hh]);
                }
            } else {
#pragma unroll
                for (int hh = 0; hh < G; ++hh) s[t][hh] = -INFINITY;
            }
        }
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            float v = m_loc[hh];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
            if (lane == 0) red_m[warp][hh] = v;
        }
    }
    __syncthreads();
    if (run) {
#pragma unroll
        for (int hh = 0; hh < G; ++hh)
            m_loc[hh] = fmaxf(fmaxf(red_m[0][hh], red_m[1][hh]), fmaxf(red_m[2][hh], red_m[3][hh]));
        // P^T[hh][key] = exp2(s - max) as bf16, swizzled K-major rows of 128 keys per tile
        const int ki = warp * 32 + lane;  // key within the tile
#pragma unroll
        for (int t = 0; t < 3; ++t) {
            if (t < nt) {
                uint8_t* pt = sP + t * kPTileBytes + (ki >> 6) * (16 * 128);
#pragma unroll
                for (int hh = 0; hh < G; ++hh) {
                    const float pe = s[t][hh] == -INFINITY ? 0.f : ex2_approx(s[t][hh] - m_loc[hh]);
                    const bf16 pb = __float2bfloat16_rn(pe);
                    l_loc[hh] += pe;
                    *reinterpret_cast<bf16*>(pt + sw128_off(hh, (ki & 63) >> 3) + (ki & 7) * 2) = pb;
                }
            }
        }
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            float v = l_loc[hh];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
            if (lane == 0) red_l[warp][hh] = v;
        }
        fence_proxy_async_smem();
        tc_fence_before();
    }
    __syncthreads();
    // O^T partial of tile t = V_t^T P_t^T into TMEM columns [64 + 16t, ...), issued by lane 0 of
    // warp t: A = V tile read MN-major (M = d_h), B = P^T; the partials are added at readout
    if (run && lane == 0 && warp < nt) {
        const int t = warp;
        tc_fence_after();
        constexpr uint32_t idesc = idesc_bf16_f32(128, 16) | (1u << 15);
        const uint32_t vt = smem_u32(sV + half_off(p.rows, t, 0));
        const uint32_t vstride = half_off(p.rows, t, 1) - half_off(p.rows, t, 0);
        const uint32_t pt = smem_u32(sP + t * kPTileBytes);
        const int steps = (min(128, nk - 128 * t) + 15) >> 4;  // 16-key steps holding keys
        for (int kk = 0; kk < steps; ++kk) {
            const uint64_t ad = sw128_mnmajor_desc(vt + kk * 16 * 128, vstride);
            const uint64_t bd = sw128_kmajor_desc(pt + (kk >> 2) * (16 * 128)) + 2 * (kk & 3);
            umma_bf16_ss(tmem + kOCol + t * 16, ad, bd, idesc, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bar_o[t]);
    }
    // Push this CTA's partial state into the inbox of the rank that merges each element slice
    // (every rank gets the per-head max and sum; those are complete since the barrier before
    // the O MMA, so they go out while it runs), then one cluster barrier (release / acquire)
    // makes every inbox complete; nothing reads another CTA's shared memory after it, so no
    // second barrier is needed before exit.
    cluster_wait();
    for (int i = tid; i < p.cs * G; i += kThreads) {
        const int q = i / G, hh = i % G;
        float mv = -INFINITY, lv = 0.f;
        if (run) {
            mv = fmaxf(fmaxf(red_m[0][hh], red_m[1][hh]), fmaxf(red_m[2][hh], red_m[3][hh]));
            lv = red_l[0][hh] + red_l[1][hh] + red_l[2][hh] + red_l[3][hh];
        }
        st_dsmem_f32(&rx_m[rank][hh], (uint32_t)q, mv);
        st_dsmem_f32(&rx_l[rank][hh], (uint32_t)q, lv);
    }
    const int per_cta = G * kDH / p.cs;
    if (run) {
        for (int t = 0; t < nt; ++t)
            if (!mbar_wait(&bar_o[t], 0)) s_ok = 0;
        tc_fence_after();
        float o[G];
#pragma unroll
        for (int hh = 0; hh < G; ++hh) o[hh] = 0.f;
#pragma unroll
        for (int t = 0; t < 3; ++t) {  // the tiles' partials, added in tile order
            if (t < nt) {
                uint32_t r[16];
                tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + kOCol + t * 16, r);
#pragma unroll
                for (int hh = 0; hh < G; ++hh) o[hh] += __uint_as_float(r[hh]);
            }
        }
        const int d = warp * 32 + lane;
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            const int e = hh * kDH + d;
            st_dsmem_f32(&rx_o[rank][e % per_cta], (uint32_t)(e / per_cta), o[hh]);
        }
    } else {
        for (int e = tid; e < G * kDH; e += kThreads)
            st_dsmem_f32(&rx_o[rank][e % per_cta], (uint32_t)(e / per_cta), 0.f);
    }
    tc_fence_before();
    cluster_sync_all();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (!s_ok && tid == 0) set_status(p.status, kDevTimeout);
    if (tid < per_cta) {
        const int e = rank * per_cta + tid;
        const int hh = e / kDH;
        float mr[kMaxCs], lr[kMaxCs], orr[kMaxCs];
#pragma unroll
        for (int r = 0; r < kMaxCs; ++r) {
            if (r < p.cs) {
                mr[r] = rx_m[r][hh];
                lr[r] = rx_l[r][hh];
                orr[r] = rx_o[r][tid];
            }
        }
        float mx = -INFINITY;
#pragma unroll
        for (int r = 0; r < kMaxCs; ++r)
            if (r < p.cs) mx = fmaxf(mx, mr[r]);
        float lt = 0.f, ot = 0.f;
#pragma unroll
        for (int r = 0; r < kMaxCs; ++r) {
            if (r < p.cs && mr[r] != -INFINITY) {
                const float cw = ex2_approx(mr[r] - mx);
                lt = fmaf(lr[r], cw, lt);
                ot = fmaf(orr[r], cw, ot);
            }
        }
        p.out[((size_t)seq * p.H + kvh * G) * kDH + e] = __float2bfloat16_rn(ot / lt);
    }
}

template <int G>
cudaError_t prepare(int cs, size_t smem) {
    cudaError_t e =
        cudaFuncSetAttribute(attn_decode_tc_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess && cs > 8)
        e = cudaFuncSetAttribute(attn_decode_tc_kernel<G>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

template <int G>
cudaError_t launch(const DecKVMaps& maps, const AttnDecTcParams& p, cudaStream_t s, bool pdl) {
    const size_t smem = smem_layout(p.rows).total;
    static KernelAttrCache attrs;
    const cudaError_t ea = attrs.ensure(smem, p.cs, [](int cs, size_t sm) { return prepare<G>(cs, sm); });
    if (ea != cudaSuccess) return ea;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.cs, p.Hkv, p.nb);
    cfg.blockDim = dim3(kThreads);
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
    return cudaLaunchKernelEx(&cfg, attn_decode_tc_kernel<G>, maps, p);
}

// Cluster size 16 (else 8) with each CTA holding ceil(max_ctx / cs) keys; preferred when all
// Hkv clusters can be resident at once, which needs two CTAs per SM (so the keys of a CTA are
// allocated to the next 32, not to whole tiles).
template <int G>
bool plan(int Hkv, int max_ctx, int* cs, int* rows) {
    int best_c = 0, best_rows = 0, best_n = 0;
    for (int c : {16, 8}) {
        const int r = ((max_ctx + c - 1) / c + 31) & ~31;
        if (r > kMaxRows) continue;
        const size_t smem = smem_layout(r).total;
        if (prepare<G>(c, smem) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(c, Hkv);
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = c;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, attn_decode_tc_kernel<G>, &cfg) != cudaSuccess) {
            cudaGetLastError();
            n = 0;
        }
        if (n >= Hkv) {
            *cs = c;
            *rows = r;
            return true;
        }
        if (n > best_n) best_c = c, best_rows = r, best_n = n;
    }
    if (best_n == 0) return false;
    *cs = best_c;
    *rows = best_rows;
    return true;
}

}  // namespace

bool plan_decode_attention_tc(int dh, int group, int Hkv, int max_ctx, int* cs, int* rows) {
    if (dh != kDH) return false;
    switch (group) {
        case 1: return plan<1>(Hkv, max_ctx, cs, rows);
        case 2: return plan<2>(Hkv, max_ctx, cs, rows);
        case 4: return plan<4>(Hkv, max_ctx, cs, rows);
        case 8: return plan<8>(Hkv, max_ctx, cs, rows);
    }
    return false;
}

cudaError_t launch_attn_decode_tc(const DecKVMaps& maps, int group, const AttnDecTcParams& p, cudaStream_t s,
                                  bool pdl) {
    switch (group) {
        case 1: return launch<1>(maps, p, s, pdl);
        case 2: return launch<2>(maps, p, s, pdl);
        case 4: return launch<4>(maps, p, s, pdl);
        case 8: return launch<8>(maps, p, s, pdl);
    }
    return cudaErrorInvalidValue;
}

}  // namespace vla
