// Small kernels around the GEMMs: RMSNorm row statistics, the rotary cos/sin table, weight
// repacking at create time, and KV-length updates.
#include "common.cuh"
#include "internal.h"

namespace vla {

namespace {

// Row sums of squares in exactly the order the residual GEMM epilogue forms them for its
// stored outputs: per 32-column group an fp32 fmaf chain from zero over its columns in order;
// for WIDTH 256 the 8 group sums of a chunk are then added in group order. One thread per
// 32-column group; with WIDTH 256 the 8 threads of a chunk are consecutive lanes.
template <int WIDTH>
__global__ void row_sumsq_kernel(const bf16* __restrict__ x, int M, int groups, int ld, float* __restrict__ ss) {
    constexpr int SUB = WIDTH / 32;  // 32-column groups per partial
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    pdl_wait();  // x is the previous kernel's output
    pdl_trigger();
    const long long part = i / SUB;
    const int sub = (int)(i % SUB);
    const bool ok = part < (long long)M * groups;
    float g = 0.f;
    if (ok) {
        const int row = (int)(part / groups), t = (int)(part % groups);
        const uint4* xr = reinterpret_cast<const uint4*>(x + (size_t)row * ld + t * WIDTH + sub * 32);
        uint4 v[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) v[c] = xr[c];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint32_t w[4] = {v[c].x, v[c].y, v[c].z, v[c].w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float a = bf16_lo(w[k]), b = bf16_hi(w[k]);
                g = fmaf(a, a, g);
                g = fmaf(b, b, g);
            }
        }
    }
    if constexpr (SUB == 1) {
        if (ok) ss[part] = g;
    } else {
        // the chunk's group sums to its first lane, added in group order
        const int base = threadIdx.x & (32 - SUB);
        float sums[SUB];
#pragma unroll
        for (int k = 0; k < SUB; ++k) sums[k] = __shfl_sync(0xFFFFFFFFu, g, base + k);
        if (ok && sub == 0) {
            float t = 0.f;
#pragma unroll
            for (int k = 0; k < SUB; ++k) t += sums[k];
            ss[part] = t;
        }
    }
}

// table[pos][j] = (cos, sin)(pos * base^(-2j/dh)), angles in float64
__global__ void rope_table_kernel(float2* table, int max_ctx, int dh, double base) {
    const int half = dh / 2;
    const long long n = (long long)max_ctx * half;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const int pos = (int)(i / half), j = (int)(i % half);
        const double theta = pow(base, -2.0 * (double)j / (double)dh);
        const double ang = (double)pos * theta;
        table[i] = make_float2((float)cos(ang), (float)sin(ang));
    }
}

// Weight repack of one layer (see RepackDst in internal.h).
__global__ void repack_kernel(RepackSrc s, RepackDst d, int D, int H, int Hkv, int dh, int F, int F_pad) {
    const long long qn = (long long)H * dh, kvn = (long long)Hkv * dh;
    const long long n_qkv = (qn + 2 * kvn) * D;
    const long long n_o = (long long)D * H * dh;
    const long long n_gu = 2LL * F_pad * D;
    const long long n_d = (long long)D * F_pad;
    const long long total = n_qkv + n_o + n_gu + n_d;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        long long j = i;
        if (j < n_qkv) {
            const long long r = j / D;
            const int k = (int)(j % D);
            const float gk = __bfloat162float(s.g_attn[k]);
            float w;
            // q and k heads: row 2j + e holds source row j + e * dh/2 (rotation pairs adjacent)
            const long long rs = (r < qn + kvn) ? (r / dh) * dh + ((r % dh) >> 1) + ((r % dh) & 1) * (dh >> 1) : r;
            if (r < qn) w = __bfloat162float(s.w_q[rs * D + k]);
            else if (r < qn + kvn) w = __bfloat162float(s.w_k[(rs - qn) * D + k]);
            else w = __bfloat162float(s.w_v[(r - qn - kvn) * D + k]);
            d.w_qkv[j] = __float2bfloat16_rn(w * gk);
            continue;
        }
        j -= n_qkv;
        if (j < n_o) {
            d.w_o[j] = s.w_o[j];
            continue;
        }
        j -= n_o;
        if (j < n_gu) {
            const long long r = j / D;
            const int k = (int)(j % D);
            const long long grp = r / 256, w_in = r % 256;
            const long long f = grp * 128 + (w_in < 128 ? w_in : w_in - 128);
            float w = 0.f;
            if (f < F) w = __bfloat162float(w_in < 128 ? s.w_gate[f * D + k] : s.w_up[f * D + k]);
            d.w_gu[j] = __float2bfloat16_rn(w * __bfloat162float(s.g_mlp[k]));
            continue;
        }
        j -= n_gu;
        {
            const long long r = j / F_pad;
            const int k = (int)(j % F_pad);
            d.w_d[j] = (k < F) ? s.w_down[r * F + k] : __float2bfloat16_rn(0.f);
        }
    }
}

__global__ void set_lengths_kernel(int* d_len, int count, int value) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < count) d_len[i] = value;
}

}  // namespace

cudaError_t launch_row_sumsq(const bf16* x, int M, int D, int ld, int width, float* ss, cudaStream_t stream,
                             bool pdl) {
    if (M <= 0) return cudaSuccess;
    const int groups = D / width;
    const long long n = (long long)M * (D / 32);  // one thread per 32-column group
    const dim3 grid((unsigned)((n + 255) / 256));
    if (width == 256) return launch_ex(row_sumsq_kernel<256>, grid, dim3(256), 0, stream, pdl, x, M, groups, ld, ss);
    if (width == 32) return launch_ex(row_sumsq_kernel<32>, grid, dim3(256), 0, stream, pdl, x, M, groups, ld, ss);
    return cudaErrorInvalidValue;
}

cudaError_t launch_rope_table(float2* table, int max_ctx, int head_dim, double base, cudaStream_t stream) {
    rope_table_kernel<<<256, 256, 0, stream>>>(table, max_ctx, head_dim, base);
    return cudaGetLastError();
}

cudaError_t launch_repack(const RepackSrc& s, const RepackDst& d, int D, int H, int Hkv, int dh, int F, int F_pad,
                          cudaStream_t stream) {
    repack_kernel<<<1024, 256, 0, stream>>>(s, d, D, H, Hkv, dh, F, F_pad);
    return cudaGetLastError();
}

cudaError_t launch_set_lengths(int* d_len, int count, int value, cudaStream_t stream) {
    if (count <= 0) return cudaSuccess;
    set_lengths_kernel<<<(count + 127) / 128, 128, 0, stream>>>(d_len, count, value);
    return cudaGetLastError();
}

}  // namespace vla
