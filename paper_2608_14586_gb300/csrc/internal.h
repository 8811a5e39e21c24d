// Internal launch interface between the C-ABI runtime and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

namespace vla {

using bf16 = __nv_bfloat16;

// Launch attributes of one kernel, raised on demand: the dynamic shared-memory limit and the
// cluster size `set(cs, smem)` has been asked for only ever grow, under a lock, so host
// threads may launch concurrently. The library drives one device per process.
struct KernelAttrCache {
    std::mutex mu;
    size_t smem = 0;
    int cs = 0;
    template <class Set>
    cudaError_t ensure(size_t need_smem, int need_cs, Set&& set) {
        std::lock_guard<std::mutex> lk(mu);
        if (need_smem <= smem && need_cs <= cs) return cudaSuccess;
        const size_t s = need_smem > smem ? need_smem : smem;
        const int c = need_cs > cs ? need_cs : cs;
        const cudaError_t e = set(c, s);
        if (e == cudaSuccess) {
            smem = s;
            cs = c;
        }
        return e;
    }
};

// ---------------------------------------------------------------------------------------
// tcgen05 GEMM: C[M,N] = A[M,K] * B[N,K]^T with a fused epilogue
// ---------------------------------------------------------------------------------------
enum EpiMode : int {
    kEpiPlain = 0,   // out = bf16(acc)
    kEpiResid = 1,   // out = bf16(resid + acc)                       (O / down projections)
    kEpiQKV = 2,     // acc / rms -> RoPE(q, k); q -> out, k/v -> KV cache (QKV projection)
    kEpiSwiGLU = 3,  // gate/up tiles interleaved by 128 columns: out = silu(g/rms) * (u/rms)
};

struct EpiParams {
    int M, N;
    bf16* out;
    int ld_out;
    bf16* out_host;  // kEpiResid: a second copy of the output rows (page-locked host memory, same layout)
    const bf16* resid;
    int ld_resid;
    // RMSNorm of the GEMM's input rows: 1/rms = 1/sqrt(sum_t ss_in[row][t] / D + eps), the
    // partial sums of squares of ss_width-column groups added in group order (kEpiQKV,
    // kEpiSwiGLU). A partial is the in-order sum of its 32-column sub-groups, each an fmaf
    // chain from zero over its columns in order.
    const float* ss_in;
    int ss_width;   // 256 (tiles of 256 columns) or 32 (any tile width that is a multiple of 32)
    int ss_groups;  // D / ss_width
    int norm_dim;   // D
    float eps;
    // kEpiResid: the same partials of the stored (bf16) outputs -> ss_out[row][col / ss_width]
    // (nullptr: not wanted; ss_width 256 needs 256-wide tiles)
    float* ss_out;
    // QKV epilogue
    bf16* kcache;        // layer base, [n_kv_heads][max_ctx][head_dim]
    bf16* vcache;
    const float2* rope;  // [max_ctx][head_dim/2] (cos, sin)
    int pos0, max_ctx, head_dim, q_cols, kv_cols;
    int* len_out;   // kEpiQKV: the layer's device KV length, set to len_value (nullptr: leave)
    int len_value;
    unsigned* status;
    // Bound of every wait of the launch, in SM clock cycles (kWaitBudgetCycles unless a
    // failure-detection test shortens it), and that test's injected fault: k-block `stall_kb`
    // of each CTA's first tile is never loaded, so the waits on it run out (-1: no fault).
    long long wait_budget;
    int stall_kb;
    int tma_out;  // set by launch_gemm: the residual epilogue stores through TMA
};

// Tensor-map helper (driver entry point fetched through the runtime). rows x cols bf16,
// row stride in elements; box = box_rows x 64 columns, 128-byte swizzle, zero fill.
bool make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t row_stride,
                    uint32_t box_rows);

// 3-D bf16 map: [planes][rows][inner] with rows of `inner` elements and planes
// `plane_stride` elements apart; box = 1 plane x box_rows x 64, 128-byte swizzle, zero fill.
bool make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t planes,
                       uint64_t plane_stride, uint32_t box_rows);

// Output map of a GEMM epilogue that stores through TMA: rows x cols bf16, row stride in
// elements; box = 32 rows x 32 columns (64-byte rows), 64-byte swizzle.
bool make_tmap_bf16_store(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t row_stride);

// Programmatic dependent launch is used unless the environment sets VLA_NO_PDL (read once;
// for profilers and debuggers that serialise kernels anyway).
bool pdl_enabled();

// Launch with an N tile of bn columns: 256 (every mode), 224 (kEpiResid / kEpiPlain; row
// statistics then per 32 columns) or 192 (kEpiQKV). Returns a cudaError_t of the launch.
// pdl: programmatic dependent launch (the CTA prologue and the first weight-tile loads may
// overlap the previous kernel; A and everything the epilogue reads come after the wait).
// out_map (optional, kEpiResid / kEpiPlain): the output as a make_tmap_bf16_store map; the
// epilogue then stores through TMA (used when there is no host copy and N is a multiple of 32).
cudaError_t launch_gemm(int mode, int bn, const CUtensorMap& A, const CUtensorMap& B, int M, int N, int K,
                        const EpiParams& ep, int num_sms, cudaStream_t stream, bool pdl = false,
                        const CUtensorMap* out_map = nullptr);

// ---------------------------------------------------------------------------------------
// Prefill attention (causal GQA, flash-style online softmax, attention_tc.cu)
// ---------------------------------------------------------------------------------------
struct AttnPrefillParams {
    const bf16* q;  // [M, H*dh]
    int ld_q;
    const bf16* kc;  // layer base [Hkv][max_ctx][dh]
    const bf16* vc;
    bf16* out;  // [M, H*dh]
    int ld_out;
    int M, H, Hkv, head_dim, max_ctx, pos0;
    float scale_log2;  // log2(e) / sqrt(dh)
};
// tcgen05 kernel (S and O in tensor memory); `status` receives a timeout code
cudaError_t launch_attn_prefill_tc(const AttnPrefillParams& p, unsigned* status, cudaStream_t stream,
                                   bool pdl = false);

// ---------------------------------------------------------------------------------------
// Elementwise / setup kernels
// ---------------------------------------------------------------------------------------
// ss[row][t] = the row's sum of squares over columns [t*width, (t+1)*width) (width 256 or 32),
// in the order EpiParams describes: the same partial sums the residual GEMM epilogue writes
// for its output, so a block gets bit-identical row statistics whether its input came from
// the previous block or from the caller.
cudaError_t launch_row_sumsq(const bf16* x, int M, int D, int ld, int width, float* ss, cudaStream_t stream,
                             bool pdl = false);

// cos/sin table [max_ctx][dh/2] from float64 angles pos * base^(-2j/dh)
cudaError_t launch_rope_table(float2* table, int max_ctx, int head_dim, double base, cudaStream_t stream);

// Repacking of one layer's weights into the library's layouts (gains folded in).
struct RepackSrc {
    const bf16 *w_q, *w_k, *w_v, *w_o, *w_gate, *w_up, *w_down, *g_attn, *g_mlp;
};
struct RepackDst {
    bf16* w_qkv;  // [H*dh + 2*Hkv*dh, D], rows of q | k | v, each column scaled by g_attn; within
                  // each q and k head the rotation pairs (j, j + dh/2) sit in rows (2j, 2j + 1)
    bf16* w_o;    // [D, H*dh]
    bf16* w_gu;   // [2*F_pad, D], 256-row groups = 128 gate rows then 128 up rows, scaled by g_mlp
    bf16* w_d;    // [D, F_pad], columns >= F zero
};
cudaError_t launch_repack(const RepackSrc& s, const RepackDst& d, int D, int H, int Hkv, int dh, int F, int F_pad,
                          cudaStream_t stream);

cudaError_t launch_set_lengths(int* d_len, int count, int value, cudaStream_t stream);

// ---------------------------------------------------------------------------------------
// Decode (one token per sequence, up to kMaxDecodeBatch sequences): weight-streaming GEMVs
// and split-KV attention
// ---------------------------------------------------------------------------------------
constexpr int kMaxDecodeBatch = 4;
// One block of a decode step for nb sequences (one token each, each with its own KV cache).
struct DecodeLayer {
    const bf16 *w_qkv, *w_o, *w_gu, *w_d;
    int nb;
    bf16* kcache[kMaxDecodeBatch];  // each sequence's layer base [Hkv][max_ctx][dh]
    bf16* vcache[kMaxDecodeBatch];
    const int* d_len[kMaxDecodeBatch];  // each sequence's device length for this layer (new position)
};
struct DecodeDims {
    int D, H, Hkv, dh, F_pad, max_ctx;
    float eps;
};
struct DecodeWork {
    float* q;          // [nb][H*dh] fp32 (post-RoPE queries)
    bf16* attn;        // [nb][H*dh]
    bf16* x_mid;       // [nb][D]
    bf16* m;           // [nb][F_pad]
    const float2* rope;
    unsigned* status;
    int attn_tc;                         // 1: tcgen05 kernel (attn_cap = keys per CTA), 0: CUDA-core kernel
    int attn_cs, attn_cap, attn_stages;  // from plan_decode_attention(_tc)
};
// Decode attention on tcgen05 (head_dim 128): one cluster of `cs` CTAs per (sequence, KV
// head), each CTA holding up to `rows` keys (a multiple of 32, at most 384). K/V tensor maps:
// 3-D [Hkv][max_ctx][128] bf16 maps of each sequence's layer planes with 32-row boxes
// (make_tmap_bf16_3d).
struct DecKVMaps {
    CUtensorMap k[kMaxDecodeBatch];
    CUtensorMap v[kMaxDecodeBatch];
};
struct AttnDecTcParams {
    const float* q;  // [nb][H*dh] post-RoPE queries, fp32
    const bf16* kc[kMaxDecodeBatch];  // layer bases [Hkv][max_ctx][dh] (the new rows are read directly)
    const bf16* vc[kMaxDecodeBatch];
    const int* d_len[kMaxDecodeBatch];  // positions of the new tokens; context = d_len + 1
    int nb, H, Hkv, max_ctx, cs, rows;
    float scale_log2;
    bf16* out;  // [nb][H*dh]
    unsigned* status;
};
bool plan_decode_attention_tc(int dh, int group, int Hkv, int max_ctx, int* cs, int* rows);
cudaError_t launch_attn_decode_tc(const DecKVMaps& maps, int group, const AttnDecTcParams& p, cudaStream_t s,
                                  bool pdl);

// Decode-attention launch plan for contexts up to max_ctx: cluster size (CTAs per KV head),
// keys per shared-memory stage and stage count.
cudaError_t plan_decode_attention(int dh, int group, int Hkv, int max_ctx, int* cs, int* cap, int* stages);

// Optional per-launch hook (measurement): called with (ctx, stage, begin) around each kernel.
struct StageHook {
    void (*fn)(void* ctx, int stage, bool begin);
    void* ctx;
    void operator()(int stage, bool begin) const {
        if (fn) fn(ctx, stage, begin);
    }
};

// Stage ids of the decode kernels (match VLA_STAGE_DEC_* in vla_prefix.h)
enum : int { kStageDecQKV = 7, kStageDecAttn = 8, kStageDecO = 9, kStageDecGateUp = 10, kStageDecDown = 11 };

// pdl_first: the layer's first kernel may overlap the previous kernel in the stream (set when
// that kernel is the previous layer's down projection). The layer's later kernels always use
// programmatic dependent launch unless a stage hook is installed.
cudaError_t launch_decode_layer(const DecodeLayer& L, const DecodeDims& d, const DecodeWork& w, const bf16* x_in,
                                bf16* x_out, int num_sms, cudaStream_t stream, const StageHook& hook, bool pdl_first);

// d_len[b][i] += 1 for i < count, b < nb (after all layers of a decode step have read their
// positions)
cudaError_t launch_advance_lengths(int* const* d_len, int nb, int count, cudaStream_t stream);

}  // namespace vla
