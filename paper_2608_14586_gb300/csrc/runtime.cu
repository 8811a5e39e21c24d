// C-ABI runtime of the LLM-prefix library (include/vla_prefix.h, include/vla_ops.h).
//
// Per block l of a prefill over [layer_begin, layer_end), on the caller's stream:
//   row_sumsq(x)        (first block)  sum of x^2 per 32-column group       (RMSNorm statistics)
//   GEMM  x * Wqkv^T   [kEpiQKV]       1/rms scale, RoPE, q -> workspace,   (RMSNorm, projection,
//                                      post-RoPE k and v -> KV cache         RoPE, KV write)
//   attention(q, K, V)                 causal GQA over cache [0, p0 + M)
//   GEMM  o * Wo^T     [kEpiResid]     x_mid = x + o Wo^T, and x_mid's row statistics
//   GEMM  x_mid * Wgu^T [kEpiSwiGLU]   1/rms scale, m = silu(gate) * up
//   GEMM  m * Wd^T     [kEpiResid]     x_out = x_mid + m Wd^T -> hidden_out, and its row
//                                      statistics for block l+1
// Every kernel after the first is launched with programmatic dependent launch. Block b reads
// hidden_in; later blocks work in place in hidden_out, so the range needs one extra [M, D]
// buffer (x_mid). hidden_out after the last block is h^(layer_end) (Eq. 5). Decode runs the
// same stages as GEMVs (decode.cu, decode_attn_tc.cu), replayed as a CUDA graph per step.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/vla_ops.h"
#include "../../include/vla_prefix.h"
#include "common.cuh"
#include "internal.h"

using vla::bf16;

namespace vla {

typedef CUresult (*PFN_encodeTiled_t)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                      const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                      CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static PFN_encodeTiled_t get_encode_fn() {
    static PFN_encodeTiled_t fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_encodeTiled_t>(ptr);
    }
    return fn;
}

bool make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t row_stride,
                    uint32_t box_rows) {
    PFN_encodeTiled_t enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint64_t planes,
                       uint64_t plane_stride, uint32_t box_rows) {
    PFN_encodeTiled_t enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {inner, rows, planes};
    cuuint64_t strides[2] = {inner * 2, plane_stride * 2};
    cuuint32_t box[3] = {64, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_tmap_bf16_store(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t row_stride) {
    PFN_encodeTiled_t enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride * 2};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool pdl_enabled() {
    static const bool on = std::getenv("VLA_NO_PDL") == nullptr;
    return on;
}

static int device_sm_count() {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

}  // namespace vla

namespace {

constexpr int kBN = 256;  // N tile of every prefill GEMM


// A decode step is ~6 kernels per block (~97 for 16 blocks), each only a few to a few tens
// of microseconds long, so host launch cost would dominate. The step is captured once per
// (KV cache, layer range) as a CUDA graph that reads the token from a library-owned staging
// vector and the position from the cache's device-side lengths; every later step is one
// graph launch plus two 8 KB device copies in/out of the staging vectors.
constexpr int kMaxDecodeGraphs = 8;

struct LayerDev {
    bf16 *w_qkv, *w_o, *w_gu, *w_d;
    // tm_qkv192 / tm_o224 / tm_d224: the same weights in 192- and 224-row boxes
    CUtensorMap tm_qkv, tm_qkv192, tm_o, tm_o224, tm_gu, tm_d, tm_d224;
};

}  // namespace

struct vla_prefix {
    int device;
    vla_config cfg;
    int L;
    int qc, kvc, qkv_n, F_pad, num_sms;
    std::vector<LayerDev> layers;
    bf16* weight_pool = nullptr;
    float2* rope = nullptr;
    // prefill workspace, sized for cfg.max_ctx tokens
    bf16 *ws_q = nullptr, *ws_attn = nullptr, *ws_xmid = nullptr, *ws_m = nullptr;
    float *ws_ss_x = nullptr, *ws_ss_mid = nullptr;  // [max_ctx][D/32] row sums of squares
    // decode workspace
    float* dq = nullptr;
    bf16 *d_attn = nullptr, *d_xmid = nullptr, *d_m = nullptr;
    unsigned* d_status = nullptr;
    int last_launches = 0;
    // failure-detection test: the next prefill launch of GEMM stage `fault_stage` withholds
    // one k-block and waits at most `fault_budget` cycles (-1: none)
    int fault_stage = -1;
    long long fault_budget = 0;
    // measurement: event pairs around each kernel while timing is enabled
    unsigned timing = 0;  // bit s: time the kernels of stage s
    std::vector<cudaEvent_t> ev_pool;
    size_t ev_used = 0;
    struct Rec {
        int stage;
        cudaEvent_t a, b;
    };
    std::vector<Rec> recs;
    cudaStream_t cur_stream = nullptr;
    cudaEvent_t pending = nullptr;
    // decode graphs
    bf16 *d_xin = nullptr, *d_xout = nullptr;  // [kMaxDecodeBatch][D] staging vectors of a decode step
    cudaStream_t cap_stream = nullptr;
    struct DecodeGraph {
        const vla_kv* kv[vla::kMaxDecodeBatch];  // the step's caches, one per sequence
        int nb, lb, le;
        cudaGraphExec_t exec;
        bool uses(const vla_kv* k) const {
            for (int b = 0; b < nb; ++b)
                if (kv[b] == k) return true;
            return false;
        }
    };
    std::vector<DecodeGraph> graphs;
};

struct vla_kv {
    vla_prefix* p;
    int lb, le, max_ctx;
    size_t plane_elems;
    // decode-attention launch plan for this cache's max_ctx (plan_decode_attention(_tc))
    int attn_tc = 0, attn_cs = 0, attn_cap = 0, attn_stages = 0;
    bf16* data = nullptr;
    int* d_len = nullptr;
    std::vector<int> len;
    bf16* k_plane(int l) const { return data + ((size_t)(l - lb) * 2) * plane_elems; }
    bf16* v_plane(int l) const { return data + ((size_t)(l - lb) * 2 + 1) * plane_elems; }
};

namespace {

template <typename T>
bool dmalloc(T** p, size_t count) {
    *p = nullptr;
    if (count == 0) count = 1;
    return cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T)) == cudaSuccess;
}

void free_prefix(vla_prefix* p) {
    if (!p) return;
    cudaFree(p->weight_pool);
    cudaFree(p->rope);
    cudaFree(p->ws_q);
    cudaFree(p->ws_attn);
    cudaFree(p->ws_xmid);
    cudaFree(p->ws_m);
    cudaFree(p->ws_ss_x);
    cudaFree(p->ws_ss_mid);
    cudaFree(p->dq);
    cudaFree(p->d_attn);
    cudaFree(p->d_xmid);
    cudaFree(p->d_m);
    cudaFree(p->d_status);
    for (cudaEvent_t e : p->ev_pool) cudaEventDestroy(e);
    for (auto& g : p->graphs) cudaGraphExecDestroy(g.exec);
    if (p->cap_stream) cudaStreamDestroy(p->cap_stream);
    cudaFree(p->d_xin);
    cudaFree(p->d_xout);
    delete p;
}

cudaEvent_t pool_event(vla_prefix* p) {
    if (p->ev_used == p->ev_pool.size()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        p->ev_pool.push_back(e);
    }
    return p->ev_pool[p->ev_used++];
}

// Records the start / end event of one kernel of `stage` when timing is enabled.
void stage_mark(vla_prefix* p, int stage, bool begin) {
    if (!(p->timing & (1u << stage))) return;
    if (begin) {
        p->pending = pool_event(p);
        if (p->pending) cudaEventRecord(p->pending, p->cur_stream);
    } else if (p->pending) {
        cudaEvent_t b = pool_event(p);
        if (b) {
            cudaEventRecord(b, p->cur_stream);
            p->recs.push_back({stage, p->pending, b});
        }
        p->pending = nullptr;
    }
}

void stage_hook_fn(void* ctx, int stage, bool begin) { stage_mark(static_cast<vla_prefix*>(ctx), stage, begin); }

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

vla_status check_config(const vla_config* c) {
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

vla_status cuda_status(cudaError_t e) { return e == cudaSuccess ? VLA_OK : VLA_ERR_CUDA; }

// Range checks shared by prefill and decode; returns the common start position in *p0.
vla_status check_range(vla_prefix* p, vla_kv* kv, int lb, int le, int n_new, int* p0) {
    if (lb < 0 || le < lb || le > p->L) return VLA_ERR_RANGE;
    if (lb == le) {
        *p0 = 0;
        return VLA_OK;
    }
    if (!kv || kv->p != p) return VLA_ERR_INVALID_ARG;
    if (lb < kv->lb || le > kv->le) return VLA_ERR_RANGE;
    const int start = kv->len[lb - kv->lb];
    for (int l = lb; l < le; ++l)
        if (kv->len[l - kv->lb] != start) return VLA_ERR_RANGE;
    if ((long long)start + n_new > kv->max_ctx) return VLA_ERR_KV_FULL;
    *p0 = start;
    return VLA_OK;
}

}  // namespace

extern "C" {

const char* vla_status_str(vla_status s) {
    switch (s) {
        case VLA_OK: return "ok";
        case VLA_ERR_INVALID_ARG: return "invalid argument";
        case VLA_ERR_SHAPE: return "shape out of range";
        case VLA_ERR_RANGE: return "layer range out of range";
        case VLA_ERR_KV_FULL: return "kv cache full";
        case VLA_ERR_NOT_PINNED: return "host buffer not page-locked";
        case VLA_ERR_OOM: return "out of memory";
        case VLA_ERR_CUDA: return "cuda error";
        case VLA_ERR_TIMEOUT: return "device wait timed out";
        case VLA_ERR_UNSUPPORTED: return "unsupported model shape";
        case VLA_ERR_BUSY: return "all pipeline slots in flight";
    }
    return "unknown status";
}

vla_status vla_prefix_create(const vla_config* cfg, const vla_layer_weights* weights, int layer_count,
                             vla_prefix** out) {
    if (!out) return VLA_ERR_INVALID_ARG;
    *out = nullptr;
    if (!cfg || !weights || layer_count <= 0) return VLA_ERR_INVALID_ARG;
    vla_status st = check_config(cfg);
    if (st != VLA_OK) return st;
    for (int l = 0; l < layer_count; ++l) {
        const vla_layer_weights& w = weights[l];
        if (!w.w_q || !w.w_k || !w.w_v || !w.w_o || !w.w_gate || !w.w_up || !w.w_down || !w.g_attn || !w.g_mlp)
            return VLA_ERR_INVALID_ARG;
    }
    vla_prefix* p = new (std::nothrow) vla_prefix();
    if (!p) return VLA_ERR_OOM;
    cudaGetDevice(&p->device);
    p->cfg = *cfg;
    p->L = layer_count;
    const int D = cfg->hidden, H = cfg->n_heads, Hkv = cfg->n_kv_heads, dh = cfg->head_dim;
    p->qc = H * dh;
    p->kvc = Hkv * dh;
    p->qkv_n = p->qc + 2 * p->kvc;
    p->F_pad = (cfg->ffn + 255) / 256 * 256;
    p->num_sms = vla::device_sm_count();
    const size_t n_qkv = (size_t)p->qkv_n * D, n_o = (size_t)D * p->qc, n_gu = (size_t)2 * p->F_pad * D,
                 n_d = (size_t)D * p->F_pad;
    const size_t per_layer = n_qkv + n_o + n_gu + n_d;
    const int T = cfg->max_ctx;
    bool ok = dmalloc(&p->weight_pool, per_layer * layer_count) && dmalloc(&p->rope, (size_t)T * dh / 2) &&
              dmalloc(&p->ws_q, (size_t)T * p->qc) && dmalloc(&p->ws_attn, (size_t)T * p->qc) &&
              dmalloc(&p->ws_xmid, (size_t)T * D) && dmalloc(&p->ws_m, (size_t)T * p->F_pad) &&
              dmalloc(&p->ws_ss_x, (size_t)T * (D / 32)) &&
              dmalloc(&p->ws_ss_mid, (size_t)T * (D / 32)) && dmalloc(&p->dq, (size_t)vla::kMaxDecodeBatch * p->qc) &&
              dmalloc(&p->d_attn, (size_t)vla::kMaxDecodeBatch * p->qc) &&
              dmalloc(&p->d_xmid, (size_t)vla::kMaxDecodeBatch * D) &&
              dmalloc(&p->d_m, (size_t)vla::kMaxDecodeBatch * p->F_pad) && dmalloc(&p->d_status, 1) &&
              dmalloc(&p->d_xin, (size_t)vla::kMaxDecodeBatch * D) &&
              dmalloc(&p->d_xout, (size_t)vla::kMaxDecodeBatch * D);
    if (!ok) {
        cudaGetLastError();
        free_prefix(p);
        return VLA_ERR_OOM;
    }
    cudaError_t e = cudaMemset(p->d_status, 0, sizeof(unsigned));
    if (e == cudaSuccess) e = vla::launch_rope_table(p->rope, T, dh, (double)cfg->rope_base, 0);
    p->layers.resize(layer_count);
    for (int l = 0; l < layer_count && e == cudaSuccess; ++l) {
        LayerDev& ld = p->layers[l];
        bf16* base = p->weight_pool + per_layer * l;
        ld.w_qkv = base;
        ld.w_o = ld.w_qkv + n_qkv;
        ld.w_gu = ld.w_o + n_o;
        ld.w_d = ld.w_gu + n_gu;
        const vla_layer_weights& w = weights[l];
        vla::RepackSrc s = {(const bf16*)w.w_q,    (const bf16*)w.w_k,  (const bf16*)w.w_v,
                            (const bf16*)w.w_o,    (const bf16*)w.w_gate, (const bf16*)w.w_up,
                            (const bf16*)w.w_down, (const bf16*)w.g_attn, (const bf16*)w.g_mlp};
        vla::RepackDst d = {ld.w_qkv, ld.w_o, ld.w_gu, ld.w_d};
        e = vla::launch_repack(s, d, D, H, Hkv, dh, cfg->ffn, p->F_pad, 0);
        if (e != cudaSuccess) break;
        if (!vla::make_tmap_bf16(&ld.tm_qkv, ld.w_qkv, p->qkv_n, D, D, kBN) ||
            !vla::make_tmap_bf16(&ld.tm_qkv192, ld.w_qkv, p->qkv_n, D, D, 192) ||
            !vla::make_tmap_bf16(&ld.tm_o, ld.w_o, D, p->qc, p->qc, kBN) ||
            !vla::make_tmap_bf16(&ld.tm_o224, ld.w_o, D, p->qc, p->qc, 224) ||
            !vla::make_tmap_bf16(&ld.tm_d224, ld.w_d, D, p->F_pad, p->F_pad, 224) ||
            !vla::make_tmap_bf16(&ld.tm_gu, ld.w_gu, 2 * p->F_pad, D, D, kBN) ||
            !vla::make_tmap_bf16(&ld.tm_d, ld.w_d, D, p->F_pad, p->F_pad, kBN)) {
            free_prefix(p);
            return VLA_ERR_CUDA;
        }
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        cudaGetLastError();
        free_prefix(p);
        return VLA_ERR_CUDA;
    }
    *out = p;
    return VLA_OK;
}

vla_status vla_prefix_destroy(vla_prefix* p) {
    if (!p) return VLA_OK;
    cudaDeviceSynchronize();
    free_prefix(p);
    return VLA_OK;
}

vla_status vla_kv_create(vla_prefix* p, int layer_begin, int layer_end, int max_ctx, vla_kv** out) {
    if (!out) return VLA_ERR_INVALID_ARG;
    *out = nullptr;
    if (!p) return VLA_ERR_INVALID_ARG;
    if (layer_begin < 0 || layer_end <= layer_begin || layer_end > p->L) return VLA_ERR_RANGE;
    if (max_ctx <= 0 || max_ctx > p->cfg.max_ctx) return VLA_ERR_SHAPE;
    vla_kv* kv = new (std::nothrow) vla_kv();
    if (!kv) return VLA_ERR_OOM;
    kv->p = p;
    kv->lb = layer_begin;
    kv->le = layer_end;
    kv->max_ctx = max_ctx;
    kv->plane_elems = (size_t)p->cfg.n_kv_heads * max_ctx * p->cfg.head_dim;
    const int dh = p->cfg.head_dim, Hkv = p->cfg.n_kv_heads, G = p->cfg.n_heads / Hkv;
    kv->attn_tc = vla::plan_decode_attention_tc(dh, G, Hkv, max_ctx, &kv->attn_cs, &kv->attn_cap) ? 1 : 0;
    if (!kv->attn_tc &&
        vla::plan_decode_attention(dh, G, Hkv, max_ctx, &kv->attn_cs, &kv->attn_cap, &kv->attn_stages) != cudaSuccess) {
        cudaGetLastError();
        delete kv;
        return VLA_ERR_UNSUPPORTED;
    }
    const int nl = layer_end - layer_begin;
    kv->len.assign(nl, 0);
    if (!dmalloc(&kv->data, kv->plane_elems * 2 * nl) || !dmalloc(&kv->d_len, (size_t)nl)) {
        cudaGetLastError();
        cudaFree(kv->data);
        cudaFree(kv->d_len);
        delete kv;
        return VLA_ERR_OOM;
    }
    if (cudaMemset(kv->d_len, 0, sizeof(int) * nl) != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) {
        cudaFree(kv->data);
        cudaFree(kv->d_len);
        delete kv;
        return VLA_ERR_CUDA;
    }
    *out = kv;
    return VLA_OK;
}

vla_status vla_kv_destroy(vla_kv* kv) {
    if (!kv) return VLA_OK;
    cudaDeviceSynchronize();
    auto& gs = kv->p->graphs;
    for (size_t i = 0; i < gs.size();) {
        if (gs[i].uses(kv)) {
            cudaGraphExecDestroy(gs[i].exec);
            gs.erase(gs.begin() + i);
        } else {
            ++i;
        }
    }
    cudaFree(kv->data);
    cudaFree(kv->d_len);
    delete kv;
    return VLA_OK;
}

vla_status vla_kv_reset(vla_kv* kv, vla_stream stream) { return vla_kv_set_length(kv, 0, stream); }

vla_status vla_kv_set_length(vla_kv* kv, int length, vla_stream stream) {
    if (!kv || length < 0) return VLA_ERR_INVALID_ARG;
    if (length > kv->max_ctx) return VLA_ERR_KV_FULL;
    for (int& v : kv->len) v = length;
    return cuda_status(vla::launch_set_lengths(kv->d_len, (int)kv->len.size(), length, (cudaStream_t)stream));
}

int vla_kv_length(const vla_kv* kv) {
    if (!kv) return -1;
    int m = kv->len.empty() ? 0 : kv->len[0];
    for (int v : kv->len) m = v < m ? v : m;
    return m;
}

vla_status vla_kv_decode_plan(const vla_kv* kv, int* tensor_cores, int* cluster_size, int* keys_per_cta) {
    if (!kv) return VLA_ERR_INVALID_ARG;
    if (tensor_cores) *tensor_cores = kv->attn_tc;
    if (cluster_size) *cluster_size = kv->attn_cs;
    if (keys_per_cta) *keys_per_cta = kv->attn_cap;
    return VLA_OK;
}

int vla_kv_layer_length(const vla_kv* kv, int layer) {
    if (!kv || layer < kv->lb || layer >= kv->le) return -1;
    return kv->len[layer - kv->lb];
}

vla_status vla_kv_data(const vla_kv* kv, int layer, void** k_plane, void** v_plane) {
    if (!kv || !k_plane || !v_plane) return VLA_ERR_INVALID_ARG;
    if (layer < kv->lb || layer >= kv->le) return VLA_ERR_RANGE;
    *k_plane = kv->k_plane(layer);
    *v_plane = kv->v_plane(layer);
    return VLA_OK;
}

// Wait bound and injected fault of one GEMM launch of `stage` with num_kb k-blocks: the
// default bound, unless a failure-detection test armed this stage (consumed by one launch).
void set_waits(vla_prefix* p, vla::EpiParams& ep, int stage, int K) {
    ep.wait_budget = vla::kWaitBudgetCycles;
    ep.stall_kb = -1;
    if (p && p->fault_stage == stage) {
        ep.wait_budget = p->fault_budget;
        ep.stall_kb = (K + 63) / 64 - 1;
        p->fault_stage = -1;
    }
}

// Prefill of [layer_begin, layer_end); with host_dev set, the last block's down projection
// also stores h^(layer_end) into page-locked host memory (host_dev: its device address).
static vla_status prefill_impl(vla_prefix* p, const void* hidden_in, int n_tokens, int layer_begin, int layer_end,
                               vla_kv* kv, void* hidden_out, vla_stream stream_, bf16* host_dev, void* host_ptr) {
    if (!p || !hidden_in || !hidden_out || n_tokens < 0) return VLA_ERR_INVALID_ARG;
    if (!aligned16(hidden_in) || !aligned16(hidden_out)) return VLA_ERR_INVALID_ARG;
    if (n_tokens > p->cfg.max_ctx) return VLA_ERR_SHAPE;
    int p0 = 0;
    vla_status st = check_range(p, kv, layer_begin, layer_end, n_tokens, &p0);
    if (st != VLA_OK) return st;
    p->last_launches = 0;
    if (n_tokens == 0) return VLA_OK;
    cudaStream_t stream = (cudaStream_t)stream_;
    const int D = p->cfg.hidden, M = n_tokens;
    if (layer_begin == layer_end) {
        cudaError_t e = cudaSuccess;
        if (hidden_in != hidden_out)
            e = cudaMemcpyAsync(hidden_out, hidden_in, (size_t)M * D * 2, cudaMemcpyDeviceToDevice, stream);
        if (e == cudaSuccess && host_ptr)
            e = cudaMemcpyAsync(host_ptr, hidden_in, (size_t)M * D * 2, cudaMemcpyDeviceToHost, stream);
        return cuda_status(e);
    }
    CUtensorMap tm_in, tm_out, tm_attn, tm_xmid, tm_m;
    if (!vla::make_tmap_bf16(&tm_in, hidden_in, M, D, D, 128) || !vla::make_tmap_bf16(&tm_out, hidden_out, M, D, D, 128) ||
        !vla::make_tmap_bf16(&tm_attn, p->ws_attn, M, p->qc, p->qc, 128) ||
        !vla::make_tmap_bf16(&tm_xmid, p->ws_xmid, M, D, D, 128) ||
        !vla::make_tmap_bf16(&tm_m, p->ws_m, M, p->F_pad, p->F_pad, 128))
        return VLA_ERR_CUDA;
    // output maps of the O and down projections (epilogue stores through TMA)
    CUtensorMap tm_st_xmid, tm_st_out;
    if (!vla::make_tmap_bf16_store(&tm_st_xmid, p->ws_xmid, M, D, D) ||
        !vla::make_tmap_bf16_store(&tm_st_out, hidden_out, M, D, D))
        return VLA_ERR_CUDA;
    const float eps = p->cfg.rms_eps;
    int launches = 0;
    cudaError_t e = cudaSuccess;
    p->cur_stream = stream;
    // Programmatic dependent launch for every kernel after the call's first, except the ones
    // being timed (their start event must precede the whole kernel).
    bool first_launch = true;
    auto pdl = [&](int stage) {
        const bool r = !first_launch && !((p->timing >> stage) & 1u) && vla::pdl_enabled();
        first_launch = false;
        return r;
    };
    // QKV tile width: the one with fewer column-slots in its last wave of tiles (waves x width;
    // 192 pays where 256-wide tiles leave a mostly idle second wave, e.g. 1024 tokens of a 7B
    // block: 192 tiles of 256 on 152 SMs, 256 tiles of 192), 256 on a tie
    // The same choice for the O and down projections (N = D) between 256 and 224 columns
    // (1024 tokens: 128 tiles of 256 leave 24 SMs idle, 152 tiles of 224 fill them).
    auto wave_cost = [&](int n, int bn) {
        const long long tiles = (long long)((M + 127) / 128) * ((n + bn - 1) / bn);
        return ((tiles + p->num_sms - 1) / p->num_sms) * bn;
    };
    const int qkv_bn = wave_cost(p->qkv_n, 192) < wave_cost(p->qkv_n, kBN) ? 192 : kBN;
    const int d_bn = wave_cost(D, 224) < wave_cost(D, kBN) ? 224 : kBN;
    const int ss_w = d_bn == kBN ? 256 : 32;  // row-statistics partials: one per tile or per 32 columns
    for (int l = layer_begin; l < layer_end && e == cudaSuccess; ++l) {
        const LayerDev& ld = p->layers[l];
        const bf16* x = (l == layer_begin) ? (const bf16*)hidden_in : (const bf16*)hidden_out;
        const CUtensorMap& tm_x = (l == layer_begin) ? tm_in : tm_out;
        // RMSNorm row statistics of the range's input (later blocks get them from the previous
        // block's down-projection epilogue) + QKV projection + RoPE + KV write
        if (l == layer_begin) {
            stage_mark(p, VLA_STAGE_ROWSTAT, true);
            e = vla::launch_row_sumsq(x, M, D, D, ss_w, p->ws_ss_x, stream, pdl(VLA_STAGE_ROWSTAT));
            stage_mark(p, VLA_STAGE_ROWSTAT, false);
            if (e != cudaSuccess) break;
            ++launches;
        }
        vla::EpiParams ep = {};
        ep.M = M;
        ep.N = p->qkv_n;
        ep.out = p->ws_q;
        ep.ld_out = p->qc;
        ep.ss_in = p->ws_ss_x;
        ep.ss_width = ss_w;
        ep.ss_groups = D / ss_w;
        ep.norm_dim = D;
        ep.eps = eps;
        ep.kcache = kv->k_plane(l);
        ep.vcache = kv->v_plane(l);
        ep.rope = p->rope;
        ep.pos0 = p0;
        ep.max_ctx = kv->max_ctx;
        ep.head_dim = p->cfg.head_dim;
        ep.q_cols = p->qc;
        ep.kv_cols = p->kvc;
        ep.len_out = kv->d_len + (l - kv->lb);
        ep.len_value = p0 + M;
        ep.status = p->d_status;
        set_waits(p, ep, VLA_STAGE_GEMM_QKV, D);
        stage_mark(p, VLA_STAGE_GEMM_QKV, true);
        e = vla::launch_gemm(vla::kEpiQKV, qkv_bn, tm_x, qkv_bn == 192 ? ld.tm_qkv192 : ld.tm_qkv, M, p->qkv_n, D,
                             ep, p->num_sms, stream, pdl(VLA_STAGE_GEMM_QKV));
        stage_mark(p, VLA_STAGE_GEMM_QKV, false);
        if (e != cudaSuccess) break;
        // causal GQA attention over the cache
        vla::AttnPrefillParams ap = {};
        ap.q = p->ws_q;
        ap.ld_q = p->qc;
        ap.kc = kv->k_plane(l);
        ap.vc = kv->v_plane(l);
        ap.out = p->ws_attn;
        ap.ld_out = p->qc;
        ap.M = M;
        ap.H = p->cfg.n_heads;
        ap.Hkv = p->cfg.n_kv_heads;
        ap.head_dim = p->cfg.head_dim;
        ap.max_ctx = kv->max_ctx;
        ap.pos0 = p0;
        ap.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)p->cfg.head_dim));
        stage_mark(p, VLA_STAGE_ATTN, true);
        e = vla::launch_attn_prefill_tc(ap, p->d_status, stream, pdl(VLA_STAGE_ATTN));
        stage_mark(p, VLA_STAGE_ATTN, false);
        if (e != cudaSuccess) break;
        // output projection + residual
        vla::EpiParams eo = {};
        eo.M = M;
        eo.N = D;
        eo.out = p->ws_xmid;
        eo.ld_out = D;
        eo.resid = x;
        eo.ld_resid = D;
        eo.ss_out = p->ws_ss_mid;
        eo.ss_width = ss_w;
        eo.ss_groups = D / ss_w;
        eo.status = p->d_status;
        set_waits(p, eo, VLA_STAGE_GEMM_O, p->qc);
        stage_mark(p, VLA_STAGE_GEMM_O, true);
        e = vla::launch_gemm(vla::kEpiResid, d_bn, tm_attn, d_bn == 224 ? ld.tm_o224 : ld.tm_o, M, D, p->qc, eo,
                             p->num_sms, stream, pdl(VLA_STAGE_GEMM_O), &tm_st_xmid);
        stage_mark(p, VLA_STAGE_GEMM_O, false);
        if (e != cudaSuccess) break;
        // RMSNorm (row statistics from the O epilogue) + gate/up + SwiGLU
        vla::EpiParams eg = {};
        eg.M = M;
        eg.N = 2 * p->F_pad;
        eg.out = p->ws_m;
        eg.ld_out = p->F_pad;
        eg.ss_in = p->ws_ss_mid;
        eg.ss_width = ss_w;
        eg.ss_groups = D / ss_w;
        eg.norm_dim = D;
        eg.eps = eps;
        eg.status = p->d_status;
        set_waits(p, eg, VLA_STAGE_GEMM_GATEUP, D);
        stage_mark(p, VLA_STAGE_GEMM_GATEUP, true);
        e = vla::launch_gemm(vla::kEpiSwiGLU, kBN, tm_xmid, ld.tm_gu, M, 2 * p->F_pad, D, eg, p->num_sms, stream,
                             pdl(VLA_STAGE_GEMM_GATEUP));
        stage_mark(p, VLA_STAGE_GEMM_GATEUP, false);
        if (e != cudaSuccess) break;
        // down projection + residual -> hidden_out
        vla::EpiParams ed = {};
        ed.M = M;
        ed.N = D;
        ed.out = (bf16*)hidden_out;
        ed.ld_out = D;
        ed.resid = p->ws_xmid;
        ed.ld_resid = D;
        ed.ss_out = (l + 1 < layer_end) ? p->ws_ss_x : nullptr;  // the next block's row statistics
        ed.out_host = (l + 1 == layer_end) ? host_dev : nullptr;   // h^(layer_end) straight to the host
        ed.ss_width = ss_w;
        ed.ss_groups = D / ss_w;
        ed.status = p->d_status;
        set_waits(p, ed, VLA_STAGE_GEMM_DOWN, p->F_pad);
        stage_mark(p, VLA_STAGE_GEMM_DOWN, true);
        e = vla::launch_gemm(vla::kEpiResid, d_bn, tm_m, d_bn == 224 ? ld.tm_d224 : ld.tm_d, M, D, p->F_pad, ed,
                             p->num_sms, stream, pdl(VLA_STAGE_GEMM_DOWN), &tm_st_out);
        stage_mark(p, VLA_STAGE_GEMM_DOWN, false);
        launches += 5;
    }
    if (e != cudaSuccess) return VLA_ERR_CUDA;
    // device lengths were advanced by each layer's QKV kernel
    for (int l = layer_begin; l < layer_end; ++l) kv->len[l - kv->lb] = p0 + M;
    p->last_launches = launches;
    return VLA_OK;
}

vla_status vla_prefix_prefill(vla_prefix* p, const void* hidden_in, int n_tokens, int layer_begin, int layer_end,
                              vla_kv* kv, void* hidden_out, vla_stream stream) {
    return prefill_impl(p, hidden_in, n_tokens, layer_begin, layer_end, kv, hidden_out, stream, nullptr, nullptr);
}

vla_status vla_prefix_prefill_to_host(vla_prefix* p, const void* hidden_in, int n_tokens, int layer_begin,
                                      int layer_end, vla_kv* kv, void* hidden_out, void* pinned_dst,
                                      vla_stream stream) {
    if (!pinned_dst) return VLA_ERR_INVALID_ARG;
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, pinned_dst) != cudaSuccess) {
        cudaGetLastError();
        return VLA_ERR_NOT_PINNED;
    }
    if (attr.type != cudaMemoryTypeHost || !attr.devicePointer) return VLA_ERR_NOT_PINNED;
    if (!aligned16(attr.devicePointer)) return VLA_ERR_INVALID_ARG;
    return prefill_impl(p, hidden_in, n_tokens, layer_begin, layer_end, kv, hidden_out, stream,
                        static_cast<bf16*>(attr.devicePointer), pinned_dst);
}

// One decode step of blocks [layer_begin, layer_end) for nb sequences (hidden_in/out [nb][D],
// one token each, sequence b in cache kvs[b] at that cache's common length).
static vla_status decode_impl(vla_prefix* p, const void* hidden_in, int nb, int layer_begin, int layer_end,
                              vla_kv* const* kvs, void* hidden_out, vla_stream stream_) {
    if (!p || !hidden_in || !hidden_out || !kvs) return VLA_ERR_INVALID_ARG;
    if (nb < 1 || nb > vla::kMaxDecodeBatch) return VLA_ERR_SHAPE;
    if (!aligned16(hidden_in) || !aligned16(hidden_out)) return VLA_ERR_INVALID_ARG;
    int p0[vla::kMaxDecodeBatch];
    for (int b = 0; b < nb; ++b) {
        vla_status st = check_range(p, kvs[b], layer_begin, layer_end, 1, &p0[b]);
        if (st != VLA_OK) return st;
        for (int c = 0; c < b; ++c)
            if (layer_begin < layer_end && kvs[c] == kvs[b]) return VLA_ERR_INVALID_ARG;  // one token per cache
        if (layer_begin < layer_end &&
            (kvs[b]->max_ctx != kvs[0]->max_ctx || kvs[b]->lb != kvs[0]->lb))  // one plane stride and plan
            return VLA_ERR_SHAPE;
    }
    p->last_launches = 0;
    cudaStream_t stream = (cudaStream_t)stream_;
    const int D = p->cfg.hidden;
    const size_t vec_bytes = (size_t)nb * D * 2;
    if (layer_begin == layer_end) {
        if (hidden_in == hidden_out) return VLA_OK;
        return cuda_status(cudaMemcpyAsync(hidden_out, hidden_in, vec_bytes, cudaMemcpyDeviceToDevice, stream));
    }
    const vla_kv* kv0 = kvs[0];
    vla::DecodeDims dims = {D, p->cfg.n_heads, p->cfg.n_kv_heads, p->cfg.head_dim, p->F_pad, kv0->max_ctx,
                            p->cfg.rms_eps};
    vla::DecodeWork w = {p->dq,       p->d_attn,   p->d_xmid,    p->d_m,        p->rope,
                         p->d_status, kv0->attn_tc, kv0->attn_cs, kv0->attn_cap, kv0->attn_stages};
    const int nl = layer_end - layer_begin;
    // enqueue the whole step on stream s, reading x_in and chaining through x_out
    auto enqueue = [&](const bf16* x_in, bf16* x_out, cudaStream_t s, const vla::StageHook& hook) {
        cudaError_t e = cudaSuccess;
        for (int l = layer_begin; l < layer_end && e == cudaSuccess; ++l) {
            const LayerDev& ld = p->layers[l];
            vla::DecodeLayer L = {};
            L.w_qkv = ld.w_qkv;
            L.w_o = ld.w_o;
            L.w_gu = ld.w_gu;
            L.w_d = ld.w_d;
            L.nb = nb;
            for (int b = 0; b < nb; ++b) {
                L.kcache[b] = kvs[b]->k_plane(l);
                L.vcache[b] = kvs[b]->v_plane(l);
                L.d_len[b] = kvs[b]->d_len + (l - kvs[b]->lb);
            }
            e = vla::launch_decode_layer(L, dims, w, l == layer_begin ? x_in : x_out, x_out, p->num_sms, s, hook,
                                         l > layer_begin);
        }
        int* lens[vla::kMaxDecodeBatch];
        for (int b = 0; b < nb; ++b) lens[b] = kvs[b]->d_len + (layer_begin - kvs[b]->lb);
        if (e == cudaSuccess) e = vla::launch_advance_lengths(lens, nb, nl, s);
        return e;
    };
    cudaError_t e = cudaSuccess;
    p->cur_stream = stream;
    if (p->timing) {
        // measurement mode: direct launches with event pairs around the selected stages
        const vla::StageHook hook = {stage_hook_fn, p};
        e = enqueue((const bf16*)hidden_in, (bf16*)hidden_out, stream, hook);
    } else {
        cudaGraphExec_t exec = nullptr;
        for (const auto& g : p->graphs) {
            if (g.nb != nb || g.lb != layer_begin || g.le != layer_end) continue;
            bool same = true;
            for (int b = 0; b < nb; ++b) same = same && g.kv[b] == kvs[b];
            if (same) exec = g.exec;
        }
        if (!exec) {
            if (!p->cap_stream && cudaStreamCreateWithFlags(&p->cap_stream, cudaStreamNonBlocking) != cudaSuccess)
                return VLA_ERR_CUDA;
            cudaGraph_t graph = nullptr;
            e = cudaStreamBeginCapture(p->cap_stream, cudaStreamCaptureModeRelaxed);
            if (e == cudaSuccess) {
                cudaError_t le = enqueue(p->d_xin, p->d_xout, p->cap_stream, vla::StageHook{nullptr, nullptr});
                e = cudaStreamEndCapture(p->cap_stream, &graph);
                if (le != cudaSuccess) e = le;
            }
            if (e == cudaSuccess) e = cudaGraphInstantiate(&exec, graph, 0);
            if (graph) cudaGraphDestroy(graph);
            if (e != cudaSuccess) {
                cudaGetLastError();
                return VLA_ERR_CUDA;
            }
            if ((int)p->graphs.size() >= kMaxDecodeGraphs) {
                cudaGraphExecDestroy(p->graphs.front().exec);
                p->graphs.erase(p->graphs.begin());
            }
            vla_prefix::DecodeGraph g = {};
            for (int b = 0; b < nb; ++b) g.kv[b] = kvs[b];
            g.nb = nb;
            g.lb = layer_begin;
            g.le = layer_end;
            g.exec = exec;
            p->graphs.push_back(g);
        }
        e = cudaMemcpyAsync(p->d_xin, hidden_in, vec_bytes, cudaMemcpyDeviceToDevice, stream);
        if (e == cudaSuccess) e = cudaGraphLaunch(exec, stream);
        if (e == cudaSuccess) e = cudaMemcpyAsync(hidden_out, p->d_xout, vec_bytes, cudaMemcpyDeviceToDevice, stream);
    }
    if (e != cudaSuccess) return VLA_ERR_CUDA;
    for (int b = 0; b < nb; ++b)
        for (int l = layer_begin; l < layer_end; ++l) kvs[b]->len[l - kvs[b]->lb] = p0[b] + 1;
    p->last_launches = 5 * nl + 1;
    return VLA_OK;
}

vla_status vla_prefix_decode(vla_prefix* p, const void* hidden_in, int layer_begin, int layer_end, vla_kv* kv,
                             void* hidden_out, vla_stream stream) {
    if (layer_begin == layer_end) {  // a copy: no cache needed
        if (!p || !hidden_in || !hidden_out) return VLA_ERR_INVALID_ARG;
        vla_kv* none = nullptr;
        return decode_impl(p, hidden_in, 1, layer_begin, layer_end, &none, hidden_out, stream);
    }
    return decode_impl(p, hidden_in, 1, layer_begin, layer_end, &kv, hidden_out, stream);
}

vla_status vla_prefix_decode_batch(vla_prefix* p, const void* hidden_in, int batch, int layer_begin, int layer_end,
                                   vla_kv* const* kvs, void* hidden_out, vla_stream stream) {
    return decode_impl(p, hidden_in, batch, layer_begin, layer_end, kvs, hidden_out, stream);
}

vla_status vla_boundary_to_host(const void* hidden_out, int n_tokens, int hidden, void* pinned_dst,
                                vla_stream side_stream, vla_event ready, vla_event done) {
    if (!hidden_out || !pinned_dst || n_tokens < 0 || hidden <= 0) return VLA_ERR_INVALID_ARG;
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, pinned_dst) != cudaSuccess) {
        cudaGetLastError();
        return VLA_ERR_NOT_PINNED;
    }
    if (attr.type != cudaMemoryTypeHost) return VLA_ERR_NOT_PINNED;
    cudaStream_t s = (cudaStream_t)side_stream;
    cudaError_t e = cudaSuccess;
    if (ready) e = cudaStreamWaitEvent(s, (cudaEvent_t)ready, 0);
    if (e == cudaSuccess && n_tokens > 0)
        e = cudaMemcpyAsync(pinned_dst, hidden_out, (size_t)n_tokens * hidden * 2, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && done) e = cudaEventRecord((cudaEvent_t)done, s);
    return cuda_status(e);
}

vla_status vla_frame_to_device(const void* pinned_src, int n_tokens, int hidden, void* hidden_in,
                               vla_stream stream) {
    if (!pinned_src || !hidden_in || n_tokens < 0 || hidden <= 0) return VLA_ERR_INVALID_ARG;
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, pinned_src) != cudaSuccess) {
        cudaGetLastError();
        return VLA_ERR_NOT_PINNED;
    }
    if (attr.type != cudaMemoryTypeHost) return VLA_ERR_NOT_PINNED;
    if (n_tokens == 0) return VLA_OK;
    return cuda_status(cudaMemcpyAsync(hidden_in, pinned_src, (size_t)n_tokens * hidden * 2, cudaMemcpyHostToDevice,
                                       (cudaStream_t)stream));
}

vla_status vla_last_async_error(vla_prefix* p) {
    if (!p) return VLA_ERR_INVALID_ARG;
    unsigned code = 0;
    if (cudaMemcpy(&code, p->d_status, sizeof(unsigned), cudaMemcpyDeviceToHost) != cudaSuccess) return VLA_ERR_CUDA;
    if (code != 0 && cudaMemset(p->d_status, 0, sizeof(unsigned)) != cudaSuccess) return VLA_ERR_CUDA;
    return code == vla::kDevOk ? VLA_OK : VLA_ERR_TIMEOUT;
}

int vla_last_launch_count(const vla_prefix* p) { return p ? p->last_launches : 0; }

vla_status vla_prefix_info(const vla_prefix* p, vla_config* cfg, int* layer_count) {
    if (!p) return VLA_ERR_INVALID_ARG;
    if (cfg) *cfg = p->cfg;
    if (layer_count) *layer_count = p->L;
    return VLA_OK;
}

vla_status vla_prefix_inject_stall(vla_prefix* p, int stage, long long wait_budget_cycles) {
    if (!p) return VLA_ERR_INVALID_ARG;
    if (stage == -1) {
        p->fault_stage = -1;
        return VLA_OK;
    }
    if (stage != VLA_STAGE_GEMM_QKV && stage != VLA_STAGE_GEMM_O && stage != VLA_STAGE_GEMM_GATEUP &&
        stage != VLA_STAGE_GEMM_DOWN)
        return VLA_ERR_UNSUPPORTED;
    if (wait_budget_cycles < 100000 || wait_budget_cycles > vla::kWaitBudgetCycles) return VLA_ERR_INVALID_ARG;
    p->fault_stage = stage;
    p->fault_budget = wait_budget_cycles;
    return VLA_OK;
}

vla_status vla_prefix_set_timing(vla_prefix* p, unsigned stage_mask) {
    if (!p) return VLA_ERR_INVALID_ARG;
    p->timing = stage_mask;
    return VLA_OK;
}

vla_status vla_prefix_stage_times(vla_prefix* p, float* ms_per_stage, int* launches_per_stage, int n_stages) {
    if (!p || n_stages < 0 || (n_stages > 0 && (!ms_per_stage || !launches_per_stage))) return VLA_ERR_INVALID_ARG;
    for (int i = 0; i < n_stages; ++i) {
        ms_per_stage[i] = 0.f;
        launches_per_stage[i] = 0;
    }
    vla_status st = VLA_OK;
    for (const auto& r : p->recs) {
        if (cudaEventSynchronize(r.b) != cudaSuccess) {
            st = VLA_ERR_CUDA;
            break;
        }
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) {
            st = VLA_ERR_CUDA;
            break;
        }
        if (r.stage >= 0 && r.stage < n_stages) {
            ms_per_stage[r.stage] += ms;
            launches_per_stage[r.stage] += 1;
        }
    }
    p->recs.clear();
    p->ev_used = 0;
    return st;
}

// ------------------------------------------------------------------------------------------
// kernel-level entry points
// ------------------------------------------------------------------------------------------
vla_status vla_op_gemm_bf16(const void* A, const void* B, int M, int N, int K, void* C, vla_stream stream) {
    if (!A || !B || !C || M <= 0 || N <= 0 || K <= 0 || (K % 8) || (N % 8)) return VLA_ERR_INVALID_ARG;
    if (!aligned16(A) || !aligned16(B) || !aligned16(C)) return VLA_ERR_INVALID_ARG;
    CUtensorMap ta, tb;
    if (!vla::make_tmap_bf16(&ta, A, M, K, K, 128) || !vla::make_tmap_bf16(&tb, B, N, K, K, kBN)) return VLA_ERR_CUDA;
    vla::EpiParams ep = {};
    ep.M = M;
    ep.N = N;
    ep.out = (bf16*)C;
    ep.ld_out = N;
    set_waits(nullptr, ep, -1, K);
    static const int sms = vla::device_sm_count();
    CUtensorMap tc;
    if (!vla::make_tmap_bf16_store(&tc, C, M, N, N)) return VLA_ERR_CUDA;
    return cuda_status(vla::launch_gemm(vla::kEpiPlain, kBN, ta, tb, M, N, K, ep, sms, (cudaStream_t)stream, false, &tc));
}

vla_status vla_op_attention_prefill(const void* q, const void* k_plane, const void* v_plane, int n_tokens,
                                    int n_heads, int n_kv_heads, int head_dim, int max_ctx, int pos0, void* out,
                                    vla_stream stream) {
    if (!q || !k_plane || !v_plane || !out || n_tokens < 0 || n_heads <= 0 || n_kv_heads <= 0 || pos0 < 0 ||
        max_ctx <= 0)
        return VLA_ERR_INVALID_ARG;
    if (n_heads % n_kv_heads) return VLA_ERR_INVALID_ARG;
    if (head_dim != 64 && head_dim != 128) return VLA_ERR_UNSUPPORTED;
    if ((long long)pos0 + n_tokens > max_ctx) return VLA_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_plane) || !aligned16(v_plane) || !aligned16(out)) return VLA_ERR_INVALID_ARG;
    vla::AttnPrefillParams ap = {};
    ap.q = (const bf16*)q;
    ap.ld_q = n_heads * head_dim;
    ap.kc = (const bf16*)k_plane;
    ap.vc = (const bf16*)v_plane;
    ap.out = (bf16*)out;
    ap.ld_out = n_heads * head_dim;
    ap.M = n_tokens;
    ap.H = n_heads;
    ap.Hkv = n_kv_heads;
    ap.head_dim = head_dim;
    ap.max_ctx = max_ctx;
    ap.pos0 = pos0;
    ap.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)head_dim));
    return cuda_status(vla::launch_attn_prefill_tc(ap, nullptr, (cudaStream_t)stream));
}

}  // extern "C"
