// engine.cu - the C ABI of libssd (include/ssd.h): handle, buffers, the
// forward sequence of one decoder step, CUDA-graph capture of the draft step
// and of the verification step, and the decoding loop of self-speculative
// decoding (arxiv 2309.08168, Algorithms 1, 2 and 4).
//
// Decoding loop, one round (Sec. 3.2):
//   draft  : K_eff replays of the draft-step graph; each runs the forward of
//            one token through the sublayers outside the skip set z, writes KV
//            only in the attention sublayers it runs, and appends d_j;
//   verify : one replay of the verification graph for M = K_eff + 1 rows
//            [x_last, d_1 .. d_K_eff] at positions len .. len + K_eff, which
//            rewrites KV for every layer and ends in the acceptance kernel;
//   accept : n accepted drafts plus a correction / bonus token are emitted,
//            len <- len + 1 + n (the KV rollback is this length pointer).
// Everything between two rounds stays on the device; the host reads one int
// (tokens emitted so far) per round to size the next round.
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "ssd.h"
#include "ssd_internal.cuh"

using namespace ssd;

namespace ssd {
int sampling_configure();
}

namespace {

thread_local std::string g_err;

int fail(int code, const std::string& msg) {
    g_err = msg;
    return code;
}

#define CUDA_TRY(expr, what)                                                                    \
    do {                                                                                        \
        cudaError_t _e = (cudaError_t)(expr);                                                   \
        if (_e != cudaSuccess)                                                                  \
            return fail(SSD_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(_e));     \
    } while (0)

// Debug mode (SSD_SYNC_CHECK=1 in the environment at ssd_create): every
// launch outside graph capture is followed by a stream synchronisation, so a
// failing kernel is reported by name and layer.
#define LAUNCH(h, expr, what, layer)                                                            \
    do {                                                                                        \
        CUDA_TRY(expr, what);                                                                   \
        if ((h)->sync_check) {                                                                  \
            cudaStreamCaptureStatus _cs = cudaStreamCaptureStatusNone;                           \
            cudaStreamIsCapturing((h)->stream, &_cs);                                           \
            if (_cs == cudaStreamCaptureStatusNone) {                                           \
                cudaError_t _s = cudaStreamSynchronize((h)->stream);                            \
                if (_s != cudaSuccess)                                                          \
                    return fail(SSD_ERR_CUDA, std::string(what) + " (layer " +                 \
                                                  std::to_string(layer) + "): " + cudaGetErrorString(_s)); \
            }                                                                                   \
        }                                                                                       \
    } while (0)

enum GraphKind { G_DRAFT = 0, G_VERIFY = 1 };

}  // namespace

struct ssd_handle {
    ssd_config cfg{};
    int device = 0;
    cudaStream_t stream = nullptr;
    bool own_stream = false;

    const bf16* embed = nullptr;
    const bf16* final_norm = nullptr;
    const bf16* lm_head = nullptr;
    std::vector<const bf16*> wq, wk, wv, wo, attn_norm, w_gate, w_up, w_down, mlp_norm;
    std::vector<void*> owned;  // weight copies (on_device = 0)
    std::vector<void*> bufs;   // work buffers
    std::vector<uint8_t> mask;
    float temperature = 1.f, top_p = 1.f;
    // adaptive draft exit (ssd_set_draft_exit)
    int exit_on = 0;
    float gamma0 = 0.f, alpha = 0.f, eps = 0.f, beta1 = 0.f, beta2 = 1.f;

    // device buffers
    f16* kc = nullptr;   // [L][Hkv][max_seq][hd] fp16
    f16* vc = nullptr;
    size_t kv_layer = 0;  // elements per layer of one of K / V
    float* h = nullptr;
    bf16* xn_hi = nullptr;  // planes of h * g (input of the next normed projection) [2][16][d]
    bf16* xn_lo = nullptr;  // = xn_hi + 16 * d
    float* ss = nullptr;    // per-128-column sums of h^2 [16][d/128]
    float* q = nullptr;
    bf16* at_hi = nullptr;  // attention output planes [16][H*hd]
    bf16* at_lo = nullptr;
    bf16* ac_hi = nullptr;  // SwiGLU output planes [16][ffn]
    bf16* ac_lo = nullptr;
    int n_sms = 0;
    unsigned* bar = nullptr;            // grid-barrier counter of the forward kernel, then its sequence number
    unsigned long long* trace = nullptr;  // per-op timestamps (profiling hook, FwdParams::trace)
    int trace_op = -1;                    // op traced per unit and per CTA
    CUtensorMap* tmaps = nullptr;       // TMA descriptors (weights, input planes) in device memory
    int n_tmaps = 0;
    FwdOp* ops_full = nullptr;          // op lists in device memory
    FwdOp* ops_draft = nullptr;
    int n_ops_full = 0, n_ops_draft = 0, max_ops = 0;
    float* logits = nullptr;
    float* p_rows = nullptr;
    float* q_rows = nullptr;
    float* partial = nullptr;
    unsigned* counters = nullptr;  // [4]: the acceptance kernels' arrival counter (+ spare words)
    float* attn_part = nullptr;
    int n_chunks = 0;
    float2* rope = nullptr;
    int* tok = nullptr;  // [max_seq] prompt | [16] debug rows
    int* out = nullptr;  // [max_seq]
    int* argbuf = nullptr;
    DecodeState* st = nullptr;
    DecodeState* st_host = nullptr;  // pinned staging
    int* emitted_host = nullptr;     // pinned

    std::map<int, cudaGraphExec_t> graphs;
    std::map<int, int> graph_launches;  // kernels per replay
    std::vector<cudaEvent_t> events;

    bool prefilled = false;
    int n_prompt = 0;
    int last_prompt_token = 0;
    bool sync_check = false;
    // prefill on the tensor cores (prefill.cu): plan, per-layer arguments and
    // TMA maps (box 64 x 128); used for prompts of more than 16 rows
    bool pf_on = false;
    PrefillPlan pf{};
    std::vector<PrefillLayer> pf_layers;
    CUtensorMap* pf_tmaps = nullptr;
    // bounded waits of the forward kernel; test hook: one forward of
    // ssd_debug_forward with an unreachable grid barrier (ssd_debug_stall_barrier)
    unsigned long long wait_ns = 2000000000ull;
    int stall_barrier = 0;
    unsigned long long stall_wait_ns = 0;
};

namespace {

int graph_key(int kind, int M, int mode) { return (mode * 2 + kind) * 64 + M; }

void drop_graphs(ssd_handle* h, int kind) {
    for (auto it = h->graphs.begin(); it != h->graphs.end();) {
        if (kind < 0 || ((it->first / 64) % 2) == kind) {
            cudaGraphExecDestroy(it->second);
            h->graph_launches.erase(it->first);
            it = h->graphs.erase(it);
        } else {
            ++it;
        }
    }
}

// Gains of the RMSNorm in front of the first sublayer that runs after
// sublayer index s (s = 2l + t, t = 0 attention, 1 MLP), or the final norm.
const bf16* next_norm(const ssd_handle* h, int s, bool draft) {
    for (int n = s + 1; n < 2 * h->cfg.n_layers; ++n) {
        if (draft && h->mask[n]) continue;
        return (n & 1) ? h->mlp_norm[n >> 1] : h->attn_norm[n >> 1];
    }
    return h->final_norm;
}

// ---------------------------------------------------------------------------
// TMA descriptors.  Index layout: layer l's wq wk wv wo w_gate w_up w_down at
// 7l + 0..6, lm_head at 7L, then the input-plane maps at 7L + 1 + buf * 4 + cls
// with buf 0 = normalised rows (K = d), 1 = attention output (K = H*hd),
// 2 = SwiGLU output (K = ffn) and cls = rows per plane 1 | 4 | 8 | 12 | 16, then the
// K and V cache maps.
// ---------------------------------------------------------------------------
size_t trace_words(const ssd_handle* h) { return (size_t)kTraceCtas + 8 * (size_t)h->n_sms; }

int tmap_weight(int l, int which) { return 7 * l + which; }
int tmap_x(const ssd_handle* h, int buf, int cls) { return 7 * h->cfg.n_layers + 1 + buf * kPlaneClasses + cls; }
int tmap_kv(const ssd_handle* h, int v) { return 7 * h->cfg.n_layers + 1 + 3 * kPlaneClasses + v; }

// Checks the TMA rules and encodes a 16-bit tensor map with 64-element (128-byte)
// inner boxes, 128-byte swizzle, zero fill out of range: base 16-byte aligned,
// strides multiples of 16 bytes.
int encode_map(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap* m, const void* base, int rank,
               const cuuint64_t* dims, const cuuint64_t* strides, const cuuint32_t* box,
               CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
    if ((uintptr_t)base & 15u) return fail(SSD_ERR_INVALID_ARG, "tensor base not 16-byte aligned for TMA");
    for (int i = 0; i + 1 < rank; ++i)
        if (strides[i] % 16) return fail(SSD_ERR_INVALID_ARG, "tensor stride not a multiple of 16 bytes for TMA");
    if (dims[0] < 64 || box[0] != 64) return fail(SSD_ERR_INVALID_ARG, "tensor row shorter than one TMA box");
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = enc(m, dtype, (cuuint32_t)rank, const_cast<void*>(base), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(SSD_ERR_CUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
    return SSD_OK;
}

// weight matrix [rows][K] bf16 viewed as {K, rows}, box 64 (k) x box_rows:
// one copy per 64-wide k box of a forward-kernel work unit (128 rows; 64 for
// the gate and up halves of a SwiGLU tile), written in the 128-byte-swizzled
// K-major layout tcgen05.mma reads
int encode_weight(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap* m, const void* base, int K, int rows,
                  int box_rows) {
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    return encode_map(enc, m, base, 2, dims, strides, box);
}

// input planes [2][16][K] bf16 (hi plane, lo plane) viewed as {K, 16, 2}, box
// {64, R, 2}: one copy per 64-wide k box holds the R hi rows, then the R lo
// rows, 128 bytes each (the N side of tcgen05.mma)
int encode_planes(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap* m, const void* base, int K, int R) {
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)kMaxRows, 2};
    cuuint64_t strides[2] = {(cuuint64_t)K * 2, (cuuint64_t)K * 2 * kMaxRows};
    cuuint32_t box[3] = {64, (cuuint32_t)R, 2};
    return encode_map(enc, m, base, 3, dims, strides, box);
}

int build_tmaps(ssd_handle* h) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    CUDA_TRY(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q),
             "driver entry point");
    if (!fn || q != cudaDriverEntryPointSuccess) return fail(SSD_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    auto enc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    const ssd_config& c = h->cfg;
    const int L = c.n_layers, d = c.d_model, qd = c.n_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
    std::vector<CUtensorMap> maps((size_t)h->n_tmaps);
    int rc = 0;
    for (int l = 0; l < L && !rc; ++l) {
        const bf16* w[7] = {h->wq[l], h->wk[l], h->wv[l], h->wo[l], h->w_gate[l], h->w_up[l], h->w_down[l]};
        const int K[7] = {d, d, d, qd, d, d, c.ffn};
        const int N[7] = {qd, kvd, kvd, d, c.ffn, c.ffn, d};
        for (int i = 0; i < 7 && !rc; ++i)
            rc = encode_weight(enc, &maps[tmap_weight(l, i)], w[i], K[i], N[i], (i == 4 || i == 5) ? 64 : kFTile);
    }
    if (!rc) rc = encode_weight(enc, &maps[7 * L], h->lm_head, d, c.vocab, kFTile);
    const bf16* planes[3] = {h->xn_hi, h->at_hi, h->ac_hi};
    const int widths[3] = {d, qd, c.ffn};
    const int rows[kPlaneClasses] = {1, 4, 8, 12, 16};
    for (int b = 0; b < 3 && !rc; ++b)
        for (int cls = 0; cls < kPlaneClasses && !rc; ++cls)
            rc = encode_planes(enc, &maps[tmap_x(h, b, cls)], planes[b], widths[b], rows[cls]);
    // K / V cache [L][Hkv][max_seq][hd] fp16 as {hd, max_seq, L * Hkv}, box 64 dims x 64 positions
    for (int v = 0; v < 2 && !rc; ++v) {
        cuuint64_t dims[3] = {(cuuint64_t)c.head_dim, (cuuint64_t)c.max_seq, (cuuint64_t)L * c.n_kv_heads};
        cuuint64_t strides[2] = {(cuuint64_t)c.head_dim * 2, (cuuint64_t)c.max_seq * c.head_dim * 2};
        cuuint32_t box[3] = {64, (cuuint32_t)kAttnChunk, 1};
        rc = encode_map(enc, &maps[tmap_kv(h, v)], v ? h->vc : h->kc, 3, dims, strides, box,
                        CU_TENSOR_MAP_DATA_TYPE_FLOAT16);
    }
    if (rc) return rc;
    CUDA_TRY(cudaMemcpy(h->tmaps, maps.data(), maps.size() * sizeof(CUtensorMap), cudaMemcpyHostToDevice),
             "tensor map upload");
    return SSD_OK;
}

// TMA maps of the prefill GEMMs: every matrix [rows][K] bf16 viewed as
// {K, rows}, box 64 (k) x 128 rows, 128-byte swizzle (the tcgen05 operand
// layout); layer l's wq wk wv wo w_gate w_up w_down at 7l + 0..6, then the
// activation planes x hi / lo, attention output hi / lo, SwiGLU output hi / lo.
int build_prefill(ssd_handle* h) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    CUDA_TRY(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q),
             "driver entry point");
    if (!fn || q != cudaDriverEntryPointSuccess) return fail(SSD_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    auto enc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    const ssd_config& c = h->cfg;
    const int L = c.n_layers, d = c.d_model, qd = c.n_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
    PrefillPlan& P = h->pf;
    std::vector<CUtensorMap> maps((size_t)7 * L + 6);
    auto map2 = [&](CUtensorMap* m, const void* base, int K, int rows) {
        cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
        cuuint64_t strides[1] = {(cuuint64_t)K * 2};
        cuuint32_t box[2] = {64, 128};
        return encode_map(enc, m, base, 2, dims, strides, box);
    };
    int rc = 0;
    for (int l = 0; l < L && !rc; ++l) {
        const bf16* w[7] = {h->wq[l], h->wk[l], h->wv[l], h->wo[l], h->w_gate[l], h->w_up[l], h->w_down[l]};
        const int K[7] = {d, d, d, qd, d, d, c.ffn};
        const int N[7] = {qd, kvd, kvd, d, c.ffn, c.ffn, d};
        for (int i = 0; i < 7 && !rc; ++i) rc = map2(&maps[7 * l + i], w[i], K[i], N[i]);
    }
    const size_t a0 = (size_t)7 * L;
    if (!rc) rc = map2(&maps[a0 + 0], P.x_hi, d, P.rows);
    if (!rc) rc = map2(&maps[a0 + 1], P.x_lo, d, P.rows);
    if (!rc) rc = map2(&maps[a0 + 2], P.at_hi, qd, P.rows);
    if (!rc) rc = map2(&maps[a0 + 3], P.at_lo, qd, P.rows);
    if (!rc) rc = map2(&maps[a0 + 4], P.ac_hi, c.ffn, P.rows);
    if (!rc) rc = map2(&maps[a0 + 5], P.ac_lo, c.ffn, P.rows);
    if (rc) return rc;
    CUDA_TRY(cudaMemcpy(h->pf_tmaps, maps.data(), maps.size() * sizeof(CUtensorMap), cudaMemcpyHostToDevice),
             "prefill tensor map upload");
    h->pf_layers.resize(L);
    for (int l = 0; l < L; ++l) {
        PrefillLayer& Ly = h->pf_layers[l];
        for (int i = 0; i < 7; ++i) Ly.tm_w[i] = h->pf_tmaps + 7 * l + i;
        Ly.attn_norm = h->attn_norm[l];
        Ly.mlp_norm = h->mlp_norm[l];
        Ly.k_cache = h->kc + (size_t)l * h->kv_layer;
        Ly.v_cache = h->vc + (size_t)l * h->kv_layer;
    }
    P.tm_x[0] = h->pf_tmaps + a0 + 0;
    P.tm_x[1] = h->pf_tmaps + a0 + 1;
    P.tm_at[0] = h->pf_tmaps + a0 + 2;
    P.tm_at[1] = h->pf_tmaps + a0 + 3;
    P.tm_ac[0] = h->pf_tmaps + a0 + 4;
    P.tm_ac[1] = h->pf_tmaps + a0 + 5;
    P.layers = h->pf_layers.data();
    return SSD_OK;
}

void set_x_maps(const ssd_handle* h, GemmArgs& a, int buf) {
    for (int cls = 0; cls < kPlaneClasses; ++cls) a.tm_x[cls] = h->tmaps + tmap_x(h, buf, cls);
}

// One projection op: fills the fields every projection shares.
GemmArgs proj_args(ssd_handle* h, int N, int K, int n_tiles) {
    GemmArgs a{};
    a.N = N;
    a.K = K;
    a.n_tiles = n_tiles;
    a.n_chunks = (K + kFKC - 1) / kFKC;
    a.n_units = n_tiles * a.n_chunks;
    a.partial = h->partial;
    a.err = &h->st->err;
    a.inv_dim = 1.0f / (float)h->cfg.d_model;
    a.eps = h->cfg.rms_eps;
    return a;
}

// The op list of one forward: embedding, the sublayers that run (all of them,
// or those outside the skip set for the draft model), lm_head last.
// RMSNorm is folded into the projections: whoever produces the residual
// stream also writes the bf16 hi / lo planes of h * g_next and per-128-column
// sums of h^2; the consuming projection scales row m by rsqrt(mean(h^2) + eps).
std::vector<FwdOp> build_ops(ssd_handle* h, bool draft) {
    const ssd_config& c = h->cfg;
    const int d = c.d_model, qd = c.n_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
    const int d_tiles = d / kFTile;
    std::vector<FwdOp> ops;
    FwdOp e{};
    e.type = OP_EMBED;
    ops.push_back(e);
    for (int l = 0; l < c.n_layers; ++l) {
        const bool run_a = !(draft && h->mask[2 * l]);
        const bool run_m = !(draft && h->mask[2 * l + 1]);
        if (run_a) {
            FwdOp q{};
            q.type = OP_QKV;
            GemmArgs& a = q.g;
            a = proj_args(h, qd + 2 * kvd, d, (qd + 2 * kvd) / kFTile);
            a.w0 = h->wq[l]; a.w1 = h->wk[l]; a.w2 = h->wv[l];
            a.tm_w[0] = h->tmaps + tmap_weight(l, 0);
            a.tm_w[1] = h->tmaps + tmap_weight(l, 1);
            a.tm_w[2] = h->tmaps + tmap_weight(l, 2);
            set_x_maps(h, a, 0);
            a.ss_in = h->ss; a.ss_in_tiles = d_tiles;
            a.n_heads = c.n_heads; a.n_kv_heads = c.n_kv_heads; a.head_dim = c.head_dim;
            a.max_seq = c.max_seq; a.q_out = h->q;
            a.k_cache = h->kc + (size_t)l * h->kv_layer;
            a.v_cache = h->vc + (size_t)l * h->kv_layer;
            a.rope = h->rope;
            ops.push_back(q);
            FwdOp at{};
            at.type = OP_ATTN;
            AttnArgs& t = at.at;
            t.q = h->q;
            t.tm_k = h->tmaps + tmap_kv(h, 0); t.tm_v = h->tmaps + tmap_kv(h, 1); t.kv_z0 = l * c.n_kv_heads;
            t.out_hi = h->at_hi; t.out_lo = h->at_lo;
            t.part = h->attn_part;
            t.n_heads = c.n_heads; t.n_kv_heads = c.n_kv_heads; t.head_dim = c.head_dim;
            t.max_seq = c.max_seq; t.n_chunks = h->n_chunks;
            t.scale = 1.0f / std::sqrt((float)c.head_dim); t.st = h->st; t.err = &h->st->err;
            ops.push_back(at);
            FwdOp o{};
            o.type = OP_RESID;
            o.g = proj_args(h, d, qd, d_tiles);
            o.g.w0 = h->wo[l];
            o.g.tm_w[0] = h->tmaps + tmap_weight(l, 3);
            set_x_maps(h, o.g, 1);
            o.g.out_f32 = h->h; o.g.ldo = d;
            o.g.g_next = next_norm(h, 2 * l, draft); o.g.xo_hi = h->xn_hi; o.g.xo_lo = h->xn_lo; o.g.ss_out = h->ss;
            ops.push_back(o);
        }
        if (run_m) {
            FwdOp gu{};
            gu.type = OP_SWIGLU;
            gu.g = proj_args(h, 2 * c.ffn, d, (c.ffn + 63) / 64);
            gu.g.w0 = h->w_gate[l]; gu.g.w1 = h->w_up[l];
            gu.g.tm_w[0] = h->tmaps + tmap_weight(l, 4);
            gu.g.tm_w[1] = h->tmaps + tmap_weight(l, 5);
            set_x_maps(h, gu.g, 0);
            gu.g.ss_in = h->ss; gu.g.ss_in_tiles = d_tiles;
            gu.g.ffn = c.ffn; gu.g.xo_hi = h->ac_hi; gu.g.xo_lo = h->ac_lo;
            ops.push_back(gu);
            FwdOp w{};
            w.type = OP_RESID;
            w.g = proj_args(h, d, c.ffn, d_tiles);
            w.g.w0 = h->w_down[l];
            w.g.tm_w[0] = h->tmaps + tmap_weight(l, 6);
            set_x_maps(h, w.g, 2);
            w.g.out_f32 = h->h; w.g.ldo = d;
            w.g.g_next = next_norm(h, 2 * l + 1, draft); w.g.xo_hi = h->xn_hi; w.g.xo_lo = h->xn_lo; w.g.ss_out = h->ss;
            ops.push_back(w);
        }
    }
    FwdOp lg{};
    lg.type = OP_LOGITS;
    lg.g = proj_args(h, c.vocab, d, (c.vocab + kFTile - 1) / kFTile);
    lg.g.w0 = h->lm_head;
    lg.g.tm_w[0] = h->tmaps + 7 * c.n_layers;
    set_x_maps(h, lg.g, 0);
    lg.g.ss_in = h->ss; lg.g.ss_in_tiles = d_tiles;
    lg.g.out_f32 = h->logits; lg.g.ldo = c.vocab;
    ops.push_back(lg);
    return ops;
}

// (Re)builds the op lists in device memory (outside any stream capture).
int upload_ops(ssd_handle* h, bool draft) {
    std::vector<FwdOp> ops = build_ops(h, draft);
    FwdOp* dst = draft ? h->ops_draft : h->ops_full;
    CUDA_TRY(cudaMemcpy(dst, ops.data(), ops.size() * sizeof(FwdOp), cudaMemcpyHostToDevice), "op list upload");
    (draft ? h->n_ops_draft : h->n_ops_full) = (int)ops.size();
    return SSD_OK;
}

// One decoder forward over M rows: a single cooperative launch of the forward
// kernel over the op list (lm_head dropped when no logits are needed).
// Launches only; no host synchronisation (graph-capturable).
int forward(ssd_handle* h, int M, int src, const int* toks, int pos0, bool draft, bool logits,
            int* n_launch = nullptr, unsigned long long* trace = nullptr, int stall_barrier = 0) {
    const ssd_config& c = h->cfg;
    FwdParams p{};
    p.ops = draft ? h->ops_draft : h->ops_full;
    p.n_ops = (draft ? h->n_ops_draft : h->n_ops_full) - (logits ? 0 : 1);
    p.M = M;
    p.src = src;
    p.toks = toks;
    p.pos0_arg = pos0;
    p.st = h->st;
    p.embed = h->embed;
    p.d = c.d_model;
    p.g0 = next_norm(h, -1, draft);
    p.h = h->h;
    p.xn_hi = h->xn_hi;
    p.xn_lo = h->xn_lo;
    p.ss = h->ss;
    p.bar = h->bar;
    p.seq = h->bar + 1;
    p.err = &h->st->err;
    p.trace = trace;
    p.trace_op = h->trace_op;
    p.wait_ns = h->wait_ns;
    p.stall_barrier = stall_barrier;
    CUDA_TRY(cudaMemsetAsync(h->bar, 0, sizeof(unsigned), h->stream), "barrier reset");
    LAUNCH(h, launch_forward(p, c.head_dim, h->n_sms, h->stream), "forward kernel", -1);
    if (n_launch) *n_launch = 1;
    return SSD_OK;
}

// Weight bytes one forward streams (bf16): the matrices and norm gains of
// every sublayer that runs, one embedding row, the final norm and lm_head.
double forward_weight_bytes(const ssd_handle* h, bool draft, bool gemm_only) {
    const ssd_config& c = h->cfg;
    const double d = c.d_model, qd = (double)c.n_heads * c.head_dim, kvd = (double)c.n_kv_heads * c.head_dim;
    const double attn = (qd * d + 2 * kvd * d + d * qd) * 2 + (gemm_only ? 0 : d * 2);
    const double mlp = 3.0 * c.ffn * d * 2 + (gemm_only ? 0 : d * 2);
    double b = (double)c.vocab * d * 2 + (gemm_only ? 0 : 2 * d * 2);
    for (int l = 0; l < c.n_layers; ++l) {
        if (!(draft && h->mask[2 * l])) b += attn;
        if (!(draft && h->mask[2 * l + 1])) b += mlp;
    }
    return b;
}

unsigned* accept_counter(ssd_handle* h) { return h->counters; }

int step_launches(ssd_handle* h, int kind, int M, int mode, int* n_launch) {
    const int V = h->cfg.vocab;
    int n = 0;
    if (kind == G_DRAFT) {
        int rc = forward(h, 1, SRC_DRAFT, nullptr, 0, true, true, &n);
        if (rc) return rc;
        *n_launch = n + 1;
        if (mode == SSD_GREEDY) CUDA_TRY(launch_greedy_draft(h->logits, V, h->st, h->stream), "draft argmax");
        else CUDA_TRY(launch_sample_draft(h->logits, V, h->st, h->q_rows, h->stream), "draft sample");
        return SSD_OK;
    }
    int rc = forward(h, M, SRC_VERIFY, nullptr, 0, false, true, &n);
    if (rc) return rc;
    *n_launch = n + 1;
    if (mode == SSD_GREEDY)
        CUDA_TRY(launch_greedy_accept(h->logits, V, M, h->st, h->out, accept_counter(h), h->argbuf,
                                      h->stream), "greedy accept");
    else
        CUDA_TRY(launch_sample_accept(h->logits, V, M, h->st, h->p_rows, h->q_rows, h->out,
                                      accept_counter(h), h->stream), "sample accept");
    return SSD_OK;
}

int get_graph(ssd_handle* h, int kind, int M, int mode, cudaGraphExec_t* out, int* n_launch) {
    const int key = graph_key(kind, M, mode);
    auto it = h->graphs.find(key);
    if (it != h->graphs.end()) {
        *out = it->second;
        *n_launch = h->graph_launches[key];
        return SSD_OK;
    }
    cudaGraph_t g = nullptr;
    CUDA_TRY(cudaStreamBeginCapture(h->stream, cudaStreamCaptureModeThreadLocal), "begin capture");
    int rc = step_launches(h, kind, M, mode, n_launch);
    cudaError_t e = cudaStreamEndCapture(h->stream, &g);
    if (rc) { if (g) cudaGraphDestroy(g); return rc; }
    CUDA_TRY(e, "end capture");
    cudaGraphExec_t exec = nullptr;
    e = cudaGraphInstantiate(&exec, g, 0);
    cudaGraphDestroy(g);
    CUDA_TRY(e, "graph instantiate");
    h->graphs[key] = exec;
    h->graph_launches[key] = *n_launch;
    *out = exec;
    return SSD_OK;
}

template <typename T>
int dalloc(ssd_handle* h, T** p, size_t n, std::vector<void*>* track) {
    (void)h;
    void* v = nullptr;
    cudaError_t e = cudaMalloc(&v, n * sizeof(T) + 16);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(SSD_ERR_OOM, std::string("cudaMalloc failed: ") + cudaGetErrorString(e));
    }
    track->push_back(v);
    *p = (T*)v;
    return SSD_OK;
}

void free_all(ssd_handle* h, std::vector<void*>& v) {
    for (void* p : v) cudaFree(p);
    v.clear();
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int check_config(const ssd_config* c) {
    if (!c) return fail(SSD_ERR_INVALID_ARG, "config is NULL");
    if (c->n_layers < 1 || c->d_model < 128 || c->d_model % 128)
        return fail(SSD_ERR_INVALID_ARG, "n_layers >= 1 and d_model a positive multiple of 128 required");
    if (c->head_dim != 64 && c->head_dim != 128)
        return fail(SSD_ERR_INVALID_ARG, "head_dim must be 64 or 128");
    if (c->n_heads < 1 || c->n_kv_heads < 1 || c->n_heads % c->n_kv_heads)
        return fail(SSD_ERR_INVALID_ARG, "n_heads must be a positive multiple of n_kv_heads");
    if ((c->n_heads * c->head_dim) % 128 || (c->n_kv_heads * c->head_dim) % 128)
        return fail(SSD_ERR_INVALID_ARG, "n_heads * head_dim and n_kv_heads * head_dim must be multiples of 128");
    if (c->ffn < 64 || c->ffn % 16) return fail(SSD_ERR_INVALID_ARG, "ffn must be a multiple of 16, at least 64");
    if (c->vocab < 2 || c->vocab > 32768) return fail(SSD_ERR_INVALID_ARG, "vocab must be in [2, 32768]");
    if (c->max_seq < 2 || c->max_seq > (1 << 24)) return fail(SSD_ERR_INVALID_ARG, "max_seq out of range");
    if (!(c->rms_eps > 0.f) || !(c->rope_theta > 0.f))
        return fail(SSD_ERR_INVALID_ARG, "rms_eps and rope_theta must be positive");
    return SSD_OK;
}

}  // namespace

namespace ssd {
// Records the message that ssd_last_error() returns on this thread.
int set_last_error(int code, const char* msg) { return fail(code, msg); }
}  // namespace ssd

extern "C" {

const char* ssd_last_error(void) { return g_err.c_str(); }

void ssd_destroy(ssd_handle* h) {
    if (!h) return;
    cudaSetDevice(h->device);
    if (h->stream) cudaStreamSynchronize(h->stream);
    drop_graphs(h, -1);
    for (cudaEvent_t e : h->events) cudaEventDestroy(e);
    free_all(h, h->bufs);
    free_all(h, h->owned);
    if (h->st_host) cudaFreeHost(h->st_host);
    if (h->emitted_host) cudaFreeHost(h->emitted_host);
    if (h->own_stream && h->stream) cudaStreamDestroy(h->stream);
    delete h;
}

int ssd_create(const ssd_config* cfg, const ssd_weights* w, void* cuda_stream, ssd_handle** out) {
    if (!out) return fail(SSD_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    int rc = check_config(cfg);
    if (rc) return rc;
    if (!w || !w->embed || !w->final_norm || !w->lm_head || !w->wq || !w->wk || !w->wv || !w->wo ||
        !w->attn_norm || !w->w_gate || !w->w_up || !w->w_down || !w->mlp_norm)
        return fail(SSD_ERR_INVALID_ARG, "weights: NULL member");
    if (w->on_device != 0 && w->on_device != 1) return fail(SSD_ERR_INVALID_ARG, "weights.on_device must be 0 or 1");
    const ssd_config c = *cfg;
    const int L = c.n_layers, d = c.d_model, qd = c.n_heads * c.head_dim, kvd = c.n_kv_heads * c.head_dim;
    for (int l = 0; l < L; ++l)
        if (!w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->attn_norm[l] || !w->w_gate[l] ||
            !w->w_up[l] || !w->w_down[l] || !w->mlp_norm[l])
            return fail(SSD_ERR_INVALID_ARG, "weights: NULL layer tensor");

    ssd_handle* h = new ssd_handle();
    h->cfg = c;
    {
        const char* sc = std::getenv("SSD_SYNC_CHECK");
        h->sync_check = sc && sc[0] == '1';
    }
    cudaGetDevice(&h->device);
    auto bail = [&](int code) { ssd_destroy(h); return code; };
    if (cuda_stream) {
        h->stream = (cudaStream_t)cuda_stream;
    } else {
        cudaError_t e = cudaStreamCreateWithFlags(&h->stream, cudaStreamNonBlocking);
        if (e != cudaSuccess) return bail(fail(SSD_ERR_CUDA, std::string("stream: ") + cudaGetErrorString(e)));
        h->own_stream = true;
    }
    {
        int e1 = forward_configure(), e2 = gemm_configure(), e3 = sampling_configure();
        int e = e1 ? e1 : (e2 ? e2 : e3);
        if (!e) e = (int)cudaDeviceGetAttribute(&h->n_sms, cudaDevAttrMultiProcessorCount, h->device);
        if (e) return bail(fail(SSD_ERR_CUDA, std::string("kernel setup: ") + cudaGetErrorString((cudaError_t)e)));
    }

    // weights: borrow device pointers or copy host tensors
    auto take = [&](const void* src, size_t elems, const bf16** dst) -> int {
        if (w->on_device) {
            if (!aligned16(src)) return fail(SSD_ERR_INVALID_ARG, "device weight pointer not 16-byte aligned");
            *dst = (const bf16*)src;
            return SSD_OK;
        }
        bf16* p = nullptr;
        int r = dalloc(h, &p, elems, &h->owned);
        if (r) return r;
        cudaError_t e = cudaMemcpy(p, src, elems * 2, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return fail(SSD_ERR_CUDA, std::string("weight copy: ") + cudaGetErrorString(e));
        *dst = p;
        return SSD_OK;
    };
    const size_t V = c.vocab, F = c.ffn;
    if ((rc = take(w->embed, V * d, &h->embed)) || (rc = take(w->final_norm, d, &h->final_norm)) ||
        (rc = take(w->lm_head, V * d, &h->lm_head)))
        return bail(rc);
    h->wq.resize(L); h->wk.resize(L); h->wv.resize(L); h->wo.resize(L); h->attn_norm.resize(L);
    h->w_gate.resize(L); h->w_up.resize(L); h->w_down.resize(L); h->mlp_norm.resize(L);
    for (int l = 0; l < L; ++l) {
        if ((rc = take(w->wq[l], (size_t)qd * d, &h->wq[l])) || (rc = take(w->wk[l], (size_t)kvd * d, &h->wk[l])) ||
            (rc = take(w->wv[l], (size_t)kvd * d, &h->wv[l])) || (rc = take(w->wo[l], (size_t)d * qd, &h->wo[l])) ||
            (rc = take(w->attn_norm[l], d, &h->attn_norm[l])) ||
            (rc = take(w->w_gate[l], F * d, &h->w_gate[l])) || (rc = take(w->w_up[l], F * d, &h->w_up[l])) ||
            (rc = take(w->w_down[l], (size_t)d * F, &h->w_down[l])) ||
            (rc = take(w->mlp_norm[l], d, &h->mlp_norm[l])))
            return bail(rc);
    }
    h->mask.assign(2 * L, 0);

    // plans
    // split-K slots of the forward kernel: [tile][segment <= chunks][16][128] tagged words
    size_t part = 0;
    {
        const int Ks[5] = {d, qd, d, c.ffn, d};
        const int tiles[5] = {(qd + 2 * kvd) / kFTile, d / kFTile, (c.ffn + 63) / 64, d / kFTile,
                              (c.vocab + kFTile - 1) / kFTile};
        for (int i = 0; i < 5; ++i) {
            const size_t chunks = (size_t)(Ks[i] + kFKC - 1) / kFKC;
            part = std::max(part, chunks * kMaxRows * (size_t)tiles[i] * kFTile);
        }
    }
    h->n_chunks = (c.max_seq + kAttnChunk - 1) / kAttnChunk;
    const int G = c.n_heads / c.n_kv_heads;

    // buffers
    std::vector<void*>& B = h->bufs;
    h->kv_layer = (size_t)c.n_kv_heads * c.max_seq * c.head_dim;
    const size_t HD = c.head_dim;
    if ((rc = dalloc(h, &h->kc, h->kv_layer * L, &B)) || (rc = dalloc(h, &h->vc, h->kv_layer * L, &B)) ||
        (rc = dalloc(h, &h->h, (size_t)kMaxRows * d, &B)) ||
        (rc = dalloc(h, &h->xn_hi, (size_t)2 * kMaxRows * d, &B)) ||
        (rc = dalloc(h, &h->ss, (size_t)kMaxRows * (d / kFTile), &B)) ||
        (rc = dalloc(h, &h->q, (size_t)kMaxRows * qd, &B)) ||
        (rc = dalloc(h, &h->at_hi, (size_t)2 * kMaxRows * qd, &B)) ||
        (rc = dalloc(h, &h->ac_hi, (size_t)2 * kMaxRows * F, &B)) ||
        (rc = dalloc(h, &h->logits, (size_t)kMaxRows * V, &B)) ||
        (rc = dalloc(h, &h->p_rows, (size_t)kMaxRows * V, &B)) ||
        (rc = dalloc(h, &h->q_rows, (size_t)kMaxRows * V, &B)) ||
        (rc = dalloc(h, &h->partial, 2 * part, &B)) ||  // tagged 64-bit words in the forward kernel
        (rc = dalloc(h, &h->counters, (size_t)4, &B)) ||
        (rc = dalloc(h, &h->attn_part, (size_t)c.n_kv_heads * h->n_chunks * G * kMaxRows * attn_part_floats((int)HD), &B)) ||
        (rc = dalloc(h, &h->rope, (size_t)c.max_seq * (HD / 2), &B)) ||
        (rc = dalloc(h, &h->tok, (size_t)c.max_seq + kMaxRows, &B)) ||
        (rc = dalloc(h, &h->out, (size_t)c.max_seq, &B)) || (rc = dalloc(h, &h->argbuf, 32, &B)) ||
        (rc = dalloc(h, &h->st, 1, &B)) || (rc = dalloc(h, &h->bar, 4, &B)))
        return bail(rc);
    h->max_ops = 2 + 5 * L;
    if (h->max_ops + 1 > 1024) return bail(fail(SSD_ERR_INVALID_ARG, "too many layers (at most 204)"));
    h->n_tmaps = 7 * L + 1 + 3 * kPlaneClasses + 2;
    if ((rc = dalloc(h, &h->tmaps, (size_t)h->n_tmaps, &B)) ||
        (rc = dalloc(h, &h->ops_full, (size_t)h->max_ops, &B)) ||
        (rc = dalloc(h, &h->ops_draft, (size_t)h->max_ops, &B)) ||
        (rc = dalloc(h, &h->trace, trace_words(h), &B)))
        return bail(rc);
    // the lo plane follows the hi plane: [2][16][K]
    h->xn_lo = h->xn_hi + (size_t)kMaxRows * d;
    h->at_lo = h->at_hi + (size_t)kMaxRows * qd;
    h->ac_lo = h->ac_hi + (size_t)kMaxRows * F;
    {
        cudaError_t e = cudaMallocHost(&h->st_host, sizeof(DecodeState));
        if (e == cudaSuccess) e = cudaMallocHost(&h->emitted_host, sizeof(int) * 4);
        if (e != cudaSuccess) return bail(fail(SSD_ERR_OOM, "pinned host allocation failed"));
    }
    // RoPE table (cos, sin) of pos * theta^(-2i/hd), computed in double
    {
        std::vector<float2> tab((size_t)c.max_seq * (HD / 2));
        for (int p = 0; p < c.max_seq; ++p)
            for (size_t i = 0; i < HD / 2; ++i) {
                double a = p * std::pow((double)c.rope_theta, -(2.0 * (double)i) / (double)HD);
                tab[(size_t)p * (HD / 2) + i] = make_float2((float)std::cos(a), (float)std::sin(a));
            }
        cudaError_t e = cudaMemcpy(h->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return bail(fail(SSD_ERR_CUDA, std::string("rope table: ") + cudaGetErrorString(e)));
    }
    cudaError_t e = cudaMemsetAsync(h->counters, 0, 4 * sizeof(unsigned), h->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->st, 0, sizeof(DecodeState), h->stream);
    // barrier counter and forward sequence number; split-K slots hold no
    // valid tag (a tag is never 0: GEMM ops have an op index >= 1)
    if (e == cudaSuccess) e = cudaMemsetAsync(h->bar, 0, 4 * sizeof(unsigned), h->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->partial, 0, 2 * part * sizeof(float), h->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->kc, 0, h->kv_layer * L * sizeof(f16), h->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->vc, 0, h->kv_layer * L * sizeof(f16), h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    if (e != cudaSuccess) return bail(fail(SSD_ERR_CUDA, std::string("init: ") + cudaGetErrorString(e)));
    if ((rc = build_tmaps(h)) || (rc = upload_ops(h, false)) || (rc = upload_ops(h, true))) return bail(rc);

    // prefill on the tensor cores: needs the q / k / v widths in whole
    // 128-row boxes; otherwise prompts run through the decode kernel
    h->pf_on = true;
    if (h->pf_on) {
        PrefillPlan& P = h->pf;
        P.n_layers = L;
        P.d = d;
        P.n_heads = c.n_heads;
        P.n_kv_heads = c.n_kv_heads;
        P.head_dim = c.head_dim;
        P.ffn = c.ffn;
        P.max_seq = c.max_seq;
        P.eps = c.rms_eps;
        P.rows = std::min(c.max_seq, 2048);
        P.embed = h->embed;
        P.rope = h->rope;
        P.err = &h->st->err;
        const size_t R = (size_t)P.rows;
        if ((rc = dalloc(h, &P.h, R * d, &B)) || (rc = dalloc(h, &P.x_hi, 2 * R * d, &B)) ||
            (rc = dalloc(h, &P.q, R * qd, &B)) || (rc = dalloc(h, &P.at_hi, 2 * R * qd, &B)) ||
            (rc = dalloc(h, &P.ac_hi, 2 * R * F, &B)) ||
            (rc = dalloc(h, &h->pf_tmaps, (size_t)7 * L + 6, &B)))
            return bail(rc);
        P.x_lo = P.x_hi + R * d;
        P.at_lo = P.at_hi + R * qd;
        P.ac_lo = P.ac_hi + R * F;
        int e4 = prefill_configure();
        if (e4) return bail(fail(SSD_ERR_CUDA, std::string("prefill setup: ") + cudaGetErrorString((cudaError_t)e4)));
        if ((rc = build_prefill(h))) return bail(rc);
    }
    *out = h;
    return SSD_OK;
}

int ssd_set_skip(ssd_handle* h, const uint8_t* mask, int n_sublayers) {
    if (!h || !mask) return fail(SSD_ERR_INVALID_ARG, "NULL handle or mask");
    if (n_sublayers != 2 * h->cfg.n_layers) return fail(SSD_ERR_INVALID_ARG, "n_sublayers must be 2 * n_layers");
    for (int i = 0; i < n_sublayers; ++i)
        if (mask[i] > 1) return fail(SSD_ERR_INVALID_ARG, "mask values must be 0 or 1");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    CUDA_TRY(cudaStreamSynchronize(h->stream), "sync");
    h->mask.assign(mask, mask + n_sublayers);
    drop_graphs(h, G_DRAFT);
    return upload_ops(h, true);
}

int ssd_set_sampling(ssd_handle* h, float temperature, float top_p) {
    if (!h) return fail(SSD_ERR_INVALID_ARG, "NULL handle");
    if (!(temperature > 0.f) || !(top_p > 0.f) || top_p > 1.f)
        return fail(SSD_ERR_INVALID_ARG, "temperature > 0 and 0 < top_p <= 1 required");
    h->temperature = temperature;
    h->top_p = top_p;
    return SSD_OK;
}

int ssd_set_draft_exit(ssd_handle* h, int enable, float gamma0, float alpha, float eps, float beta1,
                       float beta2) {
    if (!h) return fail(SSD_ERR_INVALID_ARG, "NULL handle");
    if (enable != 0 && enable != 1) return fail(SSD_ERR_INVALID_ARG, "enable must be 0 or 1");
    auto unit = [](float x) { return x >= 0.f && x <= 1.f; };
    if (enable && (!(gamma0 >= 0.f) || !(eps >= 0.f) || !unit(alpha) || !unit(beta1) || !unit(beta2)))
        return fail(SSD_ERR_INVALID_ARG, "need gamma0 >= 0, eps >= 0 and alpha, beta1, beta2 in [0, 1]");
    h->exit_on = enable;
    h->gamma0 = gamma0;
    h->alpha = alpha;
    h->eps = eps;
    h->beta1 = beta1;
    h->beta2 = beta2;
    return SSD_OK;
}

int ssd_prefill(ssd_handle* h, const int32_t* prompt, int n_prompt) {
    if (!h || !prompt) return fail(SSD_ERR_INVALID_ARG, "NULL handle or prompt");
    if (n_prompt < 1) return fail(SSD_ERR_INVALID_ARG, "n_prompt must be >= 1");
    if (n_prompt > h->cfg.max_seq) return fail(SSD_ERR_CAPACITY, "prompt longer than max_seq");
    for (int i = 0; i < n_prompt; ++i)
        if (prompt[i] < 0 || prompt[i] >= h->cfg.vocab) return fail(SSD_ERR_INVALID_ARG, "prompt token out of range");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    h->prefilled = false;
    CUDA_TRY(cudaMemsetAsync(&h->st->err, 0, sizeof(int), h->stream), "error flag reset");
    // the acceptance kernels' arrival counter is left at zero by every
    // completed launch; after a failed one it may not be, so a new prompt
    // starts from clean counters
    CUDA_TRY(cudaMemsetAsync(h->counters, 0, 4 * sizeof(unsigned), h->stream),
             "counter reset");
    if (n_prompt > 1)
        CUDA_TRY(cudaMemcpyAsync(h->tok, prompt, sizeof(int) * (n_prompt - 1), cudaMemcpyHostToDevice, h->stream),
                 "prompt upload");
    if (h->pf_on && n_prompt - 1 > kMaxRows) {
        // tensor-core prefill, chunks of up to pf.rows positions
        for (int p0 = 0; p0 < n_prompt - 1; p0 += h->pf.rows) {
            const int n = std::min(h->pf.rows, n_prompt - 1 - p0);
            int e = prefill_chunk(h->pf, h->tok + p0, n, p0, h->stream);
            if (e) return fail(SSD_ERR_CUDA, std::string("prefill: ") + cudaGetErrorString((cudaError_t)e));
            if (h->sync_check) CUDA_TRY(cudaStreamSynchronize(h->stream), "prefill chunk");
        }
    } else {
        for (int p0 = 0; p0 < n_prompt - 1; p0 += kMaxRows) {
            int M = std::min(kMaxRows, n_prompt - 1 - p0);
            int rc = forward(h, M, SRC_TOKENS, h->tok + p0, p0, false, false);
            if (rc) return rc;
        }
    }
    CUDA_TRY(cudaStreamSynchronize(h->stream), "prefill");
    {
        int derr = 0;
        CUDA_TRY(cudaMemcpy(&derr, &h->st->err, sizeof(int), cudaMemcpyDeviceToHost), "error flag");
        if (derr == kDevErrTimeout) return fail(SSD_ERR_TIMEOUT, "a wait of the forward kernel timed out");
    }
#ifdef SSD_CHECKED
    {
        int derr = 0;
        CUDA_TRY(cudaMemcpy(&derr, &h->st->err, sizeof(int), cudaMemcpyDeviceToHost), "error flag");
        if (derr) return fail(SSD_ERR_CUDA, "device check failed with code " + std::to_string(derr));
    }
#endif
    h->prefilled = true;
    h->n_prompt = n_prompt;
    h->last_prompt_token = prompt[n_prompt - 1];
    return SSD_OK;
}

int ssd_generate(ssd_handle* h, const int32_t* prompt, int n_prompt, int n_new, int K, ssd_mode mode,
                 uint64_t seed, int32_t* out_tokens, ssd_stats* stats) {
    if (!h) return fail(SSD_ERR_INVALID_ARG, "NULL handle");
    if (n_new < 0 || K < 0 || K > kMaxK) return fail(SSD_ERR_INVALID_ARG, "need n_new >= 0 and 0 <= K <= 15");
    if (mode != SSD_GREEDY && mode != SSD_SAMPLE) return fail(SSD_ERR_INVALID_ARG, "bad mode");
    if (n_new > 0 && !out_tokens) return fail(SSD_ERR_INVALID_ARG, "out_tokens is NULL");
    if (prompt) {
        int rc = ssd_prefill(h, prompt, n_prompt);
        if (rc) return rc;
    } else if (!h->prefilled) {
        return fail(SSD_ERR_STATE, "no prompt given and nothing prefilled");
    }
    if (h->n_prompt + n_new > h->cfg.max_seq) return fail(SSD_ERR_CAPACITY, "n_prompt + n_new exceeds max_seq");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    if (stats) std::memset(stats, 0, sizeof(*stats));
    if (n_new == 0) return SSD_OK;

    DecodeState* init = h->st_host;
    std::memset(init, 0, sizeof(DecodeState));
    init->len = h->n_prompt - 1;
    init->x_last = h->last_prompt_token;
    init->mode = (int)mode;
    init->inv_temperature = 1.0f / h->temperature;
    init->top_p = h->top_p;
    init->seed = (unsigned long long)seed;
    const bool exit_on = h->exit_on && K > 0;
    init->exit_on = exit_on;
    init->gamma = h->gamma0;
    init->alpha = h->alpha;
    init->eps = h->eps;
    init->beta1 = h->beta1;
    init->beta2 = h->beta2;
    CUDA_TRY(cudaMemcpyAsync(h->st, init, sizeof(DecodeState), cudaMemcpyHostToDevice, h->stream), "state upload");

    // graphs needed by this call (captured once, replayed every round)
    cudaGraphExec_t g_draft = nullptr;
    int draft_launches = 0;
    long long launches = 0;
    if (K > 0) {
        int rc = get_graph(h, G_DRAFT, 1, mode, &g_draft, &draft_launches);
        if (rc) return rc;
    }
    const size_t need_events = 3 * (size_t)n_new + 2;
    while (h->events.size() < need_events) {
        cudaEvent_t ev;
        CUDA_TRY(cudaEventCreate(&ev), "event create");
        h->events.push_back(ev);
    }
    CUDA_TRY(cudaEventRecord(h->events[0], h->stream), "event");
    int emitted = 0, round = 0;
    while (emitted < n_new) {
        const int Kd = std::min(K, n_new - emitted - 1);
        // (graphs are captured while the stream is idle)
        cudaGraphExec_t g_verify = nullptr;
        int verify_launches = 0;
        if (!(exit_on && Kd > 0)) {
            int rc = get_graph(h, G_VERIFY, Kd + 1, mode, &g_verify, &verify_launches);
            if (rc) return rc;
        }
        cudaEvent_t* ev = &h->events[2 + 3 * (size_t)round];
        CUDA_TRY(cudaEventRecord(ev[0], h->stream), "event");
        for (int j = 0; j < Kd; ++j) CUDA_TRY(cudaGraphLaunch(g_draft, h->stream), "draft step");
        CUDA_TRY(cudaEventRecord(ev[1], h->stream), "event");
        // with the draft exit the round's draft count is known on the device
        // only: read it before choosing the verification's row count
        int Kv = Kd;
        if (exit_on && Kd > 0) {
            CUDA_TRY(cudaMemcpyAsync(h->emitted_host + 2, &h->st->j, sizeof(int), cudaMemcpyDeviceToHost, h->stream),
                     "draft count read");
            CUDA_TRY(cudaStreamSynchronize(h->stream), "drafting stage");
            Kv = h->emitted_host[2];
            if (Kv < 1 || Kv > Kd) return fail(SSD_ERR_CUDA, "decode state corrupted");
            int rc = get_graph(h, G_VERIFY, Kv + 1, mode, &g_verify, &verify_launches);
            if (rc) return rc;
        }
        launches += (long long)Kd * draft_launches + verify_launches;
        CUDA_TRY(cudaGraphLaunch(g_verify, h->stream), "verification step");
        CUDA_TRY(cudaEventRecord(ev[2], h->stream), "event");
        CUDA_TRY(cudaMemcpyAsync(h->emitted_host, &h->st->emitted, sizeof(int), cudaMemcpyDeviceToHost, h->stream),
                 "state read");
        CUDA_TRY(cudaMemcpyAsync(h->emitted_host + 1, &h->st->err, sizeof(int), cudaMemcpyDeviceToHost, h->stream),
                 "state read");
        CUDA_TRY(cudaStreamSynchronize(h->stream), "round");
        if (h->emitted_host[1] == kDevErrTimeout)
            return fail(SSD_ERR_TIMEOUT, "a grid barrier of the forward kernel timed out");
        const int e = *h->emitted_host;
        if (e <= emitted || e > n_new) return fail(SSD_ERR_CUDA, "decode state corrupted");
        emitted = e;
        ++round;
    }
    CUDA_TRY(cudaEventRecord(h->events[1], h->stream), "event");
    CUDA_TRY(cudaMemcpyAsync(out_tokens, h->out, sizeof(int) * n_new, cudaMemcpyDeviceToHost, h->stream), "tokens");
    CUDA_TRY(cudaMemcpyAsync(h->st_host, h->st, sizeof(DecodeState), cudaMemcpyDeviceToHost, h->stream), "stats");
    CUDA_TRY(cudaStreamSynchronize(h->stream), "generate");
    if (stats) {
        const DecodeState* s = h->st_host;
        stats->rounds = s->rounds;
        stats->drafted = s->drafted;
        stats->accepted = s->accepted;
        stats->emitted = s->emitted;
        stats->accept_rate = s->drafted ? (double)s->accepted / s->drafted : 0.0;
        for (int i = 0; i < 33; ++i) stats->hist[i] = s->hist[i];
        float dm = 0.f, vm = 0.f, t = 0.f;
        for (int r = 0; r < round; ++r) {
            cudaEvent_t* ev = &h->events[2 + 3 * (size_t)r];
            float a = 0.f, b = 0.f;
            cudaEventElapsedTime(&a, ev[0], ev[1]);
            cudaEventElapsedTime(&b, ev[1], ev[2]);
            dm += a;
            vm += b;
        }
        cudaEventElapsedTime(&t, h->events[0], h->events[1]);
        stats->draft_ms = dm;
        stats->verify_ms = vm;
        stats->total_ms = t;
        stats->kernel_launches = launches;
        stats->gamma = exit_on ? s->gamma : 0.f;
    }
    return SSD_OK;
}

int ssd_debug_forward(ssd_handle* h, int draft, const int32_t* tokens, int n_rows, int pos0, float* logits_out) {
    if (!h || !tokens || !logits_out) return fail(SSD_ERR_INVALID_ARG, "NULL argument");
    if (n_rows < 1 || n_rows > kMaxRows) return fail(SSD_ERR_INVALID_ARG, "n_rows must be in [1, 16]");
    if (pos0 < 0 || pos0 + n_rows > h->cfg.max_seq) return fail(SSD_ERR_CAPACITY, "positions beyond max_seq");
    for (int i = 0; i < n_rows; ++i)
        if (tokens[i] < 0 || tokens[i] >= h->cfg.vocab) return fail(SSD_ERR_INVALID_ARG, "token out of range");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    int* dt = h->tok + h->cfg.max_seq;
    CUDA_TRY(cudaMemsetAsync(&h->st->err, 0, sizeof(int), h->stream), "error flag reset");
    CUDA_TRY(cudaMemcpyAsync(dt, tokens, sizeof(int) * n_rows, cudaMemcpyHostToDevice, h->stream), "upload");
    const int stall = h->stall_barrier;
    const unsigned long long wait_ns = h->wait_ns;
    if (stall) {  // armed by ssd_debug_stall_barrier for this one forward
        h->wait_ns = h->stall_wait_ns;
        h->stall_barrier = 0;
    }
    int rc = forward(h, n_rows, SRC_TOKENS, dt, pos0, draft != 0, true, nullptr, nullptr, stall);
    h->wait_ns = wait_ns;
    if (rc) return rc;
    CUDA_TRY(cudaMemcpyAsync(logits_out, h->logits, sizeof(float) * n_rows * h->cfg.vocab,
                             cudaMemcpyDeviceToHost, h->stream), "logits");
    int derr = 0;
    CUDA_TRY(cudaMemcpyAsync(&h->st_host->err, &h->st->err, sizeof(int), cudaMemcpyDeviceToHost, h->stream),
             "error flag");
    CUDA_TRY(cudaStreamSynchronize(h->stream), "debug forward");
    derr = h->st_host->err;
    if (derr == kDevErrTimeout) return fail(SSD_ERR_TIMEOUT, "a wait of the forward kernel timed out");
    if (derr) return fail(SSD_ERR_CUDA, "device check failed with code " + std::to_string(derr));
    return SSD_OK;
}

int ssd_debug_stall_barrier(ssd_handle* h, int barrier, double wait_limit_s) {
    if (!h) return fail(SSD_ERR_INVALID_ARG, "NULL handle");
    if (barrier < 0 || !(wait_limit_s > 0.0) || wait_limit_s > 10.0)
        return fail(SSD_ERR_INVALID_ARG, "need barrier >= 0 and 0 < wait_limit_s <= 10");
    h->stall_barrier = barrier;
    h->stall_wait_ns = (unsigned long long)(wait_limit_s * 1e9);
    return SSD_OK;
}

// Per-op durations (us) of one forward replay from the device trace; units:
// the rest of the trace (unit and CTA stamps of h->trace_op).
int trace_forward(ssd_handle* h, cudaGraphExec_t exec, int n_ops, std::vector<float>* us,
                  std::vector<unsigned long long>* units = nullptr) {
    std::vector<unsigned long long> t(trace_words(h));
    CUDA_TRY(cudaMemsetAsync(h->trace, 0, t.size() * sizeof(unsigned long long), h->stream), "trace reset");
    CUDA_TRY(cudaGraphLaunch(exec, h->stream), "traced replay");
    CUDA_TRY(cudaMemcpyAsync(t.data(), h->trace, t.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost,
                             h->stream), "trace read");
    CUDA_TRY(cudaStreamSynchronize(h->stream), "trace");
    us->resize(n_ops);
    for (int o = 0; o < n_ops; ++o) (*us)[o] = (float)((double)(t[o + 1] - t[o]) * 1e-3);
    if (units) *units = t;
    return SSD_OK;
}

int capture_debug_forward(ssd_handle* h, int draft, int rows, bool traced, cudaGraphExec_t* exec, int* n) {
    const int pos0 = h->cfg.max_seq - rows;
    int* dt = h->tok + h->cfg.max_seq;
    CUDA_TRY(cudaMemsetAsync(dt, 0, sizeof(int) * rows, h->stream), "tokens");
    cudaGraph_t g = nullptr;
    CUDA_TRY(cudaStreamBeginCapture(h->stream, cudaStreamCaptureModeThreadLocal), "begin capture");
    int rc = forward(h, rows, SRC_TOKENS, dt, pos0, draft != 0, true, n, traced ? h->trace : nullptr);
    cudaError_t e = cudaStreamEndCapture(h->stream, &g);
    if (rc) { if (g) cudaGraphDestroy(g); return rc; }
    CUDA_TRY(e, "end capture");
    e = cudaGraphInstantiate(exec, g, 0);
    cudaGraphDestroy(g);
    CUDA_TRY(e, "graph instantiate");
    if (pos0 < h->n_prompt) h->prefilled = false;  // the prompt's KV is overwritten
    return SSD_OK;
}

int ssd_debug_time_forward(ssd_handle* h, int draft, int rows, int gemm_only, int reps, float* ms_per_forward,
                           int* launches, double* weight_bytes) {
    if (!h || !ms_per_forward || !launches || !weight_bytes) return fail(SSD_ERR_INVALID_ARG, "NULL argument");
    if (rows < 1 || rows > kMaxRows || reps < 1 || rows > h->cfg.max_seq)
        return fail(SSD_ERR_INVALID_ARG, "rows in [1, 16] and reps >= 1 required");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    cudaGraphExec_t exec = nullptr, traced = nullptr;
    int n = 0;
    int rc = capture_debug_forward(h, draft, rows, false, &exec, &n);
    if (!rc && gemm_only) rc = capture_debug_forward(h, draft, rows, true, &traced, &n);
    if (rc) {
        if (exec) cudaGraphExecDestroy(exec);
        return rc;
    }
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    cudaError_t e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    if (e == cudaSuccess) e = cudaGraphLaunch(exec, h->stream);  // warm-up
    if (e == cudaSuccess) e = cudaEventRecord(e0, h->stream);
    for (int r = 0; r < reps && e == cudaSuccess; ++r) e = cudaGraphLaunch(exec, h->stream);
    if (e == cudaSuccess) e = cudaEventRecord(e1, h->stream);
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
    float ms = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    cudaGraphExecDestroy(exec);
    if (e != cudaSuccess) {
        if (traced) cudaGraphExecDestroy(traced);
        CUDA_TRY(e, "timing");
    }
    ms /= reps;
    *launches = n;
    *weight_bytes = forward_weight_bytes(h, draft != 0, false);
    if (gemm_only) {
        // share of the projection ops in one traced replay, applied to the event-timed forward
        std::vector<float> us;
        const int n_ops = draft ? h->n_ops_draft : h->n_ops_full;
        rc = trace_forward(h, traced, n_ops, &us);
        cudaGraphExecDestroy(traced);
        if (rc) return rc;
        std::vector<FwdOp> ops = build_ops(h, draft != 0);
        double all = 0.0, proj = 0.0;
        int n_proj = 0;
        for (int o = 0; o < n_ops; ++o) {
            all += us[o];
            if (ops[o].type != OP_EMBED && ops[o].type != OP_ATTN) { proj += us[o]; ++n_proj; }
        }
        ms = (float)(ms * (all > 0 ? proj / all : 1.0));
        *launches = n_proj;
        *weight_bytes = forward_weight_bytes(h, draft != 0, true);
    }
    *ms_per_forward = ms;
    return SSD_OK;
}

int ssd_debug_trace_forward(ssd_handle* h, int draft, int rows, float* op_us, int* op_types, int max_ops,
                            int* n_ops_out, int detail_op, unsigned long long* unit_trace,
                            unsigned long long* cta_trace, int max_ctas, int* n_ctas) {
    if (!h || !op_us || !op_types || !n_ops_out) return fail(SSD_ERR_INVALID_ARG, "NULL argument");
    if (rows < 1 || rows > kMaxRows || rows > h->cfg.max_seq) return fail(SSD_ERR_INVALID_ARG, "rows in [1, 16]");
    const int n_ops = draft ? h->n_ops_draft : h->n_ops_full;
    if (max_ops < n_ops) return fail(SSD_ERR_INVALID_ARG, "max_ops smaller than the op list");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    if (cta_trace && (!n_ctas || max_ctas < h->n_sms)) return fail(SSD_ERR_INVALID_ARG, "max_ctas below the grid");
    if (detail_op >= 0 && ((detail_op & 0xffff) >= n_ops || (detail_op >> 16) >= h->n_sms))
        return fail(SSD_ERR_INVALID_ARG, "detail_op: op index below the op count, CTA below the grid");
    cudaGraphExec_t traced = nullptr;
    int n = 0;
    h->trace_op = detail_op;
    int rc = capture_debug_forward(h, draft, rows, true, &traced, &n);
    h->trace_op = -1;
    if (rc) return rc;
    std::vector<float> us;
    std::vector<unsigned long long> units;
    CUDA_TRY(cudaGraphLaunch(traced, h->stream), "warm-up");
    rc = trace_forward(h, traced, n_ops, &us, &units);
    cudaGraphExecDestroy(traced);
    if (rc) return rc;
    std::vector<FwdOp> ops = build_ops(h, draft != 0);
    for (int o = 0; o < n_ops; ++o) {
        op_us[o] = us[o];
        op_types[o] = ops[o].type;
    }
    if (unit_trace) for (int i = 0; i < kTraceCtas - kTraceUnits; ++i) unit_trace[i] = units[kTraceUnits + i];
    if (cta_trace) {
        for (int i = 0; i < 8 * h->n_sms; ++i) cta_trace[i] = units[kTraceCtas + i];
        *n_ctas = h->n_sms;
    }
    *n_ops_out = n_ops;
    return SSD_OK;
}

int ssd_debug_spec_accept(ssd_handle* h, const float* p, const float* q, int Kd, const int32_t* drafts,
                          const uint64_t* seeds, int trials, int pos0, int32_t* out) {
    if (!h || !p || !q || !drafts || !seeds || !out) return fail(SSD_ERR_INVALID_ARG, "NULL argument");
    if (Kd < 1 || Kd > kMaxK || trials < 1 || pos0 < 0) return fail(SSD_ERR_INVALID_ARG, "bad Kd / trials / pos0");
    const int V = h->cfg.vocab;
    for (size_t i = 0; i < (size_t)trials * Kd; ++i)
        if (drafts[i] < 0 || drafts[i] >= V) return fail(SSD_ERR_INVALID_ARG, "draft token out of range");
    CUDA_TRY(cudaSetDevice(h->device), "set device");
    std::vector<void*> tmp;
    float *dp = nullptr, *dq = nullptr;
    int *dd = nullptr, *dout = nullptr;
    unsigned long long* ds = nullptr;
    int rc = 0;
    if ((rc = dalloc(h, &dp, (size_t)(Kd + 1) * V, &tmp)) || (rc = dalloc(h, &dq, (size_t)Kd * V, &tmp)) ||
        (rc = dalloc(h, &dd, (size_t)trials * Kd, &tmp)) || (rc = dalloc(h, &ds, (size_t)trials, &tmp)) ||
        (rc = dalloc(h, &dout, (size_t)2 * trials, &tmp))) {
        free_all(h, tmp);
        return rc;
    }
    cudaError_t e = cudaMemcpyAsync(dp, p, sizeof(float) * (Kd + 1) * V, cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(dq, q, sizeof(float) * Kd * V, cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(dd, drafts, sizeof(int) * trials * Kd, cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(ds, seeds, sizeof(uint64_t) * trials, cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess)
        e = (cudaError_t)launch_spec_accept_batch(dp, dq, V, Kd, dd, ds, trials, pos0, dout, h->stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(out, dout, sizeof(int) * 2 * trials, cudaMemcpyDeviceToHost, h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    free_all(h, tmp);
    CUDA_TRY(e, "spec accept");
    return SSD_OK;
}

}  // extern "C"
