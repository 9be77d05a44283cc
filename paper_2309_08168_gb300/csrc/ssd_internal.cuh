// ssd_internal.cuh - shared declarations of the libssd CUDA sources (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace ssd {

typedef __nv_bfloat16 bf16;
typedef __half f16;

constexpr int kMaxRows = 16;      // rows of one forward (verification K+1 <= 16)
constexpr int kMaxK = 15;         // drafts per round
constexpr int kTileRows = 64;     // stand-alone projection kernel (gemm.cu): output rows per CTA
constexpr int kGemmThreads = 256; // 8 warps: 4 row groups x 2 k-interleaves
constexpr int kAttnChunk = 64;    // KV positions per attention CTA (absolute chunks)
constexpr int kAttnThreads = 256;
constexpr int kStreamKC = 256;    // (stand-alone projection kernel of gemm.cu) k per CTA chunk step
constexpr int kFTile = 128;       // forward kernel: weight rows per tile (tcgen05 M, TMEM lanes)
constexpr int kFKC = 128;         // forward kernel: k per work unit (128 rows x 128 k = 32 KB of weights)
constexpr int kTraceUnits = 1024, kTraceCtas = 1280;  // offsets in FwdParams::trace
// rows per input plane of a forward of M rows (the plane classes)
constexpr int fwd_plane_rows(int M) { return M == 1 ? 1 : (M <= 4 ? 4 : (M <= 8 ? 8 : (M <= 12 ? 12 : 16))); }
constexpr int kPlaneClasses = 5;

// ---------------------------------------------------------------------------
// device state of the decode loop (one per handle, in device memory)
// ---------------------------------------------------------------------------
struct DecodeState {
    int len;        // committed KV positions [0, len)
    int x_last;     // last emitted token; sits at position len
    int j;          // drafts produced in the current round
    int emitted;    // tokens written to the output buffer by this generate call
    int rounds, drafted, accepted;
    int hist[33];
    int drafts[kMaxK + 1];
    int pos0;       // first position of the forward in flight
    int mode;       // 0 greedy, 1 sampling
    float inv_temperature;
    float top_p;
    unsigned long long seed;
    int err;        // device-side error code (0 = none)
    // adaptive draft exit (Sec. 3.4, Eqs. 2-4); exit_on = 0: off
    int exit_on;
    int exited;     // the current round's drafting stage has ended
    int exit_updates;
    float gamma, ar_smooth;
    float alpha, eps, beta1, beta2;
};

// ---------------------------------------------------------------------------
// Projection arguments: the forward kernel's tcgen05 projections and the
// stand-alone swap-AB mma.sync kernel of gemm.cu (bf16 in, fp32 accumulate)
// ---------------------------------------------------------------------------
enum GemmEpi { EPI_LOGITS = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_QKV = 3 };

struct GemmArgs {
    const bf16* w0;      // weight segment 0 (wq / w_gate / the only matrix)
    const bf16* w1;      // segment 1 (wk / w_up)
    const bf16* w2;      // segment 2 (wv)
    int N;               // logical output rows
    int K;               // reduction length (row length of every segment)
    int kc;              // gemm.cu: k-chunk per CTA (multiple of 64)
    int ksplit;          // gemm.cu: ceil(K / kc)
    int n_tiles;         // row tiles
    const float* x;      // gemm.cu: activations [M][K] fp32 (split into bf16 hi + lo in the kernel)
    int M;               // gemm.cu: activation rows (1..16)
    float* partial;      // split-K partials: gemm.cu [ksplit][M][n_tiles*64] floats; forward
                         // kernel [n_tiles][n_chunks][16][128] tagged 64-bit words
    unsigned* counters;  // gemm.cu: [n_tiles] arrival counters (left at zero)
    // epilogue operands
    float* out_f32;      // EPI_LOGITS: [M][ldo]; EPI_RESID: residual h [M][ldo]
    int ldo;
    int ffn;
    // EPI_QKV
    int n_heads, n_kv_heads, head_dim, max_seq;
    float* q_out;        // [M][H*hd] fp32, rotated
    f16* k_cache;        // this layer: [Hkv][max_seq][hd] fp16
    f16* v_cache;
    const float2* rope;  // [max_seq][hd/2] (cos, sin)
    int* err;            // device error flag
    const float* ss_in;  // [M][ss_in_tiles] sums of squares of the pre-norm row (nullptr: no norm)
    int ss_in_tiles;
    float inv_dim, eps;  // RMSNorm scale of row m: rsqrt(sum(ss_in[m]) * inv_dim + eps)
    const bf16* g_next;  // EPI_RESID: gains of the next RMSNorm (nullptr: no next input)
    bf16* xo_hi;         // EPI_RESID: planes of h * g_next [M][N]; EPI_SWIGLU: act planes [M][ffn]
    bf16* xo_lo;
    float* ss_out;       // EPI_RESID: [M][n_tiles] per-tile sums of h^2
    int n_chunks;        // forward kernel: ceil(K / kFKC)
    int n_units;         // n_tiles * n_chunks
    // TMA tensor maps (in global memory), forward kernel: w maps view W as
    // {K, rows} with box {64, 128} (SwiGLU gate / up: {64, 64}), one copy per
    // 64-wide k box of a unit; x maps view the planes as {K, 16, 2} with box
    // {64, R, 2}, one copy per k box.
    const void* tm_w[3];  // w0, w1, w2
    const void* tm_x[kPlaneClasses];  // input planes for R = 1 | 4 | 8 | 12 | 16
};

// ---------------------------------------------------------------------------
// attention (decode / verification over the KV cache, split into absolute
// 64-position chunks, fixed-order combine)
// ---------------------------------------------------------------------------
// floats per attention segment partial: o[hd], max, sum, and 2 of padding so
// that every partial starts on a 16-byte boundary (vector loads in the combine)
__host__ __device__ constexpr int attn_part_floats(int hd) { return hd + 4; }

struct AttnArgs {
    const float* q;      // [M][H*hd]
    // TMA maps of the whole K / V cache viewed as {hd, max_seq, L * Hkv} fp16,
    // box {64, 64, 1}, 128-byte swizzle; this layer's KV head kvh is z = kv_z0 + kvh
    const void* tm_k;
    const void* tm_v;
    int kv_z0;
    bf16* out_hi;        // [M][H*hd] output planes: hi = rn(o), lo = rn(o - hi)
    bf16* out_lo;
    float* part;         // segment partials [Hkv][n_chunks][G*M][attn_part_floats(hd)]: o[hd], max, sum, 2 pad
    int M, n_heads, n_kv_heads, head_dim, max_seq, n_chunks;
    float scale;         // 1/sqrt(hd)
    const DecodeState* st;
    int* err;            // device error flag (checked builds)
};

// ---------------------------------------------------------------------------
// forward kernel (forward_kernel.cu): one persistent cooperative launch per
// decoder forward, walking a device-resident op list
// ---------------------------------------------------------------------------
enum OpType { OP_EMBED = 0, OP_QKV = 1, OP_ATTN = 2, OP_RESID = 3, OP_SWIGLU = 4, OP_LOGITS = 5 };
constexpr int kDevErrTimeout = 1;  // DecodeState::err: a grid barrier or a TMA wait gave up

struct alignas(16) FwdOp {  // (copied in 16-byte pieces)
    int type;
    GemmArgs g;   // projection ops
    AttnArgs at;  // attention op
};

struct FwdParams {
    const FwdOp* ops;
    int n_ops;
    int M;                // rows of this forward (1..16)
    int src;              // EmbedSrc: where the tokens and the first position come from
    const int* toks;      // SRC_TOKENS: device token ids
    int pos0_arg;         // SRC_TOKENS: first position
    DecodeState* st;
    const bf16* embed;
    int d;
    const bf16* g0;       // gains of the first RMSNorm that runs
    float* h;             // residual stream [16][d]
    bf16* xn_hi;          // planes of h * g [16][d]
    bf16* xn_lo;
    float* ss;            // per-128-column sums of h^2 [16][d/128]
    unsigned* bar;        // grid-barrier counter, zero at launch
    unsigned* seq;        // forward sequence number (tags split-K partials; +1 per launch)
    int* err;             // device error code
    // Profiling hook: nullptr, or globaltimer stamps: [0, n_ops] start, end of
    // op o (CTA 0); [1024, 1280) the first 64 units (or 31 attention items) of
    // op trace_op & 0xffff on CTA trace_op >> 16; [1280, 1280 + 8 * grid) per
    // CTA, op trace_op & 0xffff: the 8 stamps ssd_debug_trace_forward lists.
    unsigned long long* trace;
    int trace_op;  // -1: none
    // Bounded waits: a grid barrier gives up after wait_ns (error recorded).
    // Test hook: stall_barrier = n > 0 makes the n-th grid barrier of the
    // launch unreachable (0 in every production launch).
    unsigned long long wait_ns;
    int stall_barrier;
};

// ---------------------------------------------------------------------------
// prefill on the tensor cores (prefill.cu, tc_gemm.cuh)
// ---------------------------------------------------------------------------
struct PrefillLayer {
    const void* tm_w[7];  // TMA maps (box 64 x 128) of wq wk wv wo w_gate w_up w_down
    const bf16* attn_norm;
    const bf16* mlp_norm;
    f16* k_cache;  // this layer's [Hkv][max_seq][hd]
    f16* v_cache;
};
struct PrefillPlan {
    int n_layers, d, n_heads, n_kv_heads, head_dim, ffn, max_seq;
    float eps;
    int rows;  // capacity of the row buffers (prompt positions per chunk)
    const bf16* embed;
    const float2* rope;
    float* h;           // [rows][d]
    bf16* x_hi;         // [rows][d] normalised rows, hi / lo
    bf16* x_lo;
    float* q;           // [rows][H*hd]
    bf16* at_hi;        // [rows][H*hd] attention output, hi / lo
    bf16* at_lo;
    bf16* ac_hi;        // [rows][ffn] SwiGLU output, hi / lo
    bf16* ac_lo;
    const void* tm_x[2];   // TMA maps of x_hi / x_lo  (box 64 x 128)
    const void* tm_at[2];  // of at_hi / at_lo
    const void* tm_ac[2];  // of ac_hi / ac_lo
    const PrefillLayer* layers;  // host array
    int* err;
};
int prefill_configure();
int prefill_chunk(const PrefillPlan& P, const int* toks, int n, int pos0, cudaStream_t s);

int forward_configure();
int launch_forward(const FwdParams& p, int head_dim, int grid, cudaStream_t s);

// sets the thread's ssd_last_error() message and returns code
int set_last_error(int code, const char* msg);

// launchers (return cudaError_t)
int gemm_configure();
size_t gemm_smem_bytes(int kc, int M);
constexpr int gemm_half_rows(int M) { return M <= 8 ? 8 : 16; }  // padded rows of x_hi (and of x_lo)

// src for launch_embed
enum EmbedSrc { SRC_TOKENS = 0, SRC_DRAFT = 1, SRC_VERIFY = 2 };

int launch_greedy_draft(const float* logits, int V, DecodeState* st, cudaStream_t s);
int launch_greedy_accept(const float* logits, int V, int M, DecodeState* st, int* out_tokens,
                         unsigned* counter, int* argmax_buf, cudaStream_t s);
int launch_sample_draft(const float* logits, int V, DecodeState* st, float* q_rows,
                        cudaStream_t s);
int launch_sample_accept(const float* logits, int V, int M, DecodeState* st, float* p_rows,
                         const float* q_rows, int* out_tokens, unsigned* counter,
                         cudaStream_t s);
int launch_spec_accept_batch(const float* p_rows, const float* q_rows, int V, int Kd,
                             const int* drafts, const unsigned long long* seeds, int trials,
                             int pos0, int* out, cudaStream_t s);

// Checked builds (-DSSD_CHECKED): a failed alignment / bounds condition
// records `code` in the device error flag and the access is skipped.
#ifdef SSD_CHECKED
#define SSD_GUARD(errp, cond, code) if (!(cond)) { atomicCAS((errp), 0, (code)); } else
#else
#define SSD_GUARD(errp, cond, code)
#endif

// ---------------------------------------------------------------------------
// small device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float2 f16x2(uint32_t w) {
    return __half22float2(*reinterpret_cast<const __half2*>(&w));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

// 16-byte async copy global -> shared; src_bytes = 0 zero-fills the slot.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(smem_u32(smem)),
                 "l"(gmem), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}
// Programmatic dependent launch: let the next kernel in the stream start its
// prologue now / wait until the previous kernel's results are visible.
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;\n" ::);
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }

// D += A * B, m16n8k16, A row-major bf16, B column-major bf16, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Splits 8 fp32 activations into bf16 hi = rn(x) and lo = rn(x - hi), so that
// W * hi + W * lo carries ~16 mantissa bits of x through the bf16 MMA.
__device__ __forceinline__ void split8(const float4& f0, const float4& f1, uint4& hi, uint4& lo) {
    const float f[8] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w};
    uint32_t h[4], l[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        __nv_bfloat162 hv = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
        float2 hf = __bfloat1622float2(hv);
        __nv_bfloat162 lv = __floats2bfloat162_rn(f[2 * i] - hf.x, f[2 * i + 1] - hf.y);
        h[i] = *reinterpret_cast<uint32_t*>(&hv);
        l[i] = *reinterpret_cast<uint32_t*>(&lv);
    }
    hi = make_uint4(h[0], h[1], h[2], h[3]);
    lo = make_uint4(l[0], l[1], l[2], l[3]);
}

}  // namespace ssd
