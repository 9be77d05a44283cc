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
constexpr int kTileRows = 64;     // output rows per GEMM CTA
constexpr int kGemmThreads = 256; // 8 warps: 4 row groups x 2 k-interleaves
constexpr int kAttnChunk = 64;    // KV positions per attention CTA (absolute chunks)
constexpr int kAttnThreads = 256;

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
};

// ---------------------------------------------------------------------------
// GEMM (swap-AB skinny GEMM on mma.sync m16n8k16, bf16 in, fp32 accumulate)
// ---------------------------------------------------------------------------
enum GemmEpi { EPI_LOGITS = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_QKV = 3 };

struct GemmArgs {
    const bf16* w0;      // weight segment 0 (wq / w_gate / the only matrix)
    const bf16* w1;      // segment 1 (wk / w_up)
    const bf16* w2;      // segment 2 (wv)
    int N;               // logical output rows
    int K;               // reduction length (row length of every segment)
    int kc;              // k-chunk per CTA (multiple of 64)
    int ksplit;          // ceil(K / kc)
    int n_tiles;         // row tiles
    const float* x;      // activations [M][K] fp32 (split into bf16 hi + lo in the kernel)
    int M;               // activation rows (1..16)
    float* partial;      // [ksplit][M][n_tiles*64] split-K partial sums
    unsigned* counters;  // [n_tiles] arrival counters (left at zero)
    // epilogue operands
    float* out_f32;      // EPI_LOGITS: [M][ldo]; EPI_RESID: residual h [M][ldo]
    int ldo;
    float* out_act;      // EPI_SWIGLU: act [M][ffn]
    int ffn;
    // EPI_QKV
    int n_heads, n_kv_heads, head_dim, max_seq;
    float* q_out;        // [M][H*hd] fp32, rotated
    f16* k_cache;        // this layer: [Hkv][max_seq][hd] fp16
    f16* v_cache;
    const float2* rope;  // [max_seq][hd/2] (cos, sin)
    const DecodeState* st;  // pos0
    int* err;            // device error flag (checked builds)
};

// ---------------------------------------------------------------------------
// attention (decode / verification over the KV cache, split into absolute
// 64-position chunks, fixed-order combine)
// ---------------------------------------------------------------------------
struct AttnArgs {
    const float* q;      // [M][H*hd]
    const f16* k_cache;  // [Hkv][max_seq][hd] fp16
    const f16* v_cache;
    float* out;          // [M][H*hd]
    float* part;         // [Hkv][n_chunks][G*M][hd + 2]
    unsigned* counters;  // [Hkv]
    int M, n_heads, n_kv_heads, head_dim, max_seq, n_chunks;
    float scale;         // 1/sqrt(hd)
    const DecodeState* st;
    int* err;            // device error flag (checked builds)
};

// sets the thread's ssd_last_error() message and returns code
int set_last_error(int code, const char* msg);

// launchers (return cudaError_t)
int gemm_configure();
int attention_configure();
int launch_gemm(int epi, const GemmArgs& a, cudaStream_t s);
int launch_attention(const AttnArgs& a, cudaStream_t s);
size_t gemm_smem_bytes(int kc, int M);
constexpr int gemm_half_rows(int M) { return M <= 8 ? 8 : 16; }  // padded rows of x_hi (and of x_lo)

int launch_embed(const bf16* embed, int d, int M, int src, const int* tokens_dev, int pos0,
                 DecodeState* st, float* h, cudaStream_t s);
int launch_rmsnorm(const float* h, const bf16* g, int d, int M, float eps, float* out,
                   cudaStream_t s);

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

}  // namespace ssd
