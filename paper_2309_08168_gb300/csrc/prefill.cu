// prefill.cu - prompt encoding on the tensor cores (Sec. 3.1: the prompt is
// run through the full model once, filling the KV cache, before the
// decoding rounds of Algorithms 1 / 2 start).
//
// The decode forwards are HBM-bound skinny GEMMs (M <= 16 rows); a prompt of
// hundreds of rows is compute-bound, so it gets its own kernels, layer by
// layer over a chunk of up to `rows` prompt positions:
//   embed      h[r] = E[token r]
//   norm       x = RMSNorm(h) * g as bf16 hi / lo planes (fp32 statistics)
//   QKV GEMM   tcgen05 (tc_gemm.cuh), epilogue: RoPE, q (fp32) and the fp16
//              K / V cache rows of the chunk's positions
//   attention  causal flash attention of the chunk's rows over the cache
//              [0, position] (mma.sync fp16, online softmax), output as bf16
//              hi / lo planes
//   O GEMM     tcgen05, epilogue: h += D
//   norm, gate/up GEMM (epilogue: SwiGLU as bf16 hi / lo planes), down GEMM
//              (epilogue: h += D)
// Numerics follow the decode forwards (bf16 weights, fp32 residual stream,
// activations as bf16 hi + lo, fp16 KV, fp32 softmax), in another summation
// order.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <string>
#include <vector>

#include "ssd_internal.cuh"
#include "tc_gemm.cuh"

namespace ssd {
namespace {

constexpr int kNormThreads = 256;

__global__ void __launch_bounds__(kNormThreads) pf_embed_kernel(const bf16* __restrict__ embed,
                                                                 const int* __restrict__ toks, int d,
                                                                 float* __restrict__ h) {
    const int r = blockIdx.x;
    const bf16* e = embed + (size_t)toks[r] * d;
    for (int i = threadIdx.x; i < d; i += kNormThreads) h[(size_t)r * d + i] = __bfloat162float(e[i]);
}

// x = h / sqrt(mean(h^2) + eps) * g, written as bf16 hi = rn(x), lo = rn(x - hi)
__global__ void __launch_bounds__(kNormThreads) pf_norm_kernel(const float* __restrict__ h,
                                                               const bf16* __restrict__ g, int d, float eps,
                                                               bf16* __restrict__ x_hi, bf16* __restrict__ x_lo) {
    __shared__ float s_part[kNormThreads / 32];
    const int r = blockIdx.x;
    const float* hr = h + (size_t)r * d;
    float ss = 0.f;
    for (int i = threadIdx.x; i < d; i += kNormThreads) ss += hr[i] * hr[i];
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < kNormThreads / 32; ++w) tot += s_part[w];
    const float rinv = rsqrtf(tot / (float)d + eps);
    for (int i = threadIdx.x; i < d; i += kNormThreads) {
        const float x = hr[i] * rinv * __bfloat162float(g[i]);
        const bf16 xh = __float2bfloat16_rn(x);
        x_hi[(size_t)r * d + i] = xh;
        x_lo[(size_t)r * d + i] = __float2bfloat16_rn(x - __bfloat162float(xh));
    }
}

// ---------------------------------------------------------------------------
// causal attention of the chunk's rows (flash attention, fp16 tensor cores)
// ---------------------------------------------------------------------------
// CTA = 4 warps x 16 query rows of one query head; key blocks of 64
// positions from the fp16 cache, double-buffered with cp.async; S = q K^T
// with q as fp16 hi + lo, online softmax in fp32, O += P V with P as fp16
// hi + lo.  Rows r < n_rows sit at positions pos0 + r and see keys
// [0, pos0 + r].
constexpr int kAttQ = 64, kAttKB = 64, kAttThreads = 128;
template <int HD>
constexpr size_t att_smem_bytes() { return (size_t)4 * kAttKB * (HD + 8) * 2; }  // K, V double-buffered

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm4(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm4t(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(p)));
}
__device__ __forceinline__ uint32_t pack_h2(float a, float b) {
    const __half2 v = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&v);
}
// hi = rn(a, b), lo = rn((a, b) - hi), packed
__device__ __forceinline__ void split_h2(float a, float b, uint32_t& hi, uint32_t& lo) {
    const __half2 h = __floats2half2_rn(a, b);
    const float2 f = __half22float2(h);
    hi = *reinterpret_cast<const uint32_t*>(&h);
    lo = pack_h2(a - f.x, b - f.y);
}

template <int HD>
__global__ void __launch_bounds__(kAttThreads) pf_attn_kernel(const float* __restrict__ q, const f16* __restrict__ kc,
                                                              const f16* __restrict__ vc, int n_rows, int pos0,
                                                              int n_heads, int n_kv_heads, int max_seq, float scale,
                                                              bf16* __restrict__ out_hi, bf16* __restrict__ out_lo) {
    constexpr int PITCH = HD + 8;  // halves per smem row (16-byte pad: conflict-free ldmatrix)
    constexpr int KS = HD / 16;    // k steps of q K^T
    constexpr int DN = HD / 8;     // n8 tiles of the output dims
    extern __shared__ __align__(16) unsigned char att_smem[];  // K [2][64][PITCH], then V
    __half(*sk)[kAttKB * PITCH] = reinterpret_cast<__half(*)[kAttKB * PITCH]>(att_smem);
    __half(*sv)[kAttKB * PITCH] = reinterpret_cast<__half(*)[kAttKB * PITCH]>(att_smem + 2 * kAttKB * PITCH * 2);
    const int head = blockIdx.y, kvh = (int)(((long long)head * n_kv_heads) / n_heads);
    const int qr0 = blockIdx.x * kAttQ;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const int qd = n_heads * HD;
    const f16* kh = kc + (size_t)kvh * max_seq * HD;
    const f16* vh = vc + (size_t)kvh * max_seq * HD;
    const int last_row = min(n_rows, qr0 + kAttQ) - 1;
    const int n_kb = (pos0 + last_row) / kAttKB + 1;

    auto load_kv = [&](int kb, int buf) {
        constexpr int CPR = HD / 8;  // 16-byte chunks per row
        for (int c = threadIdx.x; c < kAttKB * CPR; c += kAttThreads) {
            const int r = c / CPR, cc = c - r * CPR, key = kb * kAttKB + r;
            const bool in = key < max_seq;
            const size_t off = (size_t)(in ? key : 0) * HD + cc * 8;
            cp_async16(&sk[buf][r * PITCH + cc * 8], kh + off, in ? 16 : 0);
            cp_async16(&sv[buf][r * PITCH + cc * 8], vh + off, in ? 16 : 0);
        }
        cp_async_commit();
    };
    load_kv(0, 0);

    // q fragments (rows g and g + 8 of this warp's 16), fp16 hi + lo
    const int ra = qr0 + warp * 16 + g, rb = ra + 8;
    uint32_t qh[KS][4], ql[KS][4];
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
        const int c = ks * 16 + 2 * t;
        float2 x[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        if (ra < n_rows) {
            x[0] = *reinterpret_cast<const float2*>(q + (size_t)ra * qd + head * HD + c);
            x[2] = *reinterpret_cast<const float2*>(q + (size_t)ra * qd + head * HD + c + 8);
        }
        if (rb < n_rows) {
            x[1] = *reinterpret_cast<const float2*>(q + (size_t)rb * qd + head * HD + c);
            x[3] = *reinterpret_cast<const float2*>(q + (size_t)rb * qd + head * HD + c + 8);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) split_h2(x[i].x, x[i].y, qh[ks][i], ql[ks][i]);
    }
    const int pa = pos0 + ra, pb = pos0 + rb;  // positions of rows g and g + 8

    float o[DN][4];
#pragma unroll
    for (int j = 0; j < DN; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float ma = -INFINITY, mb = -INFINITY, la = 0.f, lb = 0.f;

    for (int kb = 0; kb < n_kb; ++kb) {
        const int buf = kb & 1;
        if (kb + 1 < n_kb) {
            load_kv(kb + 1, buf ^ 1);
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        // S = q K^T over the block's 64 keys: 8 n8 tiles
        float s[8][4];
#pragma unroll
        for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
#pragma unroll
            for (int j = 0; j < 8; j += 2) {
                uint32_t b[4];
                const int key = j * 8 + (lane & 7) + ((lane >> 4) << 3);
                const int dim = ks * 16 + ((lane >> 3) & 1) * 8;
                ldsm4(b, &sk[buf][key * PITCH + dim]);
                mma16816(s[j], qh[ks][0], qh[ks][1], qh[ks][2], qh[ks][3], b[0], b[1]);
                mma16816(s[j], ql[ks][0], ql[ks][1], ql[ks][2], ql[ks][3], b[0], b[1]);
                mma16816(s[j + 1], qh[ks][0], qh[ks][1], qh[ks][2], qh[ks][3], b[2], b[3]);
                mma16816(s[j + 1], ql[ks][0], ql[ks][1], ql[ks][2], ql[ks][3], b[2], b[3]);
            }
        }
        // scale, causal mask, online softmax (rows g: s[.][0..1], g + 8: s[.][2..3])
        float bma = -INFINITY, bmb = -INFINITY;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int key = kb * kAttKB + j * 8 + 2 * t;
            s[j][0] = key <= pa ? s[j][0] * scale : -INFINITY;
            s[j][1] = key + 1 <= pa ? s[j][1] * scale : -INFINITY;
            s[j][2] = key <= pb ? s[j][2] * scale : -INFINITY;
            s[j][3] = key + 1 <= pb ? s[j][3] * scale : -INFINITY;
            bma = fmaxf(bma, fmaxf(s[j][0], s[j][1]));
            bmb = fmaxf(bmb, fmaxf(s[j][2], s[j][3]));
        }
#pragma unroll
        for (int off = 1; off < 4; off <<= 1) {
            bma = fmaxf(bma, __shfl_xor_sync(0xffffffffu, bma, off));
            bmb = fmaxf(bmb, __shfl_xor_sync(0xffffffffu, bmb, off));
        }
        const float na = fmaxf(ma, bma), nb = fmaxf(mb, bmb);
        // rows past the chunk hold no keys: keep them finite and zero
        const float ca = na == -INFINITY ? 1.f : expf(ma - na), cb = nb == -INFINITY ? 1.f : expf(mb - nb);
        ma = na;
        mb = nb;
        float sa = 0.f, sb = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            s[j][0] = s[j][0] == -INFINITY ? 0.f : expf(s[j][0] - na);
            s[j][1] = s[j][1] == -INFINITY ? 0.f : expf(s[j][1] - na);
            s[j][2] = s[j][2] == -INFINITY ? 0.f : expf(s[j][2] - nb);
            s[j][3] = s[j][3] == -INFINITY ? 0.f : expf(s[j][3] - nb);
            sa += s[j][0] + s[j][1];
            sb += s[j][2] + s[j][3];
        }
        la = la * ca + sa;  // (quad partial sums; reduced once at the end)
        lb = lb * cb + sb;
#pragma unroll
        for (int j = 0; j < DN; ++j) {
            o[j][0] *= ca;
            o[j][1] *= ca;
            o[j][2] *= cb;
            o[j][3] *= cb;
        }
        // O += P V: k steps of 16 keys; P from the S accumulators (hi + lo)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            uint32_t ph[4], pl[4];
            split_h2(s[2 * kk][0], s[2 * kk][1], ph[0], pl[0]);
            split_h2(s[2 * kk][2], s[2 * kk][3], ph[1], pl[1]);
            split_h2(s[2 * kk + 1][0], s[2 * kk + 1][1], ph[2], pl[2]);
            split_h2(s[2 * kk + 1][2], s[2 * kk + 1][3], ph[3], pl[3]);
#pragma unroll
            for (int dn = 0; dn < DN; dn += 2) {
                uint32_t b[4];
                const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int dim = dn * 8 + (lane >> 4) * 8;
                ldsm4t(b, &sv[buf][key * PITCH + dim]);
                mma16816(o[dn], ph[0], ph[1], ph[2], ph[3], b[0], b[1]);
                mma16816(o[dn], pl[0], pl[1], pl[2], pl[3], b[0], b[1]);
                mma16816(o[dn + 1], ph[0], ph[1], ph[2], ph[3], b[2], b[3]);
                mma16816(o[dn + 1], pl[0], pl[1], pl[2], pl[3], b[2], b[3]);
            }
        }
        __syncthreads();  // the buffer is refilled two blocks later
    }
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
        la += __shfl_xor_sync(0xffffffffu, la, off);
        lb += __shfl_xor_sync(0xffffffffu, lb, off);
    }
    const float ia = la > 0.f ? 1.f / la : 0.f, ib = lb > 0.f ? 1.f / lb : 0.f;
#pragma unroll
    for (int dn = 0; dn < DN; ++dn) {
        const int c = head * HD + dn * 8 + 2 * t;
        if (ra < n_rows) {
            const size_t at = (size_t)ra * qd + c;
            tc::store_hilo(out_hi + at, out_lo + at, o[dn][0] * ia);
            tc::store_hilo(out_hi + at + 1, out_lo + at + 1, o[dn][1] * ia);
        }
        if (rb < n_rows) {
            const size_t at = (size_t)rb * qd + c;
            tc::store_hilo(out_hi + at, out_lo + at, o[dn][2] * ib);
            tc::store_hilo(out_hi + at + 1, out_lo + at + 1, o[dn][3] * ib);
        }
    }
}

}  // namespace

int prefill_configure() {
    int e = (int)cudaFuncSetAttribute(pf_attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)att_smem_bytes<128>());
    if (!e)
        e = (int)cudaFuncSetAttribute(pf_attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)att_smem_bytes<64>());
    if (!e) e = tc::tc_configure<tc::TC_QKV>();
    if (!e) e = tc::tc_configure<tc::TC_RESID>();
    if (!e) e = tc::tc_configure<tc::TC_SWIGLU>();
    return e;
}

// One chunk of prompt rows at positions pos0 .. pos0 + n - 1 through every
// layer (launches only).  toks: device token ids of the chunk.
int prefill_chunk(const PrefillPlan& P, const int* toks, int n, int pos0, cudaStream_t s) {
    const int d = P.d, qd = P.n_heads * P.head_dim, kvd = P.n_kv_heads * P.head_dim;
    const int row_tiles = (n + tc::kBM - 1) / tc::kBM;
    pf_embed_kernel<<<n, kNormThreads, 0, s>>>(P.embed, toks, d, P.h);
    int e = (int)cudaGetLastError();
    for (int l = 0; l < P.n_layers && !e; ++l) {
        const PrefillLayer& L = P.layers[l];
        pf_norm_kernel<<<n, kNormThreads, 0, s>>>(P.h, L.attn_norm, d, P.eps, P.x_hi, P.x_lo);
        e = (int)cudaGetLastError();
        if (e) break;
        tc::TcArgs a{};
        a.tm_a_hi = P.tm_x[0];
        a.tm_a_lo = P.tm_x[1];
        a.tm_b[0] = L.tm_w[0];
        a.tm_b[1] = L.tm_w[1];
        a.tm_b[2] = L.tm_w[2];
        a.rows = n;
        a.K = d;
        a.n_kb = (d + tc::kBK - 1) / tc::kBK;
        a.n_tiles = (qd + 2 * kvd + tc::kBN - 1) / tc::kBN;
        a.n_heads = P.n_heads;
        a.n_kv_heads = P.n_kv_heads;
        a.head_dim = P.head_dim;
        a.max_seq = P.max_seq;
        a.pos0 = pos0;
        a.q = P.q;
        a.k_cache = L.k_cache;
        a.v_cache = L.v_cache;
        a.rope = P.rope;
        a.err = P.err;
        e = tc::tc_launch<tc::TC_QKV>(a, row_tiles, s);
        if (e) break;
        const dim3 ag((n + kAttQ - 1) / kAttQ, P.n_heads);
        const float scale = 1.0f / std::sqrt((float)P.head_dim);
        if (P.head_dim == 128)
            pf_attn_kernel<128><<<ag, kAttThreads, att_smem_bytes<128>(), s>>>(P.q, L.k_cache, L.v_cache, n, pos0, P.n_heads,
                                                           P.n_kv_heads, P.max_seq, scale, P.at_hi, P.at_lo);
        else
            pf_attn_kernel<64><<<ag, kAttThreads, att_smem_bytes<64>(), s>>>(P.q, L.k_cache, L.v_cache, n, pos0, P.n_heads,
                                                          P.n_kv_heads, P.max_seq, scale, P.at_hi, P.at_lo);
        e = (int)cudaGetLastError();
        if (e) break;
        tc::TcArgs o{};
        o.tm_a_hi = P.tm_at[0];
        o.tm_a_lo = P.tm_at[1];
        o.tm_b[0] = o.tm_b[1] = o.tm_b[2] = L.tm_w[3];
        o.rows = n;
        o.K = qd;
        o.n_kb = (qd + tc::kBK - 1) / tc::kBK;
        o.n_tiles = (d + tc::kBN - 1) / tc::kBN;
        o.N = d;
        o.out = P.h;
        o.ldo = d;
        o.err = P.err;
        e = tc::tc_launch<tc::TC_RESID>(o, row_tiles, s);
        if (e) break;
        pf_norm_kernel<<<n, kNormThreads, 0, s>>>(P.h, L.mlp_norm, d, P.eps, P.x_hi, P.x_lo);
        e = (int)cudaGetLastError();
        if (e) break;
        tc::TcArgs gu{};
        gu.tm_a_hi = P.tm_x[0];
        gu.tm_a_lo = P.tm_x[1];
        gu.tm_b[0] = L.tm_w[4];
        gu.tm_b[1] = L.tm_w[5];
        gu.tm_b[2] = L.tm_w[4];
        gu.rows = n;
        gu.K = d;
        gu.n_kb = (d + tc::kBK - 1) / tc::kBK;
        gu.n_tiles = (P.ffn + 127) / 128;
        gu.ffn = P.ffn;
        gu.act_hi = P.ac_hi;
        gu.act_lo = P.ac_lo;
        gu.err = P.err;
        e = tc::tc_launch<tc::TC_SWIGLU>(gu, row_tiles, s);
        if (e) break;
        tc::TcArgs dn{};
        dn.tm_a_hi = P.tm_ac[0];
        dn.tm_a_lo = P.tm_ac[1];
        dn.tm_b[0] = dn.tm_b[1] = dn.tm_b[2] = L.tm_w[6];
        dn.rows = n;
        dn.K = P.ffn;
        dn.n_kb = (P.ffn + tc::kBK - 1) / tc::kBK;
        dn.n_tiles = (d + tc::kBN - 1) / tc::kBN;
        dn.N = d;
        dn.out = P.h;
        dn.ldo = d;
        dn.err = P.err;
        e = tc::tc_launch<tc::TC_RESID>(dn, row_tiles, s);
    }
    return e;
}

}  // namespace ssd
