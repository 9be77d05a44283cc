// attention.cu - causal attention of M query rows over the KV cache, for the
// draft forward (M = 1), the verification forward over [x_last, d_1..d_K]
// (M = K+1, row m at position len + m attends to [0, len + m]) and prefill.
//
// Work split: one CTA per (64-position chunk of the cache, KV head).  Chunks
// are absolute (chunk c holds positions [64c, 64c + 64)), so the partial
// softmax of a row over a chunk depends on the row and the chunk only, never
// on M; the last CTA of each KV head combines the chunks of each row in chunk
// order.  Hence a verification row is bit-identical to the M = 1 forward of
// the same token at the same position (greedy lossless property, Sec. 1).
// GQA: the CTA serves all n_heads / n_kv_heads query heads of its KV head, so
// every K/V byte is read from HBM once per forward.
#include "ssd_internal.cuh"

namespace ssd {
namespace {

template <int HD>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(const AttnArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    constexpr int KP = HD * 2 + 16;  // bytes per cached row in smem (conflict-free)
    constexpr int EPL = HD / 32;     // output dims per lane
    pdl_launch_dependents();
    pdl_wait();
    const int c = blockIdx.x, kvh = blockIdx.y;
    const int G = a.n_heads / a.n_kv_heads;
    const int M = a.M, NV = G * M;
    const int pos0 = a.st->pos0;
    const int t0 = c * kAttnChunk;
    const int t_end = min(t0 + kAttnChunk, pos0 + M);
    unsigned char* ks = smem;
    unsigned char* vs = ks + kAttnChunk * KP;
    float* qs = reinterpret_cast<float*>(vs + kAttnChunk * KP);  // [NV][HD]
    float* sc = qs + NV * HD;                                     // [8][64]
    __shared__ int s_last;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* part = a.part + ((size_t)kvh * a.n_chunks) * NV * (HD + 2);

    if (t0 < t_end) {
        constexpr int CPR = HD * 2 / 16;
        const int nt = t_end - t0;
        const f16* kb = a.k_cache + ((size_t)kvh * a.max_seq + t0) * HD;
        const f16* vb = a.v_cache + ((size_t)kvh * a.max_seq + t0) * HD;
        for (int i = threadIdx.x; i < nt * CPR; i += kAttnThreads) {
            int t = i / CPR, cc = i - t * CPR;
            SSD_GUARD(a.err, ((((uintptr_t)(kb + (size_t)t * HD + cc * 8)) & 15u) == 0) &&
                                 (((uintptr_t)(vb + (size_t)t * HD + cc * 8)) & 15u) == 0 &&
                                 t < kAttnChunk && t0 + t < a.max_seq, 201) {
                cp_async16(ks + t * KP + cc * 16, kb + (size_t)t * HD + cc * 8, 16);
                cp_async16(vs + t * KP + cc * 16, vb + (size_t)t * HD + cc * 8, 16);
            }
        }
        cp_async_commit();
        for (int i = threadIdx.x; i < NV * HD; i += kAttnThreads) {
            int v = i / HD, e = i - v * HD;
            int m = v / G, gi = v - m * G;
            qs[i] = a.q[(size_t)m * a.n_heads * HD + (size_t)(kvh * G + gi) * HD + e];
        }
        cp_async_wait<0>();
        __syncthreads();

        for (int v = warp; v < NV; v += kAttnThreads / 32) {
            const int m = v / G;
            const int n_t = min(t_end, pos0 + m + 1) - t0;  // positions this row sees here
            float* out = part + ((size_t)c * NV + v) * (HD + 2);
            if (n_t <= 0) {
                for (int e = lane; e < HD; e += 32) out[e] = 0.f;
                if (lane == 0) { out[HD] = -INFINITY; out[HD + 1] = 0.f; }
                continue;
            }
            const float* q = qs + v * HD;
            float s[2];
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const int t = lane + 32 * i;
                float dot = -INFINITY;
                if (t < n_t) {
                    dot = 0.f;
                    const unsigned char* kr = ks + t * KP;
#pragma unroll
                    for (int e8 = 0; e8 < HD / 8; ++e8) {
                        uint4 kv = *reinterpret_cast<const uint4*>(kr + e8 * 16);
                        const float* qq = q + e8 * 8;
                        const float2 k0 = f16x2(kv.x), k1 = f16x2(kv.y), k2 = f16x2(kv.z), k3 = f16x2(kv.w);
                        dot += qq[0] * k0.x + qq[1] * k0.y;
                        dot += qq[2] * k1.x + qq[3] * k1.y;
                        dot += qq[4] * k2.x + qq[5] * k2.y;
                        dot += qq[6] * k3.x + qq[7] * k3.y;
                    }
                    dot *= a.scale;
                }
                s[i] = dot;
            }
            const float mx = warp_max(fmaxf(s[0], s[1]));
            float p0 = lane < n_t ? expf(s[0] - mx) : 0.f;
            float p1 = lane + 32 < n_t ? expf(s[1] - mx) : 0.f;
            const float l = warp_sum(p0 + p1);
            float* sw = sc + warp * kAttnChunk;
            sw[lane] = p0;
            sw[lane + 32] = p1;
            __syncwarp();
            float o[EPL];
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[e] = 0.f;
            for (int t = 0; t < n_t; ++t) {
                const float w = sw[t];
                const unsigned char* vr = vs + t * KP + lane * EPL * 2;
                if constexpr (EPL == 4) {
                    uint2 vv = *reinterpret_cast<const uint2*>(vr);
                    const float2 v0 = f16x2(vv.x), v1 = f16x2(vv.y);
                    o[0] += w * v0.x;
                    o[1] += w * v0.y;
                    o[2] += w * v1.x;
                    o[3] += w * v1.y;
                } else {
                    const float2 v0 = f16x2(*reinterpret_cast<const uint32_t*>(vr));
                    o[0] += w * v0.x;
                    o[1] += w * v0.y;
                }
            }
            __syncwarp();
#pragma unroll
            for (int e = 0; e < EPL; ++e) out[lane * EPL + e] = o[e];
            if (lane == 0) { out[HD] = mx; out[HD + 1] = l; }
        }
    } else {
        // nothing cached here for any row: still take part in the arrival count
    }

    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned prev = atomicAdd(&a.counters[kvh], 1u);
        s_last = (prev == gridDim.x - 1);
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();

    // combine: row m uses chunks 0 .. (pos0 + m) / 64, in chunk order
    for (int v = warp; v < NV; v += kAttnThreads / 32) {
        const int m = v / G, gi = v - m * G;
        const int nch = (pos0 + m) / kAttnChunk + 1;
        float mx = -INFINITY;
        for (int cc = 0; cc < nch; ++cc)
            mx = fmaxf(mx, __ldcg(part + ((size_t)cc * NV + v) * (HD + 2) + HD));
        float L = 0.f;
        float o[EPL];
#pragma unroll
        for (int e = 0; e < EPL; ++e) o[e] = 0.f;
        for (int cc = 0; cc < nch; ++cc) {
            const float* pp = part + ((size_t)cc * NV + v) * (HD + 2);
            const float mc = __ldcg(pp + HD);
            if (mc == -INFINITY) continue;
            const float f = expf(mc - mx);
            L += f * __ldcg(pp + HD + 1);
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[e] += f * __ldcg(pp + lane * EPL + e);
        }
        const float inv = 1.f / L;
        float* dst = a.out + (size_t)m * a.n_heads * HD + (size_t)(kvh * G + gi) * HD + lane * EPL;
#pragma unroll
        for (int e = 0; e < EPL; ++e) dst[e] = o[e] * inv;
    }
    if (threadIdx.x == 0) a.counters[kvh] = 0u;
}

template <int HD>
int launch_hd(const AttnArgs& a, cudaStream_t s) {
    const int G = a.n_heads / a.n_kv_heads;
    size_t smem = 2 * kAttnChunk * (HD * 2 + 16) + (size_t)G * a.M * HD * 4 + 8 * kAttnChunk * 4;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_chunks, a.n_kv_heads, 1);
    cfg.blockDim = dim3(kAttnThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return (int)cudaLaunchKernelEx(&cfg, attn_kernel<HD>, a);
}

}  // namespace

int attention_configure() {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         200 * 1024);
    if (e != cudaSuccess) return (int)e;
    return (int)cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     200 * 1024);
}

int launch_attention(const AttnArgs& a, cudaStream_t s) {
    if (a.head_dim == 128) return launch_hd<128>(a, s);
    if (a.head_dim == 64) return launch_hd<64>(a, s);
    return (int)cudaErrorInvalidValue;
}

}  // namespace ssd
