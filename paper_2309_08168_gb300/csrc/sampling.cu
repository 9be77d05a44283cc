// sampling.cu - the token choice and acceptance kernels that follow a
// forward in self-speculative decoding:
//   greedy draft      x_{j+1} = argmax p(x | z*, ...)              (Algorithm 2)
//   greedy accept     longest prefix d_j == argmax p_{j-1}; the first
//                     mismatch is corrected, or a bonus token added (Alg. 2)
//   sampling draft    d_j ~ q_j = nucleus(softmax(logits / T))        (Alg. 4)
//   sampling accept   accept d_j iff r < min(1, p_{j-1}(d_j) / q_j(d_j)); the
//                     first rejected one is resampled from
//                     norm(max(0, p_{j-1} - q_j)); bonus ~ p_K      (Alg. 4)
// followed by the KV rollback len <- len + 1 + n (a length pointer: later
// writes overwrite the rejected positions).
//
// Random numbers: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), key =
// 64-bit seed, counter = (position, purpose, 0, 0), purpose 0 = draft sample,
// 1 = acceptance uniform, 2 = resample / bonus; u = ((w0 >> 8) + 0.5) * 2^-24,
// a uniform on (0, 1) that is exact in fp32.
//
// Every reduction has a fixed shape (thread-contiguous segments, warp
// shuffle trees, then one warp over the warp totals), so all results are
// run-to-run deterministic.
#include "ssd_internal.cuh"

namespace ssd {
namespace {

constexpr int kRowThreads = 1024;

// ---------------------------------------------------------------------------
// Philox4x32-10
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t philox_w0(unsigned long long seed, uint32_t pos, uint32_t purpose) {
    uint32_t c0 = pos, c1 = purpose, c2 = 0u, c3 = 0u;
    uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
        const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
        const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c0;
}

__device__ __forceinline__ float uniform01(unsigned long long seed, int pos, int purpose) {
    return ((float)(philox_w0(seed, (uint32_t)pos, (uint32_t)purpose) >> 8) + 0.5f) *
           (1.0f / 16777216.0f);
}

// ---------------------------------------------------------------------------
// block reductions (blockDim = 1024, fixed order)
// ---------------------------------------------------------------------------
__device__ float block_sum(float v, float* red) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    v = warp_sum(v);
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        float r = warp_sum(red[lane]);
        if (lane == 0) red[32] = r;
    }
    __syncthreads();
    float r = red[32];
    __syncthreads();
    return r;
}

__device__ float block_max(float v, float* red) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    v = warp_max(v);
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        float r = warp_max(red[lane]);
        if (lane == 0) red[32] = r;
    }
    __syncthreads();
    float r = red[32];
    __syncthreads();
    return r;
}

// argmax with the lowest index among equal maxima (NaN never wins)
__device__ __forceinline__ void better(float& v, int& i, float v2, int i2) {
    if (v2 > v || (v2 == v && i2 < i)) { v = v2; i = i2; }
}

__device__ int block_argmax(const float* x, int V, float* redf, int* redi) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    for (int i = threadIdx.x; i < V; i += kRowThreads) better(bv, bi, x[i], i);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
        int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
        better(bv, bi, v2, i2);
    }
    if (lane == 0) { redf[warp] = bv; redi[warp] = bi; }
    __syncthreads();
    if (warp == 0) {
        bv = redf[lane];
        bi = redi[lane];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
            int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
            better(bv, bi, v2, i2);
        }
        if (lane == 0) redi[32] = bi;
    }
    __syncthreads();
    int r = redi[32];
    __syncthreads();
    return (r < 0 || r >= V) ? 0 : r;
}

// ---------------------------------------------------------------------------
// sampling distribution of one row: softmax(logits / T) restricted to the
// nucleus {x : pi(x) >= tau*}, tau* = the largest value whose upper set holds
// >= top_p of the mass, renormalised.  s: shared row [V]; thread t owns the
// contiguous segment [t*seg, t*seg + seg).  tau* is found exactly by a
// 16-ary search over the fp32 bit patterns of pi (non-negative floats order
// like their bits), eight passes of 15 candidate thresholds.
// ---------------------------------------------------------------------------
__device__ void nucleus_row(const float* logits, int V, float inv_t, float top_p, float* s,
                            float* red) {
    const int seg = (V + kRowThreads - 1) / kRowThreads;
    const int beg = min(V, threadIdx.x * seg), end = min(V, beg + seg);
    float mx = -INFINITY;
    for (int i = beg; i < end; ++i) {
        float v = logits[i] * inv_t;
        s[i] = v;
        mx = fmaxf(mx, v);
    }
    mx = block_max(mx, red);
    float z = 0.f;
    for (int i = beg; i < end; ++i) {
        float e = expf(s[i] - mx);
        s[i] = e;
        z += e;
    }
    z = block_sum(z, red);
    for (int i = beg; i < end; ++i) s[i] = s[i] / z;
    if (!(top_p < 1.f)) { __syncthreads(); return; }

    __shared__ float wsum[32][16];
    __shared__ float cand_sum[16];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t lo = 0u, hi = 0x7F800001u;  // invariant: f(lo) >= top_p > f(hi)
    while (hi - lo > 1u) {
        const uint32_t step = (hi - lo + 15u) / 16u;
        float part[15];
#pragma unroll
        for (int c = 0; c < 15; ++c) part[c] = 0.f;
        for (int i = beg; i < end; ++i) {
            const uint32_t b = __float_as_uint(s[i]);
            const float v = s[i];
#pragma unroll
            for (int c = 0; c < 15; ++c)
                if (b >= lo + (uint32_t)(c + 1) * step) part[c] += v;
        }
#pragma unroll
        for (int c = 0; c < 15; ++c) {
            const float w = warp_sum(part[c]);
            if (lane == 0) wsum[warp][c] = w;
        }
        __syncthreads();
        if (threadIdx.x < 15) {
            float tot = 0.f;
            for (int w = 0; w < 32; ++w) tot += wsum[w][threadIdx.x];
            cand_sum[threadIdx.x] = tot;
        }
        __syncthreads();
        uint32_t nlo = lo, nhi = hi;
        for (int c = 0; c < 15; ++c) {
            const uint32_t t = lo + (uint32_t)(c + 1) * step;
            if (t >= hi) break;
            if (cand_sum[c] >= top_p) nlo = t;
            else { nhi = t; break; }
        }
        lo = nlo;
        hi = nhi;
        __syncthreads();
    }
    // kept mass (deterministic recount) and renormalisation
    float kept = 0.f;
    for (int i = beg; i < end; ++i)
        if (__float_as_uint(s[i]) >= lo) kept += s[i];
    kept = block_sum(kept, red);
    for (int i = beg; i < end; ++i) s[i] = __float_as_uint(s[i]) >= lo ? s[i] / kept : 0.f;
    __syncthreads();
}

// Inverse-CDF draw over the shared row s: the first x (ascending) with
// cumsum(x) > u * total.  Thread t owns the contiguous segment of the row and
// the interval [E_t, E_{t+1}) of the cumulative mass, E the exclusive scan of
// the segment sums (E_1024 = total), so exactly one segment holds the target;
// its thread walks it.  A target at or beyond the total (rounding as u -> 1)
// takes the last token with positive mass.
__device__ int sample_row(const float* s, int V, float u, float* red, int* redi) {
    __shared__ float ex[kRowThreads];
    const int seg = (V + kRowThreads - 1) / kRowThreads;
    const int beg = min(V, threadIdx.x * seg), end = min(V, beg + seg);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float mine = 0.f;
    int last_pos = -1;
    for (int i = beg; i < end; ++i) {
        mine += s[i];
        if (s[i] > 0.f) last_pos = i;
    }
    float incl = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) red[warp] = incl;
    int lp = last_pos;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, o));
    if (lane == 0) redi[warp] = lp;
    __syncthreads();
    if (warp == 0) {
        const float wt = red[lane];
        float wi = wt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            float y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        red[lane] = wi - wt;
        if (lane == 31) red[32] = wi;
        int l2 = redi[lane];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) l2 = max(l2, __shfl_xor_sync(0xffffffffu, l2, o));
        if (lane == 0) { redi[32] = l2; redi[33] = -1; }
    }
    __syncthreads();
    const float e_mine = red[warp] + (incl - mine);
    ex[threadIdx.x] = e_mine;
    __syncthreads();
    const float total = red[32];
    const float e_next = threadIdx.x + 1 < kRowThreads ? ex[threadIdx.x + 1] : total;
    const float target = u * total;
    if (e_mine <= target && target < e_next) {
        float cum = e_mine;
        int pick = last_pos;
        for (int i = beg; i < end; ++i) {
            cum += s[i];
            if (cum > target && s[i] > 0.f) { pick = i; break; }
        }
        redi[33] = pick;
    }
    __syncthreads();
    const int r = redi[33] >= 0 ? redi[33] : redi[32];
    __syncthreads();
    return r < 0 ? 0 : r;
}

// ---------------------------------------------------------------------------
// kernels
// ---------------------------------------------------------------------------
// greedy drafting: d_{j+1} = argmax of the draft logits.  With the draft
// exit on, the draft's confidence max softmax = 1 / sum_x exp(l_x - l_max)
// below gamma ends the round's drafting (Sec. 3.4; the draft is kept); a
// drafting stage that has ended adds nothing.
__global__ void __launch_bounds__(kRowThreads) greedy_draft_kernel(const float* __restrict__ logits,
                                                                   int V, DecodeState* st) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float redf[33];
    __shared__ int redi[34];
    if (st->exited) return;
    int best = block_argmax(logits, V, redf, redi);
    bool stop = false;
    if (st->exit_on) {
        const float lmax = logits[best];
        float s = 0.f;
        for (int i = threadIdx.x; i < V; i += kRowThreads) s += expf(logits[i] - lmax);
        s = block_sum(s, redf);
        stop = 1.f / s < st->gamma;
    }
    if (threadIdx.x == 0) {
        st->drafts[st->j] = best;
        st->j = st->j + 1;
        if (stop) st->exited = 1;
    }
}

// emission + rollback shared by both acceptance kernels (one thread)
__device__ void emit_round(DecodeState* st, int n, int y, int Kd, int* out_tokens) {
    const int e = st->emitted;
    for (int i = 0; i < n; ++i) out_tokens[e + i] = st->drafts[i];
    out_tokens[e + n] = y;
    st->emitted = e + n + 1;
    st->len = st->len + n + 1;
    st->x_last = y;
    st->rounds += 1;
    st->drafted += Kd;
    st->accepted += n;
    st->hist[n] += 1;
    st->j = 0;
    // adaptive draft exit: Eqs. 2-4 after a verification that had drafts
    if (st->exit_on && Kd > 0) {
        const float ar_e = (float)n / (float)Kd;
        const float b1 = st->exit_updates == 0 ? 0.f : st->beta1;
        st->ar_smooth = b1 * st->ar_smooth + (1.f - b1) * ar_e;
        const float gt = st->ar_smooth <= st->alpha ? st->gamma + st->eps : st->gamma - st->eps;
        st->gamma = st->beta2 * st->gamma + (1.f - st->beta2) * gt;
        st->exit_updates += 1;
    }
    st->exited = 0;
}

// greedy verification: one CTA per row computes argmax p_m; the last CTA
// accepts the longest matching prefix and emits (Algorithm 2)
__global__ void __launch_bounds__(kRowThreads) greedy_accept_kernel(
    const float* __restrict__ logits, int V, int M, DecodeState* st, int* out_tokens,
    unsigned* counter, int* argbuf) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float redf[33];
    __shared__ int redi[34];
    __shared__ int s_last;
    const int m = blockIdx.x;
    int best = block_argmax(logits + (size_t)m * V, V, redf, redi);
    if (threadIdx.x == 0) {
        argbuf[m] = best;
        __threadfence();
        unsigned prev = atomicAdd(counter, 1u);
        s_last = prev == (unsigned)(M - 1);
    }
    __syncthreads();
    if (!s_last || threadIdx.x != 0) return;
    __threadfence();
    int n = 0;
    while (n < M - 1 && st->drafts[n] == __ldcg(&argbuf[n])) ++n;
    const int y = __ldcg(&argbuf[n]);
    emit_round(st, n, y, M - 1, out_tokens);
    *counter = 0u;
}

// sampling drafting: q_{j+1} row kept for the acceptance test, d ~ q
__global__ void __launch_bounds__(kRowThreads) sample_draft_kernel(const float* __restrict__ logits,
                                                                   int V, DecodeState* st,
                                                                   float* q_rows) {
    extern __shared__ float s[];
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float red[33];
    __shared__ int redi[34];
    if (st->exited) return;  // the round's drafting stage has ended
    const int j = st->j;
    nucleus_row(logits, V, st->inv_temperature, st->top_p, s, red);
    float* q = q_rows + (size_t)j * V;
    float qmax = 0.f;
    for (int i = threadIdx.x; i < V; i += kRowThreads) {
        q[i] = s[i];
        qmax = fmaxf(qmax, s[i]);
    }
    const bool stop = st->exit_on && block_max(qmax, red) < st->gamma;  // confidence = max q (Sec. 3.4)
    const float u = uniform01(st->seed, st->len + j + 1, 0);
    int d = sample_row(s, V, u, red, redi);
    if (threadIdx.x == 0) {
        st->drafts[j] = d;
        st->j = j + 1;
        if (stop) st->exited = 1;
    }
}

// Algorithm 4's verification for one round, executed by one 1024-thread CTA
// over target rows p (Kd+1 rows) and draft rows q (Kd rows).  Returns n via
// *n_out and the correction / bonus token.
__device__ int spec_accept_core(const float* p, const float* q, const int* drafts, int Kd, int V,
                                unsigned long long seed, int len, float* s, float* red,
                                int* redi, int* n_out) {
    __shared__ int s_rej;
    if (threadIdx.x == 0) {
        int rej = Kd;  // index of the first rejected draft (0-based), Kd = none
        for (int j = 0; j < Kd; ++j) {
            const int x = drafts[j];
            const float pj = __ldcg(p + (size_t)j * V + x);
            const float qj = __ldcg(q + (size_t)j * V + x);
            const float r = uniform01(seed, len + j + 1, 1);
            // r < min(1, pj / qj)  <=>  r * qj < pj  (qj > 0)
            if (qj > 0.f && !(r * qj < pj)) { rej = j; break; }
        }
        s_rej = rej;
    }
    __syncthreads();
    const int rej = s_rej;
    const int seg = (V + kRowThreads - 1) / kRowThreads;
    const int beg = min(V, threadIdx.x * seg), end = min(V, beg + seg);
    int y;
    if (rej < Kd) {
        const float* pj = p + (size_t)rej * V;
        const float* qj = q + (size_t)rej * V;
        float tot = 0.f;
        for (int i = beg; i < end; ++i) {
            const float dlt = __ldcg(pj + i) - __ldcg(qj + i);
            s[i] = dlt > 0.f ? dlt : 0.f;
            tot += s[i];
        }
        tot = block_sum(tot, red);
        if (!(tot > 1e-30f)) {
            for (int i = beg; i < end; ++i) s[i] = __ldcg(pj + i);
        }
        __syncthreads();
        y = sample_row(s, V, uniform01(seed, len + rej + 1, 2), red, redi);
    } else {
        const float* pk = p + (size_t)Kd * V;
        for (int i = beg; i < end; ++i) s[i] = __ldcg(pk + i);
        __syncthreads();
        y = sample_row(s, V, uniform01(seed, len + Kd + 1, 2), red, redi);
    }
    *n_out = rej;
    return y;
}

__global__ void __launch_bounds__(kRowThreads) sample_accept_kernel(
    const float* __restrict__ logits, int V, int M, DecodeState* st, float* p_rows,
    const float* q_rows, int* out_tokens, unsigned* counter) {
    extern __shared__ float s[];
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float red[33];
    __shared__ int redi[34];
    __shared__ int s_last;
    const int m = blockIdx.x;
    nucleus_row(logits + (size_t)m * V, V, st->inv_temperature, st->top_p, s, red);
    float* pr = p_rows + (size_t)m * V;
    for (int i = threadIdx.x; i < V; i += kRowThreads) pr[i] = s[i];
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned prev = atomicAdd(counter, 1u);
        s_last = prev == (unsigned)(M - 1);
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    int n;
    const int y = spec_accept_core(p_rows, q_rows, st->drafts, M - 1, V, st->seed, st->len, s, red,
                                   redi, &n);
    if (threadIdx.x == 0) {
        emit_round(st, n, y, M - 1, out_tokens);
        *counter = 0u;
    }
}

__global__ void __launch_bounds__(kRowThreads) spec_accept_batch_kernel(
    const float* p, const float* q, int V, int Kd, const int* drafts,
    const unsigned long long* seeds, int pos0, int* out) {
    extern __shared__ float s[];
    __shared__ float red[33];
    __shared__ int redi[34];
    const int t = blockIdx.x;
    int n;
    const int y = spec_accept_core(p, q, drafts + (size_t)t * Kd, Kd, V, seeds[t], pos0, s, red,
                                   redi, &n);
    if (threadIdx.x == 0) {
        out[2 * t] = n;
        out[2 * t + 1] = y;
    }
}

template <typename Kern, typename... Args>
int launch_pdl(Kern k, dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return (int)cudaLaunchKernelEx(&cfg, k, args...);
}

}  // namespace

int sampling_configure() {
    // load every kernel of this file now, outside any stream capture
    cudaFuncAttributes fa;
    cudaError_t e0 = cudaFuncGetAttributes(&fa, greedy_draft_kernel);
    if (e0 == cudaSuccess) e0 = cudaFuncGetAttributes(&fa, greedy_accept_kernel);
    if (e0 != cudaSuccess) return (int)e0;
    const int big = 160 * 1024;
    cudaError_t e = cudaFuncSetAttribute(sample_draft_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, big);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(sample_accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, big);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(spec_accept_batch_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, big);
    return (int)e;
}

int launch_greedy_draft(const float* logits, int V, DecodeState* st, cudaStream_t s) {
    return launch_pdl(greedy_draft_kernel, dim3(1), dim3(kRowThreads), 0, s, logits, V, st);
}

int launch_greedy_accept(const float* logits, int V, int M, DecodeState* st, int* out_tokens,
                         unsigned* counter, int* argmax_buf, cudaStream_t s) {
    return launch_pdl(greedy_accept_kernel, dim3(M), dim3(kRowThreads), 0, s, logits, V, M, st,
                      out_tokens, counter, argmax_buf);
}

int launch_sample_draft(const float* logits, int V, DecodeState* st, float* q_rows, cudaStream_t s) {
    return launch_pdl(sample_draft_kernel, dim3(1), dim3(kRowThreads), (size_t)V * 4, s, logits, V,
                      st, q_rows);
}

int launch_sample_accept(const float* logits, int V, int M, DecodeState* st, float* p_rows,
                         const float* q_rows, int* out_tokens, unsigned* counter, cudaStream_t s) {
    return launch_pdl(sample_accept_kernel, dim3(M), dim3(kRowThreads), (size_t)V * 4, s, logits, V,
                      M, st, p_rows, q_rows, out_tokens, counter);
}

int launch_spec_accept_batch(const float* p_rows, const float* q_rows, int V, int Kd,
                             const int* drafts, const unsigned long long* seeds, int trials,
                             int pos0, int* out, cudaStream_t s) {
    spec_accept_batch_kernel<<<trials, kRowThreads, (size_t)V * 4, s>>>(p_rows, q_rows, V, Kd, drafts,
                                                                        seeds, pos0, out);
    return (int)cudaGetLastError();
}

}  // namespace ssd
