// tc_gemm.cuh - the prompt-encoding GEMM on the 5th-generation tensor cores
// (tcgen05, sm_103a): D[rows x 256] = A[rows x K] * B[256 x K]^T per CTA
// tile, with the fused epilogues of the prefill.
//
// The prefill (Sec. 3.1: the prompt is encoded before Algorithms 1 / 2 start
// decoding) runs every prompt row through the full model at once, so its
// projections are dense GEMMs with M = 128 .. 2048 token rows: compute-bound,
// unlike the decode forwards.  One CTA computes a 128-row x 256-column tile:
//   warp 0, one thread : TMA producer.  Per 64-wide k block it copies the
//                        activation tile twice (bf16 hi and lo planes, 128 x 64
//                        each) and the weight tile as two 128-row boxes (so
//                        the 256 columns can come from two matrices, e.g. the
//                        gate and up rows of the same features), 128-byte
//                        swizzle, into a ring of kTcStages stages;
//   warp 1, one thread : MMA issuer.  tcgen05.mma kind::f16 (bf16 x bf16 ->
//                        fp32), M = 128, N = 256, K = 16, eight per k block
//                        (four k steps x hi and lo), accumulating in TMEM;
//                        tcgen05.commit releases each stage and finally
//                        signals the epilogue;
//   warps 0-3          : epilogue.  Warp w reads TMEM lanes 32w..32w+31 (one
//                        token row per thread) with tcgen05.ld and applies
//                        the op's epilogue.
// Operands are K-major with the canonical 128-byte-swizzle layout that TMA
// writes: row r of a tile at r * 128 bytes, 8-row groups 1024 bytes apart
// (the descriptor's stride byte offset), each k step of 16 moves the start
// address by 32 bytes inside the swizzle row.
//
// Precision: as in the decode forwards, the fp32 activations enter as bf16
// hi = rn(x) and lo = rn(x - hi); W * hi + W * lo accumulate in the same fp32
// TMEM accumulator (~16 mantissa bits of x).
//
// Every wait is bounded (~2 s): on a timeout the thread records the error
// code and stops waiting; the CTA then gives its copies and MMAs in flight
// time to finish, frees its TMEM and returns.
#pragma once

#include "ssd_internal.cuh"

namespace ssd {
namespace tc {

constexpr int kBM = 128;          // token rows per tile (TMEM lanes)
constexpr int kBN = 256;          // output columns per tile (TMEM columns)
constexpr int kBK = 64;           // k per stage: 128 bytes of bf16 = one swizzle row
constexpr int kStages = 3;
constexpr int kThreads = 128;
constexpr int kATile = kBM * kBK * 2;        // 16 KB (one plane)
constexpr int kBTile = kBN * kBK * 2;        // 32 KB
constexpr int kStage = 2 * kATile + kBTile;  // 64 KB
constexpr size_t kSmemBytes = 1024 + (size_t)kStages * kStage + 256;
constexpr unsigned long long kWaitNs = 2000000000ull;
constexpr int kErrTimeout = 1;

// epilogues of the prefill GEMMs
enum TcEpi { TC_STORE = 0, TC_RESID = 1, TC_SWIGLU = 2, TC_QKV = 3 };

struct TcArgs {
    // TMA maps: activation planes (hi, lo) viewed as {K, rows}, box {64, 128};
    // weight matrices viewed as {K, N}, box {64, 128}
    const void* tm_a_hi;
    const void* tm_a_lo;
    const void* tm_b[3];   // weight matrices (QKV: wq, wk, wv; SWIGLU: gate, up; else [0])
    int rows;              // valid token rows
    int K;
    int n_kb;              // ceil(K / 64)
    int n_tiles;           // column tiles (gridDim.y)
    int N;                 // valid output columns (STORE / RESID: width of out)
    float* out;            // STORE: [rows][ldo] fp32; RESID: residual h [rows][ldo] (+= D)
    int ldo;
    // SWIGLU: act planes [rows][ffn] bf16 hi / lo of silu(gate) * up
    int ffn;
    bf16* act_hi;
    bf16* act_lo;
    // QKV: q (fp32, rotated) [rows][H*hd]; K / V cache of the layer
    // [Hkv][max_seq][hd] fp16; RoPE table [max_seq][hd/2] (cos, sin)
    int n_heads, n_kv_heads, head_dim, max_seq, pos0;
    float* q;
    f16* k_cache;
    f16* v_cache;
    const float2* rope;
    int* err;
};

// 128-row boxes of tile t: matrix index and first row of each half
struct TcHalves {
    int s0, r0, s1, r1;
};
__device__ __forceinline__ TcHalves tc_halves(const TcArgs& a, int epi, int t) {
    if (epi == TC_SWIGLU) return {0, t * 128, 1, t * 128};  // gate rows, up rows of features t*128..
    if (epi == TC_QKV) {
        // [Wq; Wk; Wv] in 128-row boxes (q and kv widths are multiples of 128)
        const int qd = a.n_heads * a.head_dim, kvd = a.n_kv_heads * a.head_dim;
        int b[2], s[2];
        for (int h = 0; h < 2; ++h) {
            int r = (2 * t + h) * 128;
            if (r < qd) { s[h] = 0; b[h] = r; }
            else if (r < qd + kvd) { s[h] = 1; b[h] = r - qd; }
            else { s[h] = 2; b[h] = r - qd - kvd; }
        }
        return {s[0], b[0], s[1], b[1]};
    }
    return {0, t * kBN, 0, t * kBN + 128};
}

// ---------------------------------------------------------------------------
// PTX wrappers (tcgen05, TMA, mbarrier)
// ---------------------------------------------------------------------------
__device__ __forceinline__ unsigned long long gtime() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mb_init(uint64_t* b, unsigned n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void mb_arrive_tx(uint64_t* b, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mb_try(uint64_t* b, unsigned parity) {
    unsigned ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// bounded wait; false (error recorded) after kWaitNs or once another thread
// of the grid recorded an error and 20 us have passed
__device__ __forceinline__ bool mb_wait(uint64_t* b, unsigned parity, int* err) {
    if (mb_try(b, parity)) return true;
    const unsigned long long t0 = gtime();
    while (!mb_try(b, parity)) {
        const unsigned long long dt = gtime() - t0;
        if (dt > 20000ull && *(volatile int*)err) return false;
        if (dt > kWaitNs) {
            atomicCAS(err, 0, kErrTimeout);
            return false;
        }
    }
    return true;
}
// 2D tiled TMA load; x (the k coordinate) is always a multiple of 64 elements
__device__ __forceinline__ void tma2d(void* dst, const void* map, int x, int y, uint64_t* b) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_u32(dst)), "l"(map), "r"(x), "r"(y), "r"(smem_u32(b))
        : "memory");
}

// shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart; the start address may sit 32 / 64 / 96 bytes into a
// swizzle row (k steps of 16 bf16)
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
    d |= (uint64_t)1 << 16;                           // leading byte offset (unused with this swizzle)
    d |= (uint64_t)(1024 >> 4) << 32;                 // stride byte offset
    d |= (uint64_t)1 << 46;                           // descriptor version
    d |= (uint64_t)2 << 61;                           // 128-byte swizzle
    return d;
}
// instruction descriptor: kind::f16, A = B = bf16, D = fp32, both K-major,
// N = 256, M = 128
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kBN >> 3) << 17) |
                            ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t ad, uint64_t bd, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
        ::"r"(tmem_d), "l"(ad), "l"(bd), "r"(kIdesc), "r"(accumulate)
        : "memory");
}
// the mbarrier completes once every tcgen05 op this thread issued so far is done
__device__ __forceinline__ void mma_commit(uint64_t* b) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(b))
                 : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// ---------------------------------------------------------------------------
// epilogue helpers (one token row per thread, 32 columns at a time)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void store_hilo(bf16* hi, bf16* lo, float x) {
    const bf16 h = __float2bfloat16_rn(x);
    *hi = h;
    *lo = __float2bfloat16_rn(x - __bfloat162float(h));
}

// ---------------------------------------------------------------------------
// the kernel: grid = (column tiles, row tiles)
// ---------------------------------------------------------------------------
template <int EPI>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const TcArgs a) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStage);
    uint64_t* empty = full + kStages;
    uint64_t* done = empty + kStages;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
    __shared__ int s_fail;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // row tiles fastest: the CTAs that share a weight tile run together, so
    // each weight tile is read from DRAM once and from L2 by the other rows
    const int tile = blockIdx.y, m0 = blockIdx.x * kBM;
    if (threadIdx.x == 0) {
        s_fail = 0;
        for (int s = 0; s < kStages; ++s) {
            mb_init(full + s, 1);
            mb_init(empty + s, 1);
        }
        mb_init(done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 2) {  // TMEM: 256 fp32 columns x 128 lanes for the accumulator
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(kBN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = *tmem_slot;

    bool ok = true;
    if (warp == 0 && lane == 0) {
        // producer: activations (may be written by the previous kernel:
        // generic proxy) and weights through TMA
        asm volatile("fence.proxy.async.global;" ::: "memory");
        const TcHalves hv = tc_halves(a, EPI, tile);
        for (int kb = 0; kb < a.n_kb && ok; ++kb) {
            const int s = kb % kStages;
            if (kb >= kStages) ok = mb_wait(empty + s, ((kb / kStages) - 1) & 1u, a.err);
            if (!ok) break;
            unsigned char* st = smem + s * kStage;
            mb_arrive_tx(full + s, (unsigned)kStage);
            tma2d(st, a.tm_a_hi, kb * kBK, m0, full + s);
            tma2d(st + kATile, a.tm_a_lo, kb * kBK, m0, full + s);
            tma2d(st + 2 * kATile, a.tm_b[hv.s0], kb * kBK, hv.r0, full + s);
            tma2d(st + 2 * kATile + kATile, a.tm_b[hv.s1], kb * kBK, hv.r1, full + s);
        }
    } else if (warp == 1 && lane == 0) {
        // MMA issuer
        for (int kb = 0; kb < a.n_kb && ok; ++kb) {
            const int s = kb % kStages;
            ok = mb_wait(full + s, (kb / kStages) & 1u, a.err);
            if (!ok) break;
            fence_after();
            const uint32_t st = smem_u32(smem + s * kStage);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
                const uint64_t bd = sdesc(st + 2 * kATile + kk * 32);
                mma_bf16(tmem, sdesc(st + kk * 32), bd, (kb | kk) != 0);
                mma_bf16(tmem, sdesc(st + kATile + kk * 32), bd, 1u);
            }
            mma_commit(empty + s);  // the stage is free once these MMAs have read it
        }
        if (ok) mma_commit(done);
    }
    if (!ok) s_fail = 1;
    __syncwarp();

    // epilogue: wait for the accumulator (all threads)
    if (ok) ok = mb_wait(done, 0, a.err);
    if (!ok) s_fail = 1;
    fence_after();
    const int row = m0 + warp * 32 + lane;  // this thread's token row
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    __syncthreads();
    if (!s_fail) {
        if (EPI == TC_STORE || EPI == TC_RESID) {
            for (int c0 = 0; c0 < kBN; c0 += 32) {
                float v[32];
                tmem_ld32(tl + c0, v);
                const int n0 = tile * kBN + c0;
                if (row < a.rows) {
                    float* o = a.out + (size_t)row * a.ldo + n0;
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (n0 + i < a.N) o[i] = EPI == TC_RESID ? o[i] + v[i] : v[i];
                }
            }
        } else if (EPI == TC_SWIGLU) {
            for (int c0 = 0; c0 < 128; c0 += 32) {
                float g[32], u[32];
                tmem_ld32(tl + c0, g);
                tmem_ld32(tl + 128 + c0, u);
                const int f0 = tile * 128 + c0;
                if (row < a.rows) {
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        if (f0 + i >= a.ffn) break;
                        const float x = g[i] / (1.f + expf(-g[i])) * u[i];
                        const size_t at = (size_t)row * a.ffn + f0 + i;
                        store_hilo(a.act_hi + at, a.act_lo + at, x);
                    }
                }
            }
        } else {  // TC_QKV: two 128-row boxes, each whole heads of q, k or v
            const int hd = a.head_dim, half = hd >> 1;
            const int qd = a.n_heads * hd, kvd = a.n_kv_heads * hd;
            const int pos = a.pos0 + row;
            for (int h = 0; h < 2; ++h) {
                const int f0 = (2 * tile + h) * 128;  // feature of column 0 of this box
                if (f0 >= qd + 2 * kvd) break;
                const int kind = f0 < qd ? 0 : (f0 < qd + kvd ? 1 : 2);
                const int fb = kind == 0 ? f0 : (kind == 1 ? f0 - qd : f0 - qd - kvd);
                for (int hb = 0; hb < 128; hb += hd) {       // heads in this box
                    for (int c0 = 0; c0 < half; c0 += 32) {  // rotation pairs (i, i + half)
                        float x1[32], x2[32];
                        tmem_ld32(tl + h * 128 + hb + c0, x1);
                        tmem_ld32(tl + h * 128 + hb + half + c0, x2);
                        if (row >= a.rows) continue;
                        const int head = (fb + hb) / hd;
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const int ii = c0 + i;
                            if (kind == 2) {
                                f16* vrow = a.v_cache + ((size_t)head * a.max_seq + pos) * hd;
                                vrow[ii] = __float2half_rn(x1[i]);
                                vrow[ii + half] = __float2half_rn(x2[i]);
                                continue;
                            }
                            const float2 cs = a.rope[(size_t)pos * half + ii];
                            const float y1 = x1[i] * cs.x - x2[i] * cs.y;
                            const float y2 = x2[i] * cs.x + x1[i] * cs.y;
                            if (kind == 0) {
                                float* q = a.q + (size_t)row * qd + head * hd;
                                q[ii] = y1;
                                q[ii + half] = y2;
                            } else {
                                f16* krow = a.k_cache + ((size_t)head * a.max_seq + pos) * hd;
                                krow[ii] = __float2half_rn(y1);
                                krow[ii + half] = __float2half_rn(y2);
                            }
                        }
                    }
                }
            }
        }
    } else {
        // a wait gave up: let copies and MMAs in flight finish before the
        // shared memory and TMEM are released
        if (threadIdx.x == 0) {
            const unsigned long long t0 = gtime();
            while (gtime() - t0 < 2000000ull) __nanosleep(1000);
        }
    }
    fence_before();
    __syncthreads();
    if (warp == 2) {
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kBN) : "memory");
    }
}

template <int EPI>
inline int tc_configure() {
    return (int)cudaFuncSetAttribute(tc_gemm_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kSmemBytes);
}

template <int EPI>
inline int tc_launch(const TcArgs& a, int row_tiles, cudaStream_t s) {
    tc_gemm_kernel<EPI><<<dim3(row_tiles, a.n_tiles), kThreads, kSmemBytes, s>>>(a);
    return (int)cudaGetLastError();
}

}  // namespace tc
}  // namespace ssd
