// gemm.cu - the stand-alone skinny projection GEMM of ssd_linear_noalloc:
// Y[M x N] = X[M x K] * W^T with W bf16 [N][K], fp32 X and Y, M <= 16.
//
// The weights are the large operand, so the kernel is "swap-AB": 16 weight
// rows form the M side of an m16n8k16 tensor-core MMA and the <= 16
// activation rows form its N side.  The result for activation row m depends
// only on row m (the MMA computes every output column independently, and the
// split of K into CTA chunks, into k-interleaved warps and into the
// fixed-order split-K combine depends on (N, K) only).
//
// Precision: the fp32 activation rows are split into bf16 hi = rn(x) and
// lo = rn(x - hi) and both are multiplied (the MMA's N side holds the hi rows
// then the lo rows), so the product sees ~16 mantissa bits of x; the weights
// are exact bf16; accumulation is fp32.
//
// CTA = 256 threads: warp w handles the 16-row group (w & 3) of the 64-row
// tile and the k32 blocks b = (w >> 2) (mod 2) of its k-chunk.  The weight
// chunk (64 rows x kc) is streamed HBM -> shared memory with 16-byte cp.async,
// then fed to the MMA with a k-permutation: thread (g, t) reads 8 consecutive
// bf16 of a row, which the A and B fragments both interpret as the same
// logical k slots, so the product is unchanged and every load is a 128-bit LDS.
#include <mutex>
#include <string>

#include "ssd.h"
#include "ssd_internal.cuh"

namespace ssd {
namespace {

// NPH = n8 tiles per activation half (1: M <= 8, 2: M <= 16).  The MMA's N
// side holds P = 8*NPH rows of x_hi followed by P rows of x_lo.
template <int NPH>
__global__ void __launch_bounds__(kGemmThreads) gemm_kernel(const GemmArgs a) {
    constexpr int NT = 2 * NPH;
    constexpr int P = 8 * NPH;
    constexpr int RC = 2 * P;
    extern __shared__ __align__(16) unsigned char smem[];
    pdl_launch_dependents();
    const int tile = blockIdx.x, split = blockIdx.y;
    const int k0 = split * a.kc;
    const int kc_eff = min(a.kc, a.K - k0);
    const int pitch = a.kc * 2 + 64;  // bytes; pitch % 128 == 64 -> conflict-free LDS.128
    unsigned char* ws = smem;
    unsigned char* xs = smem + kTileRows * pitch;                // [2P][pitch] hi rows, then lo rows
    float* red = reinterpret_cast<float*>(xs + 2 * P * pitch);  // [64][RC]
    float* ys = reinterpret_cast<float*>(smem);                  // [64][16], reuses ws after the MMA
    __shared__ int s_last;

    // 1. stream the weight chunk (independent of the previous kernel)
    const int cpr = kc_eff >> 3;  // 16-byte chunks per row
    for (int c = threadIdx.x; c < kTileRows * cpr; c += kGemmThreads) {
        int r = c / cpr, cc = c - r * cpr;
        const int n = tile * kTileRows + r;
        const bf16* src = n < a.N ? a.w0 + (size_t)n * a.K : nullptr;
        const bf16* g = src ? src + k0 + cc * 8 : a.w0;
        SSD_GUARD(a.err, (((uintptr_t)g & 15u) == 0) && (r * pitch + cc * 16 + 16 <= kTileRows * pitch), 101)
        cp_async16(ws + r * pitch + cc * 16, g, src ? 16 : 0);
    }
    cp_async_commit();
    // 2. activations of the previous kernel: fp32 -> bf16 hi / lo rows
    pdl_wait();
    for (int c = threadIdx.x; c < P * cpr; c += kGemmThreads) {
        int n = c / cpr, cc = c - n * cpr;
        uint4 hi = make_uint4(0, 0, 0, 0), lo = make_uint4(0, 0, 0, 0);
        if (n < a.M) {
            const float4* src = reinterpret_cast<const float4*>(a.x + (size_t)n * a.K + k0 + cc * 8);
            split8(__ldcg(src), __ldcg(src + 1), hi, lo);
        }
        *reinterpret_cast<uint4*>(xs + n * pitch + cc * 16) = hi;
        *reinterpret_cast<uint4*>(xs + (P + n) * pitch + cc * 16) = lo;
    }
    cp_async_wait<0>();
    __syncthreads();

    // 3. tensor-core MMA over the chunk
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rg = warp & 3, kh = warp >> 2;
    const int g = lane >> 2, tig = lane & 3;
    float acc[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
    const unsigned char* ar0 = ws + (rg * 16 + g) * pitch;
    const unsigned char* ar1 = ar0 + 8 * pitch;
    const int nb = kc_eff >> 5;
#pragma unroll 2
    for (int b = kh; b < nb; b += 2) {
        const int off = b * 64 + tig * 16;
        uint4 wa = *reinterpret_cast<const uint4*>(ar0 + off);
        uint4 wb = *reinterpret_cast<const uint4*>(ar1 + off);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            uint4 xv = *reinterpret_cast<const uint4*>(xs + (nt * 8 + g) * pitch + off);
            mma_bf16_16816(acc[nt], wa.x, wb.x, wa.y, wb.y, xv.x, xv.y);
            mma_bf16_16816(acc[nt], wa.z, wb.z, wa.w, wb.w, xv.z, xv.w);
        }
    }
    if ((kc_eff & 31) && kh == (nb & 1)) {  // k16 tail block
        const int off = nb * 64 + tig * 8;
        uint2 wa = *reinterpret_cast<const uint2*>(ar0 + off);
        uint2 wb = *reinterpret_cast<const uint2*>(ar1 + off);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            uint2 xv = *reinterpret_cast<const uint2*>(xs + (nt * 8 + g) * pitch + off);
            mma_bf16_16816(acc[nt], wa.x, wb.x, wa.y, wb.y, xv.x, xv.y);
        }
    }

    // 4. fixed-order combines: k-interleave 0 + 1, then x_hi + x_lo -> ys[row][m]
    const int r0 = rg * 16 + g;
    if (kh == 1) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            int c = nt * 8 + 2 * tig;
            red[r0 * RC + c] = acc[nt][0];
            red[r0 * RC + c + 1] = acc[nt][1];
            red[(r0 + 8) * RC + c] = acc[nt][2];
            red[(r0 + 8) * RC + c + 1] = acc[nt][3];
        }
    }
    __syncthreads();
    if (kh == 0) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            int c = nt * 8 + 2 * tig;
            red[r0 * RC + c] = acc[nt][0] + red[r0 * RC + c];
            red[r0 * RC + c + 1] = acc[nt][1] + red[r0 * RC + c + 1];
            red[(r0 + 8) * RC + c] = acc[nt][2] + red[(r0 + 8) * RC + c];
            red[(r0 + 8) * RC + c + 1] = acc[nt][3] + red[(r0 + 8) * RC + c + 1];
        }
    }
    __syncthreads();
    const int M = a.M;
    for (int idx = threadIdx.x; idx < kTileRows * M; idx += kGemmThreads) {
        int m = idx / kTileRows, r = idx - m * kTileRows;
        ys[r * 16 + m] = red[r * RC + m] + red[r * RC + P + m];
    }
    __syncthreads();

    // 5. split-K: the last CTA of the tile sums the partials in split order
    if (a.ksplit > 1) {
        const size_t NP = (size_t)a.n_tiles * kTileRows;
        for (int idx = threadIdx.x; idx < M * kTileRows; idx += kGemmThreads) {
            int m = idx / kTileRows, r = idx - m * kTileRows;
            a.partial[((size_t)split * M + m) * NP + (size_t)tile * kTileRows + r] = ys[r * 16 + m];
        }
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            unsigned prev = atomicAdd(&a.counters[tile], 1u);
            s_last = (prev == (unsigned)(a.ksplit - 1));
        }
        __syncthreads();
        if (!s_last) return;
        __threadfence();
        for (int idx = threadIdx.x; idx < M * kTileRows; idx += kGemmThreads) {
            int m = idx / kTileRows, r = idx - m * kTileRows;
            const float* p = a.partial + (size_t)m * NP + (size_t)tile * kTileRows + r;
            float s = __ldcg(p);
            for (int sp = 1; sp < a.ksplit; ++sp) s += __ldcg(p + (size_t)sp * M * NP);
            ys[r * 16 + m] = s;
        }
        if (threadIdx.x == 0) a.counters[tile] = 0u;
        __syncthreads();
    }

    // 6. the output rows
    for (int idx = threadIdx.x; idx < M * kTileRows; idx += kGemmThreads) {
        int m = idx / kTileRows, r = idx - m * kTileRows;
        int n = tile * kTileRows + r;
        if (n < a.N) a.out_f32[(size_t)m * a.ldo + n] = ys[r * 16 + m];
    }
}

template <int NPH>
int launch_one(const GemmArgs& a, cudaStream_t s) {
    const size_t smem = gemm_smem_bytes(a.kc, a.M);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_tiles, a.ksplit, 1);
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return (int)cudaLaunchKernelEx(&cfg, gemm_kernel<NPH>, a);
}

template <int NPH>
int configure_one() {
    return (int)cudaFuncSetAttribute(gemm_kernel<NPH>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
}

}  // namespace

int gemm_configure() {
    int e = configure_one<1>();
    return e ? e : configure_one<2>();
}

size_t gemm_smem_bytes(int kc, int M) {
    const int P = gemm_half_rows(M);
    return (size_t)(kTileRows + 2 * P) * (kc * 2 + 64) + (size_t)kTileRows * 2 * P * sizeof(float);
}

}  // namespace ssd

// ---------------------------------------------------------------------------
// ssd_linear_noalloc: the projection GEMM with its split-K scratch in a fixed
// device array instead of memory the caller or the library allocates.
//
// Some callers cannot allocate device memory at the point where they need a
// projection: a serving process that reserves every byte of HBM at start-up
// and treats any later allocation as a failure, a plug-in whose host
// framework owns all device allocations, or a latency-critical loop that
// must not call cudaMalloc / cudaFree because those calls can synchronise
// the whole device.  For them this entry point takes device inputs and
// outputs only and keeps its scratch (split-K partial sums and the per-tile
// arrival counters) in the static arrays below.  Every GPU that loads the
// library holds these arrays (about 4 MiB) until the process exits.
// ---------------------------------------------------------------------------
namespace ssd {
namespace {

constexpr size_t kNoAllocPartialFloats = size_t(1) << 20;  // 4 MiB of partial sums
constexpr int kNoAllocTiles = 4096;                          // 64-row tiles: N <= 262144

static __device__ __align__(256) float g_noalloc_partial[kNoAllocPartialFloats];
static __device__ __align__(256) unsigned g_noalloc_counters[kNoAllocTiles];
static __device__ __align__(256) int g_noalloc_err;

// Host-side device addresses of the arrays, resolved once per device.  (In
// host code the array names are host stand-ins, not device addresses.)
struct NoAllocDevice {
    bool ready = false;
    float* partial = nullptr;
    unsigned* counters = nullptr;
    int* err = nullptr;
};
constexpr int kNoAllocMaxDevices = 64;
NoAllocDevice g_noalloc_dev[kNoAllocMaxDevices];
std::mutex g_noalloc_mu;

int noalloc_setup(int dev, NoAllocDevice** out) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoAllocDevice& d = g_noalloc_dev[dev];
    if (!d.ready) {
        cudaError_t e = cudaGetSymbolAddress((void**)&d.partial, g_noalloc_partial);
        if (e == cudaSuccess) e = cudaGetSymbolAddress((void**)&d.counters, g_noalloc_counters);
        if (e == cudaSuccess) e = cudaGetSymbolAddress((void**)&d.err, g_noalloc_err);
        if (e == cudaSuccess) e = (cudaError_t)configure_one<1>();
        if (e == cudaSuccess) e = (cudaError_t)configure_one<2>();
        // (the arrays start at zero when the module loads; each call clears
        // the counters it uses on its own stream)
        if (e != cudaSuccess)
            return set_last_error(SSD_ERR_CUDA, (std::string("ssd_linear_noalloc set-up: ") +
                                                 cudaGetErrorString(e)).c_str());
        d.ready = true;
    }
    *out = &d;
    return SSD_OK;
}

}  // namespace
}  // namespace ssd

extern "C" int ssd_linear_noalloc(const void* w, const float* x, float* y, int N, int K, int M,
                                  void* cuda_stream) {
    using namespace ssd;
    if (!w || !x || !y) return set_last_error(SSD_ERR_INVALID_ARG, "ssd_linear_noalloc: NULL pointer");
    if (((uintptr_t)w & 15u) || ((uintptr_t)x & 15u))
        return set_last_error(SSD_ERR_INVALID_ARG, "ssd_linear_noalloc: w and x must be 16-byte aligned");
    if (M < 1 || M > kMaxRows || N < 1 || K < 16 || K % 16)
        return set_last_error(SSD_ERR_INVALID_ARG,
                              "ssd_linear_noalloc: need 1 <= M <= 16, N >= 1, K a positive multiple of 16");
    const int kc = K >= 512 ? 512 : ((K + 63) / 64) * 64;
    const int ksplit = (K + kc - 1) / kc;
    const int n_tiles = (N + kTileRows - 1) / kTileRows;
    const size_t need = ksplit > 1 ? (size_t)ksplit * M * n_tiles * kTileRows : 0;
    if (n_tiles > kNoAllocTiles || need > kNoAllocPartialFloats)
        return set_last_error(SSD_ERR_CAPACITY,
                              ("ssd_linear_noalloc: problem needs " + std::to_string(need) +
                               " scratch floats and " + std::to_string(n_tiles) +
                               " tiles; the fixed scratch holds 1048576 floats and 4096 tiles")
                                  .c_str());
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices)
        return set_last_error(SSD_ERR_CUDA, "ssd_linear_noalloc: no usable current device");
    NoAllocDevice* d = nullptr;
    int rc = noalloc_setup(dev, &d);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)cuda_stream;
    // the arrival counters must start at zero (the array keeps the last call's contents)
    e = cudaMemsetAsync(d->counters, 0, sizeof(unsigned) * n_tiles, s);
    GemmArgs a{};
    a.w0 = (const bf16*)w;
    a.N = N;
    a.K = K;
    a.kc = kc;
    a.ksplit = ksplit;
    a.n_tiles = n_tiles;
    a.x = x;
    a.M = M;
    a.partial = d->partial;
    a.counters = d->counters;
    a.out_f32 = y;
    a.ldo = N;
    a.err = d->err;
    if (e == cudaSuccess)
        e = (cudaError_t)(M > 8 ? launch_one<2>(a, s) : launch_one<1>(a, s));
    if (e != cudaSuccess)
        return set_last_error(SSD_ERR_CUDA, (std::string("ssd_linear_noalloc: ") + cudaGetErrorString(e)).c_str());
#ifdef SSD_CHECKED
    // checked builds: the kernel's alignment / bounds guards record a code in
    // the device flag; read it back (this makes the call synchronous), clear it
    // for the next call and report it
    int derr = 0;
    e = cudaMemcpyAsync(&derr, d->err, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = cudaMemsetAsync(d->err, 0, sizeof(int), s);
    if (e != cudaSuccess)
        return set_last_error(SSD_ERR_CUDA, (std::string("ssd_linear_noalloc: ") + cudaGetErrorString(e)).c_str());
    if (derr)
        return set_last_error(SSD_ERR_CUDA,
                              ("ssd_linear_noalloc: device check failed with code " + std::to_string(derr)).c_str());
#endif
    return SSD_OK;
}

