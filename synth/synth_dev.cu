// synth_dev.cu - seeded synthetic inputs (device side).
//
// Device twin of synth_host.c: the same element-wise definition (SplitMix64
// output function, Irwin-Hall(8) sum, one fp64 multiply, double->float->bf16
// round-to-nearest-even), so a multi-GB random-init model can be written
// straight into HBM.  It is an input generator only; it holds none of the
// decoding method's arithmetic and is not part of the decode library.
#include <cstdint>
#include <cuda_runtime.h>

namespace {

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint16_t f32_to_bf16_rne(float f) {
    uint32_t u = __float_as_uint(f);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

__global__ void fill_bf16_kernel(uint16_t* out, uint64_t first, uint64_t n, uint64_t s2,
                                 uint64_t base, double c) {
    uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
    for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += stride) {
        uint64_t key = base | (first + j);
        uint64_t w0 = mix64(s2 ^ (2u * key));
        uint64_t w1 = mix64(s2 ^ (2u * key + 1u));
        int64_t s = 0;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            s += (int64_t)((w0 >> (16 * b)) & 0xFFFFu);
            s += (int64_t)((w1 >> (16 * b)) & 0xFFFFu);
        }
        double v = __dmul_rn((double)(s - 262140), c);
        out[j] = f32_to_bf16_rne(__double2float_rn(v));
    }
}

__global__ void fill_const_kernel(uint16_t* out, uint64_t n, uint16_t bits) {
    uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
    for (uint64_t j = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += stride)
        out[j] = bits;
}

uint64_t host_mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

}  // namespace

extern "C" int synth_fill_bf16_dev(void* out, uint64_t first, uint64_t n, uint64_t seed,
                                   uint32_t tensor_id, double c, void* stream) {
    if (n == 0) return 0;
    const uint64_t s2 = host_mix64(seed + 0x9E3779B97F4A7C15ull);
    const uint64_t base = ((uint64_t)tensor_id) << 40;
    uint64_t blocks = (n + 255) / 256;
    if (blocks > 152ull * 64) blocks = 152ull * 64;
    fill_bf16_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(
        (uint16_t*)out, first, n, s2, base, c);
    return (int)cudaGetLastError();
}

extern "C" int synth_fill_const_bf16_dev(void* out, uint64_t n, uint16_t bits, void* stream) {
    if (n == 0) return 0;
    uint64_t blocks = (n + 255) / 256;
    if (blocks > 152ull * 64) blocks = 152ull * 64;
    fill_const_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>((uint16_t*)out, n, bits);
    return (int)cudaGetLastError();
}
