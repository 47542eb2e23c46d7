// Exhaustive check of the epilogue's one-instruction bf16 rounding: for every
// fp32 bit pattern a, in the low and in the high half of the word (partners:
// a with its sign flipped, and a + 0x00400001), pack_bf16x2_cvt must give the
// bits of two f32_to_bf16_bits_rn calls unless one of the inputs is a NaN
// (where the instruction returns the canonical NaN and the library never
// uses it).  Prints the number of mismatching words; exit status 0 when none.
#include <cstdio>
#include <cstdint>

#include "../../paper_2606_12280_gb300/csrc/common.cuh"

using namespace w8a8;

__device__ __forceinline__ bool is_nan_bits(uint32_t u) { return (u & 0x7fffffffu) > 0x7f800000u; }

__global__ void check(unsigned long long *bad, unsigned int *first) {
    const uint64_t n = 1ull << 32;
    for (uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x) {
        const uint32_t a = static_cast<uint32_t>(i);
        const uint32_t partner[2] = {a ^ 0x80000000u, a + 0x00400001u};
        for (int k = 0; k < 2; ++k) {
            const uint32_t b = partner[k];
            if (is_nan_bits(a) || is_nan_bits(b)) continue;
            const float fa = __uint_as_float(a), fb = __uint_as_float(b);
            const uint32_t lo = pack_bf16x2_cvt(fa, fb);
            const uint32_t hi = pack_bf16x2_cvt(fb, fa);
            const uint32_t want_lo = f32_to_bf16_bits_rn(fa) | (f32_to_bf16_bits_rn(fb) << 16);
            const uint32_t want_hi = f32_to_bf16_bits_rn(fb) | (f32_to_bf16_bits_rn(fa) << 16);
            if (lo != want_lo || hi != want_hi) {
                if (atomicAdd(bad, 1ull) == 0ull) *first = a;
            }
        }
    }
}

int main() {
    unsigned long long *bad = nullptr;
    unsigned int *first = nullptr;
    if (cudaMalloc(&bad, sizeof(*bad)) != cudaSuccess || cudaMalloc(&first, sizeof(*first)) != cudaSuccess) {
        printf("allocation failed\n");
        return 2;
    }
    cudaMemset(bad, 0, sizeof(*bad));
    cudaMemset(first, 0, sizeof(*first));
    check<<<1216, 256>>>(bad, first);
    const cudaError_t e = cudaDeviceSynchronize();
    unsigned long long h = 0;
    unsigned int f = 0;
    cudaMemcpy(&h, bad, sizeof(h), cudaMemcpyDeviceToHost);
    cudaMemcpy(&f, first, sizeof(f), cudaMemcpyDeviceToHost);
    printf("status %s mismatches %llu first 0x%08x\n", cudaGetErrorString(e), h, f);
    cudaFree(bad);
    cudaFree(first);
    return (e == cudaSuccess && h == 0ull) ? 0 : 1;
}
