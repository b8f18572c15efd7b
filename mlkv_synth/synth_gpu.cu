// Device implementation of the seeded input generator of mlkv_synth/gen.py, for filling caches
// of many GiB in place.  It holds no attention arithmetic.  Definition (see gen.py):
//
//   out(s, n) = mix64(s + (n + 1) * GAMMA)                        SplitMix64, n-th output
//   s_row = out(out(seed, tensor_id), row)
//   element (row, col): x_k = out(s_row, 3*col + k), k = 0..2; the twelve 16-bit fields summed,
//   z = (sum - 6*65536) / 65536 in fp32 (exact), value = bf16_rne(sigma * z).
//
// C ABI:
//   int synth_fill_bf16(void* dst, long long rows, long long cols, long long pitch,
//                       long long row0, long long col0, unsigned long long seed,
//                       unsigned long long tensor_id, float sigma, void* stream)
//   writes dst[r*pitch + c] = value(row0 + r, col0 + c) for r < rows, c < cols (bf16 elements).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__host__ __device__ __forceinline__ uint64_t sm_out(uint64_t s, uint64_t n)
{
    return mix64(s + (n + 1) * kGamma);
}

__device__ __forceinline__ uint32_t sum16(uint64_t x)
{
    return static_cast<uint32_t>((x & 0xffff) + ((x >> 16) & 0xffff) + ((x >> 32) & 0xffff) +
                                 (x >> 48));
}

__global__ void fill_kernel(__nv_bfloat16 *dst, long long rows, long long cols, long long pitch,
                            long long row0, long long col0, uint64_t s_tensor, float sigma)
{
    for (long long r = blockIdx.y; r < rows; r += gridDim.y) {
        const uint64_t s_row = sm_out(s_tensor, static_cast<uint64_t>(row0 + r));
        for (long long c = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; c < cols;
             c += static_cast<long long>(gridDim.x) * blockDim.x) {
            const uint64_t n = 3ull * static_cast<uint64_t>(col0 + c);
            const uint32_t total = sum16(sm_out(s_row, n)) + sum16(sm_out(s_row, n + 1)) +
                                   sum16(sm_out(s_row, n + 2));
            const float z = static_cast<float>(static_cast<int>(total) - 6 * 65536) *
                            (1.0f / 65536.0f);
            dst[r * pitch + c] = __float2bfloat16_rn(sigma * z);
        }
    }
}

}  // namespace

extern "C" int synth_fill_bf16(void *dst, long long rows, long long cols, long long pitch,
                               long long row0, long long col0, unsigned long long seed,
                               unsigned long long tensor_id, float sigma, void *stream)
{
    if (dst == nullptr || rows < 0 || cols < 0 || pitch < cols)
        return -1;
    if (rows == 0 || cols == 0)
        return 0;
    const uint64_t s_tensor = sm_out(seed, tensor_id);
    const int threads = 256;
    long long bx = (cols + threads - 1) / threads;
    if (bx > 4096)
        bx = 4096;
    long long by = rows < 65535 ? rows : 65535;
    fill_kernel<<<dim3(static_cast<unsigned>(bx), static_cast<unsigned>(by)), threads, 0,
                  static_cast<cudaStream_t>(stream)>>>(static_cast<__nv_bfloat16 *>(dst), rows,
                                                       cols, pitch, row0, col0, s_tensor, sigma);
    return cudaGetLastError() == cudaSuccess ? 0 : -2;
}
