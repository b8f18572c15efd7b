// Copies between page-locked host memory (through its device-mapped address) and device memory,
// as kernels: for the small tensors of one decode step (a few MB), a copy-engine transfer costs
// ~12 us of fixed latency each, while a kernel of plain 16-byte loads and stores over the
// CPU-GPU link costs a launch.  Used by mlkv_decode_step_host to bring a step's Q and new K/V in
// (one launch for all three); the decode kernels store the outputs into host memory themselves.
#include <cuda_runtime.h>
#include <stdint.h>

#include "mlkv_internal.h"

namespace mlkv {
namespace {

__global__ void __launch_bounds__(256) stage_copy_kernel(const __grid_constant__ StageParams p)
{
    // The next launch (the step's decode) may start at once: it reads nothing this kernel writes
    // before its own dependency wait, which returns only once this grid has finished.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
    for (int s = 0; s < p.n; ++s) {
        const uint4 *src = static_cast<const uint4 *>(p.src[s]);
        uint4 *dst = static_cast<uint4 *>(p.dst[s]);
        const size_t n16 = p.bytes[s] >> 4;
        for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n16;
             i += stride)
            dst[i] = src[i];
    }
}

}  // namespace

cudaError_t launch_stage_copy(const StageParams &p, cudaStream_t stream)
{
    size_t total = 0;
    for (int s = 0; s < p.n; ++s)
        total += p.bytes[s] >> 4;
    // One 16-byte transfer per thread, so that every load over the link is in flight at once
    // (a host-memory round trip is ~1-2 us); beyond 16 CTAs per SM, threads loop.
    size_t blocks = (total + 255) / 256;
    if (blocks < 1)
        blocks = 1;
    if (blocks > 152 * 16)
        blocks = 152 * 16;
    stage_copy_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace mlkv
