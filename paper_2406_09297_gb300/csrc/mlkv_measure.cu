// Read-bandwidth probe (benchmark support, not part of the decode path): the roofline of a decode
// layer whose owner slot an earlier layer of its block has just brought into L2 is the rate at
// which CTAs can pull L2-resident data into shared memory.  This kernel measures that rate the way
// the decode kernel moves data -- bulk asynchronous copies into a shared-memory ring completed on
// mbarriers -- without any arithmetic: every CTA streams its share of a caller's buffer `reps`
// times through a two-stage ring of 32 KiB copies.
#include <cuda_runtime.h>
#include <stdint.h>

#include "mlkv.h"
#include "mlkv_internal.h"

#include "mlkv_device.cuh"

namespace mlkv {
namespace {

constexpr int kProbeChunk = 32 * 1024;
constexpr int kProbeStages = 2;

// One thread per CTA issues and waits; the others exit at once.  Every wait is bounded: on expiry
// the CTA stops issuing, waits (again bounded) for the copies it has in flight and exits.
__global__ void __launch_bounds__(32) read_probe_kernel(const uint8_t *buf, size_t per_cta, int reps)
{
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ __align__(8) uint64_t bars[kProbeStages];
    if (threadIdx.x != 0)
        return;
    const uint32_t bar0 = smem_addr(&bars[0]);
    for (int s = 0; s < kProbeStages; ++s)
        mbar_init(bar0 + 8 * s, 1);
    fence_barrier_init();
    const uint8_t *base = buf + static_cast<size_t>(blockIdx.x) * per_cta;
    const long long chunks = static_cast<long long>(per_cta / kProbeChunk);
    const long long n = chunks * reps;
    long long issued = 0;
    bool ok = true;
    for (long long k = 0; k < n && ok; ++k) {
        const int s = static_cast<int>(k % kProbeStages);
        if (k >= kProbeStages)
            ok = mbar_wait(bar0 + 8 * s, static_cast<uint32_t>(((k - kProbeStages) / kProbeStages) & 1));
        if (!ok)
            break;
        mbar_arrive_expect_tx(bar0 + 8 * s, kProbeChunk);
        bulk_load(smem_addr(ring + static_cast<size_t>(s) * kProbeChunk),
                  base + static_cast<size_t>(k % chunks) * kProbeChunk, kProbeChunk, bar0 + 8 * s);
        ++issued;
    }
    // no copy may be in flight when the CTA exits
    for (long long k = issued > kProbeStages ? issued - kProbeStages : 0; k < issued; ++k)
        mbar_wait(bar0 + 8 * (k % kProbeStages),
                  static_cast<uint32_t>((k / kProbeStages) & 1));
}

}  // namespace
}  // namespace mlkv

extern "C" int mlkv_read_bandwidth_probe(const void *buf, int64_t bytes, int reps,
                                         int64_t *bytes_read, void *cuda_stream)
{
    if (buf == nullptr || bytes_read == nullptr || (reinterpret_cast<uintptr_t>(buf) & 15u) ||
        bytes <= 0 || reps < 1) {
        mlkv::set_last_error("buf and bytes_read must be non-NULL, buf 16-byte aligned, bytes and "
                             "reps positive");
        return MLKV_ERR_INVALID_ARG;
    }
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(mlkv::read_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 mlkv::kProbeStages * mlkv::kProbeChunk);
    if (e != cudaSuccess) {
        mlkv::set_last_error(cudaGetErrorString(e));
        return MLKV_ERR_CUDA;
    }
    const int grid = 2 * sms;   // two CTAs per SM: two issuing threads per SM
    const size_t per_cta = static_cast<size_t>(bytes) / grid / mlkv::kProbeChunk * mlkv::kProbeChunk;
    if (per_cta == 0) {
        mlkv::set_last_error("bytes must hold at least one 32 KiB chunk per CTA (2 per SM)");
        return MLKV_ERR_INVALID_ARG;
    }
    mlkv::read_probe_kernel<<<grid, 32, mlkv::kProbeStages * mlkv::kProbeChunk,
                              static_cast<cudaStream_t>(cuda_stream)>>>(
        static_cast<const uint8_t *>(buf), per_cta, reps);
    e = cudaGetLastError();
    if (e != cudaSuccess) {
        mlkv::set_last_error(cudaGetErrorString(e));
        return MLKV_ERR_CUDA;
    }
    *bytes_read = static_cast<int64_t>(per_cta) * grid * reps;
    return MLKV_OK;
}
