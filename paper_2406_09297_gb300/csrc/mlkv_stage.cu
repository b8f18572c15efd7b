// Copies between page-locked host memory (through its device-mapped address) and device memory,
// as kernels: for the small tensors of one decode step (a few MB), a copy-engine transfer costs
// ~12 us of fixed latency each, while a kernel of plain 16-byte loads and stores over the
// CPU-GPU link costs a launch.  Used by mlkv_decode_step_host to bring a step's Q and new K/V in
// (one launch for all three); the decode kernels store the outputs into host memory themselves.
// Also the store of every owner's new token into its slot for the fused step (one launch for all
// owners, Sec. 3: only owner layers store K/V).
#include <cuda_bf16.h>
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

// The new token of owner slots slot .. slot + n_slots - 1 (K[s], V[s] [b][g][D]) at position
// L_beta - 1 of each (sequence, KV head): one thread per 16-byte vector.
__global__ void __launch_bounds__(256) append_slots_kernel(const __grid_constant__ AppendParams p)
{
    // Earlier kernels of the stream may still read the cache: nothing is stored before they end.
    // The dependent (the fused decode) is let go after that wait, or at once when it is told to
    // read only what no kernel in flight writes (trigger_first).
    if (p.trigger_first)
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (!p.trigger_first)
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int vecs = p.d / 8;
    const long long total = 2LL * p.n_slots * p.b * p.g * vecs;
    const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= total)
        return;
    const int v = static_cast<int>(idx % vecs);
    long long row = idx / vecs;   // (slot, K or V, sequence, KV head)
    const int j = static_cast<int>(row % p.g);
    row /= p.g;
    const int beta = static_cast<int>(row % p.b);
    row /= p.b;
    const int kv = static_cast<int>(row & 1);
    const int s = static_cast<int>(row >> 1);
    const int pos = p.seq_len[beta] - 1;
    const uint4 *src = reinterpret_cast<const uint4 *>(kv ? p.V : p.K) +
                       ((static_cast<size_t>(s) * p.b + beta) * p.g + j) * vecs + v;
    uint4 *dst = reinterpret_cast<uint4 *>(p.cache) +
                 ((((static_cast<size_t>(p.slot + s) * 2 + kv) * p.b + beta) * p.g + j) *
                      static_cast<size_t>(p.max_seq) + pos) * vecs + v;
    *dst = *src;
}

}  // namespace

cudaError_t launch_append_slots(const AppendParams &p, cudaStream_t stream)
{
    const long long total = 2LL * p.n_slots * p.b * p.g * (p.d / 8);
    const int threads = 256;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>((total + threads - 1) / threads));
    cfg.blockDim = dim3(threads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void *args[] = {const_cast<AppendParams *>(&p)};
    return cudaLaunchKernelExC(&cfg, reinterpret_cast<const void *>(&append_slots_kernel), args);
}

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
