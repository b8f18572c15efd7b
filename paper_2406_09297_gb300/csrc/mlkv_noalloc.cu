// mlkv_decode_attention_static: decode attention for callers that cannot allocate device memory.
//
// The regular path keeps its merge scratch (partial outputs, their log-sum-exps, per-segment
// counters, an error word) in memory that mlkv_cache_create allocates.  Some callers may not
// allocate at all: a runtime whose own allocator owns every byte of device memory, or a serving
// loop that must not call cudaMalloc once it runs (cudaMalloc can synchronise the device and stall
// every stream).  This entry point takes the cache slot, Q and out from the caller and keeps its
// scratch in one fixed array compiled into the library, so it allocates nothing.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#include "mlkv.h"
#include "mlkv_internal.h"

namespace {

// The scratch every call of this entry point shares.  Its address on a device is only known to
// device code directly; host code obtains it with cudaGetSymbolAddress (below).
static __device__ __align__(256) unsigned char g_static_scratch[MLKV_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

struct DeviceSetup {
    std::once_flag once;
    int status = MLKV_OK;
    std::string error;
    void *scratch = nullptr;   // device address of g_static_scratch on this device
    int sm_count = 0;
    size_t max_smem = 0;
};

DeviceSetup g_setup[kMaxDevices];

int fail(int code, const char *msg)
{
    mlkv::set_last_error(msg);
    return code;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return static_cast<EncodeTiledFn>(nullptr);
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// Runs once per device, with that device current: looks up the scratch address and the device
// limits, and raises the kernels' shared-memory limits.
void setup_device(int dev, DeviceSetup &st)
{
    cudaError_t e = cudaGetSymbolAddress(&st.scratch, g_static_scratch);
    if (e != cudaSuccess) {
        st.status = MLKV_ERR_CUDA;
        st.error = std::string("cudaGetSymbolAddress(static scratch): ") + cudaGetErrorString(e);
        return;
    }
    int smem_optin = 0;
    if ((e = cudaDeviceGetAttribute(&st.sm_count, cudaDevAttrMultiProcessorCount, dev)) !=
            cudaSuccess ||
        (e = cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) !=
            cudaSuccess) {
        st.status = MLKV_ERR_CUDA;
        st.error = std::string("cudaDeviceGetAttribute: ") + cudaGetErrorString(e);
        return;
    }
    st.max_smem = static_cast<size_t>(smem_optin);
    // The error word (and the counters after it) start at zero; calls then clear only the
    // counters, so an error stays recorded until mlkv_static_status reads it.
    if ((e = cudaMemset(st.scratch, 0, 256)) != cudaSuccess ||
        (e = cudaDeviceSynchronize()) != cudaSuccess) {
        st.status = MLKV_ERR_CUDA;
        st.error = std::string("clearing the static scratch: ") + cudaGetErrorString(e);
        return;
    }
    for (int d : {64, 128})
        for (int T : {64, 128, 256}) {
            const mlkv::DecodeVariant *v = mlkv::find_decode_variant(d, T);
            if (v != nullptr && (e = mlkv::prepare_decode_variant(*v, st.max_smem)) != cudaSuccess) {
                st.status = MLKV_ERR_CUDA;
                st.error = std::string("cudaFuncSetAttribute: ") + cudaGetErrorString(e);
                return;
            }
        }
}

}  // namespace

extern "C" int mlkv_decode_attention_static(const void *kv_slot, int batch, int n_q_heads,
                                            int kv_heads, int head_dim, int max_seq,
                                            const void *Q, void *out, const int *seq_lens,
                                            void *cuda_stream)
{
    if (kv_slot == nullptr || Q == nullptr || out == nullptr || seq_lens == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "kv_slot, Q, out and seq_lens must be non-NULL");
    if ((reinterpret_cast<uintptr_t>(kv_slot) | reinterpret_cast<uintptr_t>(Q) |
         reinterpret_cast<uintptr_t>(out)) & 15u)
        return fail(MLKV_ERR_INVALID_ARG, "kv_slot, Q and out must be 16-byte aligned");
    if (batch < 1 || n_q_heads < 1 || kv_heads < 1 || max_seq < 1)
        return fail(MLKV_ERR_INVALID_ARG, "sizes must be positive");
    {
        // The kernel reads Q after other CTAs may have written out: they must not overlap.
        const size_t qbytes = static_cast<size_t>(batch) * n_q_heads * head_dim * 2;
        const char *qs = static_cast<const char *>(Q);
        const char *os = static_cast<const char *>(out);
        if (qs < os + qbytes && os < qs + qbytes)
            return fail(MLKV_ERR_INVALID_ARG, "out overlaps Q");
    }
    if (batch > MLKV_MAX_BATCH)
        return fail(MLKV_ERR_UNSUPPORTED, "batch exceeds MLKV_MAX_BATCH");
    if (kv_heads > n_q_heads || n_q_heads % kv_heads != 0)
        return fail(MLKV_ERR_MAP, "kv_heads must divide n_q_heads");
    const int G = n_q_heads / kv_heads;
    if (G > MLKV_MAX_GROUP)
        return fail(MLKV_ERR_UNSUPPORTED, "query group exceeds MLKV_MAX_GROUP");
    if (head_dim != 64 && head_dim != 128)
        return fail(MLKV_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    long long len_sum = 0;
    bool uniform = true;
    for (int beta = 0; beta < batch; ++beta) {
        if (seq_lens[beta] < 1 || seq_lens[beta] > max_seq)
            return fail(MLKV_ERR_RANGE, "a sequence length is outside [1, max_seq]");
        len_sum += seq_lens[beta];
        uniform = uniform && seq_lens[beta] == seq_lens[0];
    }

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return fail(MLKV_ERR_CUDA, "no usable current device");
    DeviceSetup &st = g_setup[dev];
    std::call_once(st.once, setup_device, dev, std::ref(st));
    if (st.status != MLKV_OK)
        return fail(st.status, st.error.c_str());

    // Tile length by the regular path's default rule (mlkv::default_tile_tokens, over the
    // batch * kv_heads segments); 64 when the per-sequence tables do not fit beside the ring.
    const double mean_len = static_cast<double>(len_sum) / batch;
    int T = mlkv::default_tile_tokens(head_dim, mean_len, batch * kv_heads);
    const mlkv::DecodeVariant *v = mlkv::find_decode_variant(head_dim, T);
    if (v == nullptr)
        return fail(MLKV_ERR_UNSUPPORTED, "no decode variant");
    if (!uniform && v->smem_bytes + mlkv::table_bytes(batch) > st.max_smem) {
        T = 64;
        v = mlkv::find_decode_variant(head_dim, T);
        if (v == nullptr || v->smem_bytes + mlkv::table_bytes(batch) > st.max_smem)
            return fail(MLKV_ERR_UNSUPPORTED, "batch too large for varied lengths");
    }

    static thread_local mlkv::DecodeParams p;
    long long tiles = 0;
    for (int beta = 0; beta < batch; ++beta) {
        p.tile_start[beta] = static_cast<int>(tiles);
        p.seq_len[beta] = seq_lens[beta];
        tiles += static_cast<long long>(kv_heads) * ((seq_lens[beta] + T - 1) / T);
    }
    if (tiles > 0x7fffffffLL)
        return fail(MLKV_ERR_UNSUPPORTED, "too many tiles");
    p.tile_start[batch] = static_cast<int>(tiles);

    // Carve the scratch: error word, counters[S], lse[pieces][G], o[pieces][G][D], pieces = S + P.
    const long long S = static_cast<long long>(batch) * kv_heads;
    const size_t head_bytes = 256 + ((static_cast<size_t>(S) * 4 + 255) & ~size_t(255));
    const size_t per_piece = static_cast<size_t>(G) * (head_dim + 1) * 4;
    if (head_bytes + static_cast<size_t>(S + 1) * per_piece + 256 > MLKV_STATIC_SCRATCH_BYTES)
        return fail(MLKV_ERR_UNSUPPORTED,
                    "request exceeds MLKV_STATIC_SCRATCH_BYTES (batch * kv_heads too large)");
    const long long fit = static_cast<long long>(
        (MLKV_STATIC_SCRATCH_BYTES - head_bytes - 256) / per_piece) - S;
    int ctas_per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&ctas_per_sm, v->fn, v->threads,
                                                      v->smem_bytes);
    if (e != cudaSuccess || ctas_per_sm < 1)
        return fail(MLKV_ERR_CUDA, "decode kernel cannot be resident");
    long long wave = std::min<long long>(static_cast<long long>(ctas_per_sm) * st.sm_count, tiles);
    wave = std::min(wave, fit);
    const long long per = (tiles + wave - 1) / wave;
    const int grid = std::min(static_cast<int>((tiles + per - 1) / per),
                              mlkv::kCombineMaxPiecesHost);

    char *base = static_cast<char *>(st.scratch);
    int *err = reinterpret_cast<int *>(base);
    unsigned *counters = reinterpret_cast<unsigned *>(base + 256);
    float *part_lse = reinterpret_cast<float *>(base + head_bytes);
    const size_t lse_bytes =
        (static_cast<size_t>(S + grid) * G * 4 + 255) & ~size_t(255);
    float *part_o = reinterpret_cast<float *>(base + head_bytes + lse_bytes);

    // The array keeps whatever the previous call left: the counters must start at zero.  The
    // error word is left alone (mlkv_static_status reads and clears it).
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    e = cudaMemsetAsync(base + 256, 0, head_bytes - 256, stream);
    if (e != cudaSuccess)
        return fail(MLKV_ERR_CUDA, "clearing the static scratch failed");

    EncodeTiledFn encode = encode_fn();
    if (encode == nullptr)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    CUtensorMap tmap, tmap_rows;
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(head_dim),
                                static_cast<cuuint64_t>(max_seq),
                                static_cast<cuuint64_t>(2 * S)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(head_dim) * 2,
                                   static_cast<cuuint64_t>(max_seq) * head_dim * 2};
    const cuuint32_t estr[3] = {1u, 1u, 1u};
    for (int k = 0; k < 2; ++k) {
        const cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(k == 0 ? T : 64), 1u};
        if (encode(k == 0 ? &tmap : &tmap_rows, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                   const_cast<void *>(kv_slot), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
            CUDA_SUCCESS)
            return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled failed");
    }

    p.Q = static_cast<const __nv_bfloat16 *>(Q);
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.K_new = nullptr;
    p.V_new = nullptr;
    p.cache = nullptr;
    p.max_seq = max_seq;
    p.part_o = part_o;
    p.part_lse = part_lse;
    p.counters = counters;
    p.err = err;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(head_dim)));
    p.b = batch;
    p.h = n_q_heads;
    p.g = kv_heads;
    p.G = G;
    p.slot = 0;
    p.num_tiles = static_cast<int>(tiles);
    p.uniform_len = uniform ? seq_lens[0] : 0;
    p.cluster_k = 0;
    p.tile_tokens = T;
    p.decode_grid = grid;
    p.early_fetch = 0;
    p.newest_ready = 0;
    p.store_new = 0;
    p.pf_own = 0;
    p.ml_layers = 0;
    p.ml_chunks = 1;
    p.ml_seg_major = 0;
    p.ml_snake = 0;
    p.ml_slots = 0;
    p.ml_q_stride = 0;
    p.ml_kv_stride = 0;
    p.Q_next = nullptr;
    p.deferred_merge =
        mlkv::max_pieces_per_segment(p, T, grid) > mlkv::kInlineMergeMaxPieces ? 1 : 0;
    const size_t smem = v->smem_bytes + (uniform ? 0 : mlkv::table_bytes(batch));
    e = mlkv::launch_decode(*v, grid, smem, stream, &tmap, &tmap_rows, p, nullptr);
    if (e != cudaSuccess)
        return fail(MLKV_ERR_CUDA, "decode launch failed");
    if (p.deferred_merge && mlkv::launch_combine(p, head_dim, stream) != cudaSuccess)
        return fail(MLKV_ERR_CUDA, "combine launch failed");
    return MLKV_OK;
}

extern "C" int mlkv_static_status(void *cuda_stream)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return fail(MLKV_ERR_CUDA, "no usable current device");
    DeviceSetup &st = g_setup[dev];
    std::call_once(st.once, setup_device, dev, std::ref(st));
    if (st.status != MLKV_OK)
        return fail(st.status, st.error.c_str());
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    int word = 0;
    if ((e = cudaMemcpyAsync(&word, st.scratch, sizeof(word), cudaMemcpyDeviceToHost, stream)) !=
            cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess)
        return fail(MLKV_ERR_CUDA, (std::string("reading the static error word: ") +
                                    cudaGetErrorString(e)).c_str());
    if (word == 0)
        return MLKV_OK;
    if ((e = cudaMemsetAsync(st.scratch, 0, sizeof(word), stream)) != cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess)
        return fail(MLKV_ERR_CUDA, (std::string("clearing the static error word: ") +
                                    cudaGetErrorString(e)).c_str());
    char msg[96];
    std::snprintf(msg, sizeof(msg), "a static decode launch reported device error bits 0x%x", word);
    return fail(MLKV_ERR_DEVICE, msg);
}
