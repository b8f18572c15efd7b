// Host side of libmlkv: argument validation, the MLKV cache manager and the C ABI of mlkv.h.
//
// The cache of an MLKV model (arXiv 2406.09297, Sec. 3) holds K and V only for the m owner
// layers.  It is one device allocation laid out [m][2][b][g][max_seq][d] (bf16), so that the
// keys (or values) of one (slot, sequence, KV head) are max_seq*d contiguous elements: a decode
// tile of T positions is one contiguous T*d*2-byte block, fetched by a 3-D TMA tensor map over
// (d, max_seq, m*2*b*g).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "mlkv.h"
#include "mlkv_internal.h"

namespace {

thread_local std::string g_last_error;

int fail(int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return code;
}

int fail_cuda(cudaError_t e, const char *what)
{
    return fail(MLKV_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetDeviceFn = CUresult (*)(CUdevice *);

template <typename Fn>
Fn driver_entry(const char *name)
{
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return nullptr;
    return reinterpret_cast<Fn>(fn);
}

// The device of the CUDA context current on this thread (e.g. the one PyTorch made current);
// falls back to this runtime's current device.
int current_device()
{
    static CtxGetCurrentFn get_ctx = driver_entry<CtxGetCurrentFn>("cuCtxGetCurrent");
    static CtxGetDeviceFn get_dev = driver_entry<CtxGetDeviceFn>("cuCtxGetDevice");
    CUcontext ctx = nullptr;
    if (get_ctx != nullptr && get_dev != nullptr && get_ctx(&ctx) == CUDA_SUCCESS && ctx) {
        CUdevice dev;
        if (get_dev(&dev) == CUDA_SUCCESS)
            return static_cast<int>(dev);
    }
    int d = 0;
    cudaGetDevice(&d);
    return d;
}

struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev)
    {
        if (cudaGetDevice(&prev) != cudaSuccess)
            prev = -1;
        if (prev != dev)
            ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard()
    {
        int now = -1;
        if (prev >= 0 && cudaGetDevice(&now) == cudaSuccess && now != prev)
            cudaSetDevice(prev);
    }
};

}  // namespace

struct mlkv_cache {
    int l = 0, h = 0, d = 0, g = 0, G = 0, b = 0, max_seq = 0, m = 0;
    std::vector<int> owner, slot;
    int device = 0;
    int sm_count = 0;
    int l2_bytes = 0;
    int window_max = 0;
    size_t max_smem = 0;        // opt-in dynamic shared memory per block
    void *cache = nullptr;      // [m][2][b][g][max_seq][d] bf16
    size_t cache_bytes = 0;
    float *part_o = nullptr;    // [pieces][G][d]
    float *part_lse = nullptr;  // [pieces][G]
    unsigned *counters = nullptr;
    int *err = nullptr;
    int max_ctas = 0;           // capacity of the partial buffers beyond b*g pieces
    long long records = 0;      // partial records the scratch holds
    // options
    int tile_tokens = 0;
    int grid = 0;
    int l2_persist = 0;
    size_t persist_bytes = 0;   // the context's persisting-L2 set-aside while l2_persist is on
    size_t persist_prev = 0;    // the set-aside before l2_persist was switched on
    int l2_prefetch = 0;        // multi-layer step: prefetch the step's slots into L2 when they fit
    int step_kernel = 1;        // mlkv_decode_step: one multi-layer launch where it applies
    int last_step_kernel = 0;   // 1 if the most recent step ran as one multi-layer launch
    int last_seg_major = 0;     // 1 if that launch ranked its items segment-major
    int cluster = 1;            // allow the DSMEM cluster merge
    int pdl = 1;                // programmatic dependent launch
    int early_fetch = 1;        // per-layer step: later layers read Q and tiles before the wait
    int tc = 0;                 // 1: the tcgen05 kernel where a variant exists (slower here)
    int prefill_ready = 0;      // the prefill kernel's shared-memory limit is set
    int fused_ready = 0;        // the same for the fused-decode forms (bit 1 << form)
    int fused_deep = 1;         // fused decode: the deep one-tile form where one unit per SM
    float *fused_part = nullptr;   // context-chunk partials of the fused decode
    size_t fused_part_floats = 0;
    int step_fused = 1;         // mlkv_decode_step: the cross-layer fused form where it pays (1),
                                // wherever the map allows it (2), never (0)
    int last_step_fused = 0;    // 1 if the most recent step ran in that form
    int last_step_launches = 0;   // this library's launches in the most recent step
    int last_fused_kc = 0;      // key tiles per unit (chunk) of the most recent fused decode
    int fused_kc = 0;           // > 0: key tiles per unit of the fused decode, else planned
    // mlkv_decode_step's recorded graph and the arguments it was recorded for
    int step_graph = 2;         // 2: direct when one multi-layer launch, else record/replay
    cudaStream_t record_stream = nullptr;   // private stream the step graph is recorded on
    cudaGraphExec_t step_exec = nullptr;
    struct StepKey {
        const void *Q = nullptr, *K = nullptr, *V = nullptr;
        void *out = nullptr;
        std::vector<int> lens;
        int tile = -1, grid = -1, cluster = -1, pdl = -1, l2 = -1, tc = -1, pf = -1, sk = -1;
        int sg = -1;   // step_graph: a graph recorded under one mode is not replayed under another
        int ef = -1, sf = -1;
        bool operator==(const StepKey &o) const
        {
            return Q == o.Q && K == o.K && V == o.V && out == o.out && lens == o.lens &&
                   tile == o.tile && grid == o.grid && cluster == o.cluster && pdl == o.pdl &&
                   l2 == o.l2 && tc == o.tc && pf == o.pf && sk == o.sk && sg == o.sg &&
                   ef == o.ef && sf == o.sf;
        }
    } step_key, pending_key;   // recorded arguments; arguments seen once, not yet recorded
    int step_graph_replays = 0;
    // mlkv_decode_step_host: device staging of the step's inputs and outputs, its own graph
    void *stage = nullptr;     // Q [l][b][h][d], K, V [m][b][g][d], out [l][b][h][d]
    cudaGraphExec_t host_exec = nullptr;
    cudaStream_t side = nullptr;   // the copies that overlap the step's layers
    cudaEvent_t ev[2] = {nullptr, nullptr};   // fork, the later layers' queries in
    StepKey host_key, host_pending;
    // the most recent decode launch (read-only options, for tests and tuning)
    int last_grid = 0, last_tile = 0, last_cluster_k = 0, last_deferred = 0, last_tc = 0;
    int last_l2_prefetch = 0;
    // per-variant launch state
    struct Variant {
        const mlkv::DecodeVariant *v = nullptr;
        CUtensorMap tmap;        // boxes of tile_tokens positions
        CUtensorMap tmap_rows;   // boxes of 64 positions (a partly visible last tile)
        int ctas_per_sm = 0;
        int clusters[5] = {0, 0, 0, 0, 0};   // resident k-CTA clusters, k = 2, 4
    };
    std::vector<Variant> variants;
    std::vector<int> tile_start_scratch;
};

namespace {

int check_seq_lens(const mlkv_cache *c, const int *seq_lens)
{
    if (seq_lens == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "seq_lens is NULL");
    for (int beta = 0; beta < c->b; ++beta) {
        if (seq_lens[beta] < 1 || seq_lens[beta] > c->max_seq)
            return fail(MLKV_ERR_RANGE, "seq_lens[%d] = %d outside [1, %d]", beta, seq_lens[beta],
                        c->max_seq);
    }
    return MLKV_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

mlkv_cache::Variant *pick_variant(mlkv_cache *c, double mean_len = -1.0, int force_T = 0)
{
    const int T = force_T > 0            ? force_T
                  : c->tile_tokens > 0 ? c->tile_tokens
                                       : mlkv::default_tile_tokens(c->d, mean_len, c->b * c->g);
    mlkv_cache::Variant *plain = nullptr;
    for (auto &v : c->variants) {
        if (v.v->tile_tokens != T)
            continue;
        if (v.v->tc == c->tc)
            return &v;
        if (!v.v->tc)
            plain = &v;
    }
    return plain;   // no tcgen05 variant for this tile: the mma.sync kernel
}

int encode_tmap(mlkv_cache *c, int rows, CUtensorMap *out)
{
    static EncodeTiledFn encode = driver_entry<EncodeTiledFn>("cuTensorMapEncodeTiled");
    if (encode == nullptr)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(c->d), static_cast<cuuint64_t>(c->max_seq),
                                static_cast<cuuint64_t>(c->m) * 2 * c->b * c->g};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(c->d) * 2,
                                   static_cast<cuuint64_t>(c->max_seq) * c->d * 2};
    const cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(rows), 1u};
    const cuuint32_t estr[3] = {1u, 1u, 1u};
    CUresult r = encode(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, c->cache, dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", static_cast<int>(r));
    return MLKV_OK;
}

void free_all(mlkv_cache *c)
{
    if (c->cache) cudaFree(c->cache);
    if (c->part_o) cudaFree(c->part_o);
    if (c->part_lse) cudaFree(c->part_lse);
    if (c->counters) cudaFree(c->counters);
    if (c->err) cudaFree(c->err);
    c->cache = nullptr;
    c->part_o = nullptr;
    c->part_lse = nullptr;
    c->counters = nullptr;
    c->err = nullptr;
}

// The owner map's shape in c: sizes, owners, and each layer's slot (the rank of its owner among
// the distinct owners, Eq. 18's k); c->m the number of slots.
void assign_map(mlkv_cache *c, int l, int h, int d, const int *owner, int g, int b, int max_seq)
{
    c->l = l;
    c->h = h;
    c->d = d;
    c->g = g;
    c->G = h / g;
    c->b = b;
    c->max_seq = max_seq;
    c->owner.assign(owner, owner + l);
    c->slot.assign(l, -1);
    c->m = 0;
    for (int n = 0; n < l; ++n) {
        if (c->owner[n] == n) {
            for (int q = 0; q < l; ++q)
                if (c->owner[q] == n)
                    c->slot[q] = c->m;
            ++c->m;
        }
    }
}

int validate_map(int l, int h, int d, const int *owner, int g, int b, int max_seq)
{
    if (l < 1 || h < 1 || g < 1 || b < 1 || max_seq < 1 || d < 1)
        return fail(MLKV_ERR_INVALID_ARG,
                    "sizes must be positive (l=%d h=%d d=%d g=%d b=%d max_seq=%d)", l, h, d, g, b,
                    max_seq);
    if (owner == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "layer_owner is NULL");
    if (g > h || h % g != 0)
        return fail(MLKV_ERR_MAP, "kv_heads_per_owner %d must divide n_q_heads %d", g, h);
    for (int n = 0; n < l; ++n) {
        const int o = owner[n];
        if (o < 0 || o > n)
            return fail(MLKV_ERR_MAP, "layer_owner[%d] = %d: an owner must be a layer <= %d", n,
                        o, n);
        if (owner[o] != o)
            return fail(MLKV_ERR_MAP, "layer_owner[%d] = %d, but layer %d is not its own owner",
                        n, o, o);
    }
    if (d != 64 && d != 128)
        return fail(MLKV_ERR_UNSUPPORTED, "head_dim %d: this build supports 64 and 128", d);
    if (h / g > MLKV_MAX_GROUP)
        return fail(MLKV_ERR_UNSUPPORTED, "query group h/g = %d exceeds %d", h / g,
                    MLKV_MAX_GROUP);
    if (b > MLKV_MAX_BATCH)
        return fail(MLKV_ERR_UNSUPPORTED, "batch %d exceeds %d", b, MLKV_MAX_BATCH);
    return MLKV_OK;
}

}  // namespace

void mlkv::set_last_error(const char *msg) { g_last_error = msg; }

extern "C" {

int mlkv_version(void) { return 100; }

const char *mlkv_last_error(void) { return g_last_error.c_str(); }

int mlkv_block_owner_map(int n_layers, int n_owners, int *layer_owner)
{
    if (layer_owner == nullptr || n_layers < 1 || n_owners < 1)
        return fail(MLKV_ERR_INVALID_ARG, "bad arguments to mlkv_block_owner_map");
    if (n_owners > n_layers || n_layers % n_owners != 0)
        return fail(MLKV_ERR_MAP, "n_owners %d must divide n_layers %d", n_owners, n_layers);
    const int per = n_layers / n_owners;   // layers per KV block (Eq. 18's l/m)
    for (int n = 0; n < n_layers; ++n)
        layer_owner[n] = (n / per) * per;
    return MLKV_OK;
}

int mlkv_cache_create(mlkv_cache_t *out, int n_layers, int n_q_heads, int head_dim,
                      const int *layer_owner, int kv_heads_per_owner, int batch, int max_seq)
{
    if (out == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "out is NULL");
    int rc = validate_map(n_layers, n_q_heads, head_dim, layer_owner, kv_heads_per_owner, batch,
                          max_seq);
    if (rc != MLKV_OK)
        return rc;

    mlkv_cache *c = new mlkv_cache();
    assign_map(c, n_layers, n_q_heads, head_dim, layer_owner, kv_heads_per_owner, batch, max_seq);
    const long long rows = static_cast<long long>(c->m) * 2 * c->b * c->g;
    if (rows > 0x7fffffffLL) {
        delete c;
        return fail(MLKV_ERR_UNSUPPORTED, "m*2*b*g = %lld rows exceed the TMA coordinate range",
                    rows);
    }

    c->device = current_device();
    DeviceGuard guard(c->device);
    cudaDeviceProp prop;
    cudaError_t e = cudaGetDeviceProperties(&prop, c->device);
    if (e != cudaSuccess) {
        delete c;
        return fail_cuda(e, "cudaGetDeviceProperties");
    }
    c->sm_count = prop.multiProcessorCount;
    c->l2_bytes = prop.l2CacheSize;
    c->window_max = prop.accessPolicyMaxWindowSize;
    c->max_smem = prop.sharedMemPerBlockOptin;

    for (int vi = 0; vi < 6; ++vi) {
        const int T = 64 << (vi % 3);
        const mlkv::DecodeVariant *v = mlkv::find_decode_variant(c->d, T, vi / 3);
        if (v == nullptr)
            continue;
        e = mlkv::prepare_decode_variant(*v, c->max_smem);
        if (e != cudaSuccess) {
            delete c;
            return fail_cuda(e, "cudaFuncSetAttribute(decode)");
        }
        mlkv_cache::Variant var;
        var.v = v;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&var.ctas_per_sm, v->fn, v->threads,
                                                          v->smem_bytes);
        if (e != cudaSuccess || var.ctas_per_sm < 1) {
            delete c;
            return fail(MLKV_ERR_CUDA, "decode variant d=%d T=%d cannot be resident", head_dim, T);
        }
        c->max_ctas = std::max(c->max_ctas, var.ctas_per_sm * c->sm_count);
        for (int k : {2, 4}) {
            if (v->smem_bytes + (k - 1) * v->res_bytes > c->max_smem ||
                mlkv::max_active_clusters(*v, k, &var.clusters[k]) != cudaSuccess) {
                cudaGetLastError();
                var.clusters[k] = 0;
            }
        }
        c->variants.push_back(var);
    }
    c->max_ctas = std::max(c->max_ctas, 4 * c->sm_count);

    c->cache_bytes = static_cast<size_t>(rows) * c->max_seq * c->d * 2;
    // partial records: a stream-K layer needs b g + grid; a chunked multi-layer step l b g C,
    // C chosen to fit (about 2.5 waves of chunks)
    const size_t pieces =
        std::max(static_cast<size_t>(c->b) * c->g + c->max_ctas, 3 * static_cast<size_t>(c->max_ctas));
    c->records = static_cast<long long>(pieces);
    if ((e = cudaMalloc(&c->cache, c->cache_bytes)) != cudaSuccess ||
        (e = cudaMalloc(reinterpret_cast<void **>(&c->part_o),
                        pieces * c->G * c->d * sizeof(float))) != cudaSuccess ||
        (e = cudaMalloc(reinterpret_cast<void **>(&c->part_lse), pieces * c->G * sizeof(float))) !=
            cudaSuccess ||
        (e = cudaMalloc(reinterpret_cast<void **>(&c->counters),
                        static_cast<size_t>(c->b) * c->g * sizeof(unsigned))) != cudaSuccess ||
        (e = cudaMalloc(reinterpret_cast<void **>(&c->err), sizeof(int))) != cudaSuccess) {
        cudaGetLastError();
        free_all(c);
        const size_t need = c->cache_bytes;
        delete c;
        return fail(e == cudaErrorMemoryAllocation ? MLKV_ERR_OOM : MLKV_ERR_CUDA,
                    "cudaMalloc for a %zu-byte cache: %s", need, cudaGetErrorString(e));
    }
    if ((e = cudaMemset(c->cache, 0, c->cache_bytes)) != cudaSuccess ||
        (e = cudaMemset(c->counters, 0, static_cast<size_t>(c->b) * c->g * sizeof(unsigned))) !=
            cudaSuccess ||
        (e = cudaMemset(c->err, 0, sizeof(int))) != cudaSuccess ||
        (e = cudaDeviceSynchronize()) != cudaSuccess) {
        free_all(c);
        delete c;
        return fail_cuda(e, "initialising the cache");
    }
    for (auto &var : c->variants) {
        rc = encode_tmap(c, var.v->tile_tokens, &var.tmap);
        if (rc == MLKV_OK)
            rc = encode_tmap(c, 64, &var.tmap_rows);
        if (rc != MLKV_OK) {
            free_all(c);
            delete c;
            return rc;
        }
    }
    c->tile_start_scratch.resize(static_cast<size_t>(c->b) + 1);
    *out = c;
    return MLKV_OK;
}

int mlkv_cache_destroy(mlkv_cache_t c)
{
    if (c == nullptr)
        return MLKV_OK;
    DeviceGuard guard(c->device);
    cudaDeviceSynchronize();
    if (c->l2_persist) {
        cudaCtxResetPersistingL2Cache();
        cudaDeviceSetLimit(cudaLimitPersistingL2CacheSize, c->persist_prev);
        cudaGetLastError();
    }
    if (c->step_exec)
        cudaGraphExecDestroy(c->step_exec);
    if (c->host_exec)
        cudaGraphExecDestroy(c->host_exec);
    for (cudaEvent_t ev : c->ev)
        if (ev)
            cudaEventDestroy(ev);
    if (c->side)
        cudaStreamDestroy(c->side);
    if (c->stage)
        cudaFree(c->stage);
    if (c->fused_part)
        cudaFree(c->fused_part);
    if (c->record_stream)
        cudaStreamDestroy(c->record_stream);
    free_all(c);
    delete c;
    return MLKV_OK;
}

int mlkv_append(mlkv_cache_t c, int layer, const void *K, const void *V, const int *seq_lens,
                void *cuda_stream)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (layer < 0 || layer >= c->l)
        return fail(MLKV_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, c->l);
    if (c->owner[layer] != layer)
        return MLKV_OK;   // Sec. 3: a layer without KV heads of its own stores nothing
    if (K == nullptr || V == nullptr || !aligned16(K) || !aligned16(V))
        return fail(MLKV_ERR_INVALID_ARG, "K and V must be non-NULL and 16-byte aligned");
    int rc = check_seq_lens(c, seq_lens);
    if (rc != MLKV_OK)
        return rc;
    mlkv::AppendParams p;
    p.K = static_cast<const __nv_bfloat16 *>(K);
    p.V = static_cast<const __nv_bfloat16 *>(V);
    p.cache = static_cast<__nv_bfloat16 *>(c->cache);
    p.b = c->b;
    p.g = c->g;
    p.d = c->d;
    p.max_seq = c->max_seq;
    p.slot = c->slot[layer];
    p.n_slots = 1;
    p.trigger_first = 0;
    std::memcpy(p.seq_len, seq_lens, sizeof(int) * c->b);
    DeviceGuard guard(c->device);
    cudaError_t e = mlkv::launch_append(p, static_cast<cudaStream_t>(cuda_stream));
    if (e != cudaSuccess)
        return fail_cuda(e, "append launch");
    return MLKV_OK;
}

static int decode_impl(mlkv_cache_t c, int layer, const void *K_new, const void *V_new,
                       const void *Q, void *out, const int *seq_lens, void *cuda_stream,
                       int early_fetch = 0, const void *Q_next = nullptr,
                       int newest_ready = 0, int store_new = 1, int in_step = 0)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (layer < 0 || layer >= c->l)
        return fail(MLKV_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, c->l);
    if (Q == nullptr || out == nullptr || !aligned16(Q) || !aligned16(out))
        return fail(MLKV_ERR_INVALID_ARG, "Q and out must be non-NULL and 16-byte aligned");
    const size_t qbytes = static_cast<size_t>(c->b) * c->h * c->d * 2;
    const char *qs = static_cast<const char *>(Q);
    const char *os = static_cast<const char *>(out);
    if (qs < os + qbytes && os < qs + qbytes)
        return fail(MLKV_ERR_INVALID_ARG, "out overlaps Q");
    if (K_new != nullptr && (V_new == nullptr || !aligned16(K_new) || !aligned16(V_new)))
        return fail(MLKV_ERR_INVALID_ARG, "K and V must be non-NULL and 16-byte aligned");
    int rc = check_seq_lens(c, seq_lens);
    if (rc != MLKV_OK)
        return rc;
    double mean_len = 0.0;
    for (int beta = 0; beta < c->b; ++beta)
        mean_len += seq_lens[beta];
    mean_len /= c->b;
    // Inside a decode step, a layer that is one long segment (d = 64) runs on the 128-position
    // tile (two CTAs per SM) over 64 CTAs, so the next layers' grids stream beside it (measured,
    // batch 1, 131072 positions, 12 layers: MLKV-2 81.9 us against 96.3 us for the 256-position
    // tile on the one-wave split, MQA 95.8 against 119.7; 48 or 76 CTAs were slower than 64).
    const bool single_long = in_step && c->tile_tokens == 0 && c->grid <= 0 && c->d == 64 &&
                             c->b * c->g == 1 && seq_lens[0] >= 16384;
    mlkv_cache::Variant *var = pick_variant(c, mean_len, single_long ? 128 : 0);
    if (var == nullptr)
        return fail(MLKV_ERR_UNSUPPORTED, "no decode variant for d=%d tile_tokens=%d", c->d,
                    c->tile_tokens);
    bool uniform = true;
    for (int beta = 1; beta < c->b; ++beta)
        uniform = uniform && seq_lens[beta] == seq_lens[0];
    if (!uniform && var->v->smem_bytes + mlkv::table_bytes(c->b) > c->max_smem) {
        // The per-sequence tables do not fit beside this variant's ring: take the 64-position
        // tile variant, whose ring is small.
        var = nullptr;
        for (auto &v : c->variants)
            if (v.v->tile_tokens == 64 && v.v->smem_bytes + mlkv::table_bytes(c->b) <= c->max_smem)
                var = &v;
        if (var == nullptr)
            return fail(MLKV_ERR_UNSUPPORTED, "batch %d too large for varied lengths", c->b);
    }
    const int T = var->v->tile_tokens;

    // Stream-K style split: tiles of all (beta, j) segments end to end, equal runs per CTA.
    static thread_local mlkv::DecodeParams p;
    long long tiles = 0;
    for (int beta = 0; beta < c->b; ++beta) {
        p.tile_start[beta] = static_cast<int>(tiles);
        p.seq_len[beta] = seq_lens[beta];
        tiles += static_cast<long long>(c->g) * ((seq_lens[beta] + T - 1) / T);
    }
    p.uniform_len = uniform ? seq_lens[0] : 0;
    if (tiles > 0x7fffffffLL)
        return fail(MLKV_ERR_UNSUPPORTED, "%lld tiles exceed the int32 tile index", tiles);
    p.tile_start[c->b] = static_cast<int>(tiles);
    // The launch shape.  A one-wave stream-K grid (the fewest CTAs with the makespan of one wave
    // of resident CTAs) fits large layers, where every SM streams many tiles and the merge of the
    // few split segments is amortised.  When every sequence has one length two more shapes can
    // be better for a small layer: whole segments per CTA (no merge at all), or each segment in k
    // equal pieces run as one k-CTA cluster and merged over DSMEM.  They are chosen with a cost
    // model in units of one tile's consumer work (~0.5 us on GB300 when the tile is in L2):
    // a DSMEM cluster merge costs ~2 tiles, the last-CTA merge of up to 4 partial records ~6 (a
    // global write, an atomic and the reads, after the previous layer has finished) and the
    // separate combine launch ~7.
    const long long wave = std::min<long long>(
        std::min(var->ctas_per_sm * c->sm_count, c->max_ctas), tiles);
    const long long per_wave = (tiles + wave - 1) / wave;
    int cluster_k = 0;
    int grid;
    const long long slots = std::min<long long>(var->ctas_per_sm * c->sm_count, c->max_ctas);
    const long long S_all = static_cast<long long>(c->b) * c->g;
    long long whole = 0;   // CTAs of a whole-segment grid inside a decode step, or 0
    if (c->grid <= 0 && c->cluster == 1 && uniform && early_fetch == 1) {
        // Inside a decode step the layers' grids overlap (each triggers the next at once), so
        // a layer need not fill the GPU: a grid of whole segments (no merge, hence no wait for
        // the previous layer before writing partials) of at most half the resident slots lets
        // several layers stream at once.  It pays while the one-wave split would cut at least
        // half the segments (S <= 2 waves) and the segments are enough to stream (S >= 32).
        // Measured per step: 64 segments of 16 tiles of 128, 64 CTAs 59.1 us against 64.8 us
        // for 2-CTA clusters; 256 segments of 32 tiles of 256, 64 CTAs of 4 segments 872 us
        // against 917 us; but 3072 segments 13.9 ms against 10.3 ms, and 8 or 24 segments
        // (batch 8) 2-4% slower than the clusters.
        if (S_all >= 32 && S_all <= 2 * wave) {
            for (long long gw = std::min(S_all, slots / 2); gw >= 1; --gw) {
                if (S_all % gw == 0) {
                    whole = gw;
                    break;
                }
            }
        }
    }
    if (c->grid > 0) {
        grid = static_cast<int>(std::min<long long>(std::min(c->grid, c->max_ctas), tiles));
    } else if (single_long && var->v->tile_tokens == 128) {
        grid = static_cast<int>(std::min<long long>(64, tiles));
    } else if (whole > 0) {
        grid = static_cast<int>(whole);
    } else {
        grid = static_cast<int>((tiles + per_wave - 1) / per_wave);
        if (uniform) {
            const long long nt = (seq_lens[0] + T - 1) / T;
            const long long S = static_cast<long long>(c->b) * c->g;
            const long long per = tiles / grid;
            const long long pieces = per > 0 ? (nt - 1 + per - 1) / per + 1 : grid;
            long long best = per_wave + (pieces <= 1 ? 0 : pieces <= mlkv::kInlineMergeMaxPieces ? 6 : 7);
            if (S <= wave && nt < best) {
                best = nt;   // whole segments: grid S, each CTA exactly one segment
                grid = static_cast<int>(S);
            }
            if (c->cluster) {
                // Inside a step whose next layer reads its tiles early (early_fetch), with two
                // CTAs per SM, a grid that fits twice lets the next layer's CTAs all be resident,
                // streaming their tiles, while this layer's finish; that hides the ramp of each
                // layer, which the tile-unit model does not see.  So there the largest cluster
                // size whose grid fits twice wins while each CTA keeps >= 4 tiles and the grid
                // still holds a quarter of the resident CTAs, enough copies in flight to stream
                // (measured, 64 segments of 16 tiles of 128: 2-CTA clusters 80.5 us per 12-layer
                // step against 84.7 us for 4-CTA clusters; with 32 segments 4-CTA clusters, 128
                // CTAs, stay the better).  A layer that nothing overlaps (a standalone call, the
                // first layer of a step, a step without early fetch) takes the model's choice:
                // 4-CTA clusters there, 99.8 against 123.9 us for the default workload's 12
                // layers one after another.
                if (c->cluster == 1 && var->ctas_per_sm >= 2 && early_fetch == 1) {
                    for (int k : {4, 2}) {
                        if (cluster_k == 0 && nt % k == 0 && nt / k >= 4 && 2 * S * k <= wave &&
                            4 * S * k >= wave && var->clusters[k] >= 2 * S)
                            cluster_k = k;
                    }
                }
                const bool by_rule = cluster_k > 1;
                for (int k : {2, 4}) {
                    if (by_rule)
                        break;      // chosen above
                    if (c->cluster > 1 && k != c->cluster)
                        continue;   // one cluster size asked for
                    if (nt % k == 0 && S * k <= wave && var->clusters[k] >= S &&
                        (c->cluster > 1 || nt / k + 2 < best)) {
                        best = nt / k + 2;
                        cluster_k = k;
                    }
                }
                if (cluster_k > 1)
                    grid = static_cast<int>(S * cluster_k);
            }
        }
    }
    grid = std::max(std::min(grid, mlkv::kCombineMaxPiecesHost), 1);

    p.Q = static_cast<const __nv_bfloat16 *>(Q);
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.K_new = static_cast<const __nv_bfloat16 *>(K_new);
    p.V_new = static_cast<const __nv_bfloat16 *>(V_new);
    p.cache = static_cast<__nv_bfloat16 *>(c->cache);
    p.max_seq = c->max_seq;
    p.part_o = c->part_o;
    p.part_lse = c->part_lse;
    p.counters = c->counters;
    p.err = c->err;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c->d)));
    p.b = c->b;
    p.h = c->h;
    p.g = c->g;
    p.G = c->G;
    p.slot = c->slot[layer];
    p.num_tiles = static_cast<int>(tiles);
    p.cluster_k = cluster_k;
    p.tile_tokens = T;
    p.decode_grid = grid;
    p.early_fetch = early_fetch;
    p.newest_ready = newest_ready;
    p.store_new = K_new != nullptr ? store_new : 0;
    p.Q_next = static_cast<const __nv_bfloat16 *>(Q_next);
    // Segments split over many CTAs are merged by a separate parallel kernel: one warp merging
    // dozens of partials would serialise on its loads.
    p.deferred_merge = (cluster_k <= 1 &&
                        mlkv::max_pieces_per_segment(p, T, grid) > mlkv::kInlineMergeMaxPieces)
                           ? 1
                           : 0;

    p.pf_own = 0;
    p.ml_layers = 0;
    p.ml_chunks = 1;
    p.ml_seg_major = 0;
    p.ml_snake = 0;
    p.ml_slots = 0;
    p.ml_q_stride = 0;
    p.ml_kv_stride = 0;

    // L2 persistence (option l2_persist): every layer of an owner's block reads the slot through
    // an access-policy window over the slot's first bytes (at most the device's window size),
    // persisting as large a share of it as the set-aside holds (hitRatio = set-aside / window),
    // so the lines the owner layer brings in stay for the block's later layers.  The block's last
    // layer marks its hits normal again, which frees the set-aside for the next block's owner.
    cudaAccessPolicyWindow win = {};
    const cudaAccessPolicyWindow *winp = nullptr;
    if (c->l2_persist && c->window_max > 0 && c->persist_bytes > 0) {
        const size_t slot_bytes = c->cache_bytes / c->m;
        win.base_ptr = static_cast<char *>(c->cache) + slot_bytes * p.slot;
        win.num_bytes = std::min<size_t>(slot_bytes, static_cast<size_t>(c->window_max));
        win.hitRatio = static_cast<float>(
            std::min(1.0, static_cast<double>(c->persist_bytes) / win.num_bytes));
        bool last_of_block = true;
        for (int k = layer + 1; k < c->l; ++k)
            last_of_block = last_of_block && c->owner[k] != c->owner[layer];
        win.hitProp = last_of_block ? cudaAccessPropertyNormal : cudaAccessPropertyPersisting;
        win.missProp = cudaAccessPropertyStreaming;
        winp = &win;
    }
    DeviceGuard guard(c->device);
    const size_t smem = var->v->smem_bytes +
                        (cluster_k > 1 ? (cluster_k - 1) * var->v->res_bytes
                                       : (uniform ? 0 : mlkv::table_bytes(c->b)));
    cudaError_t e = mlkv::launch_decode(*var->v, grid, smem, static_cast<cudaStream_t>(cuda_stream),
                                        &var->tmap, &var->tmap_rows, p, winp, c->pdl != 0);
    if (e != cudaSuccess)
        return fail_cuda(e, "decode launch");
    if (p.deferred_merge) {
        e = mlkv::launch_combine(p, c->d, static_cast<cudaStream_t>(cuda_stream), c->pdl != 0);
        if (e != cudaSuccess)
            return fail_cuda(e, "combine launch");
    }
    c->last_grid = grid;
    c->last_tile = T;
    c->last_cluster_k = cluster_k;
    c->last_tc = var->v->tc;
    c->last_deferred = p.deferred_merge;
    c->last_l2_prefetch = 0;
    return MLKV_OK;
}

int mlkv_decode_attention(mlkv_cache_t c, int layer, const void *Q, void *out,
                          const int *seq_lens, void *cuda_stream)
{
    return decode_impl(c, layer, nullptr, nullptr, Q, out, seq_lens, cuda_stream);
}

int mlkv_append_decode_attention(mlkv_cache_t c, int layer, const void *K, const void *V,
                                 const void *Q, void *out, const int *seq_lens,
                                 void *cuda_stream)
{
    if (c != nullptr && layer >= 0 && layer < c->l && c->owner[layer] == layer) {
        if (K == nullptr || V == nullptr)
            return fail(MLKV_ERR_INVALID_ARG, "K and V must be non-NULL for an owner layer");
        return decode_impl(c, layer, K, V, Q, out, seq_lens, cuda_stream);
    }
    return decode_impl(c, layer, nullptr, nullptr, Q, out, seq_lens, cuda_stream);
}

// The fused decode's context split for nblk blocks: kc key tiles of 128 positions a unit; *units
// (if given) the units it makes.  Measured on GB300 (batch 64 x 2048 positions, 72 rows a unit):
// one CTA keeps an SM's softmax and tensor core about as busy as two do, while every unit costs
// ~5 us outside its key tiles (start, first loads, output) and a split adds the merge launch (16
// tiles a unit, 128 units: 31 us per step; 8 tiles, 256 units: 39; 4: 43; 1: 63).  So a sequence is
// split only as far as the units still fit one per SM: the smallest kc whose units number at most
// the SMs; no split when the (sequence, KV head, block) units alone exceed them.  The unit word
// holds chunk indices below kFusedMaxChunks.
static int fused_plan(const mlkv_cache *c, const int *seq_lens, int nblk, long long *units)
{
    int n_kt_max = 0;
    bool uniform = true;
    for (int beta = 0; beta < c->b; ++beta) {
        n_kt_max = std::max(n_kt_max, (seq_lens[beta] + 127) / 128);
        uniform = uniform && seq_lens[beta] == seq_lens[0];
    }
    const long long per_seq = static_cast<long long>(nblk) * c->g;
    const int kc_min = std::max(1, (n_kt_max + mlkv::kFusedMaxChunks - 2) /
                                       (mlkv::kFusedMaxChunks - 1));
    auto units_for = [&](int k) {
        if (uniform)
            return per_seq * c->b * ((n_kt_max + k - 1) / k);
        long long u = 0;
        for (int beta = 0; beta < c->b; ++beta)
            u += per_seq * (((seq_lens[beta] + 127) / 128 + k - 1) / k);
        return u;
    };
    int kc = n_kt_max;
    if (units_for(n_kt_max) < c->sm_count) {
        // units_for falls as k grows: the smallest k with units <= SMs, by bisection
        int lo = kc_min, hi = n_kt_max;
        while (lo < hi) {
            const int mid = lo + (hi - lo) / 2;
            if (units_for(mid) <= c->sm_count)
                hi = mid;
            else
                lo = mid + 1;
        }
        kc = lo;
    }
    if (c->fused_kc > 0)
        kc = std::max(kc_min, std::min(c->fused_kc, n_kt_max));
    if (units != nullptr)
        *units = units_for(kc);
    return kc;
}

// The fused decode's CTA form for blocks of L layers and n_units units: one query tile when the
// block's rows fit one (head_dim 64); then with at most one unit per SM one CTA per SM with a deep
// ring and two S buffers (its tiles come from HBM one after another), else two CTAs per SM.  Rows
// past one tile: two query tiles.
static int fused_cta_form(const mlkv_cache *c, int L, long long n_units)
{
    const bool one = c->d == 64 && L <= 128 / c->G;
    if (!one)
        return mlkv::kFusedTwoTiles;
    return n_units <= c->sm_count && c->fused_deep ? mlkv::kFusedOneDeep : mlkv::kFusedOneTile;
}

// The cross-layer fused decode (the fused form of prefill_kernel) over nblk owner blocks of L
// layers each: block k reads slot slot0 + k and attends for the layers k*L .. k*L + L - 1 of Q and
// out ([n_q_layers][b][h][d]).  A unit (sequence, KV head, block, chunk of the context) loads each
// K/V tile of its chunk once for all L*G query rows of the block (Sec. 3: the block's layers read
// one cache); a sequence's chunks are merged by one combine_fused launch.  Launches issued are
// added to *launches.
static int fused_issue(mlkv_cache_t c, const void *Q, void *out, int n_q_layers, int L, int nblk,
                       int slot0, const int *seq_lens, cudaStream_t stream, int *launches,
                       int after_store = 0, bool q_in_host = false)
{
    const int L1 = 128 / c->G;
    long long n_units = 0;
    const int kc = fused_plan(c, seq_lens, nblk, &n_units);
    const int form = fused_cta_form(c, L, n_units);
    cudaError_t e;
    if (!(c->fused_ready & (1 << form))) {
        if ((e = mlkv::prepare_fused(c->d, form)) != cudaSuccess)
            return fail_cuda(e, "cudaFuncSetAttribute(fused decode)");
        c->fused_ready |= 1 << form;
    }
    static EncodeTiledFn encode = driver_entry<EncodeTiledFn>("cuTensorMapEncodeTiled");
    if (encode == nullptr)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
    // Q [layers][b][h][d] as (channel, head in group, group, sequence, layer); a box of 64
    // channels x G heads x min(L1, L) layers is one tile's rows, layer-major.
    CUtensorMap tmap_q;
    const cuuint64_t dims[5] = {static_cast<cuuint64_t>(c->d), static_cast<cuuint64_t>(c->G),
                                static_cast<cuuint64_t>(c->g), static_cast<cuuint64_t>(c->b),
                                static_cast<cuuint64_t>(n_q_layers)};
    const cuuint64_t strides[4] = {static_cast<cuuint64_t>(c->d) * 2,
                                   static_cast<cuuint64_t>(c->G) * c->d * 2,
                                   static_cast<cuuint64_t>(c->h) * c->d * 2,
                                   static_cast<cuuint64_t>(c->b) * c->h * c->d * 2};
    const cuuint32_t box[5] = {64u, static_cast<cuuint32_t>(c->G), 1u, 1u,
                               static_cast<cuuint32_t>(L < L1 ? L : L1)};
    const cuuint32_t estr[5] = {1u, 1u, 1u, 1u, 1u};
    CUresult r = encode(&tmap_q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(Q), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled(fused Q) failed (CUresult %d)",
                    static_cast<int>(r));
    const CUtensorMap *tmap_kv = nullptr;
    for (auto &v : c->variants)
        if (v.v->tile_tokens == 128)
            tmap_kv = &v.tmap;
    if (tmap_kv == nullptr)
        return fail(MLKV_ERR_UNSUPPORTED, "no 128-position cache map for d=%d", c->d);

    static thread_local mlkv::PrefillParams p;
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.err = c->err;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c->d)));
    p.b = c->b;
    p.h = c->h;
    p.g = c->g;
    p.G = c->G;
    p.s_max = c->max_seq;
    p.slot = slot0;
    p.head_pairs = 0;
    p.fused_L = L;
    p.fused_L1 = L1;
    p.fused_nblk = nblk;
    p.fused_early = after_store;
    // queries in page-locked host memory (Q is its device-mapped address): read row by row
    p.q_host = q_in_host ? static_cast<const __nv_bfloat16 *>(Q) : nullptr;
    int n_kt_max = 0;
    bool uniform = true;
    for (int beta = 0; beta < c->b; ++beta) {
        p.prompt_len[beta] = seq_lens[beta];
        n_kt_max = std::max(n_kt_max, (seq_lens[beta] + 127) / 128);
        uniform = uniform && seq_lens[beta] == seq_lens[0];
    }
    const int cmax = (n_kt_max + kc - 1) / kc;
    p.fused_kc = kc;
    p.fused_cmax = cmax;
    // merge: one warp per output row up to 8 chunks, then 2, 4 or 8 warps sharing a row's chunks
    p.fused_combine_w = cmax <= 8 ? 1 : cmax <= 16 ? 2 : cmax <= 32 ? 4 : 8;
    p.part = p.part_lse = nullptr;
    if (cmax > 1) {
        const size_t rows = static_cast<size_t>(nblk) * c->b * c->g * cmax * L * c->G;
        const size_t floats = rows * (c->d + 1);
        if (floats > c->fused_part_floats) {
            if (c->fused_part)
                cudaFree(c->fused_part);
            c->fused_part = nullptr;
            c->fused_part_floats = 0;
            if ((e = cudaMalloc(&c->fused_part, floats * sizeof(float))) != cudaSuccess) {
                c->fused_part = nullptr;
                return fail(MLKV_ERR_OOM, "fused-decode partials (%zu bytes): %s",
                            floats * sizeof(float), cudaGetErrorString(e));
            }
            c->fused_part_floats = floats;
        }
        p.part = c->fused_part;
        p.part_lse = c->fused_part + rows * c->d;
    }
    // Units: the longest sequences first; within a sequence block, KV head, chunk.
    static thread_local std::vector<int> order;
    order.resize(c->b);
    for (int beta = 0; beta < c->b; ++beta)
        order[beta] = beta;
    if (!uniform)
        std::stable_sort(order.begin(), order.end(),
                         [&](int x, int y) { return seq_lens[x] > seq_lens[y]; });
    int n = 0;
    long long total_units = 0;
    for (int beta : order)
        for (int blk = 0; blk < nblk; ++blk)
            for (int j = 0; j < c->g; ++j)
                for (int ch = 0; ch * kc < (seq_lens[beta] + 127) / 128; ++ch) {
                    p.units[n] = static_cast<uint32_t>(beta) | (static_cast<uint32_t>(ch) << 10) |
                                 (static_cast<uint32_t>(blk) << 18) |
                                 (static_cast<uint32_t>(j) << 24);
                    ++total_units;
                    if (++n == mlkv::kPrefillMaxUnits) {
                        p.n_units = n;
                        if ((e = mlkv::launch_fused(c->d, form, &tmap_q, tmap_kv, p, stream)) !=
                            cudaSuccess)
                            return fail_cuda(e, "fused decode launch");
                        ++*launches;
                        n = 0;
                    }
                }
    if (n > 0) {
        p.n_units = n;
        if ((e = mlkv::launch_fused(c->d, form, &tmap_q, tmap_kv, p, stream)) != cudaSuccess)
            return fail_cuda(e, "fused decode launch");
        ++*launches;
    }
    if (cmax > 1) {
        if ((e = mlkv::launch_fused_combine(c->d, p, stream)) != cudaSuccess)
            return fail_cuda(e, "fused decode merge launch");
        ++*launches;
    }
    c->last_grid = static_cast<int>(std::min<long long>(total_units, 0x7fffffffLL));
    c->last_tile = 128;
    c->last_deferred = cmax > 1 ? 1 : 0;
    c->last_fused_kc = kc;
    return MLKV_OK;
}

// Whether mlkv_decode_step takes the cross-layer fused form for these lengths: maps of equal
// contiguous blocks (owner[n] = n - n mod L, the paper's Eq. 18 layout) whose L*G query rows fit
// two 128-row tiles, under the options (step_fused; no tile length or L2 prefetch forced), and
// with step_fused = 1 where the estimates below favour it.  host_inputs: the step's buffers are
// page-locked host memory read in place.
static bool fused_step_applies(const mlkv_cache *c, const int *seq_lens, bool host_inputs)
{
    if (!c->step_fused || c->tile_tokens > 0 || c->l2_prefetch || c->m > mlkv::kFusedMaxBlocks ||
        c->g > 255 || c->h > mlkv::kPrefillMaxHeads || (c->d != 64 && c->d != 128))
        return false;
    const int L = c->l / c->m;
    const int L1 = 128 / c->G;
    if (L * c->m != c->l || L1 < 1 || L > 2 * L1)
        return false;
    for (int n = 0; n < c->l; ++n)
        if (c->owner[n] != n - n % L || c->slot[n] != n / L)
            return false;
    if (c->step_fused == 1) {
        // Where the fused form pays, from measurements on GB300 against the decode kernel's
        // launch.  A block of one layer shares nothing across layers (MHA, GQA-4, MQA at batch
        // 256 and 1: 7-16% slower fused); blocks of two saved little or lost (batch 64 x 2000
        // positions 49 vs 53 us, batch 256 x 8192 535 vs 548, batch 1 x 131072 66 vs 62, batch
        // 1 x 128 11.6 vs 10.3; with the split-key CTA form 53.2 vs 52.6, 548.9 vs 548.0, 60.3
        // vs 59.3, 12.5 vs 10.7).  For blocks of >= 3 layers the estimates in us per step, from the
        // same measurements: the fused form ~1.1 per key tile its busiest SM takes plus ~6 fixed
        // (+3 for the merge of a split); the decode kernel ~0.55 per (layer, sequence, KV head,
        // 128 positions) item per SM plus ~3.  They pick the measured winner at batch 8, 64, 128
        // and 256, batch 1 x 131072 and Llama-2-7B shapes.
        if (L < 3)
            return false;
        long long units = 0;
        const int kc = fused_plan(c, seq_lens, c->m, &units);
        long long tiles = 0;
        int n_kt_max = 0;
        bool uniform = true;
        for (int beta = 0; beta < c->b; ++beta) {
            tiles += (seq_lens[beta] + 127) / 128;
            n_kt_max = std::max(n_kt_max, (seq_lens[beta] + 127) / 128);
            uniform = uniform && seq_lens[beta] == seq_lens[0];
        }
        // the busiest SM's key tiles: whole waves of equal units with one length; with varied
        // lengths (units longest first) about the mean, and at least one unit
        const long long busiest =
            uniform ? (units + c->sm_count - 1) / c->sm_count * kc
                    : std::max<long long>(kc, (tiles * c->m * c->g + c->sm_count - 1) /
                                                  c->sm_count);
        const double fused_us =
            1.1 * static_cast<double>(busiest) + 6.0 + (kc < n_kt_max ? 3.0 : 0.0);
        const double ml_us = 0.55 * static_cast<double>(tiles) * c->l * c->g / c->sm_count + 3.0;
        if (fused_us >= ml_us)
            return false;
    }
    if (host_inputs) {
        // Inputs read in place only when no sequence is split: every chunk of a split sequence
        // would read its query rows over the CPU-GPU link again (measured at batch 1 x 131072
        // positions, MLKV-1: 47.7 us end to end against 36.9 on the device); the caller copies
        // them in instead.
        int n_kt_max = 0;
        for (int beta = 0; beta < c->b; ++beta)
            n_kt_max = std::max(n_kt_max, (seq_lens[beta] + 127) / 128);
        if (fused_plan(c, seq_lens, c->m, nullptr) < n_kt_max)
            return false;
    }
    return true;
}

// mlkv_decode_step in the cross-layer fused form, where fused_step_applies: one append launch for
// every owner's new token, then the fused decode of every block in one launch (and one merge);
// otherwise *done stays false.
static int issue_step_fused(mlkv_cache_t c, const char *Q, const char *K, const char *V, char *out,
                            const int *seq_lens, void *stream, cudaEvent_t in_ready, bool *done,
                            const mlkv::StageParams *stage, bool host_inputs = false)
{
    *done = false;
    if (!fused_step_applies(c, seq_lens, host_inputs))
        return MLKV_OK;
    bool has_map = false;   // the cache's tensor map of 128-position tiles
    for (auto &v : c->variants)
        has_map = has_map || v.v->tile_tokens == 128;
    if (!has_map)
        return MLKV_OK;
    const int L = c->l / c->m;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    DeviceGuard guard(c->device);
    if (in_ready != nullptr && (e = cudaStreamWaitEvent(s, in_ready, 0)) != cudaSuccess)
        return fail_cuda(e, "step event");
    int launches = 0;
    if (stage != nullptr) {
        if ((e = mlkv::launch_stage_copy(*stage, s)) != cudaSuccess)
            return fail_cuda(e, "copy-in of the step's inputs");
        ++launches;
    }
    // Every owner's new token at position L_beta - 1 of its slot, before any block reads it.
    mlkv::AppendParams ap;
    ap.K = reinterpret_cast<const __nv_bfloat16 *>(K);
    ap.V = reinterpret_cast<const __nv_bfloat16 *>(V);
    ap.cache = static_cast<__nv_bfloat16 *>(c->cache);
    ap.b = c->b;
    ap.g = c->g;
    ap.d = c->d;
    ap.max_seq = c->max_seq;
    ap.slot = 0;
    ap.n_slots = c->m;
    // After this library's input copy (host buffers) the fused launch goes at once and fetches
    // cache tiles while the copy runs; otherwise it follows the store's dependency wait and also
    // fetches the queries at once.
    ap.trigger_first = stage != nullptr ? 1 : 0;
    std::memcpy(ap.seq_len, seq_lens, sizeof(int) * c->b);
    if ((e = mlkv::launch_append_slots(ap, s)) != cudaSuccess)
        return fail_cuda(e, "append launch (fused step)");
    ++launches;
    // With the inputs in page-locked host memory (host_inputs: Q, K, V and out are device-mapped
    // addresses) the store reads the new tokens and the fused units their query rows from there.
    const int rc = fused_issue(c, Q, out, c->l, L, c->m, 0, seq_lens, s, &launches,
                               stage != nullptr ? 2 : 1, host_inputs);
    if (rc != MLKV_OK)
        return rc;
    c->last_cluster_k = 0;
    c->last_tc = 0;
    c->last_l2_prefetch = 0;
    c->last_step_kernel = 1;
    c->last_step_fused = 1;
    c->last_seg_major = 0;
    c->last_step_launches = launches - (stage != nullptr ? 1 : 0);
    *done = true;
    return MLKV_OK;
}

// The options under which mlkv_decode_step may issue a step as one launch (the decode kernel's
// multi-layer launch or the fused form): the mma.sync kernel, default grid, no L2-persistence
// windows (they are per layer), at most kMaxStepLayers layers.
static bool step_launch_allowed(const mlkv_cache *c)
{
    return c->step_kernel && !c->tc && c->grid <= 0 && !c->l2_persist &&
           c->l <= mlkv::kMaxStepLayers;
}

// The whole decode step in one launch: the cross-layer fused form where it applies
// (issue_step_fused), else one launch of the decode kernel over every (layer, segment) item
// (DecodeParams::ml_layers) where that applies: every sequence has one length and the makespan is
// no longer than the per-layer launches' (below).  Items are whole segments, so nothing is merged
// and no scratch is shared; every layer takes its segments' newest rows from the step's new
// tokens, and owner layers store them.  *done tells whether it was issued.  With in_ready, the
// launch waits for it (queries still arriving).  With `stage`, the copy of the step's inputs it
// describes is launched right before the step's kernel, which may then start (and fetch its first
// cache tiles) while the copy runs.
static int issue_step_ml(mlkv_cache_t c, const char *Q, const char *K, const char *V, char *out,
                         const int *seq_lens, void *stream, cudaEvent_t in_ready, bool *done,
                         const mlkv::StageParams *stage = nullptr, bool host_inputs = false)
{
    *done = false;
    c->last_step_kernel = 0;
    c->last_step_fused = 0;
    c->last_step_launches = 0;
    if (!step_launch_allowed(c))
        return MLKV_OK;
    {
        const int rc =
            issue_step_fused(c, Q, K, V, out, seq_lens, stream, in_ready, done, stage, host_inputs);
        if (rc != MLKV_OK || *done || host_inputs)
            return rc;   // host inputs: only the fused form reads them where they are
    }
    bool uniform = true;
    long long len_sum = 0;
    for (int beta = 0; beta < c->b; ++beta) {
        uniform = uniform && seq_lens[beta] == seq_lens[0];
        len_sum += seq_lens[beta];
    }
    const double mean_len = static_cast<double>(len_sum) / c->b;
    mlkv_cache::Variant *var = pick_variant(c, mean_len);
    if (var == nullptr || var->v->tc)
        return MLKV_OK;
    if (!uniform && var->v->smem_bytes + mlkv::table_bytes(c->b) > c->max_smem) {
        var = nullptr;   // the per-sequence tables need the small-ring variant
        for (auto &v : c->variants)
            if (v.v->tile_tokens == 64 && !v.v->tc &&
                v.v->smem_bytes + mlkv::table_bytes(c->b) <= c->max_smem)
                var = &v;
        if (var == nullptr)
            return MLKV_OK;
    }
    const long long S = static_cast<long long>(c->b) * c->g;
    // Sequences longest first (stable); items ranked segment-major over them.
    static thread_local std::vector<int> perm;
    perm.resize(c->b);
    for (int beta = 0; beta < c->b; ++beta)
        perm[beta] = beta;
    if (!uniform)
        std::stable_sort(perm.begin(), perm.end(),
                         [&](int x, int y) { return seq_lens[x] > seq_lens[y]; });
    // Segment-major ranks when the slots' visible rows do not fit in L2 (the block's layers then
    // share each segment's K/V while it is in L2); layer-major otherwise.  A snake deal balances
    // varied lengths.
    const long long all_kv = static_cast<long long>(c->m) * 2 * c->g * len_sum * c->d * 2;
    const int seg_major = all_kv > static_cast<long long>(c->l2_bytes) * 5 / 8 ? 1 : 0;
    const int snake = uniform ? 0 : 1;
    // A plan: tile length, chunks per segment, grid; its makespan in tiles is the heaviest CTA's
    // items under the deal.  Grid: with one length the fewest CTAs that keep ceil(items / slots)
    // items each; otherwise every resident slot.
    struct Plan {
        mlkv_cache::Variant *var;
        int T, chunks, grid;
        long long items, heaviest, per_layer;
    };
    auto plan_for = [&](mlkv_cache::Variant *v, int chunks) {
        Plan pl{v, v->v->tile_tokens, chunks, 0, S * c->l * chunks, 0, 0};
        const long long slots = static_cast<long long>(v->ctas_per_sm) * c->sm_count;
        const long long per = (pl.items + slots - 1) / slots;
        pl.grid = static_cast<int>(uniform ? (pl.items + per - 1) / per : std::min(pl.items, slots));
        long long total_tiles = 0;
        for (int beta = 0; beta < c->b; ++beta)
            total_tiles += static_cast<long long>(c->g) * ((seq_lens[beta] + pl.T - 1) / pl.T);
        // per-layer launches split every layer over the machine but pay a launch, a ramp and
        // merges per layer (about 4 tiles' time each; they overlap only in part)
        pl.per_layer = c->l * ((total_tiles + slots - 1) / slots + 4);
        static thread_local std::vector<long long> load;
        load.assign(pl.grid, 0);
        const long long per_seq = static_cast<long long>(c->g) * c->l;
        for (long long r = 0; r < pl.items; ++r) {
            const long long k = r / pl.grid, i = r - k * pl.grid;
            const long long cta = (snake && (k & 1)) ? pl.grid - 1 - i : i;
            const long long rb = r / chunks, ch = r - rb * chunks;
            const long long pb = seg_major ? rb / per_seq : (rb % S) / c->g;
            const long long nt = (seq_lens[perm[pb]] + pl.T - 1) / pl.T;
            load[cta] += (ch + 1) * nt / chunks - ch * nt / chunks;
        }
        for (long long x : load)
            pl.heaviest = std::max(pl.heaviest, x);
        if (chunks > 1)
            pl.heaviest += 4;   // the merge launch
        return pl;
    };
    Plan pl = plan_for(var, 1);
    if (uniform && pl.heaviest > pl.per_layer) {
        // Few long segments (batch 1 at long context): split every segment into C chunks, each a
        // partial record, merged by one combine launch for the whole step.  C: chunks of >= 8
        // tiles, 2 to 4 waves of items, rounded so that the items fill whole waves of resident
        // CTAs where that is possible; per tile size the plan with the lightest heaviest CTA (its
        // tiles, plus one tile's worth for each partial record it writes) is taken.  Between the
        // 256-position tile (one CTA per SM, three stages) and the 128-position one (two CTAs per
        // SM) the 256 one is taken unless it gives a CTA more than one item beyond the 128 one's
        // (measured at batch 1, 131072 positions: MLKV-2 59.4 -> 52.9 us, MLKV-6 71.6 -> 62.8,
        // MQA 93.4 -> 89.4; GQA-4, 9 items a CTA against 5: 250 -> 260, so 128 there).  A forced
        // tile size (option "tile") is used as it is.
        struct Chunked {
            bool ok = false;
            Plan plan{};
            long long per = 0;
        };
        auto best_chunks = [&](int T_chunk) {
            Chunked best;
            mlkv_cache::Variant *vch = pick_variant(c, -1.0, T_chunk);
            if (vch == nullptr || vch->v->tc)
                return best;
            const long long slots = static_cast<long long>(vch->ctas_per_sm) * c->sm_count;
            const long long nt = (seq_lens[0] + T_chunk - 1) / T_chunk;
            const long long sl = S * c->l;
            long long a = slots, bq = sl;   // gcd: C a multiple of slots / gcd fills whole waves
            while (bq != 0) {
                const long long r = a % bq;
                a = bq;
                bq = r;
            }
            const long long unit = slots / a;
            const long long c_max = std::min<long long>(
                {nt / 8, mlkv::kCombineMaxPiecesHost, static_cast<long long>(c->records) / sl});
            long long best_cost = -1;
            for (int waves = 2; waves <= 4; ++waves) {
                long long C = (waves * slots + sl - 1) / sl;
                const long long Cr = (C + unit - 1) / unit * unit;
                C = Cr <= c_max ? Cr : std::min(C, c_max);
                if (C <= 1)
                    continue;
                Plan pc = plan_for(vch, static_cast<int>(C));
                if (pc.heaviest > pc.per_layer)
                    continue;
                const long long per = (pc.items + pc.grid - 1) / pc.grid;
                const long long cost = pc.heaviest + per;
                if (best_cost < 0 || cost < best_cost) {
                    best_cost = cost;
                    best.ok = true;
                    best.plan = pc;
                    best.per = per;
                }
            }
            return best;
        };
        Chunked pick;
        if (c->tile_tokens > 0) {
            pick = best_chunks(c->tile_tokens);
        } else {
            const Chunked c256 = best_chunks(256), c128 = best_chunks(128);
            pick = (c256.ok && (!c128.ok || c256.per <= c128.per + 1)) ? c256 : c128;
        }
        if (pick.ok)
            pl = pick.plan;
    }
    if (pl.heaviest > pl.per_layer || pl.items > 0x7fffffffLL ||
        pl.items * pl.heaviest > 0x7fffffffLL)
        return MLKV_OK;
    var = pl.var;
    const int T = pl.T;
    const int grid = pl.grid;
    long long total_tiles = 0;
    for (int beta = 0; beta < c->b; ++beta)
        total_tiles += static_cast<long long>(c->g) * ((seq_lens[beta] + T - 1) / T);

    static thread_local mlkv::DecodeParams p;
    p.Q = reinterpret_cast<const __nv_bfloat16 *>(Q);
    p.out = reinterpret_cast<__nv_bfloat16 *>(out);
    p.K_new = reinterpret_cast<const __nv_bfloat16 *>(K);
    p.V_new = reinterpret_cast<const __nv_bfloat16 *>(V);
    p.cache = static_cast<__nv_bfloat16 *>(c->cache);
    p.max_seq = c->max_seq;
    p.part_o = c->part_o;
    p.part_lse = c->part_lse;
    p.counters = c->counters;
    p.err = c->err;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c->d)));
    p.b = c->b;
    p.h = c->h;
    p.g = c->g;
    p.G = c->G;
    p.slot = 0;
    p.num_tiles = static_cast<int>(total_tiles * c->l);
    p.uniform_len = uniform ? seq_lens[0] : 0;
    for (int beta = 0; beta < c->b; ++beta) {
        p.seq_len[beta] = seq_lens[beta];
        p.tile_start[beta] = perm[beta];
    }
    p.tile_start[c->b] = 0;
    p.cluster_k = 0;
    p.deferred_merge = pl.chunks > 1 ? 1 : 0;
    p.tile_tokens = T;
    p.decode_grid = grid;
    p.Q_next = nullptr;
    // After this library's input copy the first tile of each CTA goes out before the wait.
    p.early_fetch = (stage != nullptr && c->pdl) ? 2 : 0;
    p.newest_ready = 1;
    p.store_new = 0;
    // L2 prefetch of every slot's visible rows when they all fit with room to spare.
    p.pf_own = (c->l2_prefetch && uniform &&
                all_kv <= static_cast<long long>(c->l2_bytes) * 5 / 8) ? 1 : 0;
    p.ml_slots = c->m;
    p.ml_seg_major = seg_major;
    p.ml_snake = snake;
    p.ml_chunks = pl.chunks;
    p.ml_layers = c->l;
    p.ml_q_stride = static_cast<long long>(c->b) * c->h * c->d;
    p.ml_kv_stride = static_cast<long long>(c->b) * c->g * c->d;
    for (int n = 0; n < c->l; ++n) {
        p.ml_slot[n] = static_cast<unsigned char>(c->slot[n]);
        p.ml_store[n] = c->owner[n] == n ? 1 : 0;
    }
    // the layers of one owner block next to each other, blocks in slot order
    {
        int k = 0;
        for (int s = 0; s < c->m; ++s)
            for (int n = 0; n < c->l; ++n)
                if (c->slot[n] == s)
                    p.ml_order[k++] = static_cast<unsigned char>(n);
    }
    cudaError_t e = cudaSuccess;
    if (in_ready != nullptr)
        e = cudaStreamWaitEvent(static_cast<cudaStream_t>(stream), in_ready, 0);
    if (e != cudaSuccess)
        return fail_cuda(e, "step event");
    DeviceGuard guard(c->device);
    if (stage != nullptr && (e = mlkv::launch_stage_copy(*stage, static_cast<cudaStream_t>(stream))) !=
                                cudaSuccess)
        return fail_cuda(e, "copy-in of the step's inputs");
    const size_t smem = var->v->smem_bytes + (uniform ? 0 : mlkv::table_bytes(c->b));
    e = mlkv::launch_decode(*var->v, grid, smem, static_cast<cudaStream_t>(stream), &var->tmap,
                            &var->tmap_rows, p, nullptr, c->pdl != 0);
    if (e != cudaSuccess)
        return fail_cuda(e, "decode launch (multi-layer step)");
    if (p.deferred_merge) {
        e = mlkv::launch_combine(p, c->d, static_cast<cudaStream_t>(stream), c->pdl != 0);
        if (e != cudaSuccess)
            return fail_cuda(e, "combine launch (multi-layer step)");
    }
    c->last_grid = grid;
    c->last_tile = T;
    c->last_cluster_k = 0;
    c->last_tc = 0;
    c->last_deferred = p.deferred_merge;
    c->last_l2_prefetch = p.pf_own;
    c->last_step_kernel = 1;
    c->last_seg_major = seg_major;
    c->last_step_launches = p.deferred_merge ? 2 : 1;
    *done = true;
    return MLKV_OK;
}

// The layer calls of one decode step, issued on `stream` (one multi-layer launch where
// issue_step_ml applies).
// With in_ready, layer 1 onwards waits for it (the later layers' queries still arriving); with
// before_last, it is recorded once every layer but the last has been issued.
static int issue_step(mlkv_cache_t c, const char *Q, const char *K, const char *V, char *out,
                      const int *seq_lens, void *stream, cudaEvent_t in_ready = nullptr,
                      cudaEvent_t before_last = nullptr)
{
    c->last_step_kernel = 0;
    c->last_step_fused = 0;
    c->last_step_launches = 0;
    if (before_last == nullptr) {
        bool done = false;
        const int rc = issue_step_ml(c, Q, K, V, out, seq_lens, stream, in_ready, &done);
        if (rc != MLKV_OK || done)
            return rc;
    }
    const size_t qo = static_cast<size_t>(c->b) * c->h * c->d * 2;   // bytes of one layer's Q
    const size_t kv = static_cast<size_t>(c->b) * c->g * c->d * 2;   // one owner's new token
    for (int n = 0; n < c->l; ++n) {
        int rc;
        cudaError_t e = cudaSuccess;
        if (n == 1 && in_ready != nullptr)
            e = cudaStreamWaitEvent(static_cast<cudaStream_t>(stream), in_ready, 0);
        if (e == cudaSuccess && n == c->l - 1 && before_last != nullptr)
            e = cudaEventRecord(before_last, static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess)
            return fail_cuda(e, "step event");
        // Layers after the first follow this library's own launch of the preceding layer.
        // 1: queries and tiles before the previous layers' grids end; 2: only the first cache
        // tile (the queries after) -- what a layer whose queries come from the previous layer
        // may do
        const int early = (n > 0 && c->pdl) ? c->early_fetch : 0;
        const char *q_next = (early == 1 && n + 1 < c->l) ? Q + qo * (n + 1) : nullptr;
        // A segment's newest row is the step's new token of the owner: the owner layer appends
        // it itself (fused); a later layer of the block replaces that row of its tiles from the
        // same input without storing it.  So no layer waits for another's launch to store it
        // (newest_ready).  The tcgen05 kernel does neither and keeps the plain wait.
        const int patch = (early && c->tc == 0) ? 1 : 0;
        const int newest_ready = patch;
        const size_t ks = kv * c->slot[c->owner[n]];
        if (c->owner[n] == n)
            rc = decode_impl(c, n, K + ks, V + ks, Q + qo * n, out + qo * n, seq_lens, stream,
                             early, q_next, newest_ready, 1, 1);
        else if (patch)
            rc = decode_impl(c, n, K + ks, V + ks, Q + qo * n, out + qo * n, seq_lens, stream,
                             early, q_next, newest_ready, 0, 1);
        else
            rc = decode_impl(c, n, nullptr, nullptr, Q + qo * n, out + qo * n, seq_lens, stream,
                             early, q_next, newest_ready, 1, 1);
        if (rc != MLKV_OK)
            return rc;
    }
    return MLKV_OK;
}

}  // extern "C"

namespace {

mlkv_cache::StepKey step_key_of(const mlkv_cache *c, const void *Q, const void *K, const void *V,
                                void *out, const int *seq_lens)
{
    mlkv_cache::StepKey key;
    key.Q = Q;
    key.K = K;
    key.V = V;
    key.out = out;
    key.lens.assign(seq_lens, seq_lens + c->b);
    key.tile = c->tile_tokens;
    key.grid = c->grid;
    key.cluster = c->cluster;
    key.pdl = c->pdl;
    key.tc = c->tc;
    key.l2 = c->l2_persist;
    key.pf = c->l2_prefetch;
    key.sk = c->step_kernel;
    key.sg = c->step_graph;
    key.ef = c->early_fetch;
    key.sf = c->step_fused;
    return key;
}

// Runs a step's work: replayed from `exec` when `key` is what it was recorded with; issued directly
// when these arguments were not seen on the previous call (about half the host time of recording,
// and in a decode loop lengths change every step); recorded when they come back.  Recording runs
// on a private stream (the caller's may be the legacy default stream, which cannot be captured);
// the replay goes to the caller's stream.
template <class Issue>
int record_or_replay(mlkv_cache *c, const mlkv_cache::StepKey &key, mlkv_cache::StepKey &recorded,
                     mlkv_cache::StepKey &pending, cudaGraphExec_t &exec, cudaStream_t stream,
                     Issue issue)
{
    cudaError_t e;
    if (exec == nullptr || !(key == recorded)) {
        if (!(key == pending)) {
            pending = key;
            return issue(stream);
        }
        if (c->record_stream == nullptr &&
            (e = cudaStreamCreateWithFlags(&c->record_stream, cudaStreamNonBlocking)) != cudaSuccess)
            return fail_cuda(e, "cudaStreamCreateWithFlags");
        e = cudaStreamBeginCapture(c->record_stream, cudaStreamCaptureModeThreadLocal);
        if (e != cudaSuccess)
            return fail_cuda(e, "cudaStreamBeginCapture");
        int rc = issue(c->record_stream);
        cudaGraph_t graph = nullptr;
        e = cudaStreamEndCapture(c->record_stream, &graph);
        if (rc != MLKV_OK) {
            if (graph)
                cudaGraphDestroy(graph);
            return rc;
        }
        if (e != cudaSuccess)
            return fail_cuda(e, "cudaStreamEndCapture");
        bool updated = false;
        if (exec != nullptr) {
            cudaGraphExecUpdateResultInfo info;
            updated = cudaGraphExecUpdate(exec, graph, &info) == cudaSuccess;
            if (!updated) {
                cudaGetLastError();
                cudaGraphExecDestroy(exec);
                exec = nullptr;
            }
        }
        if (!updated) {
            e = cudaGraphInstantiate(&exec, graph, 0);
            if (e != cudaSuccess) {
                cudaGraphDestroy(graph);
                exec = nullptr;
                return fail_cuda(e, "cudaGraphInstantiate");
            }
        }
        cudaGraphDestroy(graph);
        recorded = key;
    }
    e = cudaGraphLaunch(exec, stream);
    if (e != cudaSuccess)
        return fail_cuda(e, "cudaGraphLaunch");
    ++c->step_graph_replays;
    return MLKV_OK;
}

}  // namespace

extern "C" {

int mlkv_plan_step(int n_layers, int n_q_heads, int head_dim, const int *layer_owner,
                   int kv_heads_per_owner, int batch, int max_seq, const int *seq_lens,
                   int sm_count, int step_fused, int fused_kc, int fused_deep, int64_t plan[4])
{
    if (plan == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "plan is NULL");
    int rc = validate_map(n_layers, n_q_heads, head_dim, layer_owner, kv_heads_per_owner, batch,
                          max_seq);
    if (rc != MLKV_OK)
        return rc;
    if (sm_count < 1)
        return fail(MLKV_ERR_INVALID_ARG, "sm_count %d must be positive", sm_count);
    if (step_fused < -1 || step_fused > 2 || fused_deep < -1 || fused_deep > 1 || fused_kc < -1 ||
        fused_kc > (1 << 20))
        return fail(MLKV_ERR_INVALID_ARG, "step_fused %d, fused_kc %d or fused_deep %d out of range",
                    step_fused, fused_kc, fused_deep);
    // The decision of mlkv_decode_step, on a cache description that holds nothing on a device.
    mlkv_cache c;
    assign_map(&c, n_layers, n_q_heads, head_dim, layer_owner, kv_heads_per_owner, batch, max_seq);
    c.sm_count = sm_count;
    if (step_fused >= 0)
        c.step_fused = step_fused;
    if (fused_kc >= 0)
        c.fused_kc = fused_kc;
    if (fused_deep >= 0)
        c.fused_deep = fused_deep;
    if ((rc = check_seq_lens(&c, seq_lens)) != MLKV_OK)
        return rc;
    plan[0] = 0;
    plan[1] = -1;
    plan[2] = 0;
    plan[3] = 0;
    if (step_launch_allowed(&c) && fused_step_applies(&c, seq_lens, false)) {
        long long units = 0;
        const int kc = fused_plan(&c, seq_lens, c.m, &units);
        plan[0] = 1;
        plan[1] = fused_cta_form(&c, c.l / c.m, units);
        plan[2] = kc;
        plan[3] = units;
    }
    return MLKV_OK;
}

int mlkv_decode_step(mlkv_cache_t c, const void *Q, const void *K, const void *V, void *out,
                     const int *seq_lens, void *cuda_stream)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (Q == nullptr || K == nullptr || V == nullptr || out == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "Q, K, V and out must be non-NULL");
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(out))
        return fail(MLKV_ERR_INVALID_ARG, "Q, K, V and out must be 16-byte aligned");
    int rc = check_seq_lens(c, seq_lens);
    if (rc != MLKV_OK)
        return rc;
    DeviceGuard guard(c->device);
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(stream, &cap);
    if (e != cudaSuccess)
        return fail_cuda(e, "cudaStreamIsCapturing");
    const char *q = static_cast<const char *>(Q);
    const char *k = static_cast<const char *>(K);
    const char *v = static_cast<const char *>(V);
    char *o = static_cast<char *>(out);
    if (!c->step_graph || cap != cudaStreamCaptureStatusNone)
        return issue_step(c, q, k, v, o, seq_lens, cuda_stream);   // the caller records us
    if (c->step_graph == 2) {
        // One multi-layer launch (and its merge) is issued directly: replaying a one-node graph
        // measured ~2 us slower per step than the launch itself.
        bool done = false;
        rc = issue_step_ml(c, q, k, v, o, seq_lens, cuda_stream, nullptr, &done);
        if (rc != MLKV_OK || done)
            return rc;
    }

    mlkv_cache::StepKey key = step_key_of(c, Q, K, V, out, seq_lens);
    return record_or_replay(c, key, c->step_key, c->pending_key, c->step_exec, stream,
                            [&](cudaStream_t s) { return issue_step(c, q, k, v, o, seq_lens, s); });
}

int mlkv_decode_step_host(mlkv_cache_t c, const void *Q, const void *K, const void *V, void *out,
                          const int *seq_lens, void *cuda_stream)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (Q == nullptr || K == nullptr || V == nullptr || out == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "Q, K, V and out must be non-NULL");
    int rc = check_seq_lens(c, seq_lens);
    if (rc != MLKV_OK)
        return rc;
    DeviceGuard guard(c->device);
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    cudaError_t e;
    mlkv_cache::StepKey key = step_key_of(c, Q, K, V, out, seq_lens);
    if (c->host_exec != nullptr && c->step_graph && key == c->host_key) {
        // The arguments this step was recorded with (their buffers were checked then).
        cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
        if ((e = cudaStreamIsCapturing(stream, &cap)) != cudaSuccess)
            return fail_cuda(e, "cudaStreamIsCapturing");
        if (cap == cudaStreamCaptureStatusNone) {
            if ((e = cudaGraphLaunch(c->host_exec, stream)) != cudaSuccess)
                return fail_cuda(e, "cudaGraphLaunch");
            ++c->step_graph_replays;
            return MLKV_OK;
        }
    }
    const size_t qo_bytes = static_cast<size_t>(c->l) * c->b * c->h * c->d * 2;
    const size_t kv_bytes = static_cast<size_t>(c->m) * c->b * c->g * c->d * 2;
    if (c->stage == nullptr && (e = cudaMalloc(&c->stage, 2 * qo_bytes + 2 * kv_bytes)) != cudaSuccess) {
        c->stage = nullptr;
        return fail(MLKV_ERR_OOM, "staging buffers (%zu bytes): %s", 2 * qo_bytes + 2 * kv_bytes,
                    cudaGetErrorString(e));
    }
    char *dq = static_cast<char *>(c->stage);
    char *dk = dq + qo_bytes;
    char *dv = dk + kv_bytes;
    char *dout = dv + kv_bytes;
    // Page-locked, 16-byte-aligned buffers are read by copy kernels and written by the layers
    // themselves through their device-mapped addresses; anything else takes one cudaMemcpyAsync
    // per tensor (a copy-engine transfer has ~12 us of fixed latency).
    const void *dev[4] = {nullptr, nullptr, nullptr, nullptr};
    bool mapped = true;
    {
        const void *hp[4] = {Q, K, V, out};
        for (int k = 0; k < 4; ++k) {
            cudaPointerAttributes at;
            if (cudaPointerGetAttributes(&at, hp[k]) != cudaSuccess ||
                at.type != cudaMemoryTypeHost || at.devicePointer == nullptr ||
                !aligned16(at.devicePointer)) {
                cudaGetLastError();
                mapped = false;
                break;
            }
            dev[k] = at.devicePointer;
        }
    }
    if (mapped && c->side == nullptr) {
        if ((e = cudaStreamCreateWithFlags(&c->side, cudaStreamNonBlocking)) != cudaSuccess)
            return fail_cuda(e, "cudaStreamCreateWithFlags");
        for (cudaEvent_t &ev : c->ev)
            if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming)) != cudaSuccess)
                return fail_cuda(e, "cudaEventCreateWithFlags");
    }
    auto issue = [&](cudaStream_t s) {
        if (mapped) {
            // The fused form reads the inputs where they are: no copy.
            bool direct = false;
            int r0 = issue_step_ml(c, static_cast<const char *>(dev[0]),
                                   static_cast<const char *>(dev[1]),
                                   static_cast<const char *>(dev[2]),
                                   static_cast<char *>(const_cast<void *>(dev[3])), seq_lens, s,
                                   nullptr, &direct, nullptr, true);
            if (r0 != MLKV_OK || direct)
                return r0;
            // One multi-layer launch: a single copy of every input right before it.
            mlkv::StageParams all{};
            all.n = 3;
            all.src[0] = dev[0]; all.dst[0] = dq; all.bytes[0] = qo_bytes;
            all.src[1] = dev[1]; all.dst[1] = dk; all.bytes[1] = kv_bytes;
            all.src[2] = dev[2]; all.dst[2] = dv; all.bytes[2] = kv_bytes;
            bool done = false;
            const int rc = issue_step_ml(c, dq, dk, dv,
                                         static_cast<char *>(const_cast<void *>(dev[3])), seq_lens,
                                         s, nullptr, &done, &all);
            if (rc != MLKV_OK || done)
                return rc;
            // Per-layer launches: layer 0's queries and the new tokens first; the other layers'
            // queries on a side branch while layer 0 runs (joined before layer 1).
            const size_t q1 = qo_bytes / c->l;   // one layer
            const bool split = c->l > 1;
            mlkv::StageParams a{};
            a.n = 3;
            a.src[0] = dev[0]; a.dst[0] = dq; a.bytes[0] = split ? q1 : qo_bytes;
            a.src[1] = dev[1]; a.dst[1] = dk; a.bytes[1] = kv_bytes;
            a.src[2] = dev[2]; a.dst[2] = dv; a.bytes[2] = kv_bytes;
            cudaError_t err = cudaSuccess;
            if (split) {
                err = cudaEventRecord(c->ev[0], s);
                if (err == cudaSuccess)
                    err = cudaStreamWaitEvent(c->side, c->ev[0], 0);
                mlkv::StageParams b{};
                b.n = 1;
                b.src[0] = static_cast<const char *>(dev[0]) + q1; b.dst[0] = dq + q1;
                b.bytes[0] = qo_bytes - q1;
                if (err == cudaSuccess)
                    err = mlkv::launch_stage_copy(b, c->side);
                if (err == cudaSuccess)
                    err = cudaEventRecord(c->ev[1], c->side);
            }
            if (err == cudaSuccess)
                err = mlkv::launch_stage_copy(a, s);
            if (err != cudaSuccess)
                return fail_cuda(err, "copy-in of the step's inputs");
            // The layers write their outputs straight into the page-locked buffer: every store of a
            // decode output is a plain global store, which reaches host memory through its mapped
            // address as well as device memory.
            return issue_step(c, dq, dk, dv, static_cast<char *>(const_cast<void *>(dev[3])),
                              seq_lens, s, split ? c->ev[1] : nullptr, nullptr);
        }
        cudaError_t err = cudaMemcpyAsync(dq, Q, qo_bytes, cudaMemcpyHostToDevice, s);
        if (err == cudaSuccess)
            err = cudaMemcpyAsync(dk, K, kv_bytes, cudaMemcpyHostToDevice, s);
        if (err == cudaSuccess)
            err = cudaMemcpyAsync(dv, V, kv_bytes, cudaMemcpyHostToDevice, s);
        if (err != cudaSuccess)
            return fail_cuda(err, "host-to-device copy of the step's inputs");
        int r = issue_step(c, dq, dk, dv, dout, seq_lens, s);
        if (r != MLKV_OK)
            return r;
        err = cudaMemcpyAsync(out, dout, qo_bytes, cudaMemcpyDeviceToHost, s);
        if (err != cudaSuccess)
            return fail_cuda(err, "device-to-host copy of the step's outputs");
        return MLKV_OK;
    };
    if (mapped && c->step_graph == 2) {
        cudaStreamCaptureStatus cap0 = cudaStreamCaptureStatusNone;
        if ((e = cudaStreamIsCapturing(stream, &cap0)) != cudaSuccess)
            return fail_cuda(e, "cudaStreamIsCapturing");
        if (cap0 == cudaStreamCaptureStatusNone) {
            // The fused form, reading the inputs where they are, issued directly.
            bool direct = false;
            rc = issue_step_ml(c, static_cast<const char *>(dev[0]),
                               static_cast<const char *>(dev[1]),
                               static_cast<const char *>(dev[2]),
                               static_cast<char *>(const_cast<void *>(dev[3])), seq_lens, stream,
                               nullptr, &direct, nullptr, true);
            if (rc != MLKV_OK || direct)
                return rc;
            // One multi-layer launch: its input copy and the launch, issued directly.
            mlkv::StageParams all{};
            all.n = 3;
            all.src[0] = dev[0]; all.dst[0] = dq; all.bytes[0] = qo_bytes;
            all.src[1] = dev[1]; all.dst[1] = dk; all.bytes[1] = kv_bytes;
            all.src[2] = dev[2]; all.dst[2] = dv; all.bytes[2] = kv_bytes;
            bool done = false;
            rc = issue_step_ml(c, dq, dk, dv, static_cast<char *>(const_cast<void *>(dev[3])),
                               seq_lens, stream, nullptr, &done, &all);
            if (rc != MLKV_OK || done)
                return rc;
        }
    }
    // Only page-locked host memory can be recorded into a graph; anything else runs directly.
    bool pinned = c->step_graph != 0;
    for (const void *ptr : {Q, K, V, static_cast<const void *>(out)}) {
        cudaPointerAttributes at;
        if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess || at.type != cudaMemoryTypeHost) {
            cudaGetLastError();
            pinned = false;
        }
    }
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if ((e = cudaStreamIsCapturing(stream, &cap)) != cudaSuccess)
        return fail_cuda(e, "cudaStreamIsCapturing");
    if (!pinned || cap != cudaStreamCaptureStatusNone)
        return issue(stream);
    return record_or_replay(c, key, c->host_key, c->host_pending, c->host_exec, stream, issue);
}

int mlkv_load_prefix(mlkv_cache_t c, int layer, const void *K, const void *V, int len,
                     void *cuda_stream)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (layer < 0 || layer >= c->l)
        return fail(MLKV_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, c->l);
    if (c->owner[layer] != layer)
        return MLKV_OK;
    if (len < 0 || len > c->max_seq)
        return fail(MLKV_ERR_RANGE, "prefix length %d outside [0, %d]", len, c->max_seq);
    if (len == 0)
        return MLKV_OK;
    if (K == nullptr || V == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "K and V must be non-NULL");
    DeviceGuard guard(c->device);
    const size_t row = static_cast<size_t>(len) * c->d * 2;
    const size_t pitch = static_cast<size_t>(c->max_seq) * c->d * 2;
    const size_t slot_bytes = c->cache_bytes / c->m;
    char *base = static_cast<char *>(c->cache) + slot_bytes * c->slot[layer];
    const size_t rows = static_cast<size_t>(c->b) * c->g;
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    cudaError_t e = cudaMemcpy2DAsync(base, pitch, K, row, row, rows, cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemcpy2DAsync(base + slot_bytes / 2, pitch, V, row, row, rows,
                              cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess)
        return fail_cuda(e, "prefix copy");
    return MLKV_OK;
}

int mlkv_prefill(mlkv_cache_t c, int layer, const void *Q, const void *K, const void *V, void *out,
                 const int *prompt_lens, int s_max, void *cuda_stream)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (layer < 0 || layer >= c->l)
        return fail(MLKV_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, c->l);
    if (s_max < 1 || s_max > c->max_seq)
        return fail(MLKV_ERR_RANGE, "s_max %d outside [1, %d]", s_max, c->max_seq);
    if (Q == nullptr || out == nullptr || !aligned16(Q) || !aligned16(out))
        return fail(MLKV_ERR_INVALID_ARG, "Q and out must be non-NULL and 16-byte aligned");
    if (prompt_lens == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "prompt_lens must be non-NULL");
    if (c->h > mlkv::kPrefillMaxHeads || s_max > mlkv::kPrefillMaxBlocks * 128)
        return fail(MLKV_ERR_UNSUPPORTED, "prefill handles at most %d query heads and %d positions",
                    mlkv::kPrefillMaxHeads, mlkv::kPrefillMaxBlocks * 128);
    int max_len = 0;
    for (int beta = 0; beta < c->b; ++beta) {
        if (prompt_lens[beta] < 1 || prompt_lens[beta] > s_max)
            return fail(MLKV_ERR_RANGE, "prompt length %d of sequence %d outside [1, %d]",
                        prompt_lens[beta], beta, s_max);
        max_len = std::max(max_len, prompt_lens[beta]);
    }
    const size_t qbytes = static_cast<size_t>(c->b) * s_max * c->h * c->d * 2;
    const char *qs = static_cast<const char *>(Q);
    const char *os = static_cast<const char *>(out);
    if (os < qs + qbytes && qs < os + qbytes)
        return fail(MLKV_ERR_INVALID_ARG, "out overlaps Q");
    const bool owner = c->owner[layer] == layer;
    if (owner && (K == nullptr || V == nullptr || !aligned16(K) || !aligned16(V)))
        return fail(MLKV_ERR_INVALID_ARG, "K and V must be non-NULL and 16-byte aligned");
    DeviceGuard guard(c->device);
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    // Sec. 3: only an owner layer stores K/V -- the prompt's, at positions [0, s_max).
    if (owner) {
        int rc = mlkv_load_prefix(c, layer, K, V, s_max, cuda_stream);
        if (rc != MLKV_OK)
            return rc;
    }
    cudaError_t e;
    if (!c->prefill_ready) {
        if ((e = mlkv::prepare_prefill(c->d)) != cudaSuccess)
            return fail_cuda(e, "cudaFuncSetAttribute(prefill)");
        c->prefill_ready = 1;
    }
    // The queries, position-major [b][s_max][h][d]: boxes of 64 channels x 1 head x 128 positions.
    static EncodeTiledFn encode = driver_entry<EncodeTiledFn>("cuTensorMapEncodeTiled");
    if (encode == nullptr)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
    CUtensorMap tmap_q;
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(c->d), static_cast<cuuint64_t>(c->h),
                                static_cast<cuuint64_t>(s_max), static_cast<cuuint64_t>(c->b)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(c->d) * 2,
                                   static_cast<cuuint64_t>(c->h) * c->d * 2,
                                   static_cast<cuuint64_t>(s_max) * c->h * c->d * 2};
    const cuuint32_t box[4] = {64u, 1u, 128u, 1u};
    const cuuint32_t estr[4] = {1u, 1u, 1u, 1u};
    CUresult r = encode(&tmap_q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(Q), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(MLKV_ERR_CUDA, "cuTensorMapEncodeTiled(Q) failed (CUresult %d)",
                    static_cast<int>(r));
    // The cache, with boxes of 128 positions (the map of the 128-position decode variant).
    const CUtensorMap *tmap_kv = nullptr;
    for (auto &v : c->variants)
        if (v.v->tile_tokens == 128)
            tmap_kv = &v.tmap;
    if (tmap_kv == nullptr)
        return fail(MLKV_ERR_UNSUPPORTED, "no 128-position cache map for d=%d", c->d);

    static thread_local mlkv::PrefillParams p;
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.err = c->err;
    p.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c->d)));
    p.b = c->b;
    p.h = c->h;
    p.g = c->g;
    p.G = c->G;
    p.s_max = s_max;
    p.slot = c->slot[layer];
    p.fused_L = p.fused_L1 = 0;
    for (int beta = 0; beta < c->b; ++beta)
        p.prompt_len[beta] = prompt_lens[beta];
    // Work units, those that see the most keys first.  head_dim 64: one query block of one head
    // per CTA (two CTAs per SM).  head_dim 128: two heads of a group at the same block when the
    // group size is even, else the blocks 2p and 2p+1 of one head (the unit of block 2p+1).
    const bool one_tile = c->d == 64;
    p.head_pairs = (!one_tile && c->G % 2 == 0) ? 1 : 0;
    const int sels = p.head_pairs ? c->h / 2 : c->h;
    const int max_blocks = (max_len + 127) / 128;
    int n = 0;
    for (int qb = max_blocks - 1; qb >= 0; --qb) {
        for (int beta = 0; beta < c->b; ++beta) {
            const int nb = (prompt_lens[beta] + 127) / 128;
            if (qb >= nb || (!one_tile && !p.head_pairs && qb % 2 == 0 && qb != nb - 1))
                continue;
            for (int sel = 0; sel < sels; ++sel) {
                p.units[n] = static_cast<uint32_t>(beta) | (static_cast<uint32_t>(qb) << 10) |
                             (static_cast<uint32_t>(sel) << 24);
                if (++n == mlkv::kPrefillMaxUnits) {
                    p.n_units = n;
                    if ((e = mlkv::launch_prefill(c->d, &tmap_q, tmap_kv, p, stream)) !=
                        cudaSuccess)
                        return fail_cuda(e, "prefill launch");
                    n = 0;
                }
            }
        }
    }
    if (n > 0) {
        p.n_units = n;
        if ((e = mlkv::launch_prefill(c->d, &tmap_q, tmap_kv, p, stream)) != cudaSuccess)
            return fail_cuda(e, "prefill launch");
    }
    return MLKV_OK;
}

int mlkv_decode_block_fused(mlkv_cache_t c, int owner_layer, const void *Q, void *out,
                            const int *seq_lens, void *cuda_stream)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (owner_layer < 0 || owner_layer >= c->l || c->owner[owner_layer] != owner_layer)
        return fail(MLKV_ERR_INVALID_ARG, "layer %d is not an owner layer", owner_layer);
    if (Q == nullptr || out == nullptr || !aligned16(Q) || !aligned16(out))
        return fail(MLKV_ERR_INVALID_ARG, "Q and out must be non-NULL and 16-byte aligned");
    if (seq_lens == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "seq_lens must be non-NULL");
    int L = 0;
    for (int n = 0; n < c->l; ++n)
        L += c->owner[n] == owner_layer;
    // Rows of one KV head: G heads in each of the block's L layers, in at most two 128-row tiles
    // of whole layers.
    const int L1 = 128 / c->G;
    if (L > 2 * L1)
        return fail(MLKV_ERR_UNSUPPORTED,
                    "%d layers x %d heads per KV head exceed two tiles of 128 query rows", L, c->G);
    if (c->h > mlkv::kPrefillMaxHeads || c->g > 255)
        return fail(MLKV_ERR_UNSUPPORTED, "fused decode handles at most 255 KV heads");
    for (int beta = 0; beta < c->b; ++beta)
        if (seq_lens[beta] < 1 || seq_lens[beta] > c->max_seq)
            return fail(MLKV_ERR_RANGE, "sequence length %d of sequence %d outside [1, %d]",
                        seq_lens[beta], beta, c->max_seq);
    const size_t qbytes = static_cast<size_t>(L) * c->b * c->h * c->d * 2;
    const char *qs = static_cast<const char *>(Q);
    const char *os = static_cast<const char *>(out);
    if (os < qs + qbytes && qs < os + qbytes)
        return fail(MLKV_ERR_INVALID_ARG, "out overlaps Q");
    DeviceGuard guard(c->device);
    int launches = 0;
    return fused_issue(c, Q, out, L, L, 1, c->slot[owner_layer], seq_lens,
                       static_cast<cudaStream_t>(cuda_stream), &launches);
}

int mlkv_merge_kv_weights(const int *layer_owner, int n_layers, int n_q_heads, int n_kv_heads,
                          int64_t row_elems, const void *W, void *W_merged, void *cuda_stream)
{
    if (layer_owner == nullptr || W == nullptr || W_merged == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "layer_owner, W and W_merged must be non-NULL");
    if (n_layers < 1 || n_q_heads < 1 || n_kv_heads < 1)
        return fail(MLKV_ERR_INVALID_ARG, "sizes must be positive (l=%d h=%d g=%d)", n_layers,
                    n_q_heads, n_kv_heads);
    if (n_layers > mlkv::kMergeMaxLayers)
        return fail(MLKV_ERR_UNSUPPORTED, "%d layers exceed %d", n_layers, mlkv::kMergeMaxLayers);
    if (row_elems < 8 || row_elems % 8 != 0 || !aligned16(W) || !aligned16(W_merged))
        return fail(MLKV_ERR_INVALID_ARG,
                    "row_elems (%lld) must be a positive multiple of 8 and W, W_merged 16-byte "
                    "aligned", static_cast<long long>(row_elems));
    if (n_kv_heads > n_q_heads || n_q_heads % n_kv_heads != 0)
        return fail(MLKV_ERR_MAP, "n_kv_heads %d must divide n_q_heads %d", n_kv_heads, n_q_heads);
    static thread_local mlkv::MergeParams p;
    int m = 0;
    for (int n = 0; n < n_layers; ++n) {
        const int o = layer_owner[n];
        if (o < 0 || o > n || layer_owner[o] != o)
            return fail(MLKV_ERR_MAP, "layer_owner[%d] = %d is not a layer <= %d that owns itself",
                        n, o, n);
        if (o == n)
            ++m;
    }
    if (static_cast<long long>(m) * n_kv_heads > 65535)
        return fail(MLKV_ERR_UNSUPPORTED, "%d owners x %d KV heads exceed 65535 merged heads", m,
                    n_kv_heads);
    // Sec. 4.2: the members of owner o are the layers of its block, in layer order.
    int k = 0, sidx = 0;
    for (int o = 0; o < n_layers; ++o) {
        if (layer_owner[o] != o)
            continue;
        p.slot_begin[sidx++] = k;
        for (int n = o; n < n_layers; ++n)
            if (layer_owner[n] == o)
                p.member[k++] = n;
    }
    p.slot_begin[sidx] = k;
    const size_t in_bytes = static_cast<size_t>(n_layers) * n_q_heads * row_elems * 2;
    const size_t out_bytes = static_cast<size_t>(m) * n_kv_heads * row_elems * 2;
    const char *wi = static_cast<const char *>(W);
    const char *wo = static_cast<const char *>(W_merged);
    if (wo < wi + in_bytes && wi < wo + out_bytes)
        return fail(MLKV_ERR_INVALID_ARG, "W_merged overlaps W");
    p.W = static_cast<const __nv_bfloat16 *>(W);
    p.out = static_cast<__nv_bfloat16 *>(W_merged);
    p.row = row_elems;
    p.h = n_q_heads;
    p.g = n_kv_heads;
    p.G = n_q_heads / n_kv_heads;
    cudaError_t e = mlkv::launch_merge(p, m, static_cast<cudaStream_t>(cuda_stream));
    if (e != cudaSuccess)
        return fail_cuda(e, "merge launch");
    return MLKV_OK;
}

int64_t mlkv_cache_bytes(mlkv_cache_t c)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    return static_cast<int64_t>(c->cache_bytes);
}

int mlkv_num_slots(mlkv_cache_t c)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    return c->m;
}

int mlkv_owner_slot(mlkv_cache_t c, int layer, int *owner, int *slot)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (layer < 0 || layer >= c->l)
        return fail(MLKV_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, c->l);
    if (owner) *owner = c->owner[layer];
    if (slot) *slot = c->slot[layer];
    return MLKV_OK;
}

int mlkv_kv_ptr(mlkv_cache_t c, int slot, void **k_base, void **v_base, int64_t strides[4])
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    if (slot < 0 || slot >= c->m)
        return fail(MLKV_ERR_INVALID_ARG, "slot %d outside [0, %d)", slot, c->m);
    const size_t slot_bytes = c->cache_bytes / c->m;
    char *base = static_cast<char *>(c->cache) + slot_bytes * slot;
    if (k_base) *k_base = base;
    if (v_base) *v_base = base + slot_bytes / 2;
    if (strides) {
        strides[3] = 1;
        strides[2] = c->d;
        strides[1] = static_cast<int64_t>(c->max_seq) * c->d;
        strides[0] = static_cast<int64_t>(c->g) * c->max_seq * c->d;
    }
    return MLKV_OK;
}

int mlkv_set_option(mlkv_cache_t c, const char *key, int64_t value)
{
    if (c == nullptr || key == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null argument");
    if (std::strcmp(key, "tile_tokens") == 0) {
        if (value != 0 && mlkv::find_decode_variant(c->d, static_cast<int>(value)) == nullptr)
            return fail(MLKV_ERR_INVALID_ARG, "tile_tokens %lld not built for d=%d",
                        static_cast<long long>(value), c->d);
        c->tile_tokens = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "grid") == 0) {
        if (value < 0 || value > c->max_ctas)
            return fail(MLKV_ERR_INVALID_ARG, "grid %lld outside [0, %d]",
                        static_cast<long long>(value), c->max_ctas);
        c->grid = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_persist") == 0) {
        if (value != 0 && value != 1)
            return fail(MLKV_ERR_INVALID_ARG, "l2_persist must be 0 or 1");
        if (value == c->l2_persist)
            return MLKV_OK;
        DeviceGuard guard(c->device);
        cudaError_t e;
        if (value == 1) {
            // Reserve the largest persisting-L2 set-aside the device allows for this process's
            // context (a per-context limit that ends with the context; no device setting changes).
            int max_persist = 0;
            e = cudaDeviceGetAttribute(&max_persist, cudaDevAttrMaxPersistingL2CacheSize, c->device);
            if (e != cudaSuccess)
                return fail_cuda(e, "cudaDeviceGetAttribute(MaxPersistingL2CacheSize)");
            if (max_persist <= 0 || c->window_max <= 0)
                return fail(MLKV_ERR_UNSUPPORTED, "the device has no persisting L2 set-aside");
            size_t prev = 0, now = 0;
            if ((e = cudaDeviceGetLimit(&prev, cudaLimitPersistingL2CacheSize)) != cudaSuccess ||
                (e = cudaDeviceSetLimit(cudaLimitPersistingL2CacheSize,
                                        static_cast<size_t>(max_persist))) != cudaSuccess ||
                (e = cudaDeviceGetLimit(&now, cudaLimitPersistingL2CacheSize)) != cudaSuccess)
                return fail_cuda(e, "cudaLimitPersistingL2CacheSize");
            c->persist_prev = prev;
            c->persist_bytes = now;
        } else {
            // Lines still marked persisting go back to normal; the earlier set-aside returns.
            if ((e = cudaCtxResetPersistingL2Cache()) != cudaSuccess ||
                (e = cudaDeviceSetLimit(cudaLimitPersistingL2CacheSize, c->persist_prev)) !=
                    cudaSuccess)
                return fail_cuda(e, "restoring the persisting L2 set-aside");
            c->persist_bytes = 0;
        }
        c->l2_persist = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_prefetch") == 0) {
        if (value != 0 && value != 1)
            return fail(MLKV_ERR_INVALID_ARG, "l2_prefetch must be 0 or 1");
        c->l2_prefetch = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_kernel") == 0) {
        if (value != 0 && value != 1)
            return fail(MLKV_ERR_INVALID_ARG, "step_kernel must be 0 or 1");
        c->step_kernel = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_fused") == 0) {
        if (value < 0 || value > 2)
            return fail(MLKV_ERR_INVALID_ARG, "step_fused must be 0, 1 or 2");
        c->step_fused = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "fused_deep") == 0) {
        if (value != 0 && value != 1)
            return fail(MLKV_ERR_INVALID_ARG, "fused_deep must be 0 or 1");
        c->fused_deep = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "fused_kc") == 0) {
        if (value < 0 || value > (1 << 20))
            return fail(MLKV_ERR_INVALID_ARG, "fused_kc must be in [0, 2^20]");
        c->fused_kc = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "cluster") == 0) {
        if (value != 0 && value != 1 && value != 2 && value != 4)
            return fail(MLKV_ERR_INVALID_ARG, "cluster must be 0, 1, 2 or 4");
        c->cluster = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "pdl") == 0) {
        if (value != 0 && value != 1)
            return fail(MLKV_ERR_INVALID_ARG, "pdl must be 0 or 1");
        c->pdl = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "early_fetch") == 0) {
        if (value < 0 || value > 2)
            return fail(MLKV_ERR_INVALID_ARG, "early_fetch must be 0, 1 or 2");
        c->early_fetch = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_graph") == 0) {
        if (value < 0 || value > 2)
            return fail(MLKV_ERR_INVALID_ARG, "step_graph must be 0, 1 or 2");
        c->step_graph = static_cast<int>(value);
        return MLKV_OK;
    }
    if (std::strcmp(key, "tc") == 0) {
        if (value != 0 && value != 1)
            return fail(MLKV_ERR_INVALID_ARG, "tc must be 0 or 1");
        c->tc = static_cast<int>(value);
        return MLKV_OK;
    }
    return fail(MLKV_ERR_INVALID_ARG, "unknown option '%s'", key);
}

int mlkv_get_option(mlkv_cache_t c, const char *key, int64_t *value)
{
    if (c == nullptr || key == nullptr || value == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null argument");
    if (std::strcmp(key, "tile_tokens") == 0) {
        *value = c->tile_tokens;
        return MLKV_OK;
    }
    if (std::strcmp(key, "grid") == 0) {
        *value = c->grid;
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_persist") == 0) {
        *value = c->l2_persist;
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_persist_bytes") == 0) {
        *value = static_cast<int64_t>(c->persist_bytes);
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_window_max") == 0) {
        *value = c->window_max;
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_prefetch") == 0) {
        *value = c->l2_prefetch;
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_kernel") == 0) {
        *value = c->step_kernel;
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_fused") == 0) {
        *value = c->step_fused;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_step_fused") == 0) {
        *value = c->last_step_fused;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_step_launches") == 0) {
        *value = c->last_step_launches;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_fused_kc") == 0) {
        *value = c->last_fused_kc;
        return MLKV_OK;
    }
    if (std::strcmp(key, "fused_kc") == 0) {
        *value = c->fused_kc;
        return MLKV_OK;
    }
    if (std::strcmp(key, "fused_deep") == 0) {
        *value = c->fused_deep;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_step_kernel") == 0) {
        *value = c->last_step_kernel;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_seg_major") == 0) {
        *value = c->last_seg_major;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_l2_prefetch") == 0) {
        *value = c->last_l2_prefetch;
        return MLKV_OK;
    }
    if (std::strcmp(key, "cluster") == 0) {
        *value = c->cluster;
        return MLKV_OK;
    }
    if (std::strcmp(key, "pdl") == 0) {
        *value = c->pdl;
        return MLKV_OK;
    }
    if (std::strcmp(key, "early_fetch") == 0) {
        *value = c->early_fetch;
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_graph") == 0) {
        *value = c->step_graph;
        return MLKV_OK;
    }
    if (std::strcmp(key, "tc") == 0) {
        *value = c->tc;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_tc") == 0) {
        *value = c->last_tc;
        return MLKV_OK;
    }
    if (std::strcmp(key, "step_graph_replays") == 0) {
        *value = c->step_graph_replays;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_grid") == 0) {
        *value = c->last_grid;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_tile_tokens") == 0) {
        *value = c->last_tile;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_cluster_k") == 0) {
        *value = c->last_cluster_k;
        return MLKV_OK;
    }
    if (std::strcmp(key, "last_deferred_merge") == 0) {
        *value = c->last_deferred;
        return MLKV_OK;
    }
    if (std::strcmp(key, "max_grid") == 0) {
        *value = c->max_ctas;
        return MLKV_OK;
    }
    if (std::strcmp(key, "sm_count") == 0) {
        *value = c->sm_count;
        return MLKV_OK;
    }
    if (std::strcmp(key, "l2_bytes") == 0) {
        *value = c->l2_bytes;
        return MLKV_OK;
    }
    if (std::strcmp(key, "ctas_per_sm") == 0) {
        mlkv_cache::Variant *var = pick_variant(c);
        *value = var ? var->ctas_per_sm : 0;
        return MLKV_OK;
    }
    return fail(MLKV_ERR_INVALID_ARG, "unknown option '%s'", key);
}

int mlkv_sync_status(mlkv_cache_t c)
{
    if (c == nullptr)
        return fail(MLKV_ERR_INVALID_ARG, "null cache handle");
    DeviceGuard guard(c->device);
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess)
        return fail_cuda(e, "cudaDeviceSynchronize");
    int word = 0;
    e = cudaMemcpy(&word, c->err, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return fail_cuda(e, "reading the device error word");
    if (word != 0) {
        // A kernel stopped early: clear the word and the merge counters it may have left behind.
        cudaMemset(c->err, 0, sizeof(int));
        cudaMemset(c->counters, 0, static_cast<size_t>(c->b) * c->g * sizeof(unsigned));
        cudaDeviceSynchronize();
        return fail(MLKV_ERR_DEVICE, "a kernel reported device error bits 0x%x", word);
    }
    return MLKV_OK;
}

}  // extern "C"
