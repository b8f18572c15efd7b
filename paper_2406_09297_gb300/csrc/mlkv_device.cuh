// Device-side building blocks shared by the decode kernels of libmlkv (mlkv_kernels.cu,
// mlkv_decode_tc.cu): PTX wrappers (mbarrier, TMA, bulk copies, cluster and grid-dependency
// control), the tile walk over (sequence, KV head) segments and the epilogue that turns a finished
// piece into the output or a partial record.  Internal; not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mlkv_internal.h"

namespace mlkv {
namespace {

constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// ------------------------------------------------------------------------------------------------
// PTX wrappers
// ------------------------------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}

// Non-blocking: whether the phase of the given parity has completed.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}

// Waits for the phase of the given parity to complete; false after kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        for (int i = 0; i < 32; ++i)
            if (mbar_try_wait(bar, parity))
                return true;
        if (global_timer_ns() - t0 > kWaitLimitNs)
            return false;
    }
}

__device__ __forceinline__ void fence_barrier_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Orders this thread's generic-proxy shared-memory writes before later async-proxy (TMA) ones.
__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint32_t bar,
                                            int x, int y, int z)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z)
        : "memory");
}

// Plain bulk copy global -> this CTA's shared memory, completing `bytes` on the mbarrier (both
// addresses 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes,
                                          uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap *map)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                              uint32_t &r2, uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D = A(16x16, row) * B(16x8, col) + D, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1)
{
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 2^x with the SFU instruction (2^-inf = 0).
__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float fast_rcp(float x)
{
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float fast_log2(float x)
{
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <int NCW>
__device__ __forceinline__ void consumer_bar_sync()
{
    asm volatile("bar.sync 1, %0;" ::"n"(NCW * 32) : "memory");
}

// Programmatic dependent launch: wait until the previous kernel of the stream has completed and
// its memory is visible; allow the next kernel of the stream to start its prologue.
// Bulk prefetch of [src, src + bytes) into L2 (src 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ void grid_dependency_wait()
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

__device__ __forceinline__ void grid_dependents_launch()
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// ------------------------------------------------------------------------------------------------
// tile walk: flattened tile index -> (beta, j, tile within segment)
// ------------------------------------------------------------------------------------------------

// With one length for every sequence (uniform_len > 0) the walk is arithmetic; otherwise it reads
// the per-sequence tables, which the kernel copies from its parameters into shared memory.
template <int T>
struct TileWalk {
    int beta, j, tt, nt, L, seg_first, layer, item;
    int kk;    // multi-layer launch: index of the current item among the CTA's
    int t0;    // first tile of the current piece's chunk (0 unless segments are chunked)
    int rec;   // multi-layer launch with chunks: the piece's partial-record index

    // Multi-layer launch: the rank of this CTA's k-th item, or -1 past its last: round k of the
    // deal gives CTA c rank k P + c, or k P + P - 1 - c in odd rounds of a snake deal.
    __device__ __forceinline__ static int ml_rank(const DecodeParams &p, int k)
    {
        const int P = static_cast<int>(gridDim.x), c = static_cast<int>(blockIdx.x);
        const int r = k * P + ((p.ml_snake && (k & 1)) ? P - 1 - c : c);
        return r < p.ml_layers * p.b * p.g * p.ml_chunks ? r : -1;
    }

    // Multi-layer launch: index into the sequence order of rank r's sequence.
    __device__ __forceinline__ static int ml_seq_pos(const DecodeParams &p, int r)
    {
        if (p.ml_chunks > 1)
            r /= p.ml_chunks;
        return p.ml_seg_major ? r / (p.g * p.ml_layers) : (r % (p.b * p.g)) / p.g;
    }

    // Multi-layer launch: tiles of chunk c of a segment of nt tiles.
    __device__ __forceinline__ static void ml_chunk(const DecodeParams &p, int nt, int c, int &a,
                                                    int &b)
    {
        a = c * nt / p.ml_chunks;   // chunks <= 1024 and nt <= 2^20: fits in 32 bits
        b = (c + 1) * nt / p.ml_chunks;
    }

    // Multi-layer launch: (layer, beta, j, L) of rank `item` (see DecodeParams).
    __device__ __forceinline__ void set_item(const DecodeParams &p, const int *s_len,
                                             const int *s_start)
    {
        const bool chunked = p.ml_chunks > 1;
        const int base = chunked ? item / p.ml_chunks : item;
        const int chunk = chunked ? item - base * p.ml_chunks : 0;
        int pb;
        if (p.ml_seg_major) {
            const int per_seq = p.g * p.ml_layers;
            pb = base / per_seq;
            const int rem = base - pb * per_seq;
            j = rem / p.ml_layers;
            layer = p.ml_order[rem - j * p.ml_layers];
        } else {
            const int S = p.b * p.g;
            layer = base / S;
            const int seg = base - layer * S;
            pb = seg / p.g;
            j = seg - pb * p.g;
        }
        if (p.uniform_len > 0) {
            beta = pb;
            L = p.uniform_len;
        } else {
            beta = s_start[pb];
            L = s_len[beta];
        }
        // the piece is tiles [t0, nt) of the segment; seg_first stays the local index its tile 0
        // would have, so that the piece is whole exactly when it is the whole segment
        const int nt_seg = (L + T - 1) / T;
        if (chunked) {
            int t1;
            ml_chunk(p, nt_seg, chunk, t0, t1);
            nt = t1;
            rec = ((layer * p.b + beta) * p.g + j) * p.ml_chunks + chunk;
        } else {
            t0 = 0;
            nt = nt_seg;
            rec = 0;
        }
    }

    // `tile`: the flattened tile of a single-layer launch, or the CTA's own tile count in a
    // multi-layer launch (its k-th item is item blockIdx.x + k gridDim.x).
    __device__ __forceinline__ void init(const DecodeParams &p, const int *s_len,
                                         const int *s_start, int tile)
    {
        if (p.ml_layers > 0) {
            // only ever started at the CTA's first tile (tile_lo = 0)
            kk = 0;
            item = ml_rank(p, 0);
            set_item(p, s_len, s_start);
            tt = t0 + tile;
            seg_first = -t0;
            return;
        }
        layer = 0;
        item = 0;
        t0 = 0;
        rec = 0;
        if (p.uniform_len > 0) {
            L = p.uniform_len;
            nt = (L + T - 1) / T;
            const int seg = tile / nt;
            tt = tile - seg * nt;
            beta = seg / p.g;
            j = seg - beta * p.g;
            seg_first = seg * nt;
            return;
        }
        int lo = 0, hi = p.b - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_start[mid] <= tile)
                lo = mid;
            else
                hi = mid - 1;
        }
        beta = lo;
        L = s_len[beta];
        nt = (L + T - 1) / T;
        const int rel = tile - s_start[beta];
        j = rel / nt;
        tt = rel - j * nt;
        seg_first = s_start[beta] + j * nt;
    }

    __device__ __forceinline__ void next(const DecodeParams &p, const int *s_len,
                                         const int *s_start)
    {
        if (++tt < nt)
            return;
        tt = 0;
        if (p.ml_layers > 0) {
            const int local_end = seg_first + nt;   // where the piece just finished ends
            item = ml_rank(p, ++kk);
            if (item >= 0) {
                set_item(p, s_len, s_start);
                tt = t0;
                seg_first = local_end - t0;
            }
            return;
        }
        if (p.uniform_len > 0) {
            seg_first += nt;
            if (++j == p.g) {
                j = 0;
                ++beta;
            }
            return;
        }
        if (++j == p.g) {
            j = 0;
            if (++beta < p.b) {
                L = s_len[beta];
                nt = (L + T - 1) / T;
            }
        }
        seg_first = (beta < p.b) ? s_start[beta] + j * nt : p.num_tiles;
    }
};

// CTA whose contiguous tile run [floor(c*N/P), floor((c+1)*N/P)) contains `tile`.
__device__ __forceinline__ int cta_of_tile(int tile, int N, int P)
{
    return static_cast<int>((static_cast<long long>(tile + 1) * P - 1) / N);
}


// Multi-layer launch with every sequence of one length: CTA `cta` of `P` prefetches into L2 its
// 1/P share of the visible rows (positions [0, L)) of every (slot, K|V, beta, j) row of slots
// 0 .. ml_slots - 1, slot by slot, so that the whole step's K/V streams from HBM at the copy
// engines' rate while the CTAs work.  Shares are 128-byte aligned; chunks of at most 1 MiB.
template <int D>
__device__ __forceinline__ void prefetch_slots_share(const DecodeParams &p, int cta, int P)
{
    const size_t row_bytes = static_cast<size_t>(p.uniform_len) * D * 2;
    const size_t rows = 2ull * p.b * p.g;                  // rows of one slot
    const size_t slot_bytes = rows * row_bytes;
    const size_t pitch = static_cast<size_t>(p.max_seq) * D * 2;
    const uint8_t *base = reinterpret_cast<const uint8_t *>(p.cache);
    for (int s = 0; s < p.ml_slots; ++s) {
        size_t lo = (slot_bytes * cta / P) & ~static_cast<size_t>(127);
        const size_t hi =
            cta + 1 == P ? slot_bytes : (slot_bytes * (cta + 1) / P) & ~static_cast<size_t>(127);
        while (lo < hi) {
            const size_t r = lo / row_bytes;
            const size_t off = lo - r * row_bytes;
            size_t n = min(hi - lo, row_bytes - off);
            n = min(n, static_cast<size_t>(1u << 20));
            bulk_prefetch_l2(base + (static_cast<size_t>(s) * rows + r) * pitch + off,
                             static_cast<uint32_t>(n));
            lo += n;
        }
    }
}

// the TMA 128-byte swizzle: the chunk index within a 128-byte row is XORed with (row mod 8).
template <int T>
__device__ __forceinline__ uint32_t swz(int row, int chunk)
{
    const int sub = chunk >> 3;
    const int c = chunk & 7;
    return static_cast<uint32_t>(sub * T * 128 + row * 128 + ((c ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Every thread of a cluster launch arrives once, right after set-up, and waits once, late: before
// its first access to another CTA's shared memory and before it exits.
// Relaxed: what the partners need from this arrival are the barrier initialisations, which
// fence.mbarrier_init.release.cluster has already published.
__device__ __forceinline__ void cluster_arrive()
{
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}

__device__ __forceinline__ void cluster_wait()
{
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Address, in the cluster's shared window, of this CTA's shared address `a` in CTA `rank`.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t a, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
    return r;
}

// Asynchronous store into another CTA's shared memory that completes `bytes` of the transaction
// count of that CTA's mbarrier `mbar` (both addresses in the cluster window).
__device__ __forceinline__ void st_async_v2(uint32_t a, float x, float y, uint32_t mbar)
{
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(a),
        "f"(x), "f"(y), "r"(mbar)
        : "memory");
}

__device__ __forceinline__ void st_async_f32(uint32_t a, float x, uint32_t mbar)
{
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.f32 [%0], %1, [%2];" ::"r"(a),
                 "f"(x), "r"(mbar)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity)
{
    if (mbar_try_wait_cluster(bar, parity))
        return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        for (int i = 0; i < 32; ++i)
            if (mbar_try_wait_cluster(bar, parity))
                return true;
        if (global_timer_ns() - t0 > kWaitLimitNs)
            return false;
    }
}

__device__ __forceinline__ unsigned atomic_add_acq_rel_gpu(unsigned *addr, unsigned v)
{
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;"
                 : "=r"(old)
                 : "l"(addr), "r"(v)
                 : "memory");
    return old;
}

enum : int { kMetaBeta = 0, kMetaJ, kMetaSeg, kMetaWhole, kMetaFirst, kMetaLast, kMetaStop,
             kMetaLayer };

// ------------------------------------------------------------------------------------------------
// epilogue warp: output, partials and the cross-CTA merge of finished pieces
// ------------------------------------------------------------------------------------------------

// One piece's result (normalised o, lse, metadata) sits in a shared-memory slot.  A whole segment
// goes straight to `out`.  Otherwise the slot becomes partial record seg + cta; the counter of the
// segment (acquire-release) tells the CTA that finished it last, which merges all its records:
//   o = sum_c 2^(lse_c - M) o_c / sum_c 2^(lse_c - M),  M = max_c lse_c.
template <int D>
__device__ __forceinline__ void epilogue_piece(const DecodeParams &p, const float *ro,
                                               const float *rlse, const int *meta, float *s_w,
                                               int cap, int lane, int cta)
{
    const int G = p.G;
    const int beta = meta[kMetaBeta], j = meta[kMetaJ], seg = meta[kMetaSeg];
    __nv_bfloat16 *ob = p.out + static_cast<size_t>(meta[kMetaLayer]) * p.ml_q_stride +
                        (static_cast<size_t>(beta) * p.h + static_cast<size_t>(j) * G) * D;
    if (meta[kMetaWhole]) {
        for (int i = lane * 4; i < G * D; i += 128) {
            const float4 v = *reinterpret_cast<const float4 *>(ro + i);
            uint2 w;
            w.x = pack_bf16x2(v.x, v.y);
            w.y = pack_bf16x2(v.z, v.w);
            *reinterpret_cast<uint2 *>(ob + i) = w;
        }
        return;
    }
    // a multi-layer launch's partial record index travels in kMetaFirst (its merge is deferred)
    const size_t piece = p.ml_layers > 0 ? static_cast<size_t>(meta[kMetaFirst])
                                         : static_cast<size_t>(seg + cta);
    float *po = p.part_o + piece * G * D;
    for (int i = lane * 4; i < G * D; i += 128)
        *reinterpret_cast<float4 *>(po + i) = *reinterpret_cast<const float4 *>(ro + i);
    if (lane < G)
        p.part_lse[piece * G + lane] = rlse[lane];
    if (p.deferred_merge)
        return;   // combine_kernel merges this segment after the launch
    __syncwarp();
    const int c_first = meta[kMetaFirst], c_last = meta[kMetaLast];
    unsigned prev = 0;
    if (lane == 0)
        prev = atomic_add_acq_rel_gpu(&p.counters[seg], 1u);
    prev = __shfl_sync(0xffffffffu, prev, 0);
    __syncwarp();
    if (prev != static_cast<unsigned>(c_last - c_first))
        return;
    // This CTA finished the segment last.  Records seg + c_first .. seg + c_last are contiguous.
    const int np = c_last - c_first + 1;
    const size_t rec0 = static_cast<size_t>(seg + c_first);
    const float NEG_INF = -__int_as_float(0x7f800000);
    if (np * G <= cap) {
        for (int i = lane; i < np * G; i += 32)
            s_w[i] = __ldcg(&p.part_lse[rec0 * G + i]);
        __syncwarp();
        for (int r = lane; r < G; r += 32) {
            float mx = NEG_INF;
            for (int k = 0; k < np; ++k)
                mx = fmaxf(mx, s_w[k * G + r]);
            float tot = 0.f;
            for (int k = 0; k < np; ++k) {
                const float w = fast_exp2(s_w[k * G + r] - mx);
                s_w[k * G + r] = w;
                tot += w;
            }
            const float inv = 1.f / tot;
            for (int k = 0; k < np; ++k)
                s_w[k * G + r] *= inv;
        }
        __syncwarp();
        // Each lane owns CH float4 columns of a 128*CH-element chunk; the loads of all its
        // columns for two pieces are in flight together.
        constexpr int CH = 8;
        const float *base = p.part_o + rec0 * G * D;
        for (int c0 = 0; c0 < G * D; c0 += 128 * CH) {
            float4 acc[CH];
#pragma unroll
            for (int u = 0; u < CH; ++u)
                acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int k = 0; k < np; k += 2) {
                float4 v0[CH], v1[CH];
#pragma unroll
                for (int u = 0; u < CH; ++u) {
                    const int i = c0 + u * 128 + lane * 4;
                    const bool in = i < G * D;
                    v0[u] = in ? __ldcg(reinterpret_cast<const float4 *>(
                                     base + static_cast<size_t>(k) * G * D + i))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
                    v1[u] = (in && k + 1 < np)
                                ? __ldcg(reinterpret_cast<const float4 *>(
                                      base + static_cast<size_t>(k + 1) * G * D + i))
                                : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int u = 0; u < CH; ++u) {
                    const int i = c0 + u * 128 + lane * 4;
                    if (i < G * D) {
                        const int row = i / D;
                        const float w0 = s_w[k * G + row];
                        const float w1 = (k + 1 < np) ? s_w[(k + 1) * G + row] : 0.f;
                        acc[u].x += w0 * v0[u].x + w1 * v1[u].x;
                        acc[u].y += w0 * v0[u].y + w1 * v1[u].y;
                        acc[u].z += w0 * v0[u].z + w1 * v1[u].z;
                        acc[u].w += w0 * v0[u].w + w1 * v1[u].w;
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < CH; ++u) {
                const int i = c0 + u * 128 + lane * 4;
                if (i < G * D) {
                    uint2 w2;
                    w2.x = pack_bf16x2(acc[u].x, acc[u].y);
                    w2.y = pack_bf16x2(acc[u].z, acc[u].w);
                    *reinterpret_cast<uint2 *>(ob + i) = w2;
                }
            }
        }
        __syncwarp();
    } else {
        // Very many pieces: the same merge, weights recomputed per element.
        for (int i = lane; i < G * D; i += 32) {
            const int row = i / D;
            float mx = NEG_INF;
            for (int k = 0; k < np; ++k)
                mx = fmaxf(mx, __ldcg(&p.part_lse[(rec0 + k) * G + row]));
            float acc = 0.f, wsum = 0.f;
            for (int k = 0; k < np; ++k) {
                const float w = fast_exp2(__ldcg(&p.part_lse[(rec0 + k) * G + row]) - mx);
                wsum += w;
                acc += w * __ldcg(&p.part_o[(rec0 + k) * G * D + i]);
            }
            ob[i] = __float2bfloat16_rn(acc / wsum);
        }
    }
    if (lane == 0)
        p.counters[seg] = 0u;
}


}  // namespace
}  // namespace mlkv
