// MLKV prefill attention on the 5th-generation tensor cores (tcgen05, tensor memory) for GB300.
//
// Prefill runs a whole prompt through one layer at once: prompt position t of query head i
// attends to positions 0 .. t of KV head j(i) = i / G of the layer's owner slot (causal
// attention, Eqs. 2-3 with the MLKV maps of Eqs. 13-18).  Owner layers first store the prompt's
// K/V in their slot (mlkv_host.cpp); every layer of the block then attends over it.
//
// Work split: one CTA per (sequence, query head, block of 128 prompt positions), longest blocks
// (those near the end of a prompt, which see the most keys) first.  Each CTA walks the key tiles
// 0 .. qb of its block's causal triangle, 128 keys per tile.
//
// Math, per key tile (all MMAs tcgen05.mma kind::f16, bf16 in, fp32 accumulate in TMEM):
//   S = Q K^T       M = 128 queries (A = the query tile, loaded once by TMA, K-major with the
//                   128-byte swizzle), N = 128 keys (B = the K tile as TMA left it), K = head_dim;
//                   double-buffered in TMEM, one query row per TMEM lane.
//   softmax         four warps, one thread per query row: the thread owns its row's 128 scores
//                   (tcgen05.ld), so the online maximum needs no exchange between threads.  The
//                   row's reference maximum is raised only when a score exceeds it by more than
//                   2^8 in the exponent; then the thread rescales its O row in TMEM (after the
//                   previous tile's product has landed).  p = 2^(s log2(e)/sqrt(d) - m) is written
//                   as bf16 to smem in the A-operand layout (K-major, 128-byte swizzle).
//   O += P V        M = 128 queries, N = head_dim (B = the V tile read MN-major), K = 128 keys;
//                   O stays in TMEM for the whole block.
// The diagonal tile masks keys after the query; keys past the prompt's end only meet such
// masked scores, and their V rows are zeroed in smem so that 0 * V stays 0.
//
// Warp roles (192 threads): warps 0-3 softmax and output, warp 4 TMA producer (query tile, then a
// ring of K/V tiles), warp 5 MMA issuer (event-driven: S of the next tile as soon as its K/V and a
// TMEM buffer are ready, P V as soon as a tile's P is written).  Every wait is bounded; on expiry
// the kernel records an error bit, stops, lets its copies and MMAs land and frees its TMEM.
#include "mlkv_device.cuh"
#include "mlkv_tcgen05.cuh"

namespace mlkv {
namespace {

template <int D>
struct PrefillPlan {
    static constexpr int kThreads = 6 * 32;
    static constexpr int kProducer = 4, kMma = 5;
    static constexpr int kSub = D / 64;                   // 64-channel blocks of a row
    static constexpr int kStages = D == 64 ? 4 : 2;
    static constexpr int kTileBytes = 128 * D * 2;        // a Q, K or V tile of 128 rows
    static constexpr int kStageBytes = 2 * kTileBytes;    // K and V
    static constexpr int kPBytes = 128 * 128 * 2;         // P: [2 key blocks][128 rows][64] bf16
    static constexpr int kQ = 0;
    static constexpr int kRing = kQ + kTileBytes;
    static constexpr int kP = kRing + kStages * kStageBytes;   // [2][kPBytes]
    static constexpr int kFlags = kP + 2 * kPBytes;            // int [4], TMEM base at +16
    // u64 barriers: q_full, full[S], empty[S], s_ready[2], s_free[2], p_ready[2], p_free[2],
    // o_ready, fin
    static constexpr int kBars = kFlags + 32;
    static constexpr int kNumBars = 1 + 2 * kStages + 10;
    static constexpr int kBytes = kBars + kNumBars * 8;
    static constexpr int kAlloc = kBytes + 1024;               // base aligned up to 1024
    static constexpr int kTmemCols = 512;                      // S: 2 x 128, O: D
    static constexpr int kColS = 0, kColO = 256;
    static_assert(D == 64 || D == 128, "head_dim 64 or 128");
    static_assert(kRing % 1024 == 0 && kP % 1024 == 0, "swizzled tiles stay 1024-byte aligned");
};

template <int D>
__global__ void __launch_bounds__(PrefillPlan<D>::kThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap tmap_q,
                   const __grid_constant__ CUtensorMap tmap_kv,
                   const __grid_constant__ PrefillParams p)
{
    using PL = PrefillPlan<D>;
    constexpr int ST = PL::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_addr(smem);
    const uint32_t bar_q = sbase + PL::kBars;
    const uint32_t bar_full = bar_q + 8;
    const uint32_t bar_empty = bar_full + 8 * ST;
    const uint32_t bar_s_ready = bar_empty + 8 * ST;   // [2]
    const uint32_t bar_s_free = bar_s_ready + 16;       // [2]
    const uint32_t bar_p_ready = bar_s_free + 16;       // [2]
    const uint32_t bar_p_free = bar_p_ready + 16;       // [2]
    const uint32_t bar_o_ready = bar_p_free + 16;
    const uint32_t bar_fin = bar_o_ready + 8;
    volatile int *flags = reinterpret_cast<volatile int *>(smem + PL::kFlags);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int item = blockIdx.x / p.h;
    const int head = blockIdx.x - item * p.h;
    const int beta = p.item_beta[item];
    const int qb = p.item_qb[item];
    const int S = p.prompt_len[beta];
    const int q0 = qb * 128;
    const int n_kt = qb + 1;                         // key tiles 0 .. qb (causal)
    const int j = head / p.G;                        // Eq. 15
    const int zk = ((p.slot * 2 + 0) * p.b + beta) * p.g + j;
    const int zv = zk + p.b * p.g;

    if (threadIdx.x == 0) {
        mbar_init(bar_q, 1);
        for (int s = 0; s < ST; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
        }
        for (int r = 0; r < 2; ++r) {
            mbar_init(bar_s_ready + 8 * r, 1);
            mbar_init(bar_s_free + 8 * r, 4);
            mbar_init(bar_p_ready + 8 * r, 4);
            mbar_init(bar_p_free + 8 * r, 1);
        }
        mbar_init(bar_o_ready, 1);
        mbar_init(bar_fin, 1);
        flags[0] = 0;
        fence_barrier_init();
    }
    if (threadIdx.x == PL::kProducer * 32) {
        prefetch_tensormap(&tmap_q);
        prefetch_tensormap(&tmap_kv);
    }
    if (warp == PL::kMma) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         sbase + PL::kFlags + 16),
                     "n"(PL::kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + PL::kFlags + 16);
    // The owner's K/V may have just been stored by the previous kernel of the stream.
    grid_dependency_wait();
    grid_dependents_launch();

    if (warp == PL::kProducer) {
        // ------------------------------------ producer ------------------------------------------
        if (lane == 0) {
            mbar_arrive_expect_tx(bar_q, PL::kTileBytes);
#pragma unroll
            for (int sub = 0; sub < PL::kSub; ++sub)
                tma_load_4d(sbase + PL::kQ + sub * 16384, &tmap_q, bar_q, sub * 64, head, q0, beta);
            int kt = 0;
            for (; kt < n_kt; ++kt) {
                const int s = kt % ST;
                if (kt >= ST && !flags[0] &&
                    !mbar_wait(bar_empty + 8 * s, ((kt / ST) & 1) ^ 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitEmpty);
                }
                if (flags[0])
                    break;
                const uint32_t fb = bar_full + 8 * s;
                mbar_arrive_expect_tx(fb, PL::kStageBytes);
                const uint32_t kdst = sbase + PL::kRing + s * PL::kStageBytes;
#pragma unroll
                for (int sub = 0; sub < PL::kSub; ++sub) {
                    tma_load_3d(kdst + sub * 16384, &tmap_kv, fb, sub * 64, kt * 128, zk);
                    tma_load_3d(kdst + PL::kTileBytes + sub * 16384, &tmap_kv, fb, sub * 64,
                                kt * 128, zv);
                }
            }
            // No copy may still be in flight when the CTA exits.
            if (!mbar_wait(bar_q, 0))
                atomicOr(p.err, kErrDrain);
            for (int k = kt > ST ? kt - ST : 0; k < kt; ++k)
                if (!mbar_wait(bar_full + 8 * (k % ST), (k / ST) & 1))
                    atomicOr(p.err, kErrDrain);
        }
        __syncwarp();
    } else if (warp == PL::kMma) {
        // ------------------------------------ MMA issuer ----------------------------------------
        constexpr uint32_t kIdS = umma_idesc(128, 128, 0, 0);
        constexpr uint32_t kIdPV = umma_idesc(128, D, 0, 1);
        int si = 0, pi = 0;
        bool ok = true;
        uint64_t idle_since = 0;
        while (pi < n_kt && ok) {
            int act = 0;   // 1: O += P V of tile pi, 2: S of tile si
            if (lane == 0) {
                if (pi < si && mbar_test_wait(bar_p_ready + 8 * (pi & 1), (pi >> 1) & 1))
                    act = 1;
                else if (si < n_kt && (si > 0 || mbar_test_wait(bar_q, 0)) &&
                         mbar_test_wait(bar_full + 8 * (si % ST), (si / ST) & 1) &&
                         (si < 2 || mbar_test_wait(bar_s_free + 8 * (si & 1), ((si >> 1) & 1) ^ 1)))
                    act = 2;
            }
            act = __shfl_sync(0xffffffffu, act, 0);
            if (act == 0) {
                if (lane == 0) {
                    const uint64_t now = global_timer_ns();
                    if (idle_since == 0)
                        idle_since = now;
                    else if (now - idle_since > kWaitLimitNs)
                        ok = false;
                }
                ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
                if (ok && flags[0])
                    ok = false;
                continue;
            }
            idle_since = 0;
            tmem_fence_after();
            if (act == 2) {
                if (lane == 0) {
                    const uint32_t kt = sbase + PL::kRing + (si % ST) * PL::kStageBytes;
#pragma unroll
                    for (int k = 0; k < D / 16; ++k)
                        umma_f16(tmem + PL::kColS + (si & 1) * 128,
                                 umma_desc(sbase + PL::kQ + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                           1024, kLayoutSw128),
                                 umma_desc(kt + (k >> 2) * 16384 + (k & 3) * 32, 16, 1024,
                                           kLayoutSw128),
                                 kIdS, k > 0 ? 1 : 0);
                    umma_commit(bar_s_ready + 8 * (si & 1));
                }
                __syncwarp();
                ++si;
            } else {
                if (lane == 0) {
                    const uint32_t vt =
                        sbase + PL::kRing + (pi % ST) * PL::kStageBytes + PL::kTileBytes;
                    const uint32_t pt = sbase + PL::kP + (pi & 1) * PL::kPBytes;
#pragma unroll
                    for (int k = 0; k < 8; ++k)
                        umma_f16(tmem + PL::kColO,
                                 umma_desc(pt + (k >> 2) * 16384 + (k & 3) * 32, 16, 1024,
                                           kLayoutSw128),
                                 umma_desc(vt + k * 2048, 16384, 1024, kLayoutSw128), kIdPV,
                                 (pi == 0 && k == 0) ? 0 : 1);
                    umma_commit(bar_empty + 8 * (pi % ST));   // the K/V stage may be refilled
                    umma_commit(bar_p_free + 8 * (pi & 1));   // the P buffer may be rewritten
                    if (pi == n_kt - 1)
                        umma_commit(bar_o_ready);
                }
                __syncwarp();
                ++pi;
            }
        }
        if (!ok) {
            flags[0] = 1;
            if (lane == 0)
                atomicOr(p.err, kErrWaitFull);
        }
        if (lane == 0)
            umma_commit(bar_fin);
        __syncwarp();
        if (!mbar_wait(bar_fin, 0) && lane == 0)
            atomicOr(p.err, kErrDrain);
        __syncwarp();
    } else {
        // ------------------------------------ softmax warps -------------------------------------
        const int r = threadIdx.x;   // query row of the block = TMEM lane
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        const float scale = p.scale_log2;
        const float NEG_INF = -__int_as_float(0x7f800000);
        float m_run = NEG_INF, l_run = 0.f;
        for (int t = 0; t < n_kt; ++t) {
            if (!flags[0] && !mbar_wait(bar_s_ready + 8 * (t & 1), (t >> 1) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
            tmem_fence_after();
            float sv[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c)
                tmem_ld32_nowait(tmem + lane_base + PL::kColS + (t & 1) * 128 + c * 32, sv[c]);
            tmem_wait_ld();
            tmem_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_s_free + 8 * (t & 1));
            const bool diag = (t == qb);
            float mx = NEG_INF;
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                    if (diag && c * 32 + k > r)
                        sv[c][k] = NEG_INF;   // a later position: causal mask
                    mx = fmaxf(mx, sv[c][k]);
                }
            const float m_tile = mx * scale;
            const bool raise = (m_run == NEG_INF) || (m_tile > m_run + 8.f);
            if (__any_sync(0xffffffffu, raise)) {
                const float m_new = raise ? fmaxf(m_run, m_tile) : m_run;
                const float alpha = fast_exp2(m_run - m_new);   // 0 while nothing is summed
                if (t > 0) {
                    // Rescale this row of O once the previous tile's product has landed.
                    const int pt = t - 1;
                    if (!flags[0] && !mbar_wait(bar_p_free + 8 * (pt & 1), (pt >> 1) & 1)) {
                        flags[0] = 1;
                        atomicOr(p.err, kErrWaitFull);
                    }
                    tmem_fence_after();
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        float ov[32];
                        tmem_ld32_nowait(tmem + lane_base + PL::kColO + c * 32, ov);
                        tmem_wait_ld();
#pragma unroll
                        for (int k = 0; k < 32; ++k)
                            ov[k] *= alpha;
                        tmem_st32(tmem + lane_base + PL::kColO + c * 32, ov);
                    }
                    tmem_fence_before();
                }
                l_run *= alpha;
                m_run = m_new;
            }
            // P row, bf16, into the A-operand layout; the row sum takes the same rounding.
            if (t >= 2 && !flags[0] &&
                !mbar_wait(bar_p_free + 8 * (t & 1), ((t >> 1) & 1) ^ 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
            uint8_t *prow = smem + PL::kP + (t & 1) * PL::kPBytes + r * 128;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t w[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float p0 = fast_exp2(fmaf(sv[c][q * 8 + 2 * u], scale, -m_run));
                        const float p1 = fast_exp2(fmaf(sv[c][q * 8 + 2 * u + 1], scale, -m_run));
                        w[u] = pack_bf16x2(p0, p1);
                        l_run += bf16_lo(w[u]) + bf16_hi(w[u]);
                    }
                    const int chunk = c * 4 + q;   // keys 8*chunk .. 8*chunk+7
                    *reinterpret_cast<uint4 *>(prow + (chunk >> 3) * 16384 +
                                               (((chunk & 7) ^ (r & 7)) << 4)) =
                        make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
            if (diag && q0 + r >= S) {
                // Key q0 + r lies past the prompt: its V row may hold anything; zero it.
                uint8_t *vrow = smem + PL::kRing + (t % ST) * PL::kStageBytes + PL::kTileBytes;
#pragma unroll
                for (int c = 0; c < 8 * PL::kSub; ++c)
                    *reinterpret_cast<uint4 *>(vrow + (c >> 3) * 16384 + r * 128 +
                                               (((c & 7) ^ (r & 7)) << 4)) = make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_p_ready + 8 * (t & 1));
        }
        // ---------------- the block's output: o = O / l ----------------
        if (!flags[0] && !mbar_wait(bar_o_ready, 0)) {
            flags[0] = 1;
            atomicOr(p.err, kErrWaitFull);
        }
        tmem_fence_after();
        const float inv = fast_rcp(l_run);
        const bool valid = q0 + r < S;
        __nv_bfloat16 *orow =
            p.out + ((static_cast<size_t>(beta) * p.s_max + (q0 + r)) * p.h + head) * D;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
            float ov[32];
            tmem_ld32_nowait(tmem + lane_base + PL::kColO + c * 32, ov);
            tmem_wait_ld();
            if (valid && !flags[0]) {
#pragma unroll
                for (int k = 0; k < 32; k += 8)
                    *reinterpret_cast<uint4 *>(orow + c * 32 + k) = make_uint4(
                        pack_bf16x2(ov[k] * inv, ov[k + 1] * inv),
                        pack_bf16x2(ov[k + 2] * inv, ov[k + 3] * inv),
                        pack_bf16x2(ov[k + 4] * inv, ov[k + 5] * inv),
                        pack_bf16x2(ov[k + 6] * inv, ov[k + 7] * inv));
            }
        }
        tmem_fence_before();
    }

    __syncthreads();
    if (warp == PL::kMma) {
        tmem_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "n"(PL::kTmemCols)
                     : "memory");
    }
}

template <int D>
const void *prefill_fn()
{
    return reinterpret_cast<const void *>(&prefill_kernel<D>);
}

}  // namespace

size_t prefill_smem_bytes(int head_dim)
{
    return head_dim == 64 ? PrefillPlan<64>::kAlloc : PrefillPlan<128>::kAlloc;
}

cudaError_t prepare_prefill(int head_dim)
{
    return cudaFuncSetAttribute(head_dim == 64 ? prefill_fn<64>() : prefill_fn<128>(),
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(prefill_smem_bytes(head_dim)));
}

cudaError_t launch_prefill(int head_dim, const CUtensorMap *tmap_q, const CUtensorMap *tmap_kv,
                           const PrefillParams &p, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.n_items * p.h));
    cfg.blockDim = dim3(static_cast<unsigned>(head_dim == 64 ? PrefillPlan<64>::kThreads
                                                             : PrefillPlan<128>::kThreads));
    cfg.dynamicSmemBytes = prefill_smem_bytes(head_dim);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void *args[] = {const_cast<CUtensorMap *>(tmap_q), const_cast<CUtensorMap *>(tmap_kv),
                    const_cast<PrefillParams *>(&p)};
    return cudaLaunchKernelExC(&cfg, head_dim == 64 ? prefill_fn<64>() : prefill_fn<128>(),
                               args);
}

}  // namespace mlkv
