// MLKV decode attention on the 5th-generation tensor cores (tcgen05, tensor memory) for GB300.
//
// Same work split, data movement, merges and launch discipline as decode_kernel (mlkv_kernels.cu):
// a persistent stream-K grid over the tiles of all (sequence, KV head) segments, one TMA producer
// warp filling a STAGES-deep ring of K and V tiles (128-byte swizzle), pieces handed to an
// epilogue warp or finished through DSMEM clusters / partial records.  What differs is the math of
// a tile, which is laid out transposed so that positions, not query heads, fill the tensor-core M
// dimension (a group holds at most 16 query heads, a tile 128 or 256 positions):
//
//   S^T[pos][h] = K[pos][:] . Q[h][:]          tcgen05.mma kind::f16, M = 128 positions, N = 16
//                                              heads, A = the K tile as TMA left it (K-major,
//                                              128-byte swizzle), B = the group's queries in smem;
//                                              the accumulator lives in tensor memory (TMEM), one
//                                              position per TMEM lane.
//   softmax                                     four warps, one thread per TMEM lane: each thread
//                                              loads its position's 16 scores (tcgen05.ld), forms
//                                              p = 2^(s * log2(e)/sqrt(d) - m[h]) and writes the
//                                              bf16 row P^T[pos][0..15] to smem.
//   O^T[d][h] += V^T[d][pos] . P^T[pos][h]      tcgen05.mma, M = head_dim, N = 16, K = positions;
//                                              A = the V tile read MN-major, B = P^T; O^T stays
//                                              in TMEM for the whole piece.
//
// The reference maximum m[h] of the online softmax (Eqs. 2-3 computed as in flash attention) is
// shared by the whole CTA, since O^T sums every position of the piece.  It is only raised when a
// score of the tile exceeds it by more than 2^8 in the exponent (one OR-reducing barrier per tile
// tells every thread); then the CTA takes the exact maximum of the tile, rescales O^T in TMEM and
// the per-thread row sums by 2^(m_old - m_new).  Between raises every p is at most 2^8, far from
// any overflow, and the final normalisation o = O / l is exact whatever the reference.
//
// Warp roles (224 threads): warps 0-3 softmax (and the piece epilogue of the CTA's last piece),
// warp 4 TMA producer, warp 5 MMA issuer (allocates and frees TMEM), warp 6 epilogue of earlier
// pieces.  S^T and P^T are double-buffered, so the tensor core computes S^T of tile t+1 and
// O^T += V^T P^T of tile t while the softmax warps work on tile t+1.  All waits are bounded as in
// decode_kernel; on expiry the kernel records an error bit, stops, lets its copies and MMAs land
// and frees its tensor memory before exit.
#include "mlkv_device.cuh"
#include "mlkv_tcgen05.cuh"

namespace mlkv {
namespace {

// Named barrier 1 over the four softmax warps.
__device__ __forceinline__ void soft_bar_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Named barrier 2 over the four softmax warps that also ORs a predicate over them.
__device__ __forceinline__ bool soft_bar_or(bool v)
{
    uint32_t out;
    asm volatile("{\n\t.reg .pred pi, po;\n\tsetp.ne.u32 pi, %1, 0;\n\t"
                 "bar.red.or.pred po, 2, 128, pi;\n\tselp.u32 %0, 1, 0, po;\n\t}"
                 : "=r"(out)
                 : "r"(v ? 1u : 0u)
                 : "memory");
    return out != 0;
}

// ------------------------------------------------------------------------------------------------
// shared-memory plan
// ------------------------------------------------------------------------------------------------

template <int D, int T, int STAGES>
struct TcPlan {
    static constexpr int kSoftWarps = 4;
    static constexpr int kProducer = 4, kMma = 5, kEpilogue = 6;
    static constexpr int kThreads = 7 * 32;
    static constexpr int kSub = D / 64;               // 64-channel column blocks of a row
    static constexpr int kHalves = T / 128;           // 128-position blocks of a tile
    static constexpr int kTileBytes = T * D * 2;      // one K (or V) tile
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kQBytes = 16 * D * 2;        // the group's queries: kSub [16][64] blocks
    static constexpr int kPBytes = T * 32;            // P^T [2][T][8] bf16
    static constexpr int kResO = 16 * D * 4;          // a piece's result: o[16][D] f32
    static constexpr int kResBytes = kResO + 16 * 4 + 32;   // + lse[16] + 8 ints of metadata
    static constexpr int kEpiCap = 64;                // epilogue merge weights (more: recomputed)
    static constexpr int kQ = STAGES * kStageBytes;   // [2][kQBytes]
    static constexpr int kP = kQ + 2 * kQBytes;       // [2][kPBytes]
    static constexpr int kRes = kP + 2 * kPBytes;     // [2][kResBytes]
    static constexpr int kEpiW = kRes + 2 * kResBytes;
    static constexpr int kLRed = kEpiW + kEpiCap * 4; // f32 [4][16] row sums per warp
    static constexpr int kMRed = kLRed + 256;         // f32 [4][16] tile maxima per warp
    static constexpr int kFlags = kMRed + 256;        // int [4], TMEM base at [4]
    // u64 barriers: full[S], empty[S], s_ready[2], s_free[2], p_ready[2], p_free[2], q_ready[2],
    // o_ready, o_free, res_full[2], res_empty[2], cluster, fin
    static constexpr int kBars = kFlags + 32;
    static constexpr int kNumBars = 2 * STAGES + 18;
    static constexpr int kTables = kBars + kNumBars * 8 + 8;
    static constexpr int kBytes = kTables;
    static constexpr int kAlloc = kBytes + 1024;      // base aligned up to 1024 in the kernel
    static constexpr int kTmemCols = 128;             // S^T: 2 x kHalves x 16, O^T: 16
    static constexpr int kColS = 0, kColO = 64;
    static_assert(T == 128 || T == 256, "tile of one or two 128-position MMA blocks");
    static_assert(D == 64 || D == 128, "head_dim 64 or 128");
    static_assert(kQ % 1024 == 0 && kQBytes % 1024 == 0, "swizzled query blocks stay aligned");
    static_assert(kResBytes % 16 == 0, "result slots stay 16-byte aligned");
};

// ------------------------------------------------------------------------------------------------
// kernel
// ------------------------------------------------------------------------------------------------

template <int D, int T, int STAGES>
__global__ void __launch_bounds__(TcPlan<D, T, STAGES>::kThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap tmap,
                     const __grid_constant__ CUtensorMap tmap_rows,
                     const __grid_constant__ DecodeParams p)
{
    using PL = TcPlan<D, T, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_addr(smem);
    const uint32_t bar_full = sbase + PL::kBars;
    const uint32_t bar_empty = bar_full + 8 * STAGES;
    const uint32_t bar_s_ready = bar_empty + 8 * STAGES;    // [2]
    const uint32_t bar_s_free = bar_s_ready + 16;           // [2]
    const uint32_t bar_p_ready = bar_s_free + 16;           // [2]
    const uint32_t bar_p_free = bar_p_ready + 16;           // [2]
    const uint32_t bar_q_ready = bar_p_free + 16;           // [2]
    const uint32_t bar_o_ready = bar_q_ready + 16;
    const uint32_t bar_o_free = bar_o_ready + 8;
    const uint32_t bar_res_full = bar_o_free + 8;           // [2]
    const uint32_t bar_res_empty = bar_res_full + 16;       // [2]
    const uint32_t bar_cluster = bar_res_empty + 16;        // leader: k-1 remote arrivals
    const uint32_t bar_fin = bar_cluster + 8;
    volatile int *flags = reinterpret_cast<volatile int *>(smem + PL::kFlags);
    int *s_len = reinterpret_cast<int *>(smem + PL::kTables);
    int *s_start = s_len + p.b;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int P = gridDim.x;
    const int cta = blockIdx.x;
    const int N = p.num_tiles;
    const int tile_lo = static_cast<int>(static_cast<long long>(cta) * N / P);
    const int tile_hi = static_cast<int>(static_cast<long long>(cta + 1) * N / P);
    const int G = p.G;
    const bool early = p.early_fetch == 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
        }
        for (int r = 0; r < 2; ++r) {
            mbar_init(bar_s_ready + 8 * r, 1);
            mbar_init(bar_s_free + 8 * r, PL::kSoftWarps);
            mbar_init(bar_p_ready + 8 * r, PL::kSoftWarps);
            mbar_init(bar_p_free + 8 * r, 1);
            mbar_init(bar_q_ready + 8 * r, PL::kSoftWarps);
            mbar_init(bar_res_full + 8 * r, 1);
            mbar_init(bar_res_empty + 8 * r, 1);
        }
        mbar_init(bar_o_ready, 1);
        mbar_init(bar_o_free, PL::kSoftWarps);
        mbar_init(bar_cluster, 1);
        mbar_init(bar_fin, 1);
        if (p.cluster_k > 1 && cluster_ctarank() == 0)
            mbar_arrive_expect_tx(bar_cluster, static_cast<uint32_t>(
                                                   (p.cluster_k - 1) * (p.G * D + p.G) * 4));
        flags[0] = 0;   // abort
        fence_barrier_init();
    }
    if (threadIdx.x == PL::kProducer * 32) {
        prefetch_tensormap(&tmap);
        prefetch_tensormap(&tmap_rows);
    }
    if (warp == PL::kMma) {
        // Tensor memory for S^T (double-buffered) and O^T; the base address lands in smem.
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         sbase + PL::kFlags + 16),
                     "n"(PL::kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (p.uniform_len <= 0) {
        for (int i = threadIdx.x; i < p.b; i += blockDim.x) {
            s_len[i] = p.seq_len[i];
            s_start[i] = p.tile_start[i];
        }
        if (threadIdx.x == 0)
            s_start[p.b] = p.tile_start[p.b];
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + PL::kFlags + 16);
    if (p.cluster_k > 1)
        cluster_arrive();   // this CTA's barriers exist; waited on before any remote access
    TileWalk<T> wk;
    if (tile_lo < tile_hi)
        wk.init(p, s_len, s_start, tile_lo);

    // Dependency discipline as in decode_kernel: with p.early_fetch (inside mlkv_decode_step) the
    // previous kernel wrote nothing this one reads but the newest row of a segment (its last tile)
    // and the merge scratch; otherwise nothing global is touched before the wait.
    if (warp == PL::kProducer) {
        // ------------------------------------ producer ------------------------------------------
        if (lane != 0) {
            grid_dependents_launch();   // only lane 0 touches global memory
        } else {
            int issued = 0;
            int tile = tile_lo;
            bool waited = !early;
            if (!early)
                grid_dependency_wait();
            if (p.Q_next != nullptr) {
                const size_t qbytes = static_cast<size_t>(p.b) * p.h * D * 2;
                const size_t lo = (qbytes * cta / P) & ~static_cast<size_t>(127);
                const size_t hi =
                    cta + 1 == P ? qbytes : (qbytes * (cta + 1) / P) & ~static_cast<size_t>(127);
                if (hi > lo)
                    bulk_prefetch_l2(reinterpret_cast<const uint8_t *>(p.Q_next) + lo,
                                     static_cast<uint32_t>(hi - lo));
            }
            for (; tile < tile_hi; ++tile) {
                if (!waited && wk.tt == wk.nt - 1) {
                    grid_dependency_wait();   // this tile holds the newest row
                    waited = true;
                }
                const int s = issued % STAGES;
                if (issued >= STAGES && !flags[0] &&
                    !mbar_wait(bar_empty + 8 * s, ((issued / STAGES) & 1) ^ 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitEmpty);
                }
                if (flags[0])
                    break;
                const uint32_t fb = bar_full + 8 * s;
                const int vis = wk.L - wk.tt * T;
                const int nbox = vis < T ? (vis + 63) / 64 : 0;
                mbar_arrive_expect_tx(fb, nbox > 0 ? static_cast<uint32_t>(nbox) * 64u * D * 4u
                                                   : static_cast<uint32_t>(PL::kStageBytes));
                const int zk = ((p.slot * 2 + 0) * p.b + wk.beta) * p.g + wk.j;
                const int zv = zk + p.b * p.g;
                const int y = wk.tt * T;
                const uint32_t kdst = sbase + s * PL::kStageBytes;
                const uint32_t vdst = kdst + PL::kTileBytes;
                if (nbox == 0) {
#pragma unroll
                    for (int sub = 0; sub < PL::kSub; ++sub) {
                        tma_load_3d(kdst + sub * T * 128, &tmap, fb, sub * 64, y, zk);
                        tma_load_3d(vdst + sub * T * 128, &tmap, fb, sub * 64, y, zv);
                    }
                } else {
                    for (int bx = 0; bx < nbox; ++bx) {
#pragma unroll
                        for (int sub = 0; sub < PL::kSub; ++sub) {
                            const uint32_t off = sub * T * 128 + bx * 64 * 128;
                            tma_load_3d(kdst + off, &tmap_rows, fb, sub * 64, y + 64 * bx, zk);
                            tma_load_3d(vdst + off, &tmap_rows, fb, sub * 64, y + 64 * bx, zv);
                        }
                    }
                }
                ++issued;
                if (issued == STAGES)
                    grid_dependents_launch();   // the first loads are in flight
                wk.next(p, s_len, s_start);
            }
            if (issued < STAGES)
                grid_dependents_launch();
            // No copy may still be in flight when the CTA exits.
            const int first = issued > STAGES ? issued - STAGES : 0;
            for (int k = first; k < issued; ++k)
                if (!mbar_wait(bar_full + 8 * (k % STAGES), (k / STAGES) & 1))
                    atomicOr(p.err, kErrDrain);
        }
        __syncwarp();
    } else if (warp == PL::kMma) {
        // ------------------------------------ MMA issuer ----------------------------------------
        // Two cursors over the CTA's tiles, driven by whichever is ready first: S^T of a tile as
        // soon as its K/V has landed and an S^T buffer is free (up to two tiles ahead of the
        // softmax), and O^T += V^T P^T of a tile as soon as its P^T is written -- which also frees
        // the tile's stage for the producer.  Lane 0 polls and decides; the warp follows.
        grid_dependents_launch();
        constexpr uint32_t kIdS = umma_idesc(128, 16, 0, 0);
        constexpr uint32_t kIdPV = umma_idesc(D, 16, 1, 1);
        const uint32_t tm_o = tmem + PL::kColO;
        const int ntiles = tile_hi - tile_lo;
        TileWalk<T> ws = wk, wp = wk;   // the S and PV cursors
        int si = 0, pi = 0;             // their tile indices within the CTA's run
        int spc = -1, ppc = -1;         // piece index of the last tile each cursor issued
        bool ok = true;
        uint64_t idle_since = 0;
        while (pi < ntiles && ok) {
            int act = 0;   // 1: O^T += V^T P^T of tile pi, 2: S^T of tile si
            if (lane == 0) {
                if (pi < si && mbar_test_wait(bar_p_ready + 8 * (pi & 1), (pi >> 1) & 1)) {
                    const bool first = (pi == 0 || wp.tt == 0);
                    // The first product of a piece overwrites O^T: the softmax warps must be
                    // done reading the previous piece's.
                    if (!first || ppc < 0 || mbar_test_wait(bar_o_free, ppc & 1))
                        act = 1;
                }
                if (act == 0 && si < ntiles &&
                    mbar_test_wait(bar_full + 8 * (si % STAGES), (si / STAGES) & 1) &&
                    (si < 2 || mbar_test_wait(bar_s_free + 8 * (si & 1), ((si >> 1) & 1) ^ 1))) {
                    const bool first = (si == 0 || ws.tt == 0);
                    if (!first || mbar_test_wait(bar_q_ready + 8 * ((spc + 1) & 1),
                                                 ((spc + 1) >> 1) & 1))
                        act = 2;
                }
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
            if (act == 1) {
                const bool first = (pi == 0 || wp.tt == 0);
                const bool last = (pi == ntiles - 1 || wp.tt == wp.nt - 1);
                if (first)
                    ++ppc;
                tmem_fence_after();
                if (lane == 0) {
                    const int sb = pi % STAGES, pb = pi & 1;
                    const uint32_t vt = sbase + sb * PL::kStageBytes + PL::kTileBytes;
                    const uint32_t pt = sbase + PL::kP + pb * PL::kPBytes;
#pragma unroll 4
                    for (int k = 0; k < T / 16; ++k)
                        umma_f16(tm_o, umma_desc(vt + k * 2048, T * 128, 1024, kLayoutSw128),
                                 umma_desc(pt + k * 256, 128, T * 16, kLayoutInterleave), kIdPV,
                                 (first && k == 0) ? 0 : 1);
                    umma_commit(bar_empty + 8 * sb);   // the K/V stage may be refilled
                    umma_commit(bar_p_free + 8 * pb);  // the P^T buffer may be rewritten
                    if (last)
                        umma_commit(bar_o_ready);      // the piece's O^T is complete
                }
                __syncwarp();
                ++pi;
                wp.next(p, s_len, s_start);
            } else {
                const int s = si % STAGES, b = si & 1;
                if (si == 0 || ws.tt == 0)
                    ++spc;
                const int vis = ws.L - ws.tt * T;
                if (p.K_new != nullptr && vis <= T) {
                    // Fused append: the tile holds position L-1, the new token.  Its K/V replace
                    // the tile row (the copy may have read the cache before the token was stored)
                    // and, in the owner layer, go to the cache for the layers that read this slot
                    // later.
                    const int r_new = vis - 1;
                    if (lane < 8 * PL::kSub) {
                        const size_t src =
                            (static_cast<size_t>(ws.beta) * p.g + ws.j) * D + lane * 8;
                        const uint4 kn = *reinterpret_cast<const uint4 *>(p.K_new + src);
                        const uint4 vn = *reinterpret_cast<const uint4 *>(p.V_new + src);
                        uint8_t *st = smem + s * PL::kStageBytes;
                        *reinterpret_cast<uint4 *>(st + swz<T>(r_new, lane)) = kn;
                        *reinterpret_cast<uint4 *>(st + PL::kTileBytes + swz<T>(r_new, lane)) = vn;
                        if (p.store_new) {
                            const size_t dst =
                                ((((static_cast<size_t>(p.slot) * 2) * p.b + ws.beta) * p.g +
                                  ws.j) * static_cast<size_t>(p.max_seq) + (ws.L - 1)) * D +
                                lane * 8;
                            *reinterpret_cast<uint4 *>(p.cache + dst) = kn;
                            *reinterpret_cast<uint4 *>(
                                p.cache + dst + static_cast<size_t>(p.b) * p.g * p.max_seq * D) = vn;
                        }
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                }
                tmem_fence_after();
                if (lane == 0) {
                    const uint32_t kt = sbase + s * PL::kStageBytes;
                    const uint32_t qt = sbase + PL::kQ + (spc & 1) * PL::kQBytes;
#pragma unroll
                    for (int hf = 0; hf < PL::kHalves; ++hf)
#pragma unroll
                        for (int k = 0; k < D / 16; ++k)
                            umma_f16(tmem + PL::kColS + (b * PL::kHalves + hf) * 16,
                                     umma_desc(kt + hf * 128 * 128 + (k >> 2) * T * 128 +
                                                   (k & 3) * 32,
                                               16, 1024, kLayoutSw128),
                                     umma_desc(qt + (k >> 2) * 2048 + (k & 3) * 32, 16, 1024,
                                               kLayoutSw128),
                                     kIdS, k > 0 ? 1 : 0);
                    umma_commit(bar_s_ready + 8 * b);
                }
                __syncwarp();
                ++si;
                ws.next(p, s_len, s_start);
            }
        }
        if (!ok) {
            flags[0] = 1;
            if (lane == 0)
                atomicOr(p.err, kErrWaitFull);
        }
        // Every MMA issued by this warp has landed before tensor memory is freed.
        if (lane == 0)
            umma_commit(bar_fin);
        __syncwarp();
        if (!mbar_wait(bar_fin, 0) && lane == 0)
            atomicOr(p.err, kErrDrain);
        __syncwarp();
    } else if (warp == PL::kEpilogue) {
        // ------------------------------------ epilogue ------------------------------------------
        if (!early)
            grid_dependency_wait();
        grid_dependents_launch();
        float *s_w = reinterpret_cast<float *>(smem + PL::kEpiW);
        for (int k = 0;; ++k) {
            const int rb = k & 1;
            int okw = 1;
            if (lane == 0 && !mbar_wait(bar_res_full + 8 * rb, (k >> 1) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
                okw = 0;
            }
            okw = __shfl_sync(0xffffffffu, okw, 0);
            if (!okw)
                break;
            const uint8_t *slot = smem + PL::kRes + rb * PL::kResBytes;
            const int *meta = reinterpret_cast<const int *>(slot + PL::kResO + 64);
            if (meta[kMetaStop])
                break;
            if (early && k == 0)
                grid_dependency_wait();   // records and merges use the shared scratch
            if (!flags[0])
                epilogue_piece<D>(p, reinterpret_cast<const float *>(slot),
                                  reinterpret_cast<const float *>(slot + PL::kResO), meta, s_w,
                                  PL::kEpiCap, lane, cta);
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_res_empty + 8 * rb);
        }
        __syncwarp();
    } else {
        // ------------------------------------ softmax warps -------------------------------------
        const int tid = threadIdx.x;   // 0..127: this thread's TMEM lane, position tid of a block
        if (!early)
            grid_dependency_wait();
        grid_dependents_launch();
        const float scale = p.scale_log2;
        const float inv_scale = 1.f / scale;   // thresholds in score units (a bound, not exact)
        const float NEG_INF = -__int_as_float(0x7f800000);
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        float *lred = reinterpret_cast<float *>(smem + PL::kLRed);
        float *mred = reinterpret_cast<float *>(smem + PL::kMRed);

        // This thread's share of a group's queries: kSub 16-byte chunks of the [16][D] block.
        uint4 qreg[PL::kSub];
        auto load_q = [&](int beta, int j) {
#pragma unroll
            for (int u = 0; u < PL::kSub; ++u) {
                const int idx = tid + 128 * u;
                const int r = idx / (8 * PL::kSub), c = idx % (8 * PL::kSub);
                qreg[u] = make_uint4(0, 0, 0, 0);
                if (r < G)
                    qreg[u] = *reinterpret_cast<const uint4 *>(
                        p.Q + ((static_cast<size_t>(beta) * p.h + static_cast<size_t>(j) * G + r) *
                                   D + c * 8));
            }
        };
        auto store_q = [&](int buf) {
            uint8_t *qb = smem + PL::kQ + buf * PL::kQBytes;
#pragma unroll
            for (int u = 0; u < PL::kSub; ++u) {
                const int idx = tid + 128 * u;
                const int r = idx / (8 * PL::kSub), c = idx % (8 * PL::kSub);
                *reinterpret_cast<uint4 *>(qb + (c >> 3) * 2048 + r * 128 +
                                           (((c & 7) ^ (r & 7)) << 4)) = qreg[u];
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_q_ready + 8 * buf);
        };

        int it = 0, pc = 0, nhand = 0;
        int tile = tile_lo;
        bool q_stored = false;   // this piece's queries are already in their buffer
        if (tile < tile_hi)
            load_q(wk.beta, wk.j);
        while (tile < tile_hi) {
            const int beta = wk.beta, j = wk.j, L = wk.L;
            const int seg = beta * p.g + j;
            const int seg_first = wk.seg_first;
            const int seg_end = seg_first + wk.nt;
            const int piece_first = tile;
            const int piece_end = seg_end < tile_hi ? seg_end : tile_hi;
            if (!q_stored)
                store_q(pc & 1);
            q_stored = false;
            if (piece_end < tile_hi) {
                // The next piece is the next segment: its queries load during this piece and go
                // to the other buffer once its tiles are done, so that the MMA warp can start the
                // next piece while this one is finished.
                const int nseg = seg + 1;
                load_q(nseg / p.g, nseg % p.g);
            }

            float m_ref[16], thr[16], l_acc[16];
#pragma unroll
            for (int h = 0; h < 16; ++h) {
                m_ref[h] = h < G ? NEG_INF : 0.f;
                thr[h] = NEG_INF;
                l_acc[h] = 0.f;
            }
            for (; tile < piece_end; ++tile, ++it) {
                const int s = it % STAGES, b = it & 1;
                const int vis = L - wk.tt * T;   // visible positions of this tile
                if (!flags[0] && !mbar_wait(bar_s_ready + 8 * b, (it >> 1) & 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitFull);
                }
                tmem_fence_after();
                float sv[PL::kHalves][16];
#pragma unroll
                for (int hf = 0; hf < PL::kHalves; ++hf)
                    tmem_ld16(tmem + lane_base + PL::kColS + (b * PL::kHalves + hf) * 16, sv[hf]);
                tmem_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(bar_s_free + 8 * b);

                // Does any visible score of the tile exceed its head's reference by 2^8?
                bool over = false;
#pragma unroll
                for (int hf = 0; hf < PL::kHalves; ++hf) {
                    const bool valid = hf * 128 + tid < vis;
#pragma unroll
                    for (int h = 0; h < 16; ++h)
                        over |= valid && h < G && sv[hf][h] > thr[h];
                }
                if (soft_bar_or(over)) {
                    // Exact maximum of the tile per head, over the four warps.
                    float mx[16];
#pragma unroll
                    for (int h = 0; h < 16; ++h) {
                        float v = NEG_INF;
#pragma unroll
                        for (int hf = 0; hf < PL::kHalves; ++hf)
                            if (hf * 128 + tid < vis)
                                v = fmaxf(v, sv[hf][h]);
                        mx[h] = v;
                    }
#pragma unroll
                    for (int h = 0; h < 16; ++h) {
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 16));
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 8));
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 4));
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 2));
                        mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 1));
                    }
                    if (lane == 0) {
#pragma unroll
                        for (int h = 0; h < 16; ++h)
                            mred[warp * 16 + h] = mx[h];
                    }
                    soft_bar_sync();
                    float alpha[16];
                    bool rescale = false;
#pragma unroll
                    for (int h = 0; h < 16; ++h) {
                        alpha[h] = 1.f;
                        if (h < G) {
                            const float t = fmaxf(fmaxf(mred[h], mred[16 + h]),
                                                  fmaxf(mred[32 + h], mred[48 + h])) * scale;
                            if (t > m_ref[h]) {
                                alpha[h] = fast_exp2(m_ref[h] - t);   // 0 when m_ref = -inf
                                rescale = rescale || m_ref[h] != NEG_INF;
                                m_ref[h] = t;
                            }
                            thr[h] = (m_ref[h] + 8.f) * inv_scale;
                        }
                    }
                    // Keep mred until every thread has read it (the next tile may write it).
                    soft_bar_sync();
                    if (rescale && tile > piece_first) {
                        // O^T and the row sums are rescaled once the product of the previous
                        // tile has landed (the next one is issued after this tile's P^T).
                        const int pt = it - 1;
                        if (!flags[0] && !mbar_wait(bar_p_free + 8 * (pt & 1), (pt >> 1) & 1)) {
                            flags[0] = 1;
                            atomicOr(p.err, kErrWaitFull);
                        }
                        tmem_fence_after();
                        float ov[16];
                        tmem_ld16(tmem + lane_base + PL::kColO, ov);
#pragma unroll
                        for (int h = 0; h < 16; ++h)
                            ov[h] *= alpha[h];
                        tmem_st16(tmem + lane_base + PL::kColO, ov);
                        tmem_fence_before();
                    }
#pragma unroll
                    for (int h = 0; h < 16; ++h)
                        l_acc[h] *= alpha[h];
                }

                // P^T rows of this thread's positions, bf16; the row sums take the same rounding.
                if (it >= 2 && !flags[0] &&
                    !mbar_wait(bar_p_free + 8 * b, ((it >> 1) & 1) ^ 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitFull);
                }
                uint8_t *pbuf = smem + PL::kP + b * PL::kPBytes;
#pragma unroll
                for (int hf = 0; hf < PL::kHalves; ++hf) {
                    const int pos = hf * 128 + tid;
                    const bool valid = pos < vis;
                    uint32_t w[8];
#pragma unroll
                    for (int h2 = 0; h2 < 8; ++h2) {
                        const float p0 = valid ? fast_exp2(fmaf(sv[hf][2 * h2], scale,
                                                                -m_ref[2 * h2])) : 0.f;
                        const float p1 = valid ? fast_exp2(fmaf(sv[hf][2 * h2 + 1], scale,
                                                                -m_ref[2 * h2 + 1])) : 0.f;
                        w[h2] = pack_bf16x2(p0, p1);
                        l_acc[2 * h2] += bf16_lo(w[h2]);
                        l_acc[2 * h2 + 1] += bf16_hi(w[h2]);
                    }
                    *reinterpret_cast<uint4 *>(pbuf + pos * 16) = make_uint4(w[0], w[1], w[2], w[3]);
                    *reinterpret_cast<uint4 *>(pbuf + T * 16 + pos * 16) =
                        make_uint4(w[4], w[5], w[6], w[7]);
                    if (!valid) {
                        // Past the sequence end the stage holds whatever the cache (or an older
                        // tile) holds: zero the V row so that 0 * V stays 0.
                        uint8_t *vrow = smem + s * PL::kStageBytes + PL::kTileBytes;
#pragma unroll
                        for (int c = 0; c < 8 * PL::kSub; ++c)
                            *reinterpret_cast<uint4 *>(vrow + swz<T>(pos, c)) =
                                make_uint4(0, 0, 0, 0);
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(bar_p_ready + 8 * b);
                wk.next(p, s_len, s_start);
            }

            if (piece_end < tile_hi) {
                store_q((pc + 1) & 1);   // its last user, piece pc - 1, is long done
                q_stored = true;
            }

            // ---------------- end of piece: o = O^T / l, lse = m + log2 l ----------------
            // Row sums over the CTA: a warp reduction, then the four warps through smem.
#pragma unroll
            for (int h = 0; h < 16; ++h) {
                float v = l_acc[h];
                v += __shfl_xor_sync(0xffffffffu, v, 16);
                v += __shfl_xor_sync(0xffffffffu, v, 8);
                v += __shfl_xor_sync(0xffffffffu, v, 4);
                v += __shfl_xor_sync(0xffffffffu, v, 2);
                v += __shfl_xor_sync(0xffffffffu, v, 1);
                l_acc[h] = v;
            }
            if (lane == 0) {
#pragma unroll
                for (int h = 0; h < 16; ++h)
                    lred[warp * 16 + h] = l_acc[h];
            }
            if (!flags[0] && !mbar_wait(bar_o_ready, pc & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
            tmem_fence_after();
            float ov[16];
            tmem_ld16(tmem + lane_base + PL::kColO, ov);
            tmem_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_o_free);
            // The result slot: the piece's normalised o and lse.  A slot is reused every other
            // piece; the epilogue warp frees it.
            const int rb = nhand & 1;
            if (tid == 0 && nhand >= 2 && !flags[0] &&
                !mbar_wait(bar_res_empty + 8 * rb, ((nhand >> 1) - 1) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitEmpty);
            }
            soft_bar_sync();   // lred complete, slot free
            uint8_t *slot = smem + PL::kRes + rb * PL::kResBytes;
            float *ro = reinterpret_cast<float *>(slot);
            float *rlse = reinterpret_cast<float *>(slot + PL::kResO);
            // This thread's TMEM lane holds channel d of O^T (head_dim 64: M = 64, so lanes
            // 0-15 of each warp hold channels 16w..16w+15; head_dim 128: lane = channel).
            const int d = D == 64 ? warp * 16 + lane : warp * 32 + lane;
            const bool has_d = D == 64 ? lane < 16 : true;
#pragma unroll
            for (int h = 0; h < 16; ++h) {
                if (h < G) {
                    const float lh = lred[h] + lred[16 + h] + lred[32 + h] + lred[48 + h];
                    if (has_d)
                        ro[h * D + d] = ov[h] * fast_rcp(lh);
                    if (tid == 0)
                        rlse[h] = m_ref[h] + fast_log2(lh);
                }
            }
            soft_bar_sync();   // slot written; lred may be reused
            const bool whole = (piece_first == seg_first && piece_end == seg_end);
            if (piece_end != tile_hi) {
                // An earlier piece: the epilogue warp writes it out while the next piece runs.
                if (tid == 0) {
                    int *meta = reinterpret_cast<int *>(slot + PL::kResO + 64);
                    meta[kMetaBeta] = beta;
                    meta[kMetaJ] = j;
                    meta[kMetaSeg] = seg;
                    meta[kMetaWhole] = whole ? 1 : 0;
                    meta[kMetaFirst] = cta_of_tile(seg_first, N, P);
                    meta[kMetaLast] = cta_of_tile(seg_end - 1, N, P);
                    meta[kMetaStop] = 0;
                    mbar_arrive(bar_res_full + 8 * rb);
                }
                ++nhand;
                ++pc;
                continue;
            }
            ++pc;
            // ---- the CTA's last piece: the softmax warps finish it from the slot ----
            __nv_bfloat16 *ob =
                p.out + (static_cast<size_t>(beta) * p.h + static_cast<size_t>(j) * G) * D;
            // mode: 0 whole, 1 cluster sender, 2 cluster leader, 3 partial record
            const int rank = p.cluster_k > 1 ? static_cast<int>(cluster_ctarank()) : 0;
            const int mode = whole ? 0 : (p.cluster_k > 1 ? (rank != 0 ? 1 : 2) : 3);
            if (p.cluster_k > 1)
                cluster_wait();   // the partner CTAs' barriers exist
            if (early && mode == 3)
                grid_dependency_wait();   // partial records and counters are shared scratch
            const uint8_t *cs = smem + PL::kTables;
            const size_t piece = static_cast<size_t>(seg + cta);
            float *po = p.part_o + piece * G * D;
            if (mode == 0) {
                for (int i = 2 * tid; i < G * D; i += 256)
                    *reinterpret_cast<uint32_t *>(ob + i) = pack_bf16x2(ro[i], ro[i + 1]);
            } else if (mode == 1) {
                const uint32_t remote =
                    map_to_rank(sbase + PL::kTables + (rank - 1) * PL::kResBytes, 0);
                const uint32_t remote_bar = map_to_rank(bar_cluster, 0);
                // the leader's barrier completes when all these bytes have landed
                for (int i = 2 * tid; i < G * D; i += 256)
                    st_async_v2(remote + i * 4, ro[i], ro[i + 1], remote_bar);
                if (tid < G)
                    st_async_f32(remote + PL::kResO + tid * 4, rlse[tid], remote_bar);
            } else if (mode == 2) {
                if (!flags[0] && !mbar_wait_cluster(bar_cluster, 0)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitFull);
                }
                const int k = p.cluster_k;   // 2 or 4
                for (int i = 2 * tid; i < G * D; i += 256) {
                    const int row = i / D;
                    float lr[4];
                    float2 x[4];
                    lr[0] = rlse[row];
                    x[0] = make_float2(ro[i], ro[i + 1]);
#pragma unroll
                    for (int r = 1; r < 4; ++r) {
                        lr[r] = NEG_INF;
                        x[r] = make_float2(0.f, 0.f);
                        if (r < k) {
                            const uint8_t *sl = cs + (r - 1) * PL::kResBytes;
                            lr[r] = reinterpret_cast<const float *>(sl + PL::kResO)[row];
                            x[r] = *reinterpret_cast<const float2 *>(sl + static_cast<size_t>(i) * 4);
                        }
                    }
                    const float mx = fmaxf(fmaxf(lr[0], lr[1]), fmaxf(lr[2], lr[3]));
                    float tot = 0.f, ax = 0.f, ay = 0.f;
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        const float w = fast_exp2(lr[r] - mx);   // 0 past k
                        tot += w;
                        ax = fmaf(w, x[r].x, ax);
                        ay = fmaf(w, x[r].y, ay);
                    }
                    const float inv = fast_rcp(tot);
                    if (!flags[0])
                        *reinterpret_cast<uint32_t *>(ob + i) = pack_bf16x2(ax * inv, ay * inv);
                }
            } else {
                for (int i = 2 * tid; i < G * D; i += 256)
                    *reinterpret_cast<float2 *>(po + i) = make_float2(ro[i], ro[i + 1]);
                if (tid < G)
                    p.part_lse[piece * G + tid] = rlse[tid];
                if (!p.deferred_merge) {
                    const int c_first = cta_of_tile(seg_first, N, P);
                    const int c_last = cta_of_tile(seg_end - 1, N, P);
                    __threadfence();
                    soft_bar_sync();
                    if (tid == 0) {
                        const unsigned prev = atomic_add_acq_rel_gpu(&p.counters[seg], 1u);
                        flags[1] = (prev == static_cast<unsigned>(c_last - c_first)) ? 1 : 0;
                    }
                    soft_bar_sync();
                    if (flags[1]) {
                        // Last finisher of the segment: merge its <= 4 records (own included).
                        const int np = c_last - c_first + 1;
                        const size_t rec0 = static_cast<size_t>(seg + c_first);
                        for (int i = 2 * tid; i < G * D; i += 256) {
                            const int row = i / D;
                            float lv[kInlineMergeMaxPieces];
                            float2 ovv[kInlineMergeMaxPieces];
                            float mx = NEG_INF;
#pragma unroll
                            for (int k = 0; k < kInlineMergeMaxPieces; ++k) {
                                lv[k] = NEG_INF;
                                ovv[k] = make_float2(0.f, 0.f);
                                if (k < np) {
                                    lv[k] = __ldcg(&p.part_lse[(rec0 + k) * G + row]);
                                    ovv[k] = __ldcg(reinterpret_cast<const float2 *>(
                                        p.part_o + (rec0 + k) * G * D + i));
                                }
                                mx = fmaxf(mx, lv[k]);
                            }
                            float tot = 0.f, ax = 0.f, ay = 0.f;
#pragma unroll
                            for (int k = 0; k < kInlineMergeMaxPieces; ++k) {
                                const float w = fast_exp2(lv[k] - mx);   // 0 past np
                                tot += w;
                                ax += w * ovv[k].x;
                                ay += w * ovv[k].y;
                            }
                            const float inv = fast_rcp(tot);
                            *reinterpret_cast<uint32_t *>(ob + i) = pack_bf16x2(ax * inv, ay * inv);
                        }
                        if (tid == 0)
                            p.counters[seg] = 0u;
                    }
                    soft_bar_sync();   // flags[1] is reused
                }
            }
        }
        if (early)
            grid_dependency_wait();   // no-op if already waited; this grid ends after the previous
        // Tell the epilogue warp that no piece follows.
        if (tid == 0) {
            const int rb = nhand & 1;
            if (nhand >= 2 && !flags[0] &&
                !mbar_wait(bar_res_empty + 8 * rb, ((nhand >> 1) - 1) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitEmpty);
            }
            int *meta = reinterpret_cast<int *>(smem + PL::kRes + rb * PL::kResBytes + PL::kResO + 64);
            meta[kMetaStop] = 1;
            mbar_arrive(bar_res_full + 8 * rb);
        }
    }

    // ------------------------------------ common exit -------------------------------------------
    if (p.cluster_k > 1 && (warp >= PL::kSoftWarps || tile_lo >= tile_hi))
        cluster_wait();   // every thread of the cluster waits once on its arrival
    tmem_fence_before();
    __syncthreads();
    if (warp == PL::kMma) {
        tmem_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "n"(PL::kTmemCols)
                     : "memory");
    }
}

template <int D, int T, int STAGES>
constexpr DecodeVariant make_tc_variant()
{
    using PL = TcPlan<D, T, STAGES>;
    return DecodeVariant{D, T, STAGES, PL::kThreads, static_cast<size_t>(PL::kAlloc),
                         static_cast<size_t>(PL::kResBytes),
                         reinterpret_cast<const void *>(&decode_tc_kernel<D, T, STAGES>), 1};
}

}  // namespace

// (head_dim, positions per tile, ring stages) of the tcgen05 kernel.
const DecodeVariant kTcVariants[] = {
    make_tc_variant<64, 128, 6>(),
    make_tc_variant<64, 256, 3>(),
    make_tc_variant<128, 128, 2>(),
};
const int kNumTcVariants = static_cast<int>(sizeof(kTcVariants) / sizeof(kTcVariants[0]));

}  // namespace mlkv
