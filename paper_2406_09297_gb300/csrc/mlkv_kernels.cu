// MLKV decode-attention kernels for GB300 (sm_103a).
//
// decode_kernel: single-token attention of one layer over the cache slot of the layer's owner
// (MLKV, arXiv 2406.09297, Sec. 3 Eqs. 13-18, attention of Eqs. 2-3).
//
//   Work split.  A "segment" is one (sequence beta, KV head j) pair: positions [0, L_beta) of one
//   K/V head, read by the G = h/g query heads of its group (Eq. 15).  Segments are cut into tiles
//   of T positions and all tiles of the layer are laid end to end (beta-major, j inside).  A
//   persistent grid of P CTAs takes equal contiguous runs of that tile list, so every CTA streams
//   the same number of bytes whatever the length mix.  The part of a segment inside one CTA's run
//   is a "piece"; a CTA that holds a whole segment writes its output directly, otherwise it
//   writes a normalised partial (o, log-sum-exp) and the last CTA to finish the segment (an atomic
//   counter, no spinning) merges the partials.
//
//   Data movement.  One producer warp issues TMA tensor copies (cp.async.bulk.tensor, 128-byte
//   swizzle) of each K and V tile into a STAGES-deep shared-memory ring, completion tracked by
//   mbarrier transaction counts.  Each tile is fetched from HBM exactly once and used by all G
//   query heads of the group.
//
//   Math.  NCW consumer warps (4 or 8) split every tile by positions.  Scores S = Q K^T and the
//   update
//   O += P V run on the tensor cores (mma.sync m16n8k16, bf16 in, fp32 accumulate) with the
//   query group padded to M = 16 rows; the softmax is online, in fp32, base 2 with the 1/sqrt(d)
//   scale folded into the exponent, with quad shuffles for row maxima.  The warps' states are
//   merged through shared memory at the end of each piece.
//
//   Launch.  Programmatic dependent launch: barrier set-up overlaps the previous kernel of the
//   stream, and no global memory is touched before griddepcontrol.wait.
//
// append_kernel: stores the new token's K/V of an owner layer at position L_beta - 1.
//
// Every wait on an mbarrier is bounded (about 2 s); on expiry the kernel sets a bit in the
// device error word, stops issuing copies, keeps its barrier sequence intact, drains the copies
// it already issued and exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mlkv_internal.h"

#include "mlkv_device.cuh"

namespace mlkv {
namespace {

// ------------------------------------------------------------------------------------------------
// shared-memory plan
// ------------------------------------------------------------------------------------------------

template <int D, int T, int STAGES, int NCW>
struct Plan {
    static constexpr int kThreads = (NCW + 2) * 32;   // consumers, one producer, one epilogue warp
    // Variants whose ring fits twice in an SM's shared memory are sized for two resident CTAs.
    static constexpr int kMinBlocks = (STAGES * 2 * T * D * 2 <= 80 * 1024) ? 2 : 1;
    static constexpr int kProducer = NCW;             // warp indices
    static constexpr int kEpilogue = NCW + 1;
    static constexpr int kSub = D / 64;               // 128-byte-wide column blocks per row
    static constexpr int kTW = T / NCW;               // positions per warp per tile
    static constexpr int kTileBytes = T * D * 2;      // one K (or V) tile
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kWarpFrag = D * 64;          // one warp's O fragments: D/8*4 f32 x 32
    static constexpr int kResO = 16 * D * 4;          // a piece's result: o[16][D] f32
    static constexpr int kResBytes = kResO + 16 * 4 + 32;   // + lse[16] + 8 ints of metadata
    static constexpr int kMerge = STAGES * kStageBytes;                 // [NCW/2][kWarpFrag]
    static constexpr int kRes = kMerge + (NCW / 2) * kWarpFrag;        // [2][kResBytes]
    static constexpr int kEpiW = kRes + 2 * kResBytes;                 // f32 [kEpiCap] weights
    static constexpr int kEpiCap = 512;
    static constexpr int kRedM = kEpiW + kEpiCap * 4;                  // f32 [NCW][16]
    static constexpr int kRedL = kRedM + NCW * 16 * 4;                 // f32 [NCW][16]
    static constexpr int kFlags = kRedL + NCW * 16 * 4;                // int [4]
    // u64 full[S], empty[S], res_full[2], res_empty[2], cluster
    static constexpr int kBars = kFlags + 16;
    // Dynamic tail: per-sequence tables (lengths differ) or, in cluster mode, the leader's
    // slots for the other ranks' results ([k-1][kResBytes]).
    // Per-stage query slots: the G rows of the segment whose first tile the stage holds, each row
    // padded by 16 bytes so that the fragment loads (8 rows apart) fall in distinct banks.
    static constexpr int kQRow = D * 2 + 16;
    static constexpr int kQSlot = 16 * kQRow;
    static constexpr int kQ = (kBars + (2 * STAGES + 5) * 8 + 8 + 127) / 128 * 128;
    static constexpr int kTables = kQ + STAGES * kQSlot;
    static constexpr int kBytes = kTables;
    static constexpr int kFinRow = D + 8;             // row stride (f32) of the last piece's sums
    static constexpr int kAlloc = kBytes + 1024;      // base aligned up to 1024 in the kernel
    static_assert(kTW % 16 == 0, "each warp takes whole 16-position mma steps");
    static_assert(NCW == 4 || NCW == 8, "tree merge over 4 or 8 warps");
    static_assert(D == 64 || D == 128, "head_dim 64 or 128");
    static_assert(T <= 256, "TMA box height");
    static_assert(kResBytes % 16 == 0, "result slots stay 16-byte aligned");
    static_assert((NCW * 16 * kFinRow + 16) * 4 <= STAGES * kStageBytes,
                  "the last piece's per-warp sums fit in the stage ring");
};


// Query fragments of one (sequence, KV head) group from global memory: the A operand of
// S = Q K^T in the mma.m16n8k16 layout, rows >= G (the padding of the group to 16 rows) zero.
template <int D>
__device__ __forceinline__ void load_q_frag(uint32_t (&qa)[D / 16][4], const DecodeParams &p,
                                            const __nv_bfloat16 *Q, int beta, int j, int lane)
{
    const int G = p.G;
    const int qr = lane >> 2, qc = (lane & 3) * 2;
    const __nv_bfloat16 *qb =
        Q + (static_cast<size_t>(beta) * p.h + static_cast<size_t>(j) * G) * D;
    const bool r0 = qr < G, r1 = qr + 8 < G;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
        const int c = ks * 16 + qc;
        qa[ks][0] = r0 ? *reinterpret_cast<const uint32_t *>(qb + qr * D + c) : 0u;
        qa[ks][1] = r1 ? *reinterpret_cast<const uint32_t *>(qb + (qr + 8) * D + c) : 0u;
        qa[ks][2] = r0 ? *reinterpret_cast<const uint32_t *>(qb + qr * D + c + 8) : 0u;
        qa[ks][3] = r1 ? *reinterpret_cast<const uint32_t *>(qb + (qr + 8) * D + c + 8) : 0u;
    }
}

// Query fragments of one (sequence, KV head) group from its shared-memory slot (16 rows of
// D bf16, row stride RS elements, rows >= G unused): the A operand of S = Q K^T in the
// mma.m16n8k16 layout, rows >= G zero.
template <int D, int RS>
__device__ __forceinline__ void load_q_frag_smem(uint32_t (&qa)[D / 16][4], const uint8_t *slot,
                                                 int G, int lane)
{
    const int qr = lane >> 2, qc = (lane & 3) * 2;
    const __nv_bfloat16 *qb = reinterpret_cast<const __nv_bfloat16 *>(slot);
    const bool r0 = qr < G, r1 = qr + 8 < G;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
        const int c = ks * 16 + qc;
        qa[ks][0] = r0 ? *reinterpret_cast<const uint32_t *>(qb + qr * RS + c) : 0u;
        qa[ks][1] = r1 ? *reinterpret_cast<const uint32_t *>(qb + (qr + 8) * RS + c) : 0u;
        qa[ks][2] = r0 ? *reinterpret_cast<const uint32_t *>(qb + qr * RS + c + 8) : 0u;
        qa[ks][3] = r1 ? *reinterpret_cast<const uint32_t *>(qb + (qr + 8) * RS + c + 8) : 0u;
    }
}

// Margin (log2 units) by which a score may exceed a row's reference maximum before the reference
// is raised: weights stay <= 2^8.
constexpr float kLazyMax = 8.f;
// Two bf16 ones, the B operand that turns P V's MMA into P's row sums.
constexpr uint32_t kOnesBf16x2 = 0x3f803f80u;

// ------------------------------------------------------------------------------------------------
// decode kernel
// ------------------------------------------------------------------------------------------------

template <int D, int T, int STAGES, int NCW>
__global__ void __launch_bounds__(Plan<D, T, STAGES, NCW>::kThreads,
                                  Plan<D, T, STAGES, NCW>::kMinBlocks)
    decode_kernel(const __grid_constant__ CUtensorMap tmap,
                  const __grid_constant__ CUtensorMap tmap_rows,
                  const __grid_constant__ DecodeParams p)
{
    using PL = Plan<D, T, STAGES, NCW>;
    constexpr int TW = PL::kTW;
    constexpr int NT = TW / 8;     // 8-position score tiles per warp
    constexpr int KS = D / 16;     // 16-wide reduction steps over the head dimension
    constexpr int NO = D / 8;      // 8-wide output column tiles

    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_addr(smem);
    const uint32_t bar_full = sbase + PL::kBars;
    const uint32_t bar_empty = bar_full + 8 * STAGES;
    const uint32_t bar_res_full = bar_empty + 8 * STAGES;    // [2]
    const uint32_t bar_res_empty = bar_res_full + 16;        // [2]
    const uint32_t bar_cluster = bar_res_empty + 16;         // leader: k-1 remote arrivals
    volatile int *flags = reinterpret_cast<volatile int *>(smem + PL::kFlags);
    int *s_len = reinterpret_cast<int *>(smem + PL::kTables);
    int *s_start = s_len + p.b;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int P = gridDim.x;
    const int cta = blockIdx.x;
    const int N = p.num_tiles;
    // floor(c N / P) in 32 bits when c N fits (a 64-bit division costs ~0.1 us at CTA start).
    // A multi-layer launch numbers each CTA's own tiles from 0: its items c, c + P, ... (whole
    // segments of nt tiles each).
    const bool ml = p.ml_layers > 0;
    const bool narrow = static_cast<long long>(P) * N < (1ll << 32);
    int tile_lo, tile_hi;
    if (ml) {
        // the tiles of this CTA's items (see TileWalk::ml_rank)
        tile_lo = 0;
        tile_hi = 0;
        for (int k = 0;; ++k) {
            const int r = TileWalk<T>::ml_rank(p, k);
            if (r < 0)
                break;
            const int L = p.uniform_len > 0
                              ? p.uniform_len
                              : p.seq_len[p.tile_start[TileWalk<T>::ml_seq_pos(p, r)]];
            if (p.ml_chunks > 1) {
                int a, b;
                TileWalk<T>::ml_chunk(p, (L + T - 1) / T, r % p.ml_chunks, a, b);
                tile_hi += b - a;
            } else {
                tile_hi += (L + T - 1) / T;
            }
        }
    } else {
        tile_lo = narrow ? static_cast<int>(static_cast<uint32_t>(cta) * N / P)
                         : static_cast<int>(static_cast<long long>(cta) * N / P);
        tile_hi = narrow ? static_cast<int>(static_cast<uint32_t>(cta + 1) * N / P)
                         : static_cast<int>(static_cast<long long>(cta + 1) * N / P);
    }
    // Per-layer pointers: a multi-layer launch reads layer `layer`'s queries, writes its outputs,
    // reads its owner's slot and new token; a single-layer launch has one of each.
    auto q_of = [&](int layer) {
        return ml ? p.Q + static_cast<size_t>(layer) * p.ml_q_stride : p.Q;
    };
    auto slot_of = [&](int layer) { return ml ? static_cast<int>(p.ml_slot[layer]) : p.slot; };

    const bool early = p.early_fetch == 1;
    const bool pre_tile = p.early_fetch != 0;   // the first tile may go out before the wait
    // The producer warp's copy of one tile into stage `s` (query rows too when a later piece
    // starts); called by all 32 lanes with the same arguments.  On GB300 one issuing thread
    // completes about one bulk copy per ~0.5 us whatever its size (measured: 8 to 64 KB, from L2
    // or HBM, 2 to 8 copies outstanding), while copies from different lanes proceed side by side;
    // so the copies of a tile -- K and V boxes, query rows -- go out from different lanes, and
    // successive stages from different groups of lanes.  Lane 0 first announces the stage's bytes.
    auto issue_tile = [&](const TileWalk<T> &w, int s, bool with_q) {
        const uint32_t fb = bar_full + 8 * s;
        const uint32_t qbytes = static_cast<uint32_t>(p.G) * D * 2;
        // A segment's last tile may be partly visible: only its boxes of 64 positions that
        // hold visible rows are fetched (the rest of the stage keeps stale rows, which the
        // consumers mask in S and zero in V).
        const int vis = w.L - w.tt * T;
        const int nbox = vis < T ? (vis + 63) / 64 : 0;
        const uint32_t kv_bytes =
            nbox > 0 ? static_cast<uint32_t>(nbox) * 64u * D * 2u * 2u : PL::kStageBytes;
        if (lane == 0)
            mbar_arrive_expect_tx(fb, kv_bytes + (with_q ? qbytes : 0u));
        __syncwarp();
        // copy i of this tile goes out from lane (i + rot) mod 32
        const int per_tile = 2 * PL::kSub * (nbox > 0 ? nbox : 1);
        const int mine = (lane - s * 2 * PL::kSub) & 31;
        const int zk = ((slot_of(w.layer) * 2 + 0) * p.b + w.beta) * p.g + w.j;
        const int zv = zk + p.b * p.g;
        const int y = w.tt * T;
        const uint32_t kdst = sbase + s * PL::kStageBytes;
        const uint32_t vdst = kdst + PL::kTileBytes;
        if (mine < per_tile) {
            // copy i: box bx = i / (2 kSub), then K or V, then the 64-column block
            const int bx = mine / (2 * PL::kSub);
            const int kv = (mine / PL::kSub) & 1;
            const int sub = mine % PL::kSub;
            const uint32_t dst = (kv ? vdst : kdst) + sub * T * 128 + bx * 64 * 128;
            if (nbox == 0)
                tma_load_3d(dst, &tmap, fb, sub * 64, y, kv ? zv : zk);
            else
                tma_load_3d(dst, &tmap_rows, fb, sub * 64, y + 64 * bx, kv ? zv : zk);
        }
        if (with_q) {
            const __nv_bfloat16 *q0 = q_of(w.layer) + (static_cast<size_t>(w.beta) * p.h +
                                                       static_cast<size_t>(w.j) * p.G) * D;
            const int r = (mine - per_tile) & 31;
            if (r < p.G)
                bulk_load(sbase + PL::kQ + s * PL::kQSlot + r * PL::kQRow, q0 + r * D, D * 2, fb);
        }
    };
    // The ring's barriers belong to the producer warp's lane 0.  With early fetch (either kind) and
    // one length for every sequence the warp also sends its first tile before the CTA barrier: a
    // CTA that got its SM late (the last ones of a layer decide the layer's end), or one that
    // starts while the step's inputs are still being copied in, then has data on the way at once.
    bool pre_issued = false;
    // The trigger comes first: the next launch (inside a decode step, the next layer's decode)
    // may start as soon as every CTA of this grid is resident.  What it reads before its own
    // dependency wait is fixed by p.early_fetch, and it finishes only after this grid.
    if (threadIdx.x == 0)
        grid_dependents_launch();
    if (warp == PL::kProducer) {
        if (lane == 0) {
            prefetch_tensormap(&tmap);   // kernel parameters: safe before the dependency wait
            prefetch_tensormap(&tmap_rows);
            for (int s = 0; s < STAGES; ++s) {
                mbar_init(bar_full + 8 * s, 1);
                mbar_init(bar_empty + 8 * s, NCW);
            }
            fence_barrier_init();
        }
        __syncwarp();
        if (pre_tile && p.uniform_len > 0 && tile_lo < tile_hi) {
            TileWalk<T> w0;
            w0.init(p, s_len, s_start, tile_lo);
            if (w0.tt != w0.nt - 1 || p.newest_ready) {   // not a newest row still to wait for
                issue_tile(w0, 0, false);
                pre_issued = true;
            }
        }
    }
    if (threadIdx.x == 0) {
        for (int r = 0; r < 2; ++r) {
            mbar_init(bar_res_full + 8 * r, 1);
            mbar_init(bar_res_empty + 8 * r, 1);
        }
        mbar_init(bar_cluster, 1);
        if (p.cluster_k > 1 && cluster_ctarank() == 0) {
            // The leader expects every other rank's result: G*D outputs and G lse values, f32.
            mbar_arrive_expect_tx(bar_cluster, static_cast<uint32_t>(
                                                   (p.cluster_k - 1) * (p.G * D + p.G) * 4));
        }
        flags[0] = 0;   // abort
        fence_barrier_init();
    }
    if (p.uniform_len <= 0) {
        for (int i = threadIdx.x; i < p.b; i += blockDim.x) {
            s_len[i] = p.seq_len[i];
            s_start[i] = p.tile_start[i];
        }
        if (threadIdx.x == 0)
            s_start[p.b] = p.tile_start[p.b];
    }
    __syncthreads();
    if (p.cluster_k > 1)
        cluster_arrive();   // this CTA's barriers exist; waited on before any remote access
    // The tile walk reads only the parameters and the shared tables: set it up before the wait.
    TileWalk<T> wk;
    if (tile_lo < tile_hi)
        wk.init(p, s_len, s_start, tile_lo);
    // Everything above overlaps the previous kernels' tails.  Normally global memory is touched
    // only after the dependency wait.  When the previous kernels still running are this library's
    // decodes of the preceding layers (p.early_fetch, inside mlkv_decode_step), they write nothing
    // this one reads except the newest row (position L-1) of the slot an owner appended to, which
    // lies in the last tile of a segment, and the merge scratch (partials, counters).  So the
    // queries and every other tile are fetched at once, and a segment's last tile too when this
    // grid replaces its newest row from K_new/V_new (p.newest_ready; else the producer waits
    // before fetching it); the epilogue warp waits before it writes its first record, and the
    // consumers before they write the last piece (scratch) or, at the latest, before they exit --
    // so this grid finishes only after the previous one, as the next layer's wait expects.
    // The first piece's query fragments come straight from global memory, before the wait when
    // the queries cannot be the previous kernel's output; later pieces find theirs in a slot.
    uint32_t qa[KS][4];
    if (early && warp < NCW && tile_lo < tile_hi)
        load_q_frag<D>(qa, p, q_of(wk.layer), wk.beta, wk.j, lane);
    if (warp != PL::kProducer && !early)
        grid_dependency_wait();
    if (warp == PL::kEpilogue && lane == 0)
        grid_dependency_wait();

    // -------------------------------- producer warp --------------------------------------------
    // Every lane walks the same tiles; lane 0 waits (dependency, free stages) and announces each
    // stage's bytes, and the copies go out from several lanes (issue_tile).
    if (warp == PL::kProducer) {
        if (ml && p.pf_own && lane == 31)
            prefetch_slots_share<D>(p, cta, P);
        int issued = pre_issued ? 1 : 0;
        int tile = tile_lo + issued;
        if (pre_issued)
            wk.next(p, s_len, s_start);
        bool waited = !early;
        if (!early)
            grid_dependency_wait();
        // The next layer's queries (an input of the whole step) go to L2 now: its CTAs load
        // them first thing, while this layer still streams.  Each CTA takes a 128-byte-aligned
        // share.  Issued from the last lane, which issues no tile copies.
        if (p.Q_next != nullptr && lane == 31) {
            const size_t qbytes = static_cast<size_t>(p.b) * p.h * D * 2;   // a multiple of 128
            const size_t lo = (qbytes * cta / P) & ~static_cast<size_t>(127);
            const size_t hi =
                cta + 1 == P ? qbytes : (qbytes * (cta + 1) / P) & ~static_cast<size_t>(127);
            if (hi > lo)
                bulk_prefetch_l2(reinterpret_cast<const uint8_t *>(p.Q_next) + lo,
                                 static_cast<uint32_t>(hi - lo));
        }
        for (; tile < tile_hi; ++tile) {
            if (!waited && wk.tt == wk.nt - 1 && !p.newest_ready) {
                grid_dependency_wait();   // this tile holds the newest row
                waited = true;
            }
            const int s = issued % STAGES;
            int stop = 0;
            if (lane == 0) {
                if (issued >= STAGES && !flags[0] &&
                    !mbar_wait(bar_empty + 8 * s, ((issued / STAGES) & 1) ^ 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitEmpty);
                }
                stop = flags[0];
            }
            if (__shfl_sync(0xffffffffu, stop, 0))
                break;
            // A later piece starts here: its query rows come with the tile.
            issue_tile(wk, s, wk.tt == wk.t0 && tile != tile_lo);
            ++issued;
            wk.next(p, s_len, s_start);
        }
        // No copy may still be in flight when the CTA exits.
        if (lane == 0) {
            const int first = issued > STAGES ? issued - STAGES : 0;
            for (int k = first; k < issued; ++k)
                if (!mbar_wait(bar_full + 8 * (k % STAGES), (k / STAGES) & 1))
                    atomicOr(p.err, kErrDrain);
        }
        __syncwarp();
        if (p.cluster_k > 1)
            cluster_wait();
        return;
    }

    // -------------------------------- epilogue warp --------------------------------------------
    if (warp == PL::kEpilogue) {
        float *s_w = reinterpret_cast<float *>(smem + PL::kEpiW);
        for (int k = 0;; ++k) {
            const int rb = k & 1;
            int ok = 1;
            if (lane == 0 && !mbar_wait(bar_res_full + 8 * rb, (k >> 1) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
                ok = 0;
            }
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok)
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
        if (p.cluster_k > 1)
            cluster_wait();
        return;
    }

    // -------------------------------- consumer warps -------------------------------------------
    float *merge = reinterpret_cast<float *>(smem + PL::kMerge);
    float *red_m = reinterpret_cast<float *>(smem + PL::kRedM);
    float *red_l = reinterpret_cast<float *>(smem + PL::kRedL);
    const int qr = lane >> 2;              // fragment row (query head within the group)
    const int qc = (lane & 3) * 2;         // fragment column pair
    const int G = p.G;
    const float scale = p.scale_log2;
    const float NEG_INF = -__int_as_float(0x7f800000);

    int it = 0;
    int nhand = 0;   // pieces handed to the epilogue warp (all but the CTA's last)
    int tile = tile_lo;

    while (tile < tile_hi) {
        const int beta = wk.beta;
        const int j = wk.j;
        const int L = wk.L;
        const int seg = beta * p.g + j;
        const int layer = wk.layer;
        const int rec = wk.rec;   // partial-record index of a chunked multi-layer piece
        const bool part = p.ml_chunks > 1;   // chunks are always partial records
        const int slot = slot_of(layer);
        const int store_new = ml ? static_cast<int>(p.ml_store[layer]) : p.store_new;
        const __nv_bfloat16 *k_new = p.K_new;
        const __nv_bfloat16 *v_new = p.V_new;
        if (ml && k_new != nullptr) {
            k_new += static_cast<size_t>(slot) * p.ml_kv_stride;
            v_new += static_cast<size_t>(slot) * p.ml_kv_stride;
        }
        const int seg_first = wk.seg_first;
        const int seg_end = seg_first + wk.nt;
        const int piece_first = tile;
        const int piece_end = seg_end < tile_hi ? seg_end : tile_hi;

        if (tile == tile_lo) {
            if (!early)
                load_q_frag<D>(qa, p, q_of(layer), beta, j, lane);
        } else {
            // A later piece: its query rows arrive with its first tile (the loop's wait for that
            // tile then returns at once).
            const int s0 = it % STAGES;
            if (!flags[0] && !mbar_wait(bar_full + 8 * s0, (it / STAGES) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
            load_q_frag_smem<D, PL::kQRow / 2>(qa, smem + PL::kQ + s0 * PL::kQSlot, G, lane);
        }

        float o[NO][4];
#pragma unroll
        for (int n = 0; n < NO; ++n)
            o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
        float m_run[2] = {NEG_INF, NEG_INF};
        // Row sums of P, accumulated on the tensor core: P times a block of ones (every column
        // of la holds its row's sum), in fp32 from the same bf16 weights P V uses.
        float la[4] = {0.f, 0.f, 0.f, 0.f};

        for (; tile < piece_end; ++tile, ++it) {
            const int s = it % STAGES;
            if (!flags[0] && !mbar_wait(bar_full + 8 * s, (it / STAGES) & 1)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
            const int row0 = warp * TW;                 // this warp's first row in the tile
            const int valid = L - (wk.tt * T + row0);   // visible rows in this warp's slice
            if (!flags[0] && valid > 0) {
                const uint32_t kt = sbase + s * PL::kStageBytes;
                const uint32_t vt = kt + PL::kTileBytes;
                if (k_new != nullptr && valid <= TW) {
                    // Fused append: this warp's slice holds position L-1, the new token.  Its K/V
                    // replace the tile rows (the copy may have read the cache before the token was
                    // stored) and, in the owner layer, are stored in the cache for the layers that
                    // read this slot later.
                    const int r_new = row0 + valid - 1;
                    if (lane < 8 * PL::kSub) {
                        const size_t src = (static_cast<size_t>(beta) * p.g + j) * D + lane * 8;
                        const uint4 kn = *reinterpret_cast<const uint4 *>(k_new + src);
                        const uint4 vn = *reinterpret_cast<const uint4 *>(v_new + src);
                        uint8_t *st = smem + s * PL::kStageBytes;
                        *reinterpret_cast<uint4 *>(st + swz<T>(r_new, lane)) = kn;
                        *reinterpret_cast<uint4 *>(st + PL::kTileBytes + swz<T>(r_new, lane)) = vn;
                        if (store_new) {
                            const size_t dst =
                                ((((static_cast<size_t>(slot) * 2) * p.b + beta) * p.g + j) *
                                     static_cast<size_t>(p.max_seq) + (L - 1)) * D + lane * 8;
                            *reinterpret_cast<uint4 *>(p.cache + dst) = kn;
                            *reinterpret_cast<uint4 *>(
                                p.cache + dst + static_cast<size_t>(p.b) * p.g * p.max_seq * D) = vn;
                        }
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                }
                if (valid < TW) {
                    // Rows past the sequence end hold whatever the cache holds there; zero the V
                    // rows so that 0-weight * V stays 0 even for non-finite contents.
                    uint8_t *vrow = smem + s * PL::kStageBytes + PL::kTileBytes;
                    const int nrows = TW - valid;
                    for (int idx = lane; idx < nrows * 8 * PL::kSub; idx += 32) {
                        const int rr = row0 + valid + idx / (8 * PL::kSub);
                        const int rem = idx % (8 * PL::kSub);
                        const int sub = rem / 8;
                        *reinterpret_cast<uint4 *>(vrow + sub * T * 128 + rr * 128 +
                                                   (rem % 8) * 16) = make_uint4(0, 0, 0, 0);
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                }

                // ---- S = Q K^T for this warp's TW positions ----
                float sc[NT][4];
#pragma unroll
                for (int n = 0; n < NT; ++n)
                    sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
                const int mi = lane >> 3;   // which 8x8 matrix this lane addresses
                const int mr = lane & 7;    // which row of it
                // The K fragments of a group of up to 8 shared-memory loads go out together and
                // the MMAs follow, so the loads' latency (~47 cycles each) is paid once per group.
                constexpr int KG = (KS * (NT / 2) <= 8) ? KS : (8 / (NT / 2) > 0 ? 8 / (NT / 2) : 1);
#pragma unroll
                for (int k0 = 0; k0 < KS; k0 += KG) {
                    uint32_t kf[KG][NT / 2][4];
#pragma unroll
                    for (int kg = 0; kg < KG; ++kg) {
#pragma unroll
                        for (int n2 = 0; n2 < NT / 2; ++n2) {
                            const int row = row0 + 8 * (2 * n2 + (mi >> 1)) + mr;
                            const int chunk = 2 * (k0 + kg) + (mi & 1);
                            ldsm_x4(kt + swz<T>(row, chunk), kf[kg][n2][0], kf[kg][n2][1],
                                    kf[kg][n2][2], kf[kg][n2][3]);
                        }
                    }
#pragma unroll
                    for (int kg = 0; kg < KG; ++kg) {
#pragma unroll
                        for (int n2 = 0; n2 < NT / 2; ++n2) {
                            mma_bf16_16816(sc[2 * n2], qa[k0 + kg], kf[kg][n2][0], kf[kg][n2][1]);
                            mma_bf16_16816(sc[2 * n2 + 1], qa[k0 + kg], kf[kg][n2][2],
                                           kf[kg][n2][3]);
                        }
                    }
                }
                // The V fragments of the first group of P V (up to 8 loads) go out now: their
                // latency overlaps the softmax below.
                constexpr int VQ = NO / 2;                         // loads per 16 positions
                constexpr int VG = (VQ * (NT / 2) <= 8) ? NT / 2 : (8 / VQ > 0 ? 8 / VQ : 1);
                uint32_t vf[VG][VQ][4];
#pragma unroll
                for (int kg = 0; kg < VG; ++kg) {
#pragma unroll
                    for (int q = 0; q < VQ; ++q) {
                        const int row = row0 + 16 * kg + 8 * (mi & 1) + mr;
                        const int chunk = 2 * q + (mi >> 1);
                        ldsm_x4_trans(vt + swz<T>(row, chunk), vf[kg][q][0], vf[kg][q][1],
                                      vf[kg][q][2], vf[kg][q][3]);
                    }
                }

                // ---- online softmax (base 2, scale folded into the exponent) ----
                float mx[2] = {NEG_INF, NEG_INF};
                if (valid < TW) {
#pragma unroll
                    for (int n = 0; n < NT; ++n) {
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const int pos_in_slice = 8 * n + qc + (c & 1);
                            if (pos_in_slice >= valid)
                                sc[n][c] = NEG_INF;
                        }
                    }
                }
#pragma unroll
                for (int n = 0; n < NT; ++n) {
                    mx[0] = fmaxf(mx[0], fmaxf(sc[n][0], sc[n][1]));
                    mx[1] = fmaxf(mx[1], fmaxf(sc[n][2], sc[n][3]));
                }
                // The reference maximum moves only when a score exceeds it by more than 2^8 (in
                // the exponent): weights then stay in [0, 256], exactly as accurate in bf16, and
                // most tiles need neither the quad reduction nor a rescale.  When one does, the
                // rows' exact maxima over this tile become the new references.
                const bool raise = mx[0] * scale > m_run[0] + kLazyMax ||
                                   mx[1] * scale > m_run[1] + kLazyMax;
                if (__any_sync(0xffffffffu, raise)) {
                    float alpha[2];
#pragma unroll
                    for (int hr = 0; hr < 2; ++hr) {
                        mx[hr] = fmaxf(mx[hr], __shfl_xor_sync(0xffffffffu, mx[hr], 1));
                        mx[hr] = fmaxf(mx[hr], __shfl_xor_sync(0xffffffffu, mx[hr], 2));
                        const float m_new = fmaxf(m_run[hr], mx[hr] * scale);
                        alpha[hr] = (m_new == NEG_INF) ? 1.f : fast_exp2(m_run[hr] - m_new);
                        m_run[hr] = m_new;
                    }
#pragma unroll
                    for (int n = 0; n < NO; ++n) {
                        o[n][0] *= alpha[0];
                        o[n][1] *= alpha[0];
                        o[n][2] *= alpha[1];
                        o[n][3] *= alpha[1];
                    }
                    la[0] *= alpha[0];
                    la[1] *= alpha[0];
                    la[2] *= alpha[1];
                    la[3] *= alpha[1];
                }
                const float m_use[2] = {m_run[0] == NEG_INF ? 0.f : m_run[0],
                                        m_run[1] == NEG_INF ? 0.f : m_run[1]};
                // P in bf16 (the mma A operand).
                uint32_t pa[NT / 2][4];
#pragma unroll
                for (int n = 0; n < NT; ++n) {
                    const float p0 = fast_exp2(fmaf(sc[n][0], scale, -m_use[0]));
                    const float p1 = fast_exp2(fmaf(sc[n][1], scale, -m_use[0]));
                    const float p2 = fast_exp2(fmaf(sc[n][2], scale, -m_use[1]));
                    const float p3 = fast_exp2(fmaf(sc[n][3], scale, -m_use[1]));
                    pa[n >> 1][(n & 1) * 2 + 0] = pack_bf16x2(p0, p1);
                    pa[n >> 1][(n & 1) * 2 + 1] = pack_bf16x2(p2, p3);
                }

                // ---- O += P V ----
#pragma unroll
                for (int kg = 0; kg < VG; ++kg) {
#pragma unroll
                    for (int q = 0; q < VQ; ++q) {
                        mma_bf16_16816(o[2 * q], pa[kg], vf[kg][q][0], vf[kg][q][1]);
                        mma_bf16_16816(o[2 * q + 1], pa[kg], vf[kg][q][2], vf[kg][q][3]);
                    }
                    mma_bf16_16816(la, pa[kg], kOnesBf16x2, kOnesBf16x2);
                }
                // the remaining 16-position groups (longer tiles), a group's loads first
#pragma unroll
                for (int k0 = VG; k0 < NT / 2; k0 += VG) {
                    uint32_t vg[VG][VQ][4];
#pragma unroll
                    for (int kg = 0; kg < VG; ++kg) {
#pragma unroll
                        for (int q = 0; q < VQ; ++q) {
                            const int row = row0 + 16 * (k0 + kg) + 8 * (mi & 1) + mr;
                            const int chunk = 2 * q + (mi >> 1);
                            ldsm_x4_trans(vt + swz<T>(row, chunk), vg[kg][q][0], vg[kg][q][1],
                                          vg[kg][q][2], vg[kg][q][3]);
                        }
                    }
#pragma unroll
                    for (int kg = 0; kg < VG; ++kg) {
#pragma unroll
                        for (int q = 0; q < VQ; ++q) {
                            mma_bf16_16816(o[2 * q], pa[k0 + kg], vg[kg][q][0], vg[kg][q][1]);
                            mma_bf16_16816(o[2 * q + 1], pa[k0 + kg], vg[kg][q][2],
                                           vg[kg][q][3]);
                        }
                        mma_bf16_16816(la, pa[k0 + kg], kOnesBf16x2, kOnesBf16x2);
                    }
                }
            }
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_empty + 8 * s);
            wk.next(p, s_len, s_start);
        }

        // ---------------- end of piece: merge the warps (no atomics) ----------------
        // Row statistics of every warp -> per-row maximum m* and total l*; each warp's
        // accumulators are weighted by 2^(m_w - m*) / l* and the warps summed.
        const float l_run[2] = {la[0], la[2]};
        if ((lane & 3) == 0) {
            red_m[warp * 16 + qr] = m_run[0];
            red_m[warp * 16 + qr + 8] = m_run[1];
            red_l[warp * 16 + qr] = l_run[0];
            red_l[warp * 16 + qr + 8] = l_run[1];
        }
        // The barrier also guarantees that every warp is done with the ring's tiles.
        consumer_bar_sync<NCW>();
        if (piece_end != tile_hi) {
            // A piece before the CTA's last: tree over warps, result to the epilogue warp, and
            // the consumers go straight on to the next piece.
            float lse[2];
    #pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
                const int row = qr + 8 * hr;
                // every piece holds at least one visible position, so mstar is finite
                float mstar = NEG_INF;
    #pragma unroll
                for (int w = 0; w < NCW; ++w)
                    mstar = fmaxf(mstar, red_m[w * 16 + row]);
                float lsum = 0.f;
    #pragma unroll
                for (int w = 0; w < NCW; ++w)
                    lsum += red_l[w * 16 + row] * fast_exp2(red_m[w * 16 + row] - mstar);
                const float f = fast_exp2(m_run[hr] - mstar) * fast_rcp(lsum);
                lse[hr] = mstar + fast_log2(lsum);
    #pragma unroll
                for (int n = 0; n < NO; ++n) {
                    o[n][2 * hr] *= f;
                    o[n][2 * hr + 1] *= f;
                }
            }
            // Tree over warps with NCW/2 slots.  First level: warp w in [NCW/2, NCW) writes slot
            // w - NCW/2 and warp r < NCW/2 adds slot r.  Later levels (half < NCW/2): warp w in
            // [half, 2 half) writes slot w and warp r < half adds slot r + half.  Every slot is
            // rewritten only by the warp that read it last, so one barrier per level suffices.
    #pragma unroll
            for (int half = NCW / 2; half >= 1; half >>= 1) {
                const bool first = (half == NCW / 2);
                if (warp >= half && warp < 2 * half) {
                    float *dst = merge + (first ? warp - half : warp) * (NO * 4 * 32);
    #pragma unroll
                    for (int n = 0; n < NO; ++n)
    #pragma unroll
                        for (int c = 0; c < 4; ++c)
                            dst[(n * 4 + c) * 32 + lane] = o[n][c];
                }
                consumer_bar_sync<NCW>();
                if (warp < half) {
                    const float *src = merge + (first ? warp : warp + half) * (NO * 4 * 32);
    #pragma unroll
                    for (int n = 0; n < NO; ++n)
    #pragma unroll
                        for (int c = 0; c < 4; ++c)
                            o[n][c] += src[(n * 4 + c) * 32 + lane];
                }
            }

            // Warp 0 hands the piece to the epilogue warp through a double-buffered slot and the
            // consumers move on to the next piece at once.
            if (warp == 0) {
                const int rb = nhand & 1;
                if (nhand >= 2 && !flags[0] &&
                    !mbar_wait(bar_res_empty + 8 * rb, ((nhand >> 1) - 1) & 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitEmpty);
                }
                uint8_t *slot = smem + PL::kRes + rb * PL::kResBytes;
                float *ro = reinterpret_cast<float *>(slot);
                float *rlse = reinterpret_cast<float *>(slot + PL::kResO);
                int *meta = reinterpret_cast<int *>(slot + PL::kResO + 64);
    #pragma unroll
                for (int hr = 0; hr < 2; ++hr) {
                    const int row = qr + 8 * hr;
                    if (row < G) {
    #pragma unroll
                        for (int n = 0; n < NO; ++n)
                            *reinterpret_cast<float2 *>(ro + row * D + n * 8 + qc) =
                                make_float2(o[n][2 * hr], o[n][2 * hr + 1]);
                        if (qc == 0)
                            rlse[row] = lse[hr];
                    }
                }
                if (lane == 0) {
                    meta[kMetaBeta] = beta;
                    meta[kMetaJ] = j;
                    meta[kMetaSeg] = seg;
                    meta[kMetaWhole] =
                        (piece_first == seg_first && piece_end == seg_end && !part) ? 1 : 0;
                    meta[kMetaFirst] = ml ? rec : cta_of_tile(seg_first, N, P);
                    meta[kMetaLast] = cta_of_tile(seg_end - 1, N, P);
                    meta[kMetaStop] = 0;
                    meta[kMetaLayer] = layer;
                }
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(bar_res_full + 8 * rb);
            }
            ++nhand;
        } else {
            // ---- the CTA's last piece: every tile has been consumed and no copy is pending, so
            // the stage ring is free.  Each warp stores its raw accumulators there; after one
            // barrier each consumer warp finishes one row per pass from every warp's statistics
            // of the row: m* = max_w m_w, l* = sum_w l_w 2^(m_w - m*), o = sum_w 2^(m_w - m*) o_w
            // / l*, lse = m* + log2 l*.
            // Rows padded to D + 8 floats: the fragment stores of a warp's 8 rows then fall in
            // distinct banks.
            constexpr int FS = PL::kFinRow;
            float *fbuf = reinterpret_cast<float *>(smem);         // [NCW][16][FS] f32
            float *flse = fbuf + NCW * 16 * FS;                     // [16]
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
                const int row = qr + 8 * hr;
                if (row < G) {
#pragma unroll
                    for (int n = 0; n < NO; ++n)
                        *reinterpret_cast<float2 *>(fbuf + (warp * 16 + row) * FS + n * 8 + qc) =
                            make_float2(o[n][2 * hr], o[n][2 * hr + 1]);
                }
            }
            if (p.cluster_k > 1)
                cluster_wait();   // the partner CTAs' barriers exist
            consumer_bar_sync<NCW>();
            const int ctid = threadIdx.x;
            const bool whole = (piece_first == seg_first && piece_end == seg_end && !part);
            __nv_bfloat16 *ob = p.out + static_cast<size_t>(layer) * p.ml_q_stride +
                                (static_cast<size_t>(beta) * p.h + static_cast<size_t>(j) * G) * D;
            constexpr int kPairs = NCW * 32;   // float2 outputs per pass
            static_assert(D == 2 * 32 || D == 4 * 32, "a warp's pass covers 64 elements of one row");
            // mode: 0 whole, 1 cluster sender, 2 cluster leader, 3 partial record
            const int rank = p.cluster_k > 1 ? static_cast<int>(cluster_ctarank()) : 0;
            const int mode = whole ? 0 : (p.cluster_k > 1 ? (rank != 0 ? 1 : 2) : 3);
            if (early && mode == 3)
                grid_dependency_wait();   // partial records and counters are shared scratch
            const uint32_t cslots = sbase + PL::kTables;
            const uint8_t *cs = smem + PL::kTables;
            uint32_t remote = 0, remote_bar = 0;
            if (mode == 1) {
                remote = map_to_rank(cslots + (rank - 1) * PL::kResBytes, 0);
                remote_bar = map_to_rank(bar_cluster, 0);
            }
            const size_t piece = ml ? static_cast<size_t>(rec) : static_cast<size_t>(seg + cta);
            float *po = p.part_o + piece * G * D;
#pragma unroll 2
            for (int i = 2 * ctid; i < G * D; i += 2 * kPairs) {
                const int row = i / D, e = i - row * D;   // row is the same across the warp
                // independent broadcast loads of the row's statistics of every warp
                float mw[NCW], lw[NCW];
#pragma unroll
                for (int w = 0; w < NCW; ++w) {
                    mw[w] = red_m[w * 16 + row];
                    lw[w] = red_l[w * 16 + row];
                }
                float ms = mw[0];   // finite: the piece holds a visible position
#pragma unroll
                for (int w = 1; w < NCW; ++w)
                    ms = fmaxf(ms, mw[w]);
                float ls = 0.f;
                float2 v = make_float2(0.f, 0.f);
#pragma unroll
                for (int w = 0; w < NCW; ++w) {
                    const float ew = fast_exp2(mw[w] - ms);
                    ls = fmaf(lw[w], ew, ls);
                    const float2 x =
                        *reinterpret_cast<const float2 *>(fbuf + (w * 16 + row) * FS + e);
                    v.x = fmaf(ew, x.x, v.x);
                    v.y = fmaf(ew, x.y, v.y);
                }
                const float inv = fast_rcp(ls);
                v.x *= inv;
                v.y *= inv;
                const float lse_row = ms + fast_log2(ls);
                const bool row_head = (e == 0 && lane == 0);   // one lane per row
                if (mode == 0) {
                    *reinterpret_cast<uint32_t *>(ob + i) = pack_bf16x2(v.x, v.y);
                } else if (mode == 1) {
                    // the leader's barrier completes when all these bytes have landed
                    st_async_v2(remote + i * 4, v.x, v.y, remote_bar);
                    if (row_head)
                        st_async_f32(remote + PL::kResO + row * 4, lse_row, remote_bar);
                } else if (mode == 2) {
                    // each element is read and rewritten by this thread alone
                    *reinterpret_cast<float2 *>(fbuf + row * FS + e) = v;
                    if (row_head)
                        flse[row] = lse_row;
                } else {
                    *reinterpret_cast<float2 *>(po + i) = v;
                    if (row_head)
                        p.part_lse[piece * G + row] = lse_row;
                }
            }
            if (mode == 2) {
                // Leader: its own result is in warp 0's rows; merge the other ranks' once landed.
                if (!flags[0] && !mbar_wait_cluster(bar_cluster, 0)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitFull);
                }
                consumer_bar_sync<NCW>();   // flse is complete
                const int k = p.cluster_k;   // 2 or 4
#pragma unroll 2
                for (int i = 2 * ctid; i < G * D; i += 2 * kPairs) {
                    const int row = i / D, e = i - row * D;
                    float lr[4];
                    float2 x[4];
                    lr[0] = flse[row];
                    x[0] = *reinterpret_cast<const float2 *>(fbuf + row * FS + e);
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
            } else if (mode == 3 && !p.deferred_merge) {
                const int c_first = cta_of_tile(seg_first, N, P);
                const int c_last = cta_of_tile(seg_end - 1, N, P);
                __threadfence();
                consumer_bar_sync<NCW>();
                if (ctid == 0) {
                    const unsigned prev = atomic_add_acq_rel_gpu(&p.counters[seg], 1u);
                    flags[1] = (prev == static_cast<unsigned>(c_last - c_first)) ? 1 : 0;
                }
                consumer_bar_sync<NCW>();
                if (flags[1]) {
                    // Last finisher of the segment: merge its <= 4 records (own included).
                    const int np = c_last - c_first + 1;
                    const size_t rec0 = static_cast<size_t>(seg + c_first);
#pragma unroll 1
                    for (int i = 2 * ctid; i < G * D; i += 2 * kPairs) {
                        const int row = i / D;
                        float lv[kInlineMergeMaxPieces];
                        float2 ov[kInlineMergeMaxPieces];
                        float mx = NEG_INF;
#pragma unroll
                        for (int k = 0; k < kInlineMergeMaxPieces; ++k) {
                            lv[k] = NEG_INF;
                            ov[k] = make_float2(0.f, 0.f);
                            if (k < np) {
                                lv[k] = __ldcg(&p.part_lse[(rec0 + k) * G + row]);
                                ov[k] = __ldcg(reinterpret_cast<const float2 *>(
                                    p.part_o + (rec0 + k) * G * D + i));
                            }
                            mx = fmaxf(mx, lv[k]);
                        }
                        float tot = 0.f, ax = 0.f, ay = 0.f;
#pragma unroll
                        for (int k = 0; k < kInlineMergeMaxPieces; ++k) {
                            const float w = fast_exp2(lv[k] - mx);   // 0 past np
                            tot += w;
                            ax += w * ov[k].x;
                            ay += w * ov[k].y;
                        }
                        const float inv = fast_rcp(tot);
                        *reinterpret_cast<uint32_t *>(ob + i) = pack_bf16x2(ax * inv, ay * inv);
                    }
                    if (ctid == 0)
                        p.counters[seg] = 0u;
                }
                consumer_bar_sync<NCW>();   // flags[1] is reused
            }
        }
    }
    if (early)
        grid_dependency_wait();   // no-op if already waited; this grid ends after the previous
    // Tell the epilogue warp that no piece follows.
    if (warp == 0) {
        const int rb = nhand & 1;
        if (nhand >= 2 && !flags[0] && !mbar_wait(bar_res_empty + 8 * rb, ((nhand >> 1) - 1) & 1)) {
            flags[0] = 1;
            atomicOr(p.err, kErrWaitEmpty);
        }
        if (lane == 0) {
            int *meta = reinterpret_cast<int *>(smem + PL::kRes + rb * PL::kResBytes + PL::kResO + 64);
            meta[kMetaStop] = 1;
            mbar_arrive(bar_res_full + 8 * rb);
        }
    }
}


// ------------------------------------------------------------------------------------------------
// combine kernel: merge of segments split over many CTAs
// ------------------------------------------------------------------------------------------------

// One CTA per (segment, query row of its group).  The CTA turns the pieces' log-sum-exps into
// weights w_c = 2^(lse_c - M) (M = max_c lse_c) and each thread sums w_c * o_c[e] for one column
// e over a strided subset of the pieces, 16 loads in flight (the first 16 issued with the
// log-sum-exps); the subsets are added through shared memory and scaled by 1 / sum_c w_c.
constexpr int kCombineThreads = 256;
constexpr int kCombineMaxPieces = 1024;

template <int D>
__global__ void __launch_bounds__(kCombineThreads)
    combine_kernel(const __grid_constant__ DecodeParams p)
{
    __shared__ float s_w[kCombineMaxPieces];
    __shared__ float s_red[kCombineThreads];
    // The next layer's decode may start at once: it reads neither the partials nor `out`, and it
    // writes partials only after its own dependency wait (after this grid).
    grid_dependents_launch();
    grid_dependency_wait();
    const int row = blockIdx.y;
    const int G = p.G;
    int seg, np;
    size_t rec0;
    __nv_bfloat16 *out = p.out;
    if (p.ml_layers > 0) {
        // a chunked multi-layer launch: blockIdx.x = layer b g + beta g + j, chunk records
        // blockIdx.x C .. blockIdx.x C + C - 1
        const int S = p.b * p.g;
        const int layer = static_cast<int>(blockIdx.x) / S;
        seg = static_cast<int>(blockIdx.x) - layer * S;
        out += static_cast<size_t>(layer) * p.ml_q_stride;
        np = p.ml_chunks;
        rec0 = static_cast<size_t>(blockIdx.x) * p.ml_chunks;
    } else {
        seg = blockIdx.x;
        const int T = p.tile_tokens;
        const int beta = seg / p.g;
        const int jj = seg - beta * p.g;
        const int L = p.uniform_len > 0 ? p.uniform_len : p.seq_len[beta];
        const int nt = (L + T - 1) / T;
        const int seg_first = p.uniform_len > 0 ? seg * nt : p.tile_start[beta] + jj * nt;
        const int c_first = cta_of_tile(seg_first, p.num_tiles, p.decode_grid);
        const int c_last = cta_of_tile(seg_first + nt - 1, p.num_tiles, p.decode_grid);
        if (c_first == c_last)
            return;   // one CTA held the whole segment and wrote the output itself
        np = c_last - c_first + 1;
        rec0 = static_cast<size_t>(seg + c_first);
    }
    const int beta = seg / p.g;
    const int j = seg - beta * p.g;
    const int tid = threadIdx.x;
    const int lane = tid & 31, wid = tid >> 5;
    constexpr int kWarps = kCombineThreads / 32;
    const float NEG_INF = -__int_as_float(0x7f800000);
    constexpr int kGroups = kCombineThreads / D;   // pieces summed side by side per column
    const int e = tid % D;
    const int grp = tid / D;
    const float *src = p.part_o + rec0 * G * D + static_cast<size_t>(row) * D + e;
    // The first 16 pieces' values of this thread go out together with the pieces' log-sum-exps:
    // one round trip to memory before the weights are known.
    float v[16];
#pragma unroll
    for (int m = 0; m < 16; ++m) {
        const int k = grp + m * kGroups;
        v[m] = k < np ? __ldcg(src + static_cast<size_t>(k) * G * D) : 0.f;
    }
    float mx = NEG_INF;
    for (int k = tid; k < np; k += kCombineThreads) {
        const float l = __ldcg(&p.part_lse[(rec0 + k) * G + row]);
        s_w[k] = l;
        mx = fmaxf(mx, l);
    }
    // block reductions: within each warp by shuffles, then across the warps through s_red
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    if (lane == 0)
        s_red[wid] = mx;
    __syncthreads();
    mx = s_red[0];
#pragma unroll
    for (int w = 1; w < kWarps; ++w)
        mx = fmaxf(mx, s_red[w]);
    float tot = 0.f;
    for (int k = tid; k < np; k += kCombineThreads) {
        const float w = fast_exp2(s_w[k] - mx);
        s_w[k] = w;
        tot += w;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
        tot += __shfl_xor_sync(0xffffffffu, tot, off);
    __syncthreads();   // every warp has read s_red's maxima; s_w holds the weights
    if (lane == 0)
        s_red[wid] = tot;
    __syncthreads();
    tot = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w)
        tot += s_red[w];
    const float inv = fast_rcp(tot);
    float acc = 0.f;
#pragma unroll
    for (int m = 0; m < 16; ++m) {
        const int k = grp + m * kGroups;
        if (k < np)
            acc += s_w[k] * v[m];
    }
    for (int k0 = grp + 16 * kGroups; k0 < np; k0 += kGroups * 16) {
#pragma unroll
        for (int m = 0; m < 16; ++m) {
            const int k = k0 + m * kGroups;
            v[m] = k < np ? __ldcg(src + static_cast<size_t>(k) * G * D) : 0.f;
        }
#pragma unroll
        for (int m = 0; m < 16; ++m) {
            const int k = k0 + m * kGroups;
            if (k < np)
                acc += s_w[k] * v[m];
        }
    }
    __syncthreads();   // every thread has read the warps' sums
    s_red[tid] = acc;
    __syncthreads();
    if (grp == 0) {
        float sum = 0.f;
#pragma unroll
        for (int q = 0; q < kGroups; ++q)
            sum += s_red[q * D + e];
        out[(static_cast<size_t>(beta) * p.h + static_cast<size_t>(j) * G + row) * D + e] =
            __float2bfloat16_rn(sum * inv);
    }
}

// ------------------------------------------------------------------------------------------------
// append kernel: one thread per 16-byte vector of the new token's K/V rows
// ------------------------------------------------------------------------------------------------

__global__ void append_kernel(const __grid_constant__ AppendParams p)
{
    grid_dependency_wait();
    grid_dependents_launch();
    const int vecs = p.d / 8;
    const long long total = 2LL * p.b * p.g * vecs;
    const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= total)
        return;
    const int v = static_cast<int>(idx % vecs);
    long long row = idx / vecs;   // (kv, beta, j)
    const int j = static_cast<int>(row % p.g);
    row /= p.g;
    const int beta = static_cast<int>(row % p.b);
    const int kv = static_cast<int>(row / p.b);
    const int pos = p.seq_len[beta] - 1;
    const uint4 *src = reinterpret_cast<const uint4 *>(kv ? p.V : p.K) +
                       (static_cast<size_t>(beta) * p.g + j) * vecs + v;
    uint4 *dst = reinterpret_cast<uint4 *>(p.cache) +
                 ((((static_cast<size_t>(p.slot) * 2 + kv) * p.b + beta) * p.g + j) *
                      static_cast<size_t>(p.max_seq) + pos) * vecs + v;
    *dst = *src;
}

template <int D, int T, int STAGES, int NCW>
constexpr DecodeVariant make_variant()
{
    using PL = Plan<D, T, STAGES, NCW>;
    return DecodeVariant{D, T, STAGES, PL::kThreads, static_cast<size_t>(PL::kAlloc),
                         static_cast<size_t>(PL::kResBytes),
                         reinterpret_cast<const void *>(&decode_kernel<D, T, STAGES, NCW>)};
}

// (head_dim, positions per tile, ring stages, consumer warps); the first match of a
// (head_dim, tile) pair is used.  <64, 128, 2, 4> fits twice on an SM (90 KB, 167 registers).
const DecodeVariant kVariants[] = {
    make_variant<64, 128, 2, 4>(),
    make_variant<64, 256, 3, 4>(),
    make_variant<64, 64, 4, 4>(),
    make_variant<128, 64, 5, 4>(),
    make_variant<128, 128, 2, 4>(),
};

}  // namespace

const DecodeVariant *find_decode_variant(int head_dim, int tile_tokens, int tc)
{
    if (tc) {
        for (int i = 0; i < kNumTcVariants; ++i)
            if (kTcVariants[i].head_dim == head_dim && kTcVariants[i].tile_tokens == tile_tokens)
                return &kTcVariants[i];
        return nullptr;
    }
    for (const DecodeVariant &v : kVariants)
        if (v.head_dim == head_dim && v.tile_tokens == tile_tokens)
            return &v;
    return nullptr;
}

cudaError_t prepare_decode_variant(const DecodeVariant &v, size_t max_smem)
{
    size_t tail = table_bytes(MLKV_MAX_BATCH);
    if (3 * v.res_bytes > tail)
        tail = 3 * v.res_bytes;   // cluster mode, k = 4
    size_t want = v.smem_bytes + tail;
    if (want > max_smem)
        want = max_smem;
    if (v.smem_bytes > want)
        return cudaErrorInvalidValue;
    return cudaFuncSetAttribute(v.fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(want));
}

cudaError_t launch_decode(const DecodeVariant &v, int grid, size_t smem, cudaStream_t stream,
                          const CUtensorMap *tmap, const CUtensorMap *tmap_rows,
                          const DecodeParams &p, const cudaAccessPolicyWindow *window, bool pdl)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(static_cast<unsigned>(v.threads));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[3];
    int na = 0;
    if (pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    if (p.cluster_k > 1) {
        attr[na].id = cudaLaunchAttributeClusterDimension;
        attr[na].val.clusterDim.x = static_cast<unsigned>(p.cluster_k);
        attr[na].val.clusterDim.y = 1;
        attr[na].val.clusterDim.z = 1;
        ++na;
    }
    if (window != nullptr) {
        attr[na].id = cudaLaunchAttributeAccessPolicyWindow;
        attr[na].val.accessPolicyWindow = *window;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    void *args[] = {const_cast<CUtensorMap *>(tmap), const_cast<CUtensorMap *>(tmap_rows),
                    const_cast<DecodeParams *>(&p)};
    return cudaLaunchKernelExC(&cfg, v.fn, args);
}

int max_pieces_per_segment(const DecodeParams &p, int T, int grid)
{
    const long long N = p.num_tiles;
    if (grid <= 1 || N <= 0)
        return 1;
    if (p.uniform_len > 0) {
        // Every CTA holds at least floor(N/grid) tiles, so a segment of nt tiles meets at most
        // ceil((nt - 1) / floor(N/grid)) + 1 of them.
        const long long nt = (p.uniform_len + T - 1) / T;
        const long long per = N / grid;
        if (per <= 0)
            return grid;
        return static_cast<int>((nt - 1 + per - 1) / per + 1);
    }
    auto cta_of = [&](long long tile) { return static_cast<int>(((tile + 1) * grid - 1) / N); };
    int worst = 1;
    for (int beta = 0; beta < p.b; ++beta) {
        const int nt = (p.seq_len[beta] + T - 1) / T;
        for (int j = 0; j < p.g; ++j) {
            const long long first =
                static_cast<long long>(p.tile_start[beta]) + static_cast<long long>(j) * nt;
            const int np = cta_of(first + nt - 1) - cta_of(first) + 1;
            worst = np > worst ? np : worst;
        }
    }
    return worst;
}

cudaError_t launch_combine(const DecodeParams &p, int head_dim, cudaStream_t stream, bool pdl)
{
    cudaLaunchConfig_t cfg = {};
    const int segs = p.b * p.g * (p.ml_layers > 0 ? p.ml_layers : 1);
    cfg.gridDim = dim3(static_cast<unsigned>(segs), static_cast<unsigned>(p.G));
    cfg.blockDim = dim3(kCombineThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    void *args[] = {const_cast<DecodeParams *>(&p)};
    const void *fn = head_dim == 64 ? reinterpret_cast<const void *>(&combine_kernel<64>)
                                    : reinterpret_cast<const void *>(&combine_kernel<128>);
    return cudaLaunchKernelExC(&cfg, fn, args);
}

cudaError_t max_active_clusters(const DecodeVariant &v, int k, int *out)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(k));
    cfg.blockDim = dim3(static_cast<unsigned>(v.threads));
    cfg.dynamicSmemBytes = v.smem_bytes + (k - 1) * v.res_bytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(k);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaOccupancyMaxActiveClusters(out, v.fn, &cfg);
}

cudaError_t launch_append(const AppendParams &p, cudaStream_t stream)
{
    const long long total = 2LL * p.b * p.g * (p.d / 8);
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
    return cudaLaunchKernelExC(&cfg, reinterpret_cast<const void *>(&append_kernel), args);
}

}  // namespace mlkv
