// MLKV prefill attention on the 5th-generation tensor cores (tcgen05, tensor memory) for GB300.
//
// Prefill runs a whole prompt through one layer at once: prompt position t of query head i
// attends to positions 0 .. t of KV head j(i) = i / G of the layer's owner slot (causal
// attention, Eqs. 2-3 with the MLKV maps of Eqs. 13-18).  Owner layers first store the prompt's
// K/V in their slot (mlkv_host.cpp); every layer of the block then attends over it.
//
// Work unit (one CTA), head_dim 128: two query tiles A and B of 128 prompt positions that read the
// same KV head, so that every K/V tile is loaded once for both.  With an even group size G they are
// two heads of one group at the same positions (identical causal triangles); otherwise they are the
// blocks 2p and 2p+1 of one head (B sees one tile more; a last block without a partner runs alone
// as B).  Prefill at head_dim 64: one query tile (as B) per CTA and two CTAs per SM, each with half
// the tensor memory; the two CTAs' starts, first loads and outputs overlap each other's key-tile
// loops (measured 8% faster than two tiles per CTA, although every K/V tile is then fetched once
// per query tile).  Units that see the most keys run first.
//
// Fused decode (one new token per sequence, every layer of an owner block at once, Sec. 3): the
// query rows of a unit are the G heads of KV head j in each of the block's L layers, row = layer * G
// + head, layers [0, L1) in tile B and [L1, L) in tile A (L1 = 128 / G); a unit takes one chunk of
// the sequence's key tiles and reads each K/V tile once for all L * G rows.  At head_dim 64 with
// L * G <= 128 a one-tile form runs it: with at most one unit per SM the deep form (one CTA per SM,
// a 12-tile ring, key tiles alternating between two softmax warpgroups), else two CTAs per SM;
// otherwise the two-tile form.
//
// Per key tile t and query tile X (all MMAs tcgen05.mma kind::f16, bf16 in, fp32 accumulate):
//   S_X = Q_X K_t^T  M = 128 queries (A = Q_X, K-major, 128-byte swizzle as TMA wrote it),
//                    N = 128 keys (B = the K tile), K = head_dim; one query row per TMEM lane.
//   softmax          a warpgroup per query tile, one thread per row: the thread owns its row's
//                    128 scores, so the running maximum needs no exchange between threads.  The
//                    reference maximum is raised only when a score exceeds it by more than 2^8
//                    (then the thread rescales its O row in TMEM); p = 2^(s log2(e)/sqrt(d) - m)
//                    goes back to TMEM as bf16 pairs.
//   O_X += P_X V_t   A = P_X read from TMEM, B = the V tile read MN-major from shared memory,
//                    N = head_dim, K = 128 keys; O_X stays in TMEM for the whole unit.
// While one warpgroup turns S into P, the tensor core works on the other query tile.
//
// TMEM (512 columns, 256 with one query tile): S per tile (128 columns), O per tile (head_dim).
// For head_dim 64, P has columns of its own (so S of the next tile can be computed while P of this
// one is being written); for head_dim 128, P overwrites the first 64 columns of its S (tcgen05.mma
// of one thread execute in order, so S of the next tile is written after P V has read P).
//
// The diagonal tile masks keys after the query; keys past the prompt's end only meet such masked
// scores, and their V rows are zeroed in shared memory so that 0 * V stays 0.
//
// Warp roles: 4 softmax warps per query tile (warps 0-3 tile A, 4-7 tile B; the one-tile CTA's
// warps 0-3 take its tile), then the TMA producer (query tiles, then K_0, V_0, K_1, V_1, ...
// through a ring), the MMA issuer (for head_dim 64 only of S, the next warp issuing the P V
// products), the rest idle.  Registers: the two-tile block launches with 168 a thread and its last
// warpgroup gives registers back (72 or 88) to the softmax warpgroups (216 or 208, head_dim 64 or
// 128): 128 * low + 256 * high <= 384 * 168; the one-tile block launches with 128 (two blocks per
// SM) and splits 56 / 200: 128 * 56 + 128 * 200 = 256 * 128.
// Every wait is bounded; on expiry the kernel records an error bit, stops, lets its copies and MMAs
// land and frees its TMEM.
#include <type_traits>

#include "mlkv_device.cuh"
#include "mlkv_tcgen05.cuh"

namespace mlkv {
namespace {

// Forms of the CTA (kForm):
//   kTwoTiles  two query tiles share every K/V tile, one CTA per SM (head_dim 128; the fused
//              decode of blocks whose rows exceed one tile);
//   kOneTile   one query tile per CTA and two CTAs per SM (prefill at head_dim 64; the fused
//              decode with more units than SMs): each CTA holds half the tensor memory and a third
//              of the registers of the two-tile form, and two independent CTAs hide each other's
//              start, first loads and output;
//   kOneDeep   one query tile, one CTA per SM (the fused decode with at most one unit per SM, its
//              K/V tiles streamed from HBM): a ring of 12 tiles keeps ~6 K/V pairs in flight, and
//              the key tiles alternate between two softmax warpgroups on the same 128 query rows,
//              each with its own S, P and O columns and its own running maximum and sum, merged
//              per row at the end -- two key tiles' softmax chains run at once, and S of the next
//              tile is computed while this one's softmax runs.
constexpr int kTwoTiles = 0, kOneTile = 1, kOneDeep = 2;

template <int D, int kForm>
struct PrefillPlan {
    static constexpr bool kOne = kForm != kTwoTiles;
    static constexpr int kTiles = kOne ? 1 : 2;              // query tiles per CTA
    static constexpr int kSBuf = kForm == kOneDeep ? 2 : 1;  // S, P and O buffers per query tile
    static constexpr int kSoftWarps = 4 * kTiles * kSBuf;    // a warpgroup per tile or buffer
    static constexpr int kThreads = (kSoftWarps + 4) * 32;
    static constexpr int kMinBlocks = kForm == kOneTile ? 2 : 1;
    // registers at launch, then the other warps' share and the softmax warps' (setmaxnreg)
    static constexpr int kRegsLaunch = kForm == kOneTile ? 128 : 168;
    static constexpr int kRegsLow = kForm == kOneTile ? 56 : (D == 64 ? 72 : 88);
    static constexpr int kRegsHigh = kForm == kOneTile ? 200 : (D == 64 ? 216 : 208);
    static constexpr int kProducer = kSoftWarps, kMma = kSoftWarps + 1;
    static constexpr int kSub = D / 64;                      // 64-channel blocks of a row
    static constexpr int kTileBytes = 128 * D * 2;           // 128 rows of Q, K or V
    // K_t and V_t alternate in the ring
    static constexpr int kRingTiles = kForm == kOneDeep ? 12 : kOne ? 5 : (D == 64 ? 8 : 4);
    static constexpr int kQ = 0;                             // [kTiles] query tiles
    static constexpr int kRing = kQ + kTiles * kTileBytes;
    static constexpr int kFlags = kRing + kRingTiles * kTileBytes;   // int [4], TMEM base at +16
    // u64 barriers: q, full[R], empty[R], s_ready[2], s_free[2], p_ready[2], pv_done[2], fin[2]
    // (s_ready and s_free per query tile, or per S buffer in the deep form)
    static constexpr int kBars = kFlags + 32;
    static constexpr int kNumBars = 1 + 2 * kRingTiles + 8 + 2;
    // the second warpgroup's running maximum and sum per row, for the merge (two buffers)
    static constexpr int kML = kBars + kNumBars * 8;
    static constexpr int kBytes = kML + (kSBuf == 2 ? 128 * 8 : 0);
    static constexpr int kAlloc = kBytes + 1024;             // base aligned up to 1024
    static_assert(kMinBlocks * (kAlloc + 1024) <= 228 * 1024, "shared memory of the resident CTAs");
    static constexpr int kTmemCols = kForm == kOneTile ? 256 : 512;
    static constexpr bool kPSep = D == 64;                   // P in columns of its own
    static constexpr int kColS = 0;                          // + 128 per query tile or buffer
    static constexpr int kColO = 128 * kTiles * kSBuf;       // + D per query tile or buffer
    static constexpr int kColP = kColO + D * kTiles * kSBuf; // + 64 per tile or buffer (kPSep)
    static_assert(D == 64 || D == 128, "head_dim 64 or 128");
    static_assert(!kOne || D == 64, "one query tile per CTA only at head_dim 64");
    static_assert(kRing % 1024 == 0 && kTileBytes % 1024 == 0, "swizzled tiles 1024-aligned");
    static_assert((kPSep ? kColP + 64 * kTiles * kSBuf : kColO + D * kTiles) <= kTmemCols,
                  "TMEM columns overlap");
    static_assert(128 * kRegsLow + 32 * kSoftWarps * kRegsHigh <= kThreads * kRegsLaunch,
                  "register split");
    static_assert(kMinBlocks * kThreads * kRegsLaunch <= 65536, "registers of the resident CTAs");
    static_assert(kSBuf == 1 || (kTiles == 1 && kPSep), "two buffers: one tile, P apart");
};

template <int N>
__device__ __forceinline__ void setmaxnreg_inc()
{
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

template <int N>
__device__ __forceinline__ void setmaxnreg_dec()
{
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}

__device__ __forceinline__ float max3f(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

template <int D, bool kFused, int kForm>
__global__ void __launch_bounds__(PrefillPlan<D, kForm>::kThreads,
                                  PrefillPlan<D, kForm>::kMinBlocks)
    prefill_kernel(const __grid_constant__ CUtensorMap tmap_q,
                   const __grid_constant__ CUtensorMap tmap_kv,
                   const __grid_constant__ PrefillParams p)
{
    using PL = PrefillPlan<D, kForm>;
    constexpr bool kSplit = PL::kSBuf == 2;   // key tiles alternate between two warpgroups
    // Query tile g's shared-memory slot and tensor-memory columns (the only tile of a one-tile CTA
    // is tile B, in slot 0).
    auto slot_of = [](int g) { return PL::kTiles == 1 ? 0 : g; };
    constexpr int R = PL::kRingTiles;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_addr(smem);
    const uint32_t bar_q = sbase + PL::kBars;
    const uint32_t bar_full = bar_q + 8;
    const uint32_t bar_empty = bar_full + 8 * R;
    const uint32_t bar_s_ready = bar_empty + 8 * R;   // [2] per query tile
    const uint32_t bar_s_free = bar_s_ready + 16;
    const uint32_t bar_p_ready = bar_s_free + 16;
    const uint32_t bar_pv_done = bar_p_ready + 16;
    const uint32_t bar_fin = bar_pv_done + 16;   // [2]: one per issuing thread
    volatile int *flags = reinterpret_cast<volatile int *>(smem + PL::kFlags);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // The unit: sequence, last query block of B, head pair or head (see PrefillParams::units).
    // Fused decode: sequence, KV head j and owner block blk; S is then the sequence length, every
    // query row sees positions [0, S), and the tiles hold the block's layers [0, L1) (B) and
    // [L1, L) (A).
    const uint32_t u = p.units[blockIdx.x];
    const int beta = static_cast<int>(u & 0x3FFu);
    const int sel = static_cast<int>(u >> 24);
    const int S = p.prompt_len[beta];
    // Fused decode: key tiles [kt0, kt0 + n_b) of the sequence (a chunk of p.fused_kc tiles).
    const int chunk = static_cast<int>((u >> 10) & (kFused ? 0xFFu : 0x3FFFu));
    const int blk = kFused ? static_cast<int>((u >> 18) & 0x3Fu) : 0;
    const int n_kt = (S + 127) / 128;
    const int kt0 = kFused ? chunk * p.fused_kc : 0;
    const int kt1 = kFused ? min(kt0 + p.fused_kc, n_kt) : 0;
    const bool has_end = !kFused || kt1 == n_kt;   // the unit holds the sequence's last tile
    const int qb_b = kFused ? kt1 - kt0 - 1 : chunk;
    const int head_a = p.head_pairs ? 2 * sel : sel;
    const int head_b = p.head_pairs ? 2 * sel + 1 : sel;
    const int n_b = qb_b + 1;                                   // key tiles 0 .. qb_b
    const int n_a = PL::kTiles == 1 ? 0
                    : kFused ? (p.fused_L > p.fused_L1 ? n_b : 0)
                             : (p.head_pairs ? n_b : ((qb_b & 1) ? qb_b : 0));   // 0: no tile A
    const int j = kFused ? sel : head_b / p.G;                  // Eq. 15
    const int zk = (((p.slot + blk) * 2 + 0) * p.b + beta) * p.g + j;
    const int zv = zk + p.b * p.g;

    if (threadIdx.x == 0) {
        // the query tiles' barrier: the producer's tensor-map copy, or every softmax warp's share
        // of the rows read from host memory
        mbar_init(bar_q, (kFused && p.q_host != nullptr) ? PL::kSoftWarps : 1);
        for (int s = 0; s < R; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
        }
        for (int g = 0; g < 2; ++g) {
            mbar_init(bar_s_ready + 8 * g, 1);
            mbar_init(bar_s_free + 8 * g, 4);
            mbar_init(bar_p_ready + 8 * g, 4);
            mbar_init(bar_pv_done + 8 * g, 1);
        }
        mbar_init(bar_fin, 1);
        mbar_init(bar_fin + 8, 1);
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
    if (kFused && warp < PL::kSoftWarps) {
        // The tiles' rows past the loaded ones (the TMA box, G x min(L1, L) rows) are never
        // written; zero them so that their (discarded) scores stay finite.
        const int grp = PL::kTiles == 1 ? 1 : warp >> 2, r = threadIdx.x & 127;
        const int box_rows = (p.fused_L < p.fused_L1 ? p.fused_L : p.fused_L1) * p.G;
        // rows the load writes: the box (tensor map), or tile A's own rows (read from host)
        const int keep = (p.q_host != nullptr && grp == 0) ? (p.fused_L - p.fused_L1) * p.G
                                                           : box_rows;
        if (r >= keep && warp < 4 * PL::kTiles) {   // one warpgroup per query tile
            uint8_t *qrow = smem + PL::kQ + slot_of(grp) * PL::kTileBytes;
#pragma unroll
            for (int c = 0; c < 8 * PL::kSub; ++c)
                *reinterpret_cast<uint4 *>(qrow + (c >> 3) * 16384 + r * 128 +
                                           (((c & 7) ^ (r & 7)) << 4)) = make_uint4(0, 0, 0, 0);
            fence_proxy_async_smem();
        }
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + PL::kFlags + 16);
    // The owner's K/V may have just been stored by the previous kernel of the stream.  In the
    // fused step that kernel stores only position L - 1 of each slot and was itself launched after
    // every earlier kernel had finished (it triggers this launch only after its own dependency
    // wait): the queries and every tile but the one holding position L - 1 are loaded at once, the
    // producer waits before that tile, and the output waits before its stores.
    const bool early = kFused && p.fused_early;
    const bool q_early = kFused && p.fused_early == 1;   // the queries before the wait too
    if (!early)
        grid_dependency_wait();
    grid_dependents_launch();
    if (warp == PL::kProducer) {
        // ------------------------------------ producer ------------------------------------------
        setmaxnreg_dec<PL::kRegsLow>();
        if (lane == 0) {
            bool waited = !early;
            // mode 2: the cache tiles that hold no new row first, as far as the ring goes
            int idx_pre = 0;
            if (early && !q_early) {
                const int n_pre = 2 * n_b < R ? 2 * n_b : R;
                for (; idx_pre < n_pre; ++idx_pre) {
                    if (has_end && (idx_pre >> 1) + kt0 == n_kt - 1)
                        break;
                    const uint32_t fb = bar_full + 8 * idx_pre;
                    mbar_arrive_expect_tx(fb, PL::kTileBytes);
                    const uint32_t dst = sbase + PL::kRing + idx_pre * PL::kTileBytes;
                    const int z = (idx_pre & 1) ? zv : zk;
#pragma unroll
                    for (int sub = 0; sub < PL::kSub; ++sub)
                        tma_load_3d(dst + sub * 16384, &tmap_kv, fb, sub * 64,
                                    ((idx_pre >> 1) + kt0) * 128, z);
                }
                grid_dependency_wait();   // the step's inputs are in place
                waited = true;
            }
            if (kFused && p.q_host != nullptr) {
                // the softmax warps read the queries from host memory
            } else if (kFused) {
                // Q [layers][b][h][D] as (channel, head in group, group, sequence, layer): a box
                // of min(L1, L) layers x G heads = the tile's rows, layer-major (row = layer*G + i),
                // from the block's first layer (tile B) and its layer L1 (tile A).
                const int box_rows = (p.fused_L < p.fused_L1 ? p.fused_L : p.fused_L1) * p.G;
                const int lay0 = blk * p.fused_L;
                mbar_arrive_expect_tx(bar_q, (n_a > 0 ? 2 : 1) * PL::kSub * box_rows * 128);
#pragma unroll
                for (int sub = 0; sub < PL::kSub; ++sub) {
                    if (n_a > 0)
                        tma_load_5d(sbase + PL::kQ + sub * 16384, &tmap_q, bar_q, sub * 64, 0, j,
                                    beta, lay0 + p.fused_L1);
                    tma_load_5d(sbase + PL::kQ + slot_of(1) * PL::kTileBytes + sub * 16384,
                                &tmap_q, bar_q, sub * 64, 0, j, beta, lay0);
                }
            } else {
                mbar_arrive_expect_tx(bar_q, (n_a > 0 ? 2 : 1) * PL::kTileBytes);
#pragma unroll
                for (int sub = 0; sub < PL::kSub; ++sub) {
                    if (n_a > 0)
                        tma_load_4d(sbase + PL::kQ + sub * 16384, &tmap_q, bar_q, sub * 64,
                                    head_a, (n_a - 1) * 128, beta);
                    tma_load_4d(sbase + PL::kQ + slot_of(1) * PL::kTileBytes + sub * 16384, &tmap_q,
                                bar_q, sub * 64, head_b, qb_b * 128, beta);
                }
            }
            const int n_idx = 2 * n_b;   // K_0, V_0, K_1, V_1, ...
            int idx = idx_pre;
            for (; idx < n_idx; ++idx) {
                const int s = idx % R;
                if (idx >= R && !flags[0] &&
                    !mbar_wait(bar_empty + 8 * s, ((idx / R) & 1) ^ 1)) {
                    flags[0] = 1;
                    atomicOr(p.err, kErrWaitEmpty);
                }
                if (flags[0])
                    break;
                if (!waited && has_end && (idx >> 1) + kt0 == n_kt - 1) {
                    grid_dependency_wait();   // the tile that holds the new row
                    waited = true;
                }
                const uint32_t fb = bar_full + 8 * s;
                mbar_arrive_expect_tx(fb, PL::kTileBytes);
                const uint32_t dst = sbase + PL::kRing + s * PL::kTileBytes;
                const int z = (idx & 1) ? zv : zk;
#pragma unroll
                for (int sub = 0; sub < PL::kSub; ++sub)
                    tma_load_3d(dst + sub * 16384, &tmap_kv, fb, sub * 64,
                                ((idx >> 1) + kt0) * 128, z);
            }
            // No copy may still be in flight when the CTA exits.
            if (!mbar_wait(bar_q, 0))
                atomicOr(p.err, kErrDrain);
            for (int k = idx > R ? idx - R : 0; k < idx; ++k)
                if (!mbar_wait(bar_full + 8 * (k % R), (k / R) & 1))
                    atomicOr(p.err, kErrDrain);
        }
        __syncwarp();
    } else if (warp == PL::kMma || (PL::kPSep && warp == PL::kMma + 1)) {
        // ------------------------------------ MMA issuers ---------------------------------------
        // With P in columns of its own (head_dim 64) warp kMma issues every S = Q K^T and warp
        // kMma + 1 every O += P V: the two never touch the same tensor-memory columns, each waits
        // only for what its own products need, and the tensor core gets both streams.  (One thread
        // issuing both spent about a third of each key tile on barrier checks while the tensor core
        // ran dry.)  With P over S (head_dim 128) one thread issues both, in order.
        setmaxnreg_dec<PL::kRegsLow>();
        const bool do_s = warp == PL::kMma, do_pv = !PL::kPSep || warp == PL::kMma + 1;
        const uint32_t my_fin = bar_fin + (warp == PL::kMma ? 0 : 8);
        if (lane == 0) {
            constexpr uint32_t kIdS = umma_idesc(128, 128, 0, 0);
            constexpr uint32_t kIdPV = umma_idesc(128, D, 0, 1);
            constexpr uint32_t kSlot = PL::kTileBytes >> 4;   // one ring slot in descriptor units
            // Descriptors of query tile A and of ring slot 0.  A tile, a slot, a K step or a
            // 64-channel block only moves the start-address field (shared addresses < 256 KB), so
            // each MMA's descriptors are one add away; the tensor core queues little, and any
            // latency between two MMAs of this thread leaves it idle.
            const uint64_t dq = umma_desc(sbase + PL::kQ, 16, 1024, kLayoutSw128);
            const uint64_t dk = umma_desc(sbase + PL::kRing, 16, 1024, kLayoutSw128);
            const uint64_t dv = umma_desc(sbase + PL::kRing, 16384, 1024, kLayoutSw128);
            bool ok = true;
            auto wait = [&](uint32_t bar, int parity) {
                const uint32_t par = static_cast<uint32_t>(parity) & 1u;
                if (ok && !mbar_test_wait(bar, par) && !mbar_wait(bar, par))
                    ok = false;
                return ok;
            };
            // Each ring tile is checked once: the K tile serves both query tiles' S, the V tile
            // both P V (a check costs ~150 cycles while the MMAs keep shared memory busy).
            int seen0 = -1, seen1 = -1;
            auto tile_full = [&](int idx) {
                if (idx == seen0 || idx == seen1)
                    return ok;
                if (wait(bar_full + 8 * (idx % R), idx / R)) {
                    seen1 = seen0;
                    seen0 = idx;
                }
                return ok;
            };
            auto issue_s = [&](int g, int t) {
                const uint64_t qa = dq + slot_of(g) * kSlot;
                const uint64_t kb = dk + ((2 * t) % R) * kSlot;
                const int sb = kSplit ? (t & 1) : g;   // S buffer and its barrier
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    const uint32_t off = (k >> 2) * 1024 + (k & 3) * 2;   // 16384 B, 32 B
                    umma_f16(tmem + PL::kColS + 128 * (kSplit ? sb : slot_of(g)), qa + off,
                             kb + off, kIdS, k > 0 ? 1 : 0);
                }
                umma_commit(bar_s_ready + 8 * sb);
            };
            auto issue_pv = [&](int g, int t, bool last) {
                const uint64_t vb = dv + ((2 * t + 1) % R) * kSlot;
                const int sg = slot_of(g);
                const int ob = kSplit ? (t & 1) : sg;   // P and O buffer (warpgroup t mod 2)
                const uint32_t pc =
                    tmem + (PL::kPSep ? PL::kColP + 64 * ob : PL::kColS + 128 * sg);
                const bool first = kSplit ? t < 2 : t == 0;   // the buffer's first product
#pragma unroll
                for (int k = 0; k < 8; ++k)   // 16 keys = 2048 B of V, 8 TMEM columns of P
                    umma_f16_ts(tmem + PL::kColO + D * ob, pc + 8 * k, vb + k * 128, kIdPV,
                                (!first || k > 0) ? 1 : 0);
                // With P over S, the next S's completion already implies this product's.
                if (PL::kPSep || last)
                    umma_commit(bar_pv_done + 8 * (kSplit ? (t & 1) : g));
            };
            if (do_s && wait(bar_q, 0) && tile_full(0)) {
                tmem_fence_after();
                if (n_a > 0)
                    issue_s(0, 0);
                issue_s(1, 0);
            }
            // Ring slots are released by tile B's softmax warps (they see every MMA that read them
            // complete), not by commits: a commit costs the tensor pipe about as much as a short MMA.
            for (int t = 0; ok && t < n_b; ++t) {
                if (PL::kPSep) {
                    // S issuer: both tiles' next S as soon as each tile's S has been read (early in
                    // its softmax).  P V issuer: both P V as their P arrive.
#pragma unroll
                    for (int g = 0; g < 2; ++g) {
                        const int ng = g ? n_b : n_a;
                        if (!do_s || !ok || t + 1 >= ng)
                            continue;
                        // S(t + 1) once its columns are free: tile t's S read (one buffer), or
                        // tile t - 1's (two buffers: S(t + 1) then runs during tile t's softmax)
                        if (kSplit ? (t >= 1 && !wait(bar_s_free + 8 * ((t + 1) & 1), (t - 1) >> 1))
                                   : !wait(bar_s_free + 8 * g, t))
                            break;
                        if (!tile_full(2 * t + 2))
                            break;
                        tmem_fence_after();
                        issue_s(g, t + 1);
                    }
#pragma unroll
                    for (int g = 0; g < 2; ++g) {
                        const int ng = g ? n_b : n_a;
                        if (!do_pv || !ok || t >= ng)
                            continue;
                        if (!tile_full(2 * t + 1) ||
                            !wait(bar_p_ready + 8 * (kSplit ? (t & 1) : g), kSplit ? (t >> 1) : t))
                            break;
                        tmem_fence_after();
                        issue_pv(g, t, t + 1 >= ng);
                    }
                    continue;
                }
#pragma unroll
                for (int g = 0; g < 2; ++g) {
                    const int ng = g ? n_b : n_a;
                    if (!ok || t >= ng)
                        continue;
                    const bool next = t + 1 < ng;
                    {
                        // Everything first, then P V and the next S back to back.
                        if (!tile_full(2 * t + 1) || (next && !tile_full(2 * t + 2)) ||
                            !wait(bar_p_ready + 8 * g, t))
                            break;
                        tmem_fence_after();
                        issue_pv(g, t, !next);
                        if (next)
                            issue_s(g, t + 1);
                    }
                }
            }
            if (!ok) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
            umma_commit(my_fin);
            if (!mbar_wait(my_fin, 0))
                atomicOr(p.err, kErrDrain);
        }
        __syncwarp();
    } else if (warp < PL::kSoftWarps) {
        // ------------------------------------ softmax warpgroups --------------------------------
        setmaxnreg_inc<PL::kRegsHigh>();
        const int grp = PL::kTiles == 1 ? 1 : warp >> 2;   // 0: query tile A, 1: query tile B
        const int r = threadIdx.x & 127;            // query row of the tile = TMEM lane
        const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const int n_g = grp ? n_b : n_a;
        const int head = grp ? head_b : head_a;
        const int q0 = (kt0 + n_g - 1) * 128;       // first position of the unit's last tile
        const int sg = slot_of(grp);
        // the warpgroup's buffer: the tile's own, or (split keys) this warpgroup's tiles t = wg,
        // wg + 2, ... with S, P and O buffer wg
        const int wg = kSplit ? warp >> 2 : 0;
        const int bsel = kSplit ? wg : grp;
        const uint32_t col_s = tmem + lane_off + PL::kColS + 128 * (kSplit ? wg : sg);
        const uint32_t col_o = tmem + lane_off + PL::kColO + D * (kSplit ? wg : sg);
        const uint32_t col_p =
            tmem + lane_off +
            (PL::kPSep ? PL::kColP + 64 * (kSplit ? wg : sg) : PL::kColS + 128 * sg);
        const uint32_t s_ready = bar_s_ready + 8 * bsel, s_free = bar_s_free + 8 * bsel;
        const uint32_t p_ready = bar_p_ready + 8 * bsel, pv_done = bar_pv_done + 8 * bsel;
        constexpr int kStep = kSplit ? 2 : 1;   // tiles between this warpgroup's
        // The prompt's last block holds keys past its end; the first tile to reach it zeroes them.
        const bool zero_v = n_g > 0 && (kFused ? has_end : n_g == (S + 127) / 128) &&
                            (grp == 0 || n_a != n_b);
        const float scale = p.scale_log2;
        const float NEG_INF = -__int_as_float(0x7f800000);
        auto wait = [&](uint32_t bar, int parity) {
            if (!flags[0] && !mbar_wait(bar, static_cast<uint32_t>(parity) & 1u)) {
                flags[0] = 1;
                atomicOr(p.err, kErrWaitFull);
            }
        };
        if (kFused && p.q_host != nullptr) {
            // The unit's query rows from page-locked host memory through its device-mapped
            // address (16 bytes a load, four in flight per thread), written into the query tiles
            // the way the tensor map would have (128-byte swizzle); rows past them stay zero.
            const int nth = 32 * PL::kSoftWarps;
            const int L1r = p.fused_L < p.fused_L1 ? p.fused_L : p.fused_L1;
            const int rows_b = L1r * p.G;
            const int rows_a = n_a > 0 ? (p.fused_L - p.fused_L1) * p.G : 0;
            constexpr int kC = D / 8;   // 16-byte chunks of a row
            const int total = (rows_b + rows_a) * kC;
            for (int k0 = threadIdx.x; k0 < total; k0 += 4 * nth) {
                uint4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int k = k0 + u * nth;
                    if (k < total) {
                        const int rr = k / kC, c = k - rr * kC;
                        const bool in_b = rr < rows_b;
                        const int rw = in_b ? rr : rr - rows_b;
                        const int lay = blk * p.fused_L + (in_b ? 0 : p.fused_L1) + rw / p.G;
                        v[u] = *reinterpret_cast<const uint4 *>(
                            p.q_host + ((static_cast<size_t>(lay) * p.b + beta) * p.h + j * p.G +
                                        rw % p.G) * D + c * 8);
                    }
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int k = k0 + u * nth;
                    if (k < total) {
                        const int rr = k / kC, c = k - rr * kC;
                        const bool in_b = rr < rows_b;
                        const int rw = in_b ? rr : rr - rows_b;
                        *reinterpret_cast<uint4 *>(smem + PL::kQ +
                                                   slot_of(in_b ? 1 : 0) * PL::kTileBytes +
                                                   (c >> 3) * 16384 + rw * 128 +
                                                   (((c & 7) ^ (rw & 7)) << 4)) = v[u];
                    }
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(bar_q);
        }
        float m_run = NEG_INF, l_run = 0.f;
        for (int t = wg; t < n_g; t += kStep) {
            const int u = kSplit ? t >> 1 : t;   // this warpgroup's use of its buffers
            wait(s_ready, u);
            // Tile B's first warp frees ring slots whose readers have all completed: K_t once S_B(t)
            // is done (S_A(t) was issued before it by the same thread); V_{t-1} once S_B(t) (P over
            // S: issued after P V_{t-1}) or P_B V_{t-1} (own P) is done.
            const bool releaser = grp == 1 && (warp & 3) == 0 && lane == 0;
            if (releaser && (t == 0 || PL::kPSep))   // K_t
                mbar_arrive(bar_empty + 8 * ((2 * t) % R));
            if (releaser && t > 0 && !PL::kPSep) {
                mbar_arrive(bar_empty + 8 * ((2 * t - 1) % R));
                mbar_arrive(bar_empty + 8 * ((2 * t) % R));
            }
            const bool diag = t == n_g - 1 && has_end;
            // This tile's scores, with the causal (or sequence-end) mask of the last tile.
            float sv[4][32];
            auto load_scores = [&]() {
                tmem_fence_after();
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    tmem_ld32_nowait(col_s + c * 32, sv[c]);
                tmem_wait_ld();
                if (diag) {
                    // Keys [0, lim) of the tile are visible: up to the sequence's end (fused
                    // decode) or to the query's own position (causal mask).
                    const int lim = kFused ? S - q0 : r + 1;
#pragma unroll
                    for (int c = 0; c < 4; ++c)
#pragma unroll
                        for (int k = 0; k < 32; ++k)
                            if (c * 32 + k >= lim)
                                sv[c][k] = NEG_INF;
                }
            };
            // Raises the reference maximum to the tile's when a score exceeds it by more than 2^8
            // (the thread then rescales its O row in TMEM).
            auto raise_to_tile_max = [&]() {
                float mx[4];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    float a = max3f(sv[c][0], sv[c][1], sv[c][2]);
                    float b = max3f(sv[c][3], sv[c][4], sv[c][5]);
#pragma unroll
                    for (int k = 6; k < 30; k += 4) {
                        a = max3f(a, sv[c][k], sv[c][k + 1]);
                        b = max3f(b, sv[c][k + 2], sv[c][k + 3]);
                    }
                    mx[c] = max3f(a, b, fmaxf(sv[c][30], sv[c][31]));
                }
                const float m_tile = max3f(mx[0], mx[1], fmaxf(mx[2], mx[3])) * scale;
                const bool raise = (m_run == NEG_INF) || (m_tile > m_run + 8.f);
                if (__any_sync(0xffffffffu, raise)) {
                    const float m_new = raise ? fmaxf(m_run, m_tile) : m_run;
                    const float alpha = fast_exp2(m_run - m_new);   // 0 while nothing is summed
                    if (u > 0) {
                        // Rescale this row of O once the previous tile's product has landed.
                        if (PL::kPSep)
                            wait(pv_done, u - 1);
                        tmem_fence_after();
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            float ov[32];
                            tmem_ld32_nowait(col_o + c * 32, ov);
                            tmem_wait_ld();
#pragma unroll
                            for (int k = 0; k < 32; ++k)
                                ov[k] *= alpha;
                            tmem_st32(col_o + c * 32, ov);
                        }
                    }
                    l_run *= alpha;
                    m_run = m_new;
                }
            };
            const float2 sc2 = make_float2(scale, scale);
            float2 acc[4];
            uint32_t w[2][32];
            // p = 2^(s log2(e)/sqrt(d) - m) as bf16 pairs, and the row's sum in fp32.
            auto weights = [&]() {
                const float m_use = m_run == NEG_INF ? 0.f : m_run;   // all masked so far: p = 0
                const float2 nm2 = make_float2(-m_use, -m_use);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    acc[q] = make_float2(0.f, 0.f);
#pragma unroll
                for (int half = 0; half < 2; ++half) {
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int c = half * 64 + 2 * i;   // keys c, c + 1
                        const float2 x = __ffma2_rn(
                            make_float2(sv[c >> 5][c & 31], sv[c >> 5][(c & 31) + 1]), sc2, nm2);
                        const float2 pr = make_float2(fast_exp2(x.x), fast_exp2(x.y));
                        acc[i & 3] = __fadd2_rn(acc[i & 3], pr);
                        w[half][i] = pack_bf16x2(pr.x, pr.y);
                    }
                }
            };
            load_scores();
            if (__any_sync(0xffffffffu, m_run == NEG_INF)) {
                raise_to_tile_max();
                weights();
            } else {
                // Most tiles: the weights against the current reference, without the tile's
                // maximum.  A row whose weights add up to more than 2^8 (or overflow) may hold one
                // above 2^8: the scores are read again (S is still in TMEM: its columns are freed
                // only below) and the reference raised as above.
                weights();
                const float2 s01 = __fadd2_rn(acc[0], acc[1]), s23 = __fadd2_rn(acc[2], acc[3]);
                const float2 s4 = __fadd2_rn(s01, s23);
                if (__any_sync(0xffffffffu, !(s4.x + s4.y <= 256.f))) {
                    load_scores();
                    raise_to_tile_max();
                    weights();
                }
            }
            if (PL::kPSep) {
                // S's columns may now take the next tile's scores.
                tmem_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(s_free);
            }
            // The P buffer of the previous tile must have been read by its P V; the weights above
            // were computed while that product ran.
            if (PL::kPSep && u > 0) {
                wait(pv_done, u - 1);
                if (releaser)   // V of this warpgroup's previous tile
                    mbar_arrive(bar_empty + 8 * ((2 * (t - kStep) + 1) % R));
            }
            tmem_fence_after();
            tmem_st32_nowait(col_p, w[0]);
            tmem_st32_nowait(col_p + 32, w[1]);
            const float2 s01 = __fadd2_rn(acc[0], acc[1]), s23 = __fadd2_rn(acc[2], acc[3]);
            const float2 s4 = __fadd2_rn(s01, s23);
            l_run += s4.x + s4.y;
            tmem_wait_st();
            if (diag && zero_v && q0 + r >= S) {
                // Key q0 + r lies past the prompt: its V row may hold anything; zero it.
                const int idx = 2 * t + 1;
                wait(bar_full + 8 * (idx % R), idx / R);
                uint8_t *vrow = smem + PL::kRing + (idx % R) * PL::kTileBytes;
#pragma unroll
                for (int c = 0; c < 8 * PL::kSub; ++c)
                    *reinterpret_cast<uint4 *>(vrow + (c >> 3) * 16384 + r * 128 +
                                               (((c & 7) ^ (r & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                fence_proxy_async_smem();
            }
            tmem_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(p_ready);
        }
        // ---------------- the tile's output: o = O / l ----------------
        if (early)
            grid_dependency_wait();   // earlier kernels of the stream have finished with out
        // Split keys: the second warpgroup hands its running maximum and sum to the first, which
        // merges the two O buffers row by row (O = O_0 2^(m_0 - M) + O_1 2^(m_1 - M), likewise l).
        const int n_mine = kSplit ? (n_g - wg + 1) / 2 : n_g;   // this warpgroup's tiles
        float a0 = 1.f, a1 = 0.f;
        if (kSplit) {
            if (n_mine > 0)
                wait(pv_done, n_mine - 1);
            float2 *ml = reinterpret_cast<float2 *>(smem + PL::kML);
            if (wg == 1)
                ml[r] = make_float2(m_run, l_run);
            asm volatile("bar.sync 1, %0;" ::"n"(8 * 32) : "memory");
            if (wg == 1)
                m_run = NEG_INF;   // done: nothing to store
            else {
                const float2 o1 = ml[r];
                if (o1.y > 0.f) {
                    const float mx = fmaxf(m_run, o1.x);
                    a0 = fast_exp2(m_run - mx);
                    a1 = fast_exp2(o1.x - mx);
                    l_run = l_run * a0 + o1.y * a1;
                    m_run = mx;
                }
            }
        }
        // O of this row, 32 columns at c: this warpgroup's buffer, merged with the second's
        auto load_o = [&](int c, float (&ov)[32]) {
            tmem_ld32_nowait(col_o + c * 32, ov);
            if (kSplit && a1 > 0.f) {
                float o1[32];
                tmem_ld32_nowait(col_o + D + c * 32, o1);
                tmem_wait_ld();
#pragma unroll
                for (int k = 0; k < 32; ++k)
                    ov[k] = ov[k] * a0 + o1[k] * a1;
            } else {
                tmem_wait_ld();
            }
        };
        if (n_g > 0 && wg == 0) {
            if (!kSplit)
                wait(pv_done, PL::kPSep ? n_g - 1 : 0);   // with P over S only the last P V commits
            tmem_fence_after();
            const float inv = fast_rcp(l_run);
            bool valid;
            __nv_bfloat16 *orow;
            if (kFused) {
                // Row r: layer (grp ? 0 : L1) + r / G of the block, head j*G + r % G; out
                // [layers][b][h][D], the block's first layer blk * L.
                const int L1 = p.fused_L < p.fused_L1 ? p.fused_L : p.fused_L1;
                valid = r < (grp ? L1 : p.fused_L - p.fused_L1) * p.G;
                const int layer = (grp ? 0 : p.fused_L1) + r / p.G;
                orow = p.out + ((static_cast<size_t>(blk * p.fused_L + layer) * p.b + beta) * p.h +
                                j * p.G + r % p.G) * D;
                if (p.fused_cmax > 1) {
                    // One chunk of the context: o = O / l and lse = m + log2(l) for the merge.
                    const size_t row = (((static_cast<size_t>(blk) * p.b + beta) * p.g + j) *
                                            p.fused_cmax + chunk) * (p.fused_L * p.G) +
                                       layer * p.G + r % p.G;
                    float *prow = p.part + row * D;
                    if (valid && !flags[0])
                        p.part_lse[row] = m_run + log2f(l_run);
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        float ov[32];
                        load_o(c, ov);
                        if (valid && !flags[0]) {
#pragma unroll
                            for (int k = 0; k < 32; k += 4)
                                *reinterpret_cast<float4 *>(prow + c * 32 + k) =
                                    make_float4(ov[k] * inv, ov[k + 1] * inv, ov[k + 2] * inv,
                                                ov[k + 3] * inv);
                        }
                    }
                    valid = false;   // nothing more to store for this row
                } else {
                    // The warp's 32 rows go through this tile's query slot (its last S has
                    // completed), 16-byte chunks swizzled by row, and out 16 bytes a lane: the G
                    // heads of a layer are contiguous rows of out, so the stores coalesce, which
                    // matters most when out is page-locked host memory.
                    uint8_t *stage = smem + PL::kQ + sg * PL::kTileBytes;
                    constexpr int kChunks = D * 2 / 16;   // 16-byte chunks of a row
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        float ov[32];
                        load_o(c, ov);
#pragma unroll
                        for (int k = 0; k < 32; k += 8)
                            *reinterpret_cast<uint4 *>(stage + r * (D * 2) +
                                                       ((((c * 32 + k) >> 3) ^ (r & 7)) << 4)) =
                                make_uint4(pack_bf16x2(ov[k] * inv, ov[k + 1] * inv),
                                           pack_bf16x2(ov[k + 2] * inv, ov[k + 3] * inv),
                                           pack_bf16x2(ov[k + 4] * inv, ov[k + 5] * inv),
                                           pack_bf16x2(ov[k + 6] * inv, ov[k + 7] * inv));
                    }
                    __syncwarp();
                    const int rw0 = (warp & 3) * 32;
                    const int n_rows = (grp ? L1 : p.fused_L - p.fused_L1) * p.G;
#pragma unroll
                    for (int it = 0; it < kChunks; ++it) {
                        const int cidx = it * 32 + lane;
                        const int rr = rw0 + cidx / kChunks, ch = cidx % kChunks;
                        if (rr < n_rows && !flags[0]) {
                            const int lay = (grp ? 0 : p.fused_L1) + rr / p.G;
                            __nv_bfloat16 *o =
                                p.out + ((static_cast<size_t>(blk * p.fused_L + lay) * p.b + beta) *
                                             p.h + j * p.G + rr % p.G) * D;
                            *reinterpret_cast<uint4 *>(o + ch * 8) = *reinterpret_cast<const uint4 *>(
                                stage + rr * (D * 2) + ((ch ^ (rr & 7)) << 4));
                        }
                    }
                    valid = false;
                }
            } else {
                valid = q0 + r < S;
                orow = p.out + ((static_cast<size_t>(beta) * p.s_max + (q0 + r)) * p.h + head) * D;
            }
#pragma unroll
            for (int c = 0; c < (kFused ? 0 : D / 32); ++c) {   // the prefill's rows
                float ov[32];
                tmem_ld32_nowait(col_o + c * 32, ov);
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
    } else {
        setmaxnreg_dec<PL::kRegsLow>();   // warp 11 (and 10 with head_dim 128): no role
    }

    __syncthreads();
    if (warp == PL::kMma) {
        tmem_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "n"(PL::kTmemCols)
                     : "memory");
    }
}

// Merges the context chunks of the fused decode: per output row (block, sequence, KV head, block
// layer, group head) o = sum_c 2^(lse_c - M) o_c / sum_c 2^(lse_c - M), M = max_c lse_c.  W warps
// per row (fused_combine_w: 1, 2, 4 or 8, more for more chunks): warp w takes chunks w, w + W, ...,
// 4 of them in flight, and each lane keeps a running maximum, sum of weights and weighted sum for
// its D / 32 columns; the W warps' states are then merged through shared memory.
template <int D>
__global__ void __launch_bounds__(256, D == 64 ? 6 : 4) combine_fused_kernel(const __grid_constant__ PrefillParams p)
{
    // Launched while the decode grid still runs: the partials are read after it has finished.
    grid_dependency_wait();
    grid_dependents_launch();
    constexpr int E = D / 32;   // columns per lane
    using Vec = typename std::conditional<E == 2, float2, float4>::type;
    __shared__ float s_m[8], s_l[8];
    __shared__ Vec s_acc[8][32];
    const int W = p.fused_combine_w;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int w = warp % W;
    const int rows_per_head = p.fused_L * p.G;
    const long long row = static_cast<long long>(blockIdx.x) * (8 / W) + warp / W;
    const bool live = row < static_cast<long long>(p.fused_nblk) * p.b * p.g * rows_per_head;
    const float NEG_INF = -__int_as_float(0x7f800000);
    int rr = 0, j = 0, beta = 0, blk = 0, chunks = 0;
    size_t base = 0;
    if (live) {
        rr = static_cast<int>(row % rows_per_head);
        const long long bj = row / rows_per_head;   // (block, sequence, KV head)
        j = static_cast<int>(bj % p.g);
        const long long bb = bj / p.g;
        beta = static_cast<int>(bb % p.b);
        blk = static_cast<int>(bb / p.b);
        const int n_kt = (p.prompt_len[beta] + 127) / 128;
        chunks = (n_kt + p.fused_kc - 1) / p.fused_kc;
        base = static_cast<size_t>(bj) * p.fused_cmax * rows_per_head + rr;
    }
    float m = NEG_INF, l = 0.f;
    float acc[E] = {};
    for (int c0 = w; c0 < chunks; c0 += 4 * W) {
        float lse[4];
        Vec v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int c = c0 + u * W;
            const size_t r = base + static_cast<size_t>(c) * rows_per_head;
            if (c < chunks) {
                lse[u] = p.part_lse[r];
                v[u] = *reinterpret_cast<const Vec *>(p.part + r * D + lane * E);
            } else {
                lse[u] = NEG_INF;
                v[u] = Vec{};
            }
        }
        const float mx = fmaxf(fmaxf(m, fmaxf(lse[0], lse[1])), fmaxf(lse[2], lse[3]));
        const float scale = m == NEG_INF ? 0.f : exp2f(m - mx);
        l *= scale;
#pragma unroll
        for (int e = 0; e < E; ++e)
            acc[e] *= scale;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const float wt = lse[u] == NEG_INF ? 0.f : exp2f(lse[u] - mx);
            l += wt;
            const float *x = reinterpret_cast<const float *>(&v[u]);
#pragma unroll
            for (int e = 0; e < E; ++e)
                acc[e] += wt * x[e];
        }
        m = mx;
    }
    if (W > 1) {
        if (lane == 0) {
            s_m[warp] = m;
            s_l[warp] = l;
        }
        Vec a;
        float *ap = reinterpret_cast<float *>(&a);
#pragma unroll
        for (int e = 0; e < E; ++e)
            ap[e] = acc[e];
        s_acc[warp][lane] = a;
        __syncthreads();
        if (w != 0 || !live)
            return;
        // warp 0 of the row: every warp of the row against the largest maximum (warp 0 holds
        // chunk 0, so M is finite)
        float M = NEG_INF;
        for (int k = 0; k < W; ++k)
            M = fmaxf(M, s_m[warp + k]);
        l = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e)
            acc[e] = 0.f;
        for (int k = 0; k < W; ++k) {
            const float wt = s_m[warp + k] == NEG_INF ? 0.f : exp2f(s_m[warp + k] - M);
            l += wt * s_l[warp + k];
            const Vec b = s_acc[warp + k][lane];
            const float *x = reinterpret_cast<const float *>(&b);
#pragma unroll
            for (int e = 0; e < E; ++e)
                acc[e] += wt * x[e];
        }
    } else if (!live) {
        return;
    }
    const float inv = 1.f / l;
    const int layer = rr / p.G, i = rr - layer * p.G;
    __nv_bfloat16 *orow =
        p.out + ((static_cast<size_t>(blk * p.fused_L + layer) * p.b + beta) * p.h + j * p.G + i) * D;
#pragma unroll
    for (int e = 0; e < E; e += 2)
        *reinterpret_cast<uint32_t *>(orow + lane * E + e) =
            pack_bf16x2(acc[e] * inv, acc[e + 1] * inv);
}

template <int D, bool kFused, int kForm>
const void *prefill_fn()
{
    return reinterpret_cast<const void *>(&prefill_kernel<D, kFused, kForm>);
}

// The forms built: prefill at head_dim 64 with one query tile per CTA, at 128 with two; the fused
// decode in the two-tile form (either head_dim) or, at head_dim 64, either one-tile form.
template <typename F>
auto plan_value(int head_dim, int form, F f)
{
    if (head_dim == 64) {
        if (form == kOneDeep)
            return f(PrefillPlan<64, kOneDeep>{});
        return form == kOneTile ? f(PrefillPlan<64, kOneTile>{}) : f(PrefillPlan<64, kTwoTiles>{});
    }
    return f(PrefillPlan<128, kTwoTiles>{});
}
int threads_of(int head_dim, int form)
{
    return plan_value(head_dim, form, [](auto pl) { return decltype(pl)::kThreads; });
}
int regs_of(int head_dim, int form)
{
    return plan_value(head_dim, form, [](auto pl) { return decltype(pl)::kRegsLaunch; });
}
size_t smem_of(int head_dim, int form)
{
    return plan_value(head_dim, form,
                      [](auto pl) { return static_cast<size_t>(decltype(pl)::kAlloc); });
}

const void *kernel_fn(int head_dim, bool fused, int form)
{
    if (fused) {
        if (head_dim == 64)
            return form == kOneDeep   ? prefill_fn<64, true, kOneDeep>()
                   : form == kOneTile ? prefill_fn<64, true, kOneTile>()
                                      : prefill_fn<64, true, kTwoTiles>();
        return prefill_fn<128, true, kTwoTiles>();
    }
    return head_dim == 64 ? prefill_fn<64, false, kOneTile>() : prefill_fn<128, false, kTwoTiles>();
}

cudaError_t launch(int head_dim, bool fused, int form, const CUtensorMap *tmap_q,
                   const CUtensorMap *tmap_kv, const PrefillParams &p, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.n_units));
    cfg.blockDim = dim3(static_cast<unsigned>(threads_of(head_dim, form)));
    cfg.dynamicSmemBytes = smem_of(head_dim, form);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void *args[] = {const_cast<CUtensorMap *>(tmap_q), const_cast<CUtensorMap *>(tmap_kv),
                    const_cast<PrefillParams *>(&p)};
    return cudaLaunchKernelExC(&cfg, kernel_fn(head_dim, fused, form), args);
}

// The prefill form of a head_dim; a fused-decode form valid for the head_dim.
int prefill_form(int head_dim) { return head_dim == 64 ? kOneTile : kTwoTiles; }
int fused_form(int head_dim, int form) { return head_dim == 64 ? form : kTwoTiles; }

}  // namespace

size_t prefill_smem_bytes(int head_dim) { return smem_of(head_dim, prefill_form(head_dim)); }

// The warpgroups' register split (setmaxnreg) adds up to the registers the block is launched with;
// a kernel built with another per-thread count would wait forever in setmaxnreg.inc, so it is
// refused here instead of launched.
cudaError_t prepare(int head_dim, bool fused, int form)
{
    cudaFuncAttributes fa;
    const void *fn = kernel_fn(head_dim, fused, form);
    cudaError_t e = cudaFuncGetAttributes(&fa, fn);
    if (e != cudaSuccess)
        return e;
    if (fa.numRegs != regs_of(head_dim, form))
        return cudaErrorInvalidKernelImage;
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem_of(head_dim, form)));
}

cudaError_t prepare_prefill(int head_dim)
{
    return prepare(head_dim, false, prefill_form(head_dim));
}

cudaError_t prepare_fused(int head_dim, int form)
{
    return prepare(head_dim, true, fused_form(head_dim, form));
}

cudaError_t launch_prefill(int head_dim, const CUtensorMap *tmap_q, const CUtensorMap *tmap_kv,
                           const PrefillParams &p, cudaStream_t stream)
{
    return launch(head_dim, false, prefill_form(head_dim), tmap_q, tmap_kv, p, stream);
}

cudaError_t launch_fused(int head_dim, int form, const CUtensorMap *tmap_q,
                         const CUtensorMap *tmap_kv, const PrefillParams &p, cudaStream_t stream)
{
    return launch(head_dim, true, fused_form(head_dim, form), tmap_q, tmap_kv, p, stream);
}

cudaError_t launch_fused_combine(int head_dim, const PrefillParams &p, cudaStream_t stream)
{
    const long long rows = static_cast<long long>(p.fused_nblk) * p.b * p.g * p.fused_L * p.G;
    const int per_cta = 8 / p.fused_combine_w;   // rows of a CTA
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>((rows + per_cta - 1) / per_cta));
    cfg.blockDim = dim3(256);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void *args[] = {const_cast<PrefillParams *>(&p)};
    const void *fn = head_dim == 64 ? reinterpret_cast<const void *>(&combine_fused_kernel<64>)
                                    : reinterpret_cast<const void *>(&combine_fused_kernel<128>);
    return cudaLaunchKernelExC(&cfg, fn, args);
}

}  // namespace mlkv
