// Internal interface between the host side of libmlkv (mlkv_host.cpp) and its kernels
// (mlkv_kernels.cu).  Not part of the public ABI (include/mlkv.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mlkv.h"

namespace mlkv {

// Error bits a kernel ORs into the cache's device error word.
enum : int {
    kErrWaitFull = 1,   // a consumer gave up waiting for a K/V tile
    kErrWaitEmpty = 2,  // the producer gave up waiting for a free stage
    kErrDrain = 4,      // the producer gave up waiting for its last copies at exit
};

// Layers one multi-layer decode launch can cover (DecodeParams::ml_layers).
constexpr int kMaxStepLayers = 128;

// Split-KV decode of one layer.  Passed by value (__grid_constant__), so a launch needs no
// device-side metadata and is stream-ordered and graph-capturable by construction.
struct DecodeParams {
    const __nv_bfloat16 *Q;   // [b][h][D]
    __nv_bfloat16 *out;       // [b][h][D]
    const __nv_bfloat16 *K_new;   // fused append: new token [b][g][D], or nullptr
    const __nv_bfloat16 *V_new;
    __nv_bfloat16 *cache;     // [m][2][b][g][max_seq][D] (written only by the fused append)
    int max_seq;
    float *part_o;            // [pieces][G][D]  normalised partial outputs
    float *part_lse;          // [pieces][G]     log2-domain log-sum-exp of each partial
    unsigned *counters;       // [b*g]           pieces finished per segment; zero between launches
    int *err;                 // device error word
    float scale_log2;         // log2(e) / sqrt(D)
    int b, h, g, G, slot;
    int num_tiles;            // total tiles over all (beta, j) segments
    int uniform_len;          // the common length when every sequence has the same, else 0
    int cluster_k;            // > 1: clusters of k CTAs, one segment each, merged over DSMEM
    int deferred_merge;       // 1: split segments only write partials; combine_kernel merges them
    int tile_tokens;          // T of the launch (the combine kernel re-derives the piece layout)
    int decode_grid;          // P of the decode launch
    const __nv_bfloat16 *Q_next;   // the next layer's queries (decode step), prefetched to L2
    int early_fetch;          // 1: the previous kernel is this library's decode of the preceding
                              // layer, which writes neither Q nor any cache row but a segment's
                              // newest: Q and the tiles without that row are read before the
                              // dependency wait.  2: the previous kernel is this library's copy of
                              // the step's inputs (Q, K_new, V_new), which writes no cache row:
                              // only the CTA's first tile is fetched before the wait
    int newest_ready;         // 1: the segments' newest rows are replaced from K_new/V_new by this
                              // grid: no wait before a segment's last tile
    int store_new;            // with K_new: 1 = also store the new token in the cache (the owner
                              // layer's fused append); 0 = only replace the tiles' newest rows (a
                              // later layer of the block, whose owner's launch stores the token)
    int pf_own;               // multi-layer launch: 1 = prefetch the step's slots into L2
    // Multi-layer launch (ml_layers > 0): one grid covers every (layer, sequence, KV head) item of
    // a decode step, each item a whole segment.  Items are ranked either layer-major (layer n's
    // segments n b g .. (n + 1) b g - 1) or, with ml_seg_major, segment-major: sequences in the
    // order tile_start[0..b) holds, then KV head j, then the step's layers in the order ml_order[]
    // lists them (owner blocks together), so the CTAs working at one time share a few segments'
    // K/V (read once from HBM, the other layers of the block find it in L2) -- the order for slots
    // larger than L2.  Sequences are ordered longest first; ranks are dealt to the CTAs round-robin
    // (round k gives rank k P + c to CTA c) or, with ml_snake, as a snake (odd rounds k P + P-1-c),
    // which balances varied lengths.  Q and out then
    // hold every layer ([layer][b][h][D], ml_q_stride elements apart) and K_new / V_new every
    // owner's new token ([slot][b][g][D], ml_kv_stride elements apart); layer n reads slot
    // ml_slot[n], and stores its new token in the cache if ml_store[n] (an owner layer), else only
    // replaces its tiles' newest rows with it.  slot, store_new and Q_next are unused; pf_own = 1
    // has every CTA prefetch its share of the visible rows of all ml_slots slots into L2 first
    // (every sequence of one length only).
    int ml_layers;
    int ml_seg_major;         // 1: ranks segment-major (below); 0: layer-major, layer by layer
    int ml_snake;             // 1: snake deal of ranks to CTAs; 0: plain round-robin
    int ml_chunks;            // C >= 1: every segment is C items (chunk c: tiles [c nt / C,
                              // (c + 1) nt / C)); rank r is chunk r mod C of the item ranked
                              // r / C.  With C > 1 every item writes a partial record at
                              // (layer b g + beta g + j) C + c and combine_kernel merges them
    int ml_slots;             // owner slots the step reads (with pf_own: all prefetched into L2)
    long long ml_q_stride, ml_kv_stride;
    unsigned char ml_slot[kMaxStepLayers];
    unsigned char ml_store[kMaxStepLayers];
    unsigned char ml_order[kMaxStepLayers];
    int seq_len[MLKV_MAX_BATCH];
    int tile_start[MLKV_MAX_BATCH + 1];  // first flattened tile of sequence beta (j-major inside);
                                         // a multi-layer launch: the sequences, longest first
};

// Causal prefill of one layer (mlkv_prefill.cu): one CTA per work unit, a unit being two query
// tiles of 128 prompt positions over one KV head.  Passed by value.
//   units[u] = beta | qb_b << 10 | sel << 24, qb_b the block (of 128 positions) of tile B.
//   head_pairs = 1 (G even): tiles A and B are heads 2 sel and 2 sel + 1 at block qb_b.
//   head_pairs = 0 (G odd):  both are head sel; A is block qb_b - 1 when qb_b is odd, else absent.
constexpr int kPrefillMaxUnits = 6144;   // units per launch (more: several launches)
// Unit word of the fused decode: sequence (10 bits), chunk (8), block (6), KV head (8).
constexpr int kFusedMaxChunks = 256;
constexpr int kFusedMaxBlocks = 64;
constexpr int kPrefillMaxHeads = 256;    // sel has 8 bits
constexpr int kPrefillMaxBlocks = 1 << 14;
struct PrefillParams {
    __nv_bfloat16 *out;       // [b][s_max][h][D]
    int *err;                 // device error word
    float scale_log2;         // log2(e) / sqrt(D)
    int b, h, g, G, s_max, slot, n_units, head_pairs;
    // Cross-layer fused decode (mlkv_decode_block_fused, and mlkv_decode_step's fused form): every
    // block has L layers, L1 of them in tile B (the rest in tile A); prompt_len holds the sequence
    // lengths.  Both 0 for prefill.  A unit's block blk (fused_nblk blocks in all) reads slot
    // slot + blk and the layers blk*L .. blk*L + L - 1 of Q and out.
    int fused_L, fused_L1, fused_nblk;
    // Split over the context: a unit holds key tiles [chunk*kc, chunk*kc + kc) of its sequence;
    // with more than one chunk (cmax > 1) it writes o = O/l (f32) and lse = m + log2(l) to part /
    // part_lse [nblk][b][g][cmax][L*G rows] and combine_fused merges the chunks.
    int fused_kc, fused_cmax;
    float *part, *part_lse;
    // What the fused launch may read before its dependency wait (the previous kernel of the
    // stream is this library's store of the new tokens): 1 -- the store triggered this launch
    // after its own wait, so everything but the tile holding the new row (the queries too);
    // 2 -- the store triggered it at once (the step's inputs still being copied in), so only
    // cache tiles that hold no new row; 0 -- nothing.
    int fused_early;
    int fused_combine_w;   // warps per output row of combine_fused (1, 2, 4 or 8)
    // Fused decode: non-null -- the queries [layers][b][h][D] are page-locked host memory (this is
    // its device-mapped address): each unit loads its rows with plain loads, not the tensor map.
    const __nv_bfloat16 *q_host;
    int prompt_len[MLKV_MAX_BATCH];
    uint32_t units[kPrefillMaxUnits];
};

// Dynamic shared memory of the prefill kernel; sets its limit (once per device); launches it with
// programmatic dependent launch on `stream`.
size_t prefill_smem_bytes(int head_dim);
cudaError_t prepare_prefill(int head_dim);
cudaError_t launch_prefill(int head_dim, const CUtensorMap *tmap_q, const CUtensorMap *tmap_kv,
                           const PrefillParams &p, cudaStream_t stream);
// Fused decode forms (head_dim 64 with L * G <= 128 may take either one-tile form; otherwise the
// two-tile form is used whatever is asked): 0 two query tiles per CTA; 1 one tile, two CTAs per
// SM; 2 one tile, one CTA per SM with a 12-tile ring and two S buffers.
constexpr int kFusedTwoTiles = 0, kFusedOneTile = 1, kFusedOneDeep = 2;
cudaError_t prepare_fused(int head_dim, int form);
cudaError_t launch_fused(int head_dim, int form, const CUtensorMap *tmap_q,
                         const CUtensorMap *tmap_kv, const PrefillParams &p, cudaStream_t stream);
cudaError_t launch_fused_combine(int head_dim, const PrefillParams &p, cudaStream_t stream);

// Copies through device-mapped page-locked host memory (mlkv_stage.cu): up to 4 segments, each a
// multiple of 16 bytes with 16-byte-aligned ends.
struct StageParams {
    const void *src[4];
    void *dst[4];
    size_t bytes[4];
    int n;
};
cudaError_t launch_stage_copy(const StageParams &p, cudaStream_t stream);

// KV-weight merge (mlkv_merge.cu).  Passed by value.
constexpr int kMergeMaxLayers = 1024;
struct MergeParams {
    const __nv_bfloat16 *W;   // [l][h][row]
    __nv_bfloat16 *out;       // [m][g][row], owners in increasing layer order
    long long row;            // elements per head row block, a multiple of 8
    int h, g, G;
    int slot_begin[kMergeMaxLayers + 1];   // members of slot s: member[slot_begin[s] .. [s+1])
    int member[kMergeMaxLayers];           // layers grouped by slot
};
cudaError_t launch_merge(const MergeParams &p, int n_slots, cudaStream_t stream);

struct AppendParams {
    const __nv_bfloat16 *K;   // [n_slots][b][g][D] (one slot for launch_append)
    const __nv_bfloat16 *V;
    __nv_bfloat16 *cache;     // [m][2][b][g][max_seq][D]
    int b, g, d, max_seq, slot;   // K[s] and V[s] go to slot + s
    int n_slots;
    int trigger_first;            // append_slots: trigger the dependent launch before the wait
    int seq_len[MLKV_MAX_BATCH];
};

// Static description of one compiled decode variant.
struct DecodeVariant {
    int head_dim;
    int tile_tokens;
    int stages;
    int threads;
    size_t smem_bytes;        // without the per-sequence tables (see table_bytes)
    size_t res_bytes;         // one piece result slot (cluster mode adds k-1 of them)
    const void *fn;
    int tc = 0;               // 1: decode_tc_kernel (tcgen05, TMEM), 0: decode_kernel (mma.sync)
};

// The tcgen05 variants (mlkv_decode_tc.cu).
extern const DecodeVariant kTcVariants[];
extern const int kNumTcVariants;

// Shared memory a launch adds for the per-sequence tables (only when lengths differ).
inline size_t table_bytes(int batch) { return ((8 * static_cast<size_t>(batch) + 4) + 15) & ~15ull; }

// Returns the compiled variant for (head_dim, tile_tokens) of the tcgen05 kernel (tc = 1) or of
// the mma.sync kernel (tc = 0), or nullptr.
const DecodeVariant *find_decode_variant(int head_dim, int tile_tokens, int tc = 0);

// Raises the variant's dynamic shared-memory limit (capped at max_smem, the device's opt-in
// per-block maximum); call once per device before the first launch.
cudaError_t prepare_decode_variant(const DecodeVariant &v, size_t max_smem);

// pdl: launch with programmatic stream serialization (the kernel's prologue may overlap the
// previous kernel of the stream; it waits on griddepcontrol.wait before touching global memory).
// tmap: the cache with boxes of {64 channels, tile_tokens positions}; tmap_rows: the same tensor
// with boxes of 64 positions, used for a segment's last tile when it is only partly visible.
cudaError_t launch_decode(const DecodeVariant &v, int grid, size_t smem, cudaStream_t stream,
                          const CUtensorMap *tmap, const CUtensorMap *tmap_rows,
                          const DecodeParams &p, const cudaAccessPolicyWindow *window,
                          bool pdl = true);

// Default positions per tile of the mma.sync decode kernel for a launch over `segments`
// (sequence, KV head) pairs of mean length mean_len.  Longer tiles move more bytes per TMA
// request and per barrier round trip; shorter ones waste less on short sequences.  For d = 64 the
// 128-position variant is small enough for two CTAs per SM, so the next layer's CTAs start (and
// fetch) while this layer's last ones finish: measured faster for many segments of moderate
// length (64 x 2048: 85 vs 89 us a step; 512 x ~2048: 527 vs 560), slower for few long segments
// or HBM-bound layers (1 x 131072, 256 x 8192).  mean_len < 0 means "unknown" (reports the
// long-sequence choice).
inline int default_tile_tokens(int d, double mean_len, int segments)
{
    if (d == 64) {
        if (mean_len >= 0 && (mean_len < 512 || (segments >= 32 && mean_len <= 4096)))
            return 128;
        return 256;
    }
    return (mean_len < 0 || mean_len >= 512) ? 128 : 64;
}

// Sets the calling thread's mlkv_last_error() text.
void set_last_error(const char *msg);

// Largest number of CTAs sharing one (sequence, KV head) segment for a stream-K launch of `grid`
// CTAs over the tiles described by p (tile_start / seq_len / uniform_len, g, b) with tile length T.
int max_pieces_per_segment(const DecodeParams &p, int T, int grid);

// Merges the partials of every split segment of the decode launch described by p (which must
// have deferred_merge = 1), launched right after it on the same stream.
cudaError_t launch_combine(const DecodeParams &p, int head_dim, cudaStream_t stream,
                           bool pdl = true);

// Pieces per segment above which the decode launch defers its merges to combine_kernel.
constexpr int kInlineMergeMaxPieces = 4;
// combine_kernel keeps one weight per piece in shared memory.
constexpr int kCombineMaxPiecesHost = 1024;

// How many k-CTA clusters of this variant can be resident at once.
cudaError_t max_active_clusters(const DecodeVariant &v, int k, int *out);

// Every owner slot's new token in one launch (mlkv_stage.cu), for the fused step.
cudaError_t launch_append_slots(const AppendParams &p, cudaStream_t stream);
cudaError_t launch_append(const AppendParams &p, cudaStream_t stream);

}  // namespace mlkv
