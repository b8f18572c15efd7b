/*
 * mlkv.h - C ABI of the GB300 (sm_103a) MLKV decode-attention library, libmlkv.so.
 *
 * MLKV (Zuhri et al., "MLKV: Multi-Layer Key-Value Heads for Memory Efficient Transformer
 * Decoding", arXiv 2406.09297) shares KV heads inside a layer (query groups, Sec. 2.3 Eq. 12)
 * and across layers (Sec. 3, Eqs. 13-18): only the m layers that own KV heads store keys and
 * values, and every other layer reads the cache of an earlier owner layer.  This library holds
 * that cache on one GPU and runs the per-layer single-token decode attention over it.
 *
 * Conventions shared by every call
 *  - Indices are 0-based (the paper counts from 1).
 *  - Return value: MLKV_OK (0) or a negative MLKV_ERR_* code; mlkv_last_error() then holds a
 *    one-line description for the calling thread.  Arguments are validated on the host before any
 *    work is queued: a call that returns an error has queued nothing.
 *  - "device" pointers are CUDA device (or managed) memory of the cache's device; "host" pointers
 *    are ordinary CPU memory read before the call returns.  The caller owns every buffer it
 *    passes; device buffers must stay valid until the stream reaches the queued work.
 *  - Tensors are bf16 (IEEE bfloat16 bit patterns), row-major, densely packed, 16-byte aligned.
 *  - cuda_stream is a cudaStream_t (NULL = legacy default stream).  Calls are asynchronous with
 *    respect to the host and ordered on that stream.  Calls on one cache must be ordered with
 *    respect to each other (one stream, or explicit events): they share the cache's merge scratch.
 *  - seq_lens (host int32[batch]) counts the token being decoded: sequence beta attends positions
 *    [0, seq_lens[beta]), 1 <= seq_lens[beta] <= max_seq.
 *  - No call allocates device memory except mlkv_cache_create; no call synchronises the device
 *    except mlkv_sync_status and mlkv_cache_destroy.
 */
#ifndef MLKV_H_
#define MLKV_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MLKV_OK 0
#define MLKV_ERR_INVALID_ARG (-1) /* null handle/pointer, misaligned buffer, bad index */
#define MLKV_ERR_MAP (-2)         /* invalid layer->owner map or head counts */
#define MLKV_ERR_RANGE (-3)       /* a sequence length outside [1, max_seq] */
#define MLKV_ERR_OOM (-4)         /* device allocation failed */
#define MLKV_ERR_CUDA (-5)        /* a CUDA runtime / driver call failed */
#define MLKV_ERR_UNSUPPORTED (-6) /* valid request outside what this build supports */
#define MLKV_ERR_DEVICE (-7)      /* a kernel reported an error (bounded wait expired) */

#define MLKV_MAX_BATCH 1024       /* largest batch a cache may hold */
#define MLKV_MAX_GROUP 16         /* largest query group h/g per KV head */
#define MLKV_STATIC_SCRATCH_BYTES (8u << 20) /* scratch of mlkv_decode_attention_static */

typedef struct mlkv_cache *mlkv_cache_t;

/*
 * mlkv_cache_create - validates an MLKV layout and allocates its KV cache on the current device.
 *
 * Paper: Sec. 3 (m owner layers, g KV heads each, cache of 2*b*s*m*g*d_k elements), Eq. 18
 * (layer -> KV block), Eq. 12 (query head -> KV head within a layer).
 *
 *   out                 receives the handle (host pointer, written on success only)
 *   n_layers            l >= 1
 *   n_q_heads           h >= 1, query heads per layer
 *   head_dim            d_k; 64 or 128 in this build (else MLKV_ERR_UNSUPPORTED)
 *   layer_owner         host int32[n_layers]: layer_owner[n] is the layer whose KV heads layer n
 *                       reads.  Must satisfy 0 <= owner[n] <= n and owner[owner[n]] == owner[n]
 *                       (owners own themselves); Eq. 18's contiguous blocks are one such map
 *                       (see mlkv_block_owner_map), non-uniform maps are accepted too.
 *   kv_heads_per_owner  g, must divide h; h/g <= MLKV_MAX_GROUP
 *   batch, max_seq      b in [1, MLKV_MAX_BATCH], s >= 1: the cache holds positions [0, max_seq)
 *
 * Device layout (bf16): [m][2 (K,V)][b][g][max_seq][d], slot = rank of the owner among owners.
 * The cache starts zeroed.  Errors: MLKV_ERR_INVALID_ARG, _MAP, _UNSUPPORTED, _OOM, _CUDA.
 */
int mlkv_cache_create(mlkv_cache_t *out, int n_layers, int n_q_heads, int head_dim,
                      const int *layer_owner, int kv_heads_per_owner, int batch, int max_seq);

/* Frees the cache and its scratch after synchronising the device.  NULL is accepted. */
int mlkv_cache_destroy(mlkv_cache_t c);

/*
 * mlkv_append - stores the new token's keys and values of an owner layer.
 *
 * Paper: Sec. 2.4 (KV caching keeps the keys/values of earlier tokens) and Sec. 3 Eq. 13 (only
 * the m owner layers have K/V projections; the other layers store nothing).
 *
 *   layer      0 <= layer < l.  For a layer that does not own KV heads the call returns MLKV_OK
 *              and queues nothing.
 *   K, V       device bf16 [batch][g][d]: the new token's key / value per sequence and KV head
 *   seq_lens   host int32[batch]; the token is written at position seq_lens[beta] - 1
 * Writing the same token twice at the same position is idempotent.
 */
int mlkv_append(mlkv_cache_t c, int layer, const void *K, const void *V, const int *seq_lens,
                void *cuda_stream);

/*
 * mlkv_decode_attention - single-token attention of every query head of one layer.
 *
 * Paper: Eqs. 2-3 (alpha = softmax(q k^T / sqrt(d_k)), o = alpha v) with the MLKV maps of
 * Eqs. 15 and 18: query head i of layer n attends over KV head floor(i / (h/g)) of the cache
 * slot of layer_owner[n], positions [0, seq_lens[beta]).
 *
 *   Q        device bf16 [batch][h][d], this layer's queries (post-projection; any positional
 *            encoding already applied)
 *   out      device bf16 [batch][h][d], may not alias Q; written with round-to-nearest-even
 *   seq_lens host int32[batch], 1 <= seq_lens[beta] <= max_seq
 * Arithmetic: bf16 inputs, fp32 accumulation and softmax, fp32 merge of split-KV partials.
 */
int mlkv_decode_attention(mlkv_cache_t c, int layer, const void *Q, void *out,
                          const int *seq_lens, void *cuda_stream);

/*
 * mlkv_append_decode_attention - mlkv_append followed by mlkv_decode_attention for one layer,
 * in one kernel launch.
 *
 * Paper: Sec. 3 -- an owner layer stores its new token (Eq. 13) and its query heads then attend
 * over positions [0, L) including that token (Eqs. 2-3, 15, 18).  For a layer that owns KV heads
 * the new token's K/V are stored at position seq_lens[beta] - 1 exactly as mlkv_append stores
 * them; for any other layer K and V are ignored (may be NULL) and the call is
 * mlkv_decode_attention.  Arguments as for those two calls.
 */
int mlkv_append_decode_attention(mlkv_cache_t c, int layer, const void *K, const void *V,
                                 const void *Q, void *out, const int *seq_lens,
                                 void *cuda_stream);

/*
 * mlkv_decode_step - one decode step of the whole model: for every layer n in order, the calls
 * mlkv_append_decode_attention (layers that own KV heads) or mlkv_decode_attention (the others).
 *
 * Paper: Sec. 3 (the layer stack of Eq. 18: owner layers store their token, every layer attends
 * over its owner's cache) and Sec. 4.5 (autoregressive decoding, one token per step).
 *
 *   Q        device bf16 [l][batch][h][d], every layer's queries
 *   K, V     device bf16 [m][batch][g][d], every owner layer's new token, in slot order
 *   out      device bf16 [l][batch][h][d]
 *   seq_lens host int32[batch], as for mlkv_decode_attention
 * All four device buffers 16-byte aligned (else MLKV_ERR_INVALID_ARG).
 * The results equal those of the layer calls up to rounding: inside a step the layers' launches
 * overlap and may split a layer's work differently (whole segments per CTA).  Every layer of an
 * owner's block reads that owner's new token from K and V (the later layers take their newest
 * row from there rather than from the cache), so K and V, like Q, must stay valid until the stream
 * has run the whole step.
 * Cross-layer fused form (option "step_fused"): for maps of equal contiguous owner blocks
 * (owner[n] = n - n mod (l/m), the layout of Sec. 3, Eq. 18) whose (l/m) * (h/g) query rows per KV
 * head fit two tiles of 128, the step is one launch that stores every owner's new token, one
 * tcgen05 launch in which each unit (sequence, KV head, block, chunk of the context) loads every
 * K/V tile of its chunk once for all the block's layers' query rows, and, when a segment is split
 * into chunks, one merge launch.  Other maps, option "step_fused" = 0, and the
 * options that select the decode kernel's shapes ("grid", "tile_tokens", "tc", "l2_prefetch",
 * "l2_persist") take the decode kernel's multi-layer launch.  Option "last_step_fused" reads
 * back 1 if the most recent step ran in the fused form, "last_step_launches" the number of this
 * library's launches of that step, "last_fused_kc" the key tiles of 128 positions per unit.
 * Option "step_graph": with 1 a call whose pointers, lengths and options equal those of the
 * previous call replays a CUDA graph of the step's launches (recorded on the second such call; new
 * values in the same buffers are fine); a call with arguments different from the previous call's
 * issues the launches directly, which costs the host about half of recording them -- the case of a
 * decode loop, whose lengths grow every step.  With 2 (default) a step that runs as one
 * multi-layer launch (and its merge launch) is always issued directly -- a replayed one-node graph
 * measured ~2 us slower per step -- and a step of per-layer launches is recorded and replayed as
 * with 1.  0 issues every step directly.  When cuda_stream is itself being captured the launches
 * are issued directly, into the caller's graph.
 */
int mlkv_decode_step(mlkv_cache_t c, const void *Q, const void *K, const void *V, void *out,
                     const int *seq_lens, void *cuda_stream);

/*
 * mlkv_plan_step - the form mlkv_decode_step takes for a map and a step's lengths, decided on the
 * host with no GPU and no cache: the same decision a cache of this map makes on a device with
 * sm_count SMs (152 on GB300), with its options "step_fused", "fused_kc" and "fused_deep" at the
 * given values (-1: the default) and every other option at its default, for device buffers.
 *
 * Paper: Sec. 3, Eq. 18 (the equal contiguous owner blocks the fused form requires).
 *
 *   layer_owner .. max_seq  as for mlkv_cache_create (same validation and error codes)
 *   seq_lens    host int32[batch], as for mlkv_decode_step (each in [1, max_seq])
 *   plan        host int64[4], written on success:
 *               [0] 1 if the step runs in the cross-layer fused form, else 0 (the decode kernel);
 *               [1] the fused launch's CTA form: 0 two 128-row query tiles per CTA, 1 one tile at
 *                   two CTAs per SM, 2 one tile at one CTA per SM with the key tiles alternating
 *                   between two softmax warpgroups; -1 when not fused;
 *               [2] key tiles of 128 positions per unit (the context split; 0 when not fused);
 *               [3] units of the fused launch (sequence, KV head, owner block, chunk), 0 when not
 *                   fused.
 * Errors: MLKV_ERR_INVALID_ARG (NULL plan, sm_count < 1, an option out of range), and those of
 * mlkv_cache_create and of the lengths' check.
 */
int mlkv_plan_step(int n_layers, int n_q_heads, int head_dim, const int *layer_owner,
                   int kv_heads_per_owner, int batch, int max_seq, const int *seq_lens,
                   int sm_count, int step_fused, int fused_kc, int fused_deep, int64_t plan[4]);

/*
 * mlkv_decode_step_host - mlkv_decode_step with the step's tensors in host memory (the user's end
 * of a step).  Layouts as for mlkv_decode_step, in host memory; everything is queued on
 * cuda_stream, and out holds the step's outputs once the stream has reached the end of the call's
 * work.
 * Page-locked, 16-byte-aligned buffers (cudaHostAlloc, cudaHostRegister) are used through their
 * device-mapped addresses: in the cross-layer fused form the kernels read the queries and the new
 * tokens and write the outputs there directly (no copy); otherwise one copy kernel brings Q, K and
 * V into device staging buffers right before the launch and the kernels write the outputs in
 * place.  With option "step_graph" = 1 the launches of a step are recorded into one CUDA graph the
 * second time the same arguments come and replayed after (as for mlkv_decode_step; with 2, the
 * default, a one-launch or fused step is issued directly).  Other buffers take one
 * cudaMemcpyAsync per tensor, in and out, and synchronise with the host as CUDA's pageable copies
 * do.  The staging buffers, 2 * (l*b*h*d + m*b*g*d) bf16, are allocated on the first call and
 * kept until mlkv_cache_destroy.
 * Errors: as mlkv_decode_step, and MLKV_ERR_OOM for the staging buffers.
 */
int mlkv_decode_step_host(mlkv_cache_t c, const void *Q, const void *K, const void *V, void *out,
                          const int *seq_lens, void *cuda_stream);

/*
 * mlkv_prefill - the prompt of every sequence through one layer at once (prefill): owner layers
 * first store the prompt's K/V at positions [0, s_max) of their slot (Sec. 3: only a layer with KV
 * heads of its own stores them); then prompt position t of query head i attends, causally, to
 * positions 0 .. t of KV head i / (h/g) of the layer's owner (Eqs. 2-3 at every prompt position,
 * maps of Eqs. 13-18).  A later mlkv_decode_step continues each sequence at length
 * prompt_lens[beta] + 1.  Runs on the tcgen05 tensor cores.
 *
 *   Q            device bf16 [batch][s_max][h][d], position-major (a token's heads contiguous)
 *   K, V         device bf16 [batch][g][s_max][d], the prompt's keys / values; read only for an
 *                owner layer (may be NULL otherwise)
 *   out          device bf16 [batch][s_max][h][d]; rows past a prompt's length are not written
 *   prompt_lens  host int32[batch], 1 <= prompt_lens[beta] <= s_max
 *   s_max        1 <= s_max <= max_seq
 * The caller keeps the buffers valid until the stream reaches the call.  Errors:
 * MLKV_ERR_INVALID_ARG (null or unaligned pointer, out overlapping Q), MLKV_ERR_RANGE (lengths),
 * MLKV_ERR_CUDA.
 */
int mlkv_prefill(mlkv_cache_t c, int layer, const void *Q, const void *K, const void *V, void *out,
                 const int *prompt_lens, int s_max, void *cuda_stream);

/*
 * mlkv_load_prefix - bulk-stores positions [0, len) of an owner layer's keys and values
 * (prefill).  K, V: device bf16 [batch][g][len][d].  No-op (MLKV_OK) for a non-owner layer.
 * Paper: Sec. 4.5 starts decoding from a pre-filled ("dummy") cache.
 */
int mlkv_load_prefix(mlkv_cache_t c, int layer, const void *K, const void *V, int len,
                     void *cuda_stream);

/* Bytes of the KV cache: 2*b*max_seq*m*g*d*2 (Sec. 3's element count times 2 bytes), or a
 * negative error code. */
int64_t mlkv_cache_bytes(mlkv_cache_t c);

/* Number m of owner layers (Sec. 3), or a negative error code. */
int mlkv_num_slots(mlkv_cache_t c);

/* owner (host int*) receives layer_owner[layer]; slot (host int*) the cache slot of that owner. */
int mlkv_owner_slot(mlkv_cache_t c, int layer, int *owner, int *slot);

/*
 * mlkv_kv_ptr - device addresses of one slot's K and V blocks, for bulk initialisation and
 * inspection.  strides (host int64[4]) receives the element strides of (beta, j, t, e).
 */
int mlkv_kv_ptr(mlkv_cache_t c, int slot, void **k_base, void **v_base, int64_t strides[4]);

/*
 * mlkv_set_option / mlkv_get_option - tuning knobs (host only, take effect on the next call):
 *   "tile_tokens"  positions per pipeline stage: 64, 128 or 256 (d=64) / 64 or 128 (d=128);
 *                  0 (default) picks per call: the longer tile when the mean length is >= 512,
 *                  except 128 for d=64 when batch x kv_heads >= 32 and the mean length <= 4096
 *   "grid"         persistent CTA count; 0 = one wave of resident CTAs (default)
 *   "l2_persist"   1 = keep part of each owner's slot in L2 for the later layers of its block:
 *                  switching it on reserves the device's largest persisting-L2 set-aside for this
 *                  process's CUDA context (cudaLimitPersistingL2CacheSize; the limit belongs to
 *                  the context, so other work in the process sees the smaller normal L2 too), and
 *                  every decode launch then reads its owner's slot through an access-policy
 *                  window over the slot's first bytes (at most the device's window size) whose
 *                  persisting share is set-aside / window; the last layer of a block marks its
 *                  hits normal again.  Switching it off (or destroying the cache) resets the
 *                  persisting lines and restores the earlier set-aside.  MLKV_ERR_UNSUPPORTED
 *                  where the device has no set-aside.  Default 0 (see the design notes for the
 *                  measurements behind the default).
 *   "l2_prefetch"  1 = when mlkv_decode_step runs as one multi-layer launch (see "step_kernel")
 *                  and the visible K/V rows of all owner slots fit in 5/8 of L2, every CTA first
 *                  prefetches its share of them into L2 (cp.async.bulk.prefetch); 0 (default) = no
 *                  prefetch, measured faster on GB300.  Results are identical.
 *   "step_kernel"  1 (default) = mlkv_decode_step issues the whole step as one launch of the
 *                  decode kernel over every (layer, sequence, KV head) item, each a whole segment,
 *                  when the tcgen05 kernel, a fixed grid and l2_persist (whose windows are per
 *                  layer) are off, the model has at most 128 layers and the estimated makespan is
 *                  no longer than per-layer launches' (a few long segments, e.g. batch 1 at long
 *                  context, keep per-layer launches).  Sequences are taken longest first; when the
 *                  owner slots' visible rows do not fit in L2 the items are ranked segment-major
 *                  (the layers of a block read each segment at about the same time, so L2 serves
 *                  all but the first), else layer by layer.  0 = always one launch per layer.
 *                  Same results within the tolerance.
 *   "step_fused"   1 (default) = where "step_kernel" gives one launch for the step, the map has
 *                  equal contiguous owner blocks of >= 3 layers whose query rows fit two 128-row
 *                  tiles, and the owner slots hold >= 4 tiles of 128 visible positions per SM, the
 *                  step runs in the cross-layer fused form (see mlkv_decode_step); 2 = that form
 *                  wherever the map allows it (blocks of any size, any step); 0 = the decode
 *                  kernel's multi-layer launch.  Same results within the tolerance.
 *   "fused_kc"     > 0 = key tiles of 128 positions per unit of the fused form (clamped to what
 *                  the unit word holds); 0 (default) = planned: a sequence is split only as far
 *                  as the units still number at most the SMs.
 *   "fused_deep"   1 (default) = a fused launch at head_dim 64 whose blocks' rows fit one 128-row
 *                  tile and whose units number at most the SMs runs one CTA per SM with a
 *                  12-tile K/V ring, its key tiles alternating between two softmax warpgroups
 *                  (S, P and O in two buffers of tensor memory, merged per row at the end); 0 =
 *                  two CTAs per SM with a 5-tile ring.  Same results within the tolerance.
 *   "cluster"      1 (default) = when every sequence has one length and each (sequence, KV head)
 *                  splits into 2 or 4 equal pieces without lengthening the one-wave makespan,
 *                  run the pieces of a segment as one thread-block cluster and merge them through
 *                  distributed shared memory (with two CTAs per SM, the largest size whose grid
 *                  fits twice, so the next layer's CTAs are resident meanwhile); 0 = always the
 *                  global-memory merge; 2 or 4 = that cluster size whenever it applies
 *   "pdl"          1 (default) = programmatic dependent launch: a decode launch's set-up overlaps
 *                  the previous kernel of the stream (it touches no global memory before that
 *                  kernel has completed); 0 = plain stream order
 *   "early_fetch"  1 (default) = in a step of per-layer launches, a layer's grid reads its queries
 *                  and every cache tile but the newest row's before the preceding layers' grids have
 *                  finished (the step is given every layer's queries); 2 = only its first cache
 *                  tile before then, its queries after (what a layer whose queries come from the
 *                  previous layer may do: the cache and the owner's new token exist already);
 *                  0 = nothing before then
 *   "step_graph"   2 (default) = mlkv_decode_step issues a one-launch step directly and replays a
 *                  recorded CUDA graph of a per-layer step; 1 = always the graph; 0 = never (see
 *                  mlkv_decode_step)
 *   "tc"           0 (default) = the decode kernel on mma.sync tensor-core instructions; 1 = the
 *                  tcgen05 kernel (tensor-memory accumulators) for 128- and 256-position tiles,
 *                  the mma.sync kernel otherwise.  Same results within the tolerance; the tcgen05
 *                  kernel is slower for query groups of <= 16 heads (see the design notes).
 * Read-only (mlkv_get_option): "sm_count", "l2_bytes", "max_grid", "ctas_per_sm", and for the most
 * recent decode launch "last_grid", "last_tile_tokens", "last_cluster_k" (0 = global merge),
 * "last_deferred_merge", "last_tc" (1 if it ran the tcgen05 kernel), and "step_graph_replays"
 * (graph launches by mlkv_decode_step), "l2_persist_bytes" (the set-aside reserved while
 * l2_persist is on, else 0), "l2_window_max" (the device's largest access-policy window),
 * "last_step_kernel" (1 if the most recent mlkv_decode_step ran as one multi-layer launch or in
 * the fused form), "last_step_fused" (1 if in the fused form; "last_grid" is then its units and
 * "last_fused_kc" the 128-position key tiles per unit), "last_step_launches" (this library's
 * launches of that step when it ran in either form, else 0), "last_seg_major" (1 if the
 * multi-layer launch ranked its items segment-major) and "last_l2_prefetch" (1 if it prefetched
 * the slots into L2).
 * Unknown keys or values return MLKV_ERR_INVALID_ARG.
 */
int mlkv_set_option(mlkv_cache_t c, const char *key, int64_t value);
int mlkv_get_option(mlkv_cache_t c, const char *key, int64_t *value);

/* Synchronises the device, then returns MLKV_ERR_DEVICE if a kernel of this cache reported an
 * error since the last call (and clears it), MLKV_ERR_CUDA on a CUDA error, else MLKV_OK. */
int mlkv_sync_status(mlkv_cache_t c);

/* One-line description of the calling thread's most recent error ("" if none). */
const char *mlkv_last_error(void);

/*
 * mlkv_block_owner_map - the contiguous map of Eq. 18: layer n (0-based) reads the KV heads of
 * the bottom layer of its block, (n / (l/m)) * (l/m).  Host only.  n_owners must divide
 * n_layers (else MLKV_ERR_MAP).  layer_owner: host int32[n_layers], written on success.
 */
int mlkv_block_owner_map(int n_layers, int n_owners, int *layer_owner);

/*
 * mlkv_decode_attention_static - decode attention over one owner slot held by the caller, for
 * callers that cannot allocate device memory.  It allocates nothing: no cudaMalloc, cudaFree or
 * allocating library call, on any call.
 *
 * The paper has no counterpart; this is a deployment variant of mlkv_decode_attention.  Some
 * callers may not allocate device memory once they run: a runtime whose own allocator owns all
 * device memory, or a serving loop that must not call cudaMalloc (it can synchronise the device
 * and stall every stream).  Such a caller keeps the cache slot itself and passes it here; the
 * merge scratch of the split-KV kernel (partial outputs, their log-sum-exps, per-(sequence, KV
 * head) counters, an error word) lives in one array compiled into the library, of
 * MLKV_STATIC_SCRATCH_BYTES (8 MiB), which every GPU that loads the library holds until exit.
 *
 *   kv_slot    device bf16 [2][batch][kv_heads][max_seq][head_dim]: the K block then the V block
 *              of one owner layer, the layout of mlkv_kv_ptr's k_base (v_base follows it)
 *   batch, n_q_heads, kv_heads, head_dim, max_seq   as for mlkv_cache_create (kv_heads = g)
 *   Q, out, seq_lens, cuda_stream                   as for mlkv_decode_attention
 * Runs on the calling thread's current device.  The first call on a device sets that device up
 * (looks up the scratch array's device address with cudaGetSymbolAddress and raises the kernels'
 * shared-memory limits); make that first call before any stream capture.  Every call clears the
 * part of the array that must start at zero, in stream order.  All calls share the one array:
 * calls whose work overlaps on the GPU (different streams, no ordering between them) race on it
 * and must not be issued.  A request whose scratch would exceed the array (roughly
 * batch * kv_heads * (h/g) * (head_dim + 1) * 4 bytes plus one record per CTA) returns
 * MLKV_ERR_UNSUPPORTED before any work is queued.
 */
int mlkv_decode_attention_static(const void *kv_slot, int batch, int n_q_heads, int kv_heads,
                                 int head_dim, int max_seq, const void *Q, void *out,
                                 const int *seq_lens, void *cuda_stream);

/*
 * mlkv_static_status - the error record of mlkv_decode_attention_static on the current device.
 * The paper has no counterpart (see mlkv_decode_attention_static).
 *
 * The kernels of mlkv_decode_attention_static report an expired bounded wait (see
 * mlkv_sync_status) by setting bits of an error word inside the library's static scratch array;
 * the word is cleared once when a device is set up and then keeps every bit set since.  This call
 * waits for cuda_stream (a cudaStream_t, NULL = legacy default stream) to finish, reads the word,
 * clears it if it is non-zero, and returns MLKV_ERR_DEVICE if it was (mlkv_last_error gives the
 * bits), MLKV_ERR_CUDA if the stream reported a CUDA error, else MLKV_OK.  It allocates nothing.
 * Call it after the static calls whose status matters have been queued on cuda_stream (with
 * several streams, after all of them have finished); the first call on a device sets the device
 * up as mlkv_decode_attention_static does, so make it outside any stream capture.
 */
int mlkv_static_status(void *cuda_stream);

/*
 * mlkv_decode_block_fused - decode attention of every layer of one owner block in one launch:
 * each K/V tile of the owner's slot is read once for the query heads of all the block's layers.
 * NOT a step of sequential decoding: layer n+1's queries depend on layer n's output, so a model
 * never has them all at once; this call measures what the shared cache (Sec. 3) would allow if it
 * did.  The result equals mlkv_decode_attention for each layer of the block (Eqs. 2-3, 15, 18).
 *
 *   owner_layer  an owner layer o; the block is every layer n with layer_owner[n] == o, in order
 *   Q            device bf16 [L][batch][n_q_heads][head_dim], L = the block's layer count, layer-
 *                major in block order; 16-byte aligned
 *   out          device bf16 [L][batch][n_q_heads][head_dim]; must not overlap Q
 *   seq_lens     host int32[batch]: positions [0, L_beta) of the owner's slot are visible (append
 *                the new token first, e.g. with mlkv_append)
 * Needs L <= 2 * floor(128 / G), G = n_q_heads / kv_heads (the L * G query rows of one KV head
 * fill at most two 128-row tiles of whole layers), else MLKV_ERR_UNSUPPORTED.
 * Errors: MLKV_ERR_INVALID_ARG (not an owner layer, null or unaligned pointers, overlap),
 * MLKV_ERR_RANGE (lengths), MLKV_ERR_UNSUPPORTED, MLKV_ERR_CUDA.
 */
int mlkv_decode_block_fused(mlkv_cache_t c, int owner_layer, const void *Q, void *out,
                            const int *seq_lens, void *cuda_stream);

/*
 * mlkv_merge_kv_weights - converts one MHA projection (K or V) to MLKV by averaging (Sec. 4.2:
 * "KV heads in the same group of the same layer, as well as the heads from subsequent layers which
 * do not have KV heads of their own, are merged by averaging"): merged KV head j of owner layer o
 * is the mean, over every layer n with layer_owner[n] == o and every query head i of group j
 * (Eq. 12: i / (n_q_heads / n_kv_heads) == j), of W[n][i][:], rounded to bf16 (nearest, ties to
 * even).  The sums are carried as pairs of floats with exact per-addition errors, so the result
 * is the bf16 nearest to the exact mean unless that mean lies within about count^2 * 2^-48
 * (relative) of a rounding boundary (count = members of the head), provided each column's sum
 * of magnitudes stays below FLT_MAX (about 3.4e38).  Needs no cache.
 *
 *   layer_owner  host int32[n_layers]: owner[n] <= n and owner[owner[n]] == owner[n] (Eq. 18 or
 *                any such map; the identity map with n_kv_heads < n_q_heads is the GQA conversion)
 *   n_q_heads    heads per layer of the MHA model (h); n_kv_heads (g) must divide it
 *   row_elems    elements of one head's rows: head_dim * d_model for a weight, head_dim for a bias;
 *                a positive multiple of 8
 *   W            device bf16 [n_layers][n_q_heads][row_elems], 16-byte aligned, read only
 *   W_merged     device bf16 [m][n_kv_heads][row_elems], m = owner layers, in increasing layer
 *                order (the slot order of mlkv_owner_slot); 16-byte aligned; must not overlap W
 *   cuda_stream  the stream the kernel is queued on (asynchronous; nothing is allocated)
 * A model's K and V projections can go through one call: stacked as 2 * n_layers layers (K's, then
 * V's) with layer_owner[n + n_layers] = layer_owner[n] + n_layers, the merged heads come out K's
 * then V's, each equal to a call of its own (no merged head mixes layers of different owners).
 * Errors: MLKV_ERR_INVALID_ARG (null or unaligned pointers, sizes, overlap), MLKV_ERR_MAP (owner
 * map, g not dividing h), MLKV_ERR_UNSUPPORTED (more than 1024 layers or 65535 merged heads),
 * MLKV_ERR_CUDA.
 */
int mlkv_merge_kv_weights(const int *layer_owner, int n_layers, int n_q_heads, int n_kv_heads,
                          int64_t row_elems, const void *W, void *W_merged, void *cuda_stream);

/*
 * mlkv_read_bandwidth_probe - benchmark support, not part of the decode path (the paper has no
 * counterpart): queues one kernel that reads [buf, buf + bytes) `reps` times the way the decode
 * kernel moves K/V -- bulk asynchronous copies of 32 KiB into a two-stage shared-memory ring,
 * two CTAs per SM, each streaming its own contiguous share -- and does nothing else with the
 * data.  Timed with CUDA events around it on an L2-resident buffer it gives the L2 read roofline
 * of the decode layers that find their owner's slot in L2; on a buffer larger than L2, the HBM
 * read rate.  Allocates nothing.
 *
 *   buf          device memory, 16-byte aligned, read only
 *   bytes        size of buf; every CTA reads bytes / (2 * SMs) rounded down to 32 KiB
 *   reps         passes over the buffer (>= 1)
 *   bytes_read   host int64*: receives the bytes the kernel reads in all passes
 * Errors: MLKV_ERR_INVALID_ARG (null, unaligned, too small), MLKV_ERR_CUDA.
 */
int mlkv_read_bandwidth_probe(const void *buf, int64_t bytes, int reps, int64_t *bytes_read,
                              void *cuda_stream);

/* Library version, major*10000 + minor*100 + patch. */
int mlkv_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MLKV_H_ */
