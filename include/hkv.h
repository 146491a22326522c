/*
 * hkv.h — C-ABI of the HeadKV decode hot path on one GB300 (sm_103a).
 *
 * HeadKV ("Head-Aware Key-Value Compression for Efficient Autoregressive
 * Image Generation") labels every attention head local or global from the
 * early attention (Sec. 4, Step 2), gives local heads a small budget and
 * global heads rho*N tokens (Sec. 5.1), trims global heads with Stratified
 * Token Eviction (Sec. 4, Eqs. 5-6) every P steps, and decodes over the
 * resulting ragged per-head cache (Eq. 1).
 *
 * Conventions for every entry point
 *  - All pointers to tensors are DEVICE pointers unless marked "host".
 *    The caller owns every buffer and the stream; the library never
 *    allocates, frees, or keeps state between calls (all state lives in the
 *    caller's buffers).
 *  - All calls are asynchronous on `stream` except hkv_allocate_budgets and
 *    hkv_check, which synchronise it.
 *  - Per-head arrays are indexed by the flat head index
 *        i = (layer * n_seqs + seq) * n_heads + head      ([L][S][H] order),
 *    so one layer's heads are contiguous.
 *  - Per-step activations q, k, v are [n_seqs][n_heads][head_dim] in the
 *    config's dtype (fp32 or bf16), contiguous.
 *  - Errors: every call validates its arguments before launching anything
 *    and returns a status; nothing aborts or throws across the ABI.
 *    Failures detected on the device (capacity, bounds, a bounded wait that
 *    ran out) set the cache's error word; hkv_check reports it.
 *  - Fault injection for tests: if the environment variable
 *    HKV_FAULT_INJECT is "<name>:<code>" (name without the hkv_ prefix, e.g.
 *    "decode_attention:7"), that call returns <code> before touching the GPU.
 */
#ifndef HKV_H
#define HKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream (cudaStream_t); NULL selects the legacy default stream. */
typedef struct CUstream_st *hkv_stream_t;

typedef enum {
  HKV_OK = 0,
  HKV_ERR_INVALID_ARG = 1, /* null pointer, bad layer index, bad enum value */
  HKV_ERR_SHAPE = 2,       /* unsupported head_dim / dtype / sizes */
  HKV_ERR_CAPACITY = 3,    /* a segment or the workspace is too small */
  HKV_ERR_STATE = 4,       /* the cache is not in the phase the call needs */
  HKV_ERR_BOUNDS = 5,      /* a segment reaches outside the arena (device) */
  HKV_ERR_TIMEOUT = 6,     /* a bounded device wait ran out (device) */
  HKV_ERR_CUDA = 7,        /* a CUDA runtime call or launch failed */
  HKV_ERR_ALIGN = 8        /* a pointer is not 16-byte aligned */
} hkv_status;

enum { HKV_FP32 = 0, HKV_BF16 = 1 };

/* flags of hkv_decode_step */
enum {
  /* The kernel launched just before this call on the same stream does not
   * write this layer's cache (its K/V rows, off/cap/len, label, nbuf).
   * The step then reads the layer's lengths and starts streaming old K/V
   * rows while that kernel is still finishing (programmatic dependent
   * launch), and waits for it only before touching q, k, v. True when the
   * previous kernel is the decode step or attention of another layer, or
   * any call of this library other than a decode step or append of the same
   * layer (hkv_evict never lets the next kernel start early). */
  HKV_STEP_PREFETCH = 1
};

/* head labels (Sec. 4, Step 2); DENSE marks heads of the uncompressed
 * prefill-phase cache (Step 1), which are never evicted from */
enum { HKV_LOCAL = 0, HKV_GLOBAL = 1, HKV_DENSE = 255 };

/*
 * Model shape and method hyperparameters (plain data, host memory).
 *  n_cond        C: conditioning tokens, always kept (Eqs. 2-4)
 *  n_image       N: image tokens per sequence (grid rows x row_len)
 *  row_len       tokens per grid row, end-of-row token included
 *  recent_w      w: recent window, two grid rows (Sec. 5.1)
 *  local_w       w_loc: a head is local iff fewer than w_loc tokens carry
 *                tau of its attention (Sec. 4, Step 2)
 *  period        P: tokens buffered between cache updates (Sec. 4,
 *                Efficient Cache Update)
 *  group_at      E: image tokens generated when heads are grouped
 *                (Appendix, More Implementation Details)
 *  global_budget B_g = floor(rho * N) image tokens kept by a global head
 *                (Sec. 5.1); must be >= recent_w
 *  budget_mode   HKV_BUDGET_PAPER (0) or HKV_BUDGET_REDISTRIBUTE (1): the
 *                rule hkv_allocate_budgets applies (below); the update calls
 *                size their scratch for the longest segment it allows
 *  tau           accumulation threshold, 0.9 in the paper (Step 2)
 *  r_s           long/near split ratio, 0.5 in the paper (Eq. 5)
 */
typedef struct {
  int32_t n_layers, n_seqs, n_heads, head_dim;
  int32_t dtype; /* HKV_FP32 or HKV_BF16 */
  int32_t n_cond, n_image, row_len;
  int32_t recent_w, local_w, period, group_at;
  int32_t global_budget;
  int32_t budget_mode;
  int32_t distance_mode; /* HKV_DIST_RASTER or HKV_DIST_GRID2D */
  int32_t reserved;      /* must be 0 */
  double tau, r_s;
} hkv_config;

/* budget rules (hkv_config.budget_mode) */
enum {
  HKV_BUDGET_PAPER = 0,      /* Sec. 5.1: B_g (global) or w (local) */
  /* not in the paper, aggregate-preserving: within each (sequence, layer)
   * group of H heads the (H - n_g)(B_g - w) image tokens the local heads do
   * not use go to its n_g global heads in equal shares, the remainder one
   * token each to the global heads of lowest head index; the group then
   * keeps H * B_g image tokens, as if every head kept B_g. A group without
   * global heads keeps the paper's budgets. */
  HKV_BUDGET_REDISTRIBUTE = 1
};

/* token distance of head identification and of Eq. 5 (hkv_config.distance_mode) */
enum {
  /* the paper's: Step 2 counts backward from the newest token in raster
   * order, Eq. 5's long-range subset is the T r_s oldest history tokens */
  HKV_DIST_RASTER = 0,
  /* not in the paper: image token i sits in grid cell (i / row_len,
   * i % row_len) and distances are squared Euclidean distances of cells.
   * Step 2 counts the image tokens outward from the newest, nearest first
   * (equal distances newer first), then the conditioning tokens newest
   * first; Eq. 5's long-range subset is the floor(T r_s) history tokens
   * farthest from the newest image token (equal distances older first).
   * hkv_decode_step_identify does not take it (HKV_ERR_INVALID_ARG). */
  HKV_DIST_GRID2D = 1
};

/*
 * A KV cache: one arena holding every head's segment back to back.
 * Segment i spans tokens [off[i], off[i] + cap[i]) of the arena; its first
 * len[i] rows are live: the conditioning tokens, the history, the recent
 * window and the buffered tokens of Eq. 2. Attention does not depend on row
 * order, so the periodic update refills evicted rows with surviving rows
 * from the end of the segment instead of shifting everything: rows are in
 * position order only in an uncompressed (HKV_DENSE) cache and among the
 * tokens appended since the last update; pos[] identifies every row.
 * All arrays are device memory owned by the caller.
 *  k, v      arena, [capacity_tokens][head_dim] in the config dtype
 *  pos       [capacity_tokens] int32: the original cache position of each
 *            live token (conditioning j -> j, image token t -> C + t)
 *  off       [L*S*H] int64 segment offsets (tokens)
 *  cap       [L*S*H] int32 segment capacities (tokens)
 *  len       [L*S*H] int32 live tokens
 *  nbuf      [L*S*H] int32 tokens buffered since the last update
 *  ntok      [L*S*H] int32 image tokens appended so far
 *  label     [L*S*H] uint8 HKV_LOCAL / HKV_GLOBAL / HKV_DENSE
 *  qbuf      [L*S*H][P][head_dim] ring of the P latest image-token queries
 *            (Q_past of Eq. 6); image token t goes to slot t mod P
 *  err       one uint32 error word (0 = none), first error wins
 *  capacity_tokens  arena size in tokens (host value), used for checks
 */
typedef struct {
  void *k;
  void *v;
  int32_t *pos;
  int64_t *off;
  int32_t *cap;
  int32_t *len;
  int32_t *nbuf;
  int32_t *ntok;
  uint8_t *label;
  void *qbuf;
  uint32_t *err;
  int64_t capacity_tokens;
} hkv_cache;

/* Human-readable name of a status code (static string). */
const char *hkv_status_str(hkv_status s);

/* Checks a config: sizes positive, head_dim in {64, 128}, dtype known,
 * recent_w <= global_budget <= n_image, period <= group_at <= n_image,
 * 0 < tau <= 1, 0 <= r_s <= 1, budget_mode one of HKV_BUDGET_*. Host
 * only. */
hkv_status hkv_validate_config(const hkv_config *cfg);

/* Sec. 5.1: the image tokens a global head keeps, B_g = floor(rho * N),
 * for rho = rho_num / rho_den (0 < rho <= 1, rho_den < 2^31) and N = n_image
 * image tokens, in exact integer arithmetic. Writes *budget_out (host).
 * Bad arguments -> HKV_ERR_INVALID_ARG. Host only. */
hkv_status hkv_global_budget(int64_t rho_num, int64_t rho_den, int32_t n_image,
                             int32_t *budget_out);

/* Whether the decode step of image token t starts with the periodic update
 * (Sec. 4, Efficient Cache Update): *due_out = 1 iff t > E and (t - E) is a
 * multiple of P (E = group_at, P = period), else 0. The grouping step of
 * token E - 1 runs the first update itself (hkv_repack); every P tokens
 * after it the buffer is full, and the update runs after that step's
 * attention, i.e. before the next step (hkv_evict, or inside
 * hkv_append_evict). Host only. */
hkv_status hkv_update_due(const hkv_config *cfg, int32_t t, int32_t *due_out);

/* Bytes of device workspace hkv_decode_attention and hkv_decode_step need
 * for this config (split-K partial results, records of the heads split
 * between CTAs, a small control block, ready flags of the partial results
 * and four barrier words per layer). The workspace must be zero-filled before
 * its first use; every call leaves it ready for the next one (after a call
 * that reported an error, zero it again). Concurrent calls must not share a
 * workspace. Host only. */
size_t hkv_workspace_size(const hkv_config *cfg);

/* Sets up the uncompressed cache of Step 1 (cache prefilling): every head
 * gets a segment of cap = C + E tokens at off = i * (C + E), len = nbuf =
 * ntok = 0, label = HKV_DENSE, and the error word is cleared. The arena
 * must hold L*S*H*(C+E) tokens. */
hkv_status hkv_init_dense(const hkv_config *cfg, const hkv_cache *cache, hkv_stream_t stream);

/* Step 1: writes the C conditioning tokens of one layer (kc, vc:
 * [S][H][C][head_dim]) at the start of every head's segment and sets
 * len = C. Only for an HKV_DENSE cache of a fresh layer. */
hkv_status hkv_prefill(const hkv_config *cfg, const hkv_cache *cache, int layer,
                       const void *kc, const void *vc, hkv_stream_t stream);

/* One decode step of one layer, before its attention (KV cache update,
 * Sec. 3; periodic update, Sec. 4):
 *  1. for a compressed head whose buffer holds P tokens, run the update
 *     first: a local head keeps its conditioning and newest w tokens
 *     (Eq. 3); a global head whose history exceeds its budget (cap - C - P
 *     - w: B_g - w under the paper's budgets) evicts the excess
 *     by STE (Eqs. 4-6: long/near split by r_s, in raster order or on the
 *     grid per cfg->distance_mode; scores from the P buffered
 *     queries, the lowest floor(M/2) / M - floor(M/2) of each subset
 *     evicted, older first on equal score); the segment shrinks in place by
 *     moving the surviving rows above the new length into the evicted rows
 *     below it;
 *  2. append k, v of the new image token at the tail (pos = C + ntok), push
 *     q into the Q_past ring, len += 1.
 * q, k, v: [S][H][head_dim]. A full segment sets HKV_ERR_CAPACITY in the
 * error word and leaves that head unchanged. */
hkv_status hkv_append_evict(const hkv_config *cfg, const hkv_cache *cache, int layer,
                            const void *q, const void *k, const void *v, hkv_stream_t stream);

/* The periodic head-aware update alone (Sec. 4, Efficient Cache Update;
 * Eqs. 3-6), for every head of the layer whose buffer holds P tokens: the
 * same update hkv_append_evict runs before its append, without the append.
 * Heads whose buffer is not full are left as they are, so the call is
 * harmless when no update is due; with hkv_decode_step it must run before
 * the step that follows the P-th buffered token. The update stages the P
 * buffered queries, then rows of keys, in shared memory: the larger of
 * P * head_dim * elem and 256 * (head_dim * elem + 16) bytes, plus 16 bytes
 * per token of the longest segment, must fit in 227 KB, else
 * HKV_ERR_CAPACITY (also for hkv_append_evict and hkv_repack). */
hkv_status hkv_evict(const hkv_config *cfg, const hkv_cache *cache, int layer, hkv_stream_t stream);

/* hkv_evict for every layer in one launch (one CTA per head of the model):
 * the same update of every head whose buffer holds P tokens, the same
 * results, the same checks and errors. All heads fill their buffers at the
 * same token, so one call before the first layer's step replaces a call
 * per layer; the per-head updates are independent and latency-bound, and
 * one launch keeps the GPU full with them. Asynchronous on `stream`. */
hkv_status hkv_evict_all(const hkv_config *cfg, const hkv_cache *cache, hkv_stream_t stream);

/* One decode step of one layer: the append of the new token (Sec. 3, KV
 * Cache) fused with the attention of Eq. 1 over the cache including that
 * token. One kernel launch when every CTA's share of the layer spans at
 * most 128 heads (bounded from the config: the heads of a layer times the
 * tiles of the longest segment it allows, over the grid), else two chained
 * kernels (attention, then a finishing kernel that combines heads split
 * across CTAs and advances the counters); hkv_decode_step_launches tells
 * which. out[s][h][:] = softmax(q k^T / sqrt(d)) V over the
 * head's len live tokens and the new one (whose K/V are read straight from
 * k and v), fp32; then k, v join the arena at row len, q joins the Q_past
 * ring, and len, ntok (and nbuf for compressed heads) advance by one.
 * q, k, v: [S][H][head_dim] in the config dtype; workspace of
 * hkv_workspace_size bytes. A compressed head whose buffer already holds P
 * tokens (hkv_evict not run) sets HKV_ERR_STATE, a full segment
 * HKV_ERR_CAPACITY, in the error word; the step is then not taken.
 * flags: 0 or HKV_STEP_PREFETCH (see above). */
hkv_status hkv_decode_step(const hkv_config *cfg, const hkv_cache *cache, int layer,
                           const void *q, const void *k, const void *v, float *out,
                           void *workspace, size_t ws_bytes, int flags, hkv_stream_t stream);

/* Kernel launches one hkv_decode_step call of this config makes on the
 * current device: 1 or 2 (see hkv_decode_step); 0 for an invalid config or
 * a failed device query. Host only. */
int hkv_decode_step_launches(const hkv_config *cfg);

/* hkv_decode_step fused with the head-type identification of Sec. 4,
 * Step 2, for the grouping step (image token E - 1) on the uncompressed
 * cache: besides everything hkv_decode_step does, each head's attention
 * mass on its newest local_w - 1 tokens (the new one included) is
 * accumulated with the softmax sum, and label_out[i] (device, [L*S*H], flat
 * head index i) becomes HKV_LOCAL iff that mass is at least tau of the
 * total, i.e. iff fewer than local_w tokens, counted back from the newest,
 * carry tau of the attention; else HKV_GLOBAL. Same decision as
 * hkv_identify_heads over the same cache (which also reports n_h; this
 * does not). A head of another label than HKV_DENSE sets HKV_ERR_STATE in
 * the error word and the step is not taken; label_out NULL ->
 * HKV_ERR_INVALID_ARG. */
hkv_status hkv_decode_step_identify(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                    const void *q, const void *k, const void *v, float *out,
                                    uint8_t *label_out, void *workspace, size_t ws_bytes,
                                    int flags, hkv_stream_t stream);

/* Eq. 1 for one new query per head over that head's live tokens (any mix
 * of lengths): out[s][h][:] = softmax(q k^T / sqrt(d)) V, fp32 accumulation,
 * written in fp32 ([S][H][head_dim]). Split-K over the layer's total token
 * count, then a second kernel combines the heads split across CTAs;
 * workspace of hkv_workspace_size bytes.
 * A head with len = 0 yields zeros. */
hkv_status hkv_decode_attention(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                const void *q, float *out, void *workspace, size_t ws_bytes,
                                hkv_stream_t stream);

/* hkv_decode_attention for callers that cannot allocate device memory:
 * the paper has no counterpart to this entry point. A plain C host program
 * without a device allocator, or a plugin inside a host framework that owns
 * and budgets all device memory, may have no way to provide the workspace
 * that hkv_decode_attention takes. Here the split-K partials, the records
 * of heads split between CTAs and the kernels' control block live in a
 * fixed device array inside the library (1.06 MiB: 1 MiB of partials,
 * 64 KiB of records, 256 bytes), which every GPU that loads the library
 * holds until the process exits. Nothing in it has to start at zero: each
 * call writes what it reads. Same inputs, outputs and results as
 * hkv_decode_attention; it allocates nothing.
 *  - The first call on a device, with that device current, looks up the
 *    array's device address and prepares the kernel; make that first call
 *    before any stream capture. The address is kept for the rest of the
 *    process: do not reset the device (cudaDeviceReset) after that call.
 *  - Every call uses the same array; calls that may overlap on the GPU
 *    (other streams, other host threads) race on it and must be serialised
 *    by the caller. */
hkv_status hkv_decode_attention_noalloc(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                        const void *q, float *out, hkv_stream_t stream);

/* Sec. 4, Step 2 for one layer of an HKV_DENSE cache (heads of any other
 * label set HKV_ERR_STATE in the error word): for each head, the
 * attention of q over the live keys is accumulated backward from the newest
 * token (or outward on the grid, HKV_DIST_GRID2D) until tau is reached; n_h
 * is the number of tokens needed and the head is HKV_LOCAL iff n_h < w_loc.
 * Writes label_out[i] and, if non-null,
 * nh_out[i] for the layer's heads (i = flat head index; both arrays are
 * [L*S*H]). */
hkv_status hkv_identify_heads(const hkv_config *cfg, const hkv_cache *cache, int layer,
                              const void *q, uint8_t *label_out, int32_t *nh_out,
                              hkv_stream_t stream);

/* A variant of Sec. 4, Step 2 that the paper does not have: the decision
 * from the attention of several recent queries instead of the current one.
 * For each head of one layer of an HKV_DENSE cache, the newest
 * Pe = min(period, ntok) queries of the cache's query ring (written by the
 * decode steps; the newest is the current token's) each attend over the keys
 * that existed at their own step: the p-th oldest (p = 0 .. Pe-1) over the
 * oldest len - (Pe - 1 - p) keys. Their softmax rows are averaged, the
 * average is accumulated backward from the newest token (or outward on the
 * grid, HKV_DIST_GRID2D) until tau is
 * reached, n_h is the number of tokens needed, and the head is HKV_LOCAL iff
 * n_h < w_loc. With period = 1 this is hkv_identify_heads. Call it after the
 * grouping token's decode step, like hkv_identify_heads. Writes
 * label_out[i] and, if non-null, nh_out[i] for the layer's heads (device
 * arrays of [L*S*H]).
 *  - a head with another label than HKV_DENSE, or with ntok = 0 (no query
 *    buffered yet): HKV_ERR_STATE in the error word, head not decided;
 *  - len above n_cond + group_at: HKV_ERR_CAPACITY in the error word;
 *  - n_cond + group_at tokens that do not fit one block's shared memory
 *    (36 bytes a token for a period of 48 or more, else 20; 12 more with
 *    HKV_DIST_GRID2D; 227 KB in all): HKV_ERR_CAPACITY returned, nothing
 *    launched;
 *  - label_out NULL or layer out of range: HKV_ERR_INVALID_ARG. */
hkv_status hkv_identify_heads_multi(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                    uint8_t *label_out, int32_t *nh_out, hkv_stream_t stream);

/* Sec. 5.1 budgets for all L*S*H heads from their labels: budget = B_g
 * (global) or w (local) image tokens (or the redistributed budgets, per
 * cfg->budget_mode), cap = C + budget + P, off = exclusive prefix sum of cap
 * (tokens). The periodic update reads each global head's history budget
 * from its capacity (cap - C - P - w). Writes budget, cap, off (device) and the
 * arena size in tokens to *total_tokens (host); synchronises the stream.
 * A label other than HKV_LOCAL / HKV_GLOBAL yields HKV_ERR_STATE. */
hkv_status hkv_allocate_budgets(const hkv_config *cfg, const uint8_t *label, int32_t *budget,
                                int32_t *cap, int64_t *off, int64_t *total_tokens,
                                hkv_stream_t stream);


/* Head-aware compression of one layer after grouping (Step 3): copies
 * every head of the dense cache into its segment of the ragged cache (whose
 * off, cap and label arrays the caller filled from hkv_allocate_budgets and
 * hkv_identify_heads) and applies the first update there: local heads keep
 * the conditioning and newest w tokens; global heads keep a history of at
 * most cap - C - P - w tokens (B_g - w under the paper's budgets) chosen by
 * STE with the P latest queries. Sets len,
 * nbuf = 0 and ntok on the ragged side. The two caches share the qbuf ring
 * layout; the ragged cache's qbuf must be the dense cache's qbuf. */
hkv_status hkv_repack(const hkv_config *cfg, const hkv_cache *dense, const hkv_cache *ragged,
                      int layer, hkv_stream_t stream);

/* Synchronises the stream and returns the status recorded in the cache's
 * error word (HKV_OK if none), or HKV_ERR_CUDA if the stream failed. */
hkv_status hkv_check(const hkv_cache *cache, hkv_stream_t stream);

/* Copies one layer's cache state to host memory, for a checkpoint or for
 * comparing the cache with a reference at any step (the paper has no
 * counterpart). For the layer's S*H heads, in flat order s*H + h: label,
 * len, nbuf and ntok (host arrays of S*H entries each, any of them NULL to
 * skip), and the positions of every head's live tokens, head after head, in
 * the order they sit in the head's segment (pos_out: host int32 array of
 * pos_capacity entries, or NULL). *pos_count (if not NULL) receives the
 * layer's live token count, the entries written to pos_out. Host memory may
 * be pageable. Synchronises the stream; the work queued before it on the
 * stream is included.
 *  - pos_out given and pos_capacity below the live token count ->
 *    HKV_ERR_CAPACITY (nothing written to pos_out);
 *  - a segment with len < 0 or outside the arena -> HKV_ERR_BOUNDS. */
hkv_status hkv_export_state(const hkv_config *cfg, const hkv_cache *cache, int layer,
                            uint8_t *label_out, int32_t *len_out, int32_t *nbuf_out,
                            int32_t *ntok_out, int32_t *pos_out, int64_t pos_capacity,
                            int64_t *pos_count, hkv_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* HKV_H */
