/* memdecay.h -- C ABI of the GB300 (sm_103a) MemDecay decode-time eviction loop.
 *
 * MemDecay ("MemDecay: Region-Aware KV Cache Eviction for Efficient LLM Agent
 * Inference", arXiv 2607.10582) keeps, for every cached token i of a paged KV
 * cache, a region label r(i), an attention importance a_i and a decay clock
 * t_ref_i.  At every observation step (Algorithm 1) it updates a_i with an
 * EWMA of the attention mass the token received (Eq. 2), restarts the clock of
 * tokens attended above a threshold (Eq. 3), scores every token with its
 * region's decayed base priority plus its weighted importance (Eq. 4), reduces
 * token scores to page scores (Eq. 5) and, when the cache holds more pages than
 * the budget, evicts the lowest-scoring non-pinned pages (Sec. III-D).
 *
 * This library implements that loop on one GPU, in four stages run by
 * md_decode_step and md_evict:
 *   1. paged GQA decode attention that also produces each cached token's
 *      attention mass (Sec. III-C, observation of Abar_i);
 *   2. per-token retention priority (Eqs. 2-4);
 *   3. token -> page priority (Eq. 5, pinning protects whole pages, Sec. IV-A);
 *   4. budgeted selection of the lowest-priority pages (radix select) and
 *      compaction of the block table and free list (Sec. III-D, Algorithm 1).
 *
 * Conventions shared by every call
 * --------------------------------
 * - Memory: the library allocates no device memory.  The caller passes one
 *   device workspace (md_config.workspace) of md_workspace_size() bytes, which
 *   holds the KV page pool and all per-token / per-page state.  Device
 *   pointers passed to calls are borrowed for the duration of the call's GPU
 *   work only; K/V are copied into the pool.
 * - Streams: every call enqueues its GPU work on md_config.stream (a
 *   cudaStream_t) and returns without synchronising, except where stated.
 * - Host mirror: sequence token/page counts, the free-stack top and the step
 *   counter are tracked exactly on the host, so argument and capacity errors
 *   are returned synchronously, before anything is launched, and nothing is
 *   changed when a call fails.
 * - Device errors (an exchange wait that timed out) are recorded in a sticky
 *   device status word, read by md_sync(); after one, the handle refuses
 *   further work (MD_ERR_STATE) and must be destroyed.  No kernel traps.
 * - Threading: a handle is used from one host thread and one stream.
 * - Layouts are row-major; bf16 tensors are passed as raw 16-bit patterns.
 */
#ifndef MEMDECAY_H
#define MEMDECAY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct md_ctx md_ctx; /* opaque, host-owned */

typedef enum {
  MD_OK = 0,
  MD_WARN_OVER_BUDGET = 1,     /* pinned pages alone exceed a budget: every
                                  evictable page was evicted, state is valid */
  MD_ERR_INVALID_ARG = -1,
  MD_ERR_CAPACITY = -2,        /* block table row or page pool would overflow */
  MD_ERR_WORKSPACE = -3,       /* workspace missing, misaligned or too small */
  MD_ERR_CUDA = -4,            /* a CUDA runtime call failed */
  MD_ERR_DEVICE_TIMEOUT = -5,  /* a bounded device-side wait ran out */
  MD_ERR_STATE = -6            /* call not valid in the handle's state */
} md_status;

/* Region labels, in the order Sec. III-A lists them. */
enum {
  MD_REGION_SYSTEM = 0,
  MD_REGION_PLAN = 1,
  MD_REGION_USER = 2,
  MD_REGION_TOOL_IN = 3,
  MD_REGION_TOOL_OUT = 4,
  MD_REGION_RETRIEVAL = 5,
  MD_REGION_SCRATCHPAD = 6,
  MD_NUM_REGIONS = 7
};

#define MD_MAX_BATCH 256          /* sequences per handle                     */
#define MD_HEAD_DIM 128           /* the only supported head dimension        */
#define MD_MAX_GROUP 8            /* query heads per KV head (GQA group)      */
#define MD_MAX_CHUNKS 64          /* attention splits per (seq, layer, head)  */
#define MD_MAX_CHUNK_TOKENS 4096  /* tokens per attention split               */
#define MD_CALIB_BUCKETS 256      /* age buckets of the calibration histogram  */
#define MD_CALIB_BUCKET_WIDTH 4   /* decode steps per age bucket (Fig. 3)      */

typedef struct {
  /* Geometry: L layers (1..255), Hq query heads, Hkv KV heads (Hq / Hkv <= 8,
   * L * Hq < 65,536), head_dim must be 128, page_size 16 or 32 tokens
   * (Sec. III-D, fixed-size pages). */
  int num_layers, num_q_heads, num_kv_heads, head_dim, page_size;
  /* Capacity: sequences, block-table width (pages per sequence, at most
   * MD_MAX_CHUNKS * MD_MAX_CHUNK_TOKENS / page_size), pages in the pool. */
  int max_batch, max_pages_per_seq, num_phys_pages;
  /* Policy (Sec. IV-A uses rho 0.9, gamma = 1 - rho, tau = 2 / |K_t|):
   *   a_i <- rho a_i + gamma Abar_i                           (Eq. 2)
   *   refresh when Abar_i >= tau_scale / |K_t|                 (Eq. 3)
   *   score_mode 0: s_i = b_r 2^(-dt/h_r) + attn_weight a_i    (Eq. 4)
   *   score_mode 1: s_i = (b_r + attn_weight a_i) 2^(-dt/h_r)
   *   score_mode 2: s_i = b_r 2^(-dt/h_r) + attn_weight a_i |K_t|: the
   *                 attention term relative to the uniform level 1/|K_t|, the
   *                 change the paper's ablation points to (Sec. IV-D, Sec. V)
   *   score_mode 3: s_i = t_ins_i (recency; the streaming baseline, Sec. IV-C)
   *   score_mode 4: s_i = uniform draw per token and observation step from
   *                 random_seed (the random baseline, Sec. IV-C)
   *   (the H2O-style baseline of Sec. IV-C is score_mode 0 with rho = gamma
   *    = 1, every b_r = 0 and no pinned region: accumulated attention)
   *   Pinned regions score +inf in every mode.
   *   page_reduce 0: S_p = mean over the page's tokens (Eq. 5); 1: max. */
  float rho, gamma, tau_scale, attn_weight;
  int score_mode, page_reduce;
  int keep_token_prio;        /* 1: store s_i per token (md_get_state) */
  void *workspace;            /* device memory, 256-byte aligned, caller-owned */
  size_t workspace_bytes;
  void *stream;               /* cudaStream_t (NULL = legacy default stream) */
  uint64_t random_seed;       /* score_mode 4 only */
  /* 1: region-aligned page allocation -- a token whose region differs from
   * the page being written opens a fresh page, so no page holds two regions
   * (the allocator variant Sec. III-D leaves to future work).  Pages may then
   * be partly filled; every stage masks by each page's fill. */
  int region_aligned_pages;
} md_config;

/* Bytes of device workspace md_create needs for cfg (0 if cfg is invalid).
 * Pure host arithmetic; no CUDA call. */
size_t md_workspace_size(const md_config *cfg);

/* Validates cfg, lays out the workspace, and enqueues its initialisation
 * (empty cache, free stack [P-1, ..., 0] so the first page taken is 0).
 * Region parameters start as b = 0, half-life = +inf, not pinned.
 * MD_ERR_CAPACITY if the device holds fewer than MD_MAX_CHUNKS attention CTAs
 * at once (every chunk of an item must fit in one round of the grid). */
md_status md_create(const md_config *cfg, md_ctx **out);

/* Structural prior of one region (Sec. III-B, Table 1): base priority
 * b_r >= 0 and half-life h_r > 0 in decode steps (lambda_r = ln 2 / h_r,
 * Eq. 7; h_r = +INFINITY means lambda_r = 0).  pinned != 0 puts the region in
 * the never-evicted set F (Eq. 1).  The pinned flag can only change while no
 * sequence holds tokens (MD_ERR_STATE otherwise); b_r and h_r at any time. */
md_status md_set_region_params(md_ctx *ctx, int region, float base_priority,
                               float half_life_steps, int pinned);

/* Appends n tokens to sequence seq (the prompt from the orchestrator, Fig. 1
 * "append KV"; Sec. III-A: every token carries a region label and an
 * insertion step).
 *   regions_host      [n] region label per token (host memory)
 *   insert_steps_host [n] insertion step per token (host), each <= the current
 *                     step; NULL means the current step for all
 *   k_dev, v_dev      bf16 [L][Hkv][n][D] (device)
 * Each token starts with a_i = 0 and t_ref_i = its insertion step.  New pages
 * are taken from the free stack. */
md_status md_append_tokens(md_ctx *ctx, int seq, int n_tokens, const uint8_t *regions_host,
                           const int32_t *insert_steps_host, const void *k_dev,
                           const void *v_dev);

/* One decode step for sequences [0, batch): advances the step counter t,
 * appends each sequence's new token (region new_region_host[b], inserted at
 * t), then runs stage 1: for every layer and query head, attention over every
 * cached token of the sequence (the new one included; no mask), writing the
 * output and accumulating each token's attention mass for the observation
 * window (Sec. III-C).
 *   q_dev               bf16 [batch][L][Hq][D]    (device)
 *   k_new_dev, v_new_dev bf16 [batch][L][Hkv][D]  (device)
 *   new_region_host     [batch]                   (host)
 *   out_dev             bf16 [batch][L][Hq][D]    (device, written)
 * All steps of one observation window must use the same batch. */
md_status md_decode_step(md_ctx *ctx, int batch, const void *q_dev, const void *k_new_dev,
                         const void *v_new_dev, const uint8_t *new_region_host, void *out_dev);

/* md_decode_step with the step's tensors in host memory.  The query rows
 * are copied into the workspace before the step.  The new tokens' K/V and
 * the output are used where they are when the device can reach them: the
 * kernels read the K/V rows and write the output over the host link (on a
 * GB300, NVLink-C2C), with no copy.  The device reaches pinned (page-locked)
 * or registered host memory, and, where it accesses pageable memory
 * coherently (cudaDevAttrPageableMemoryAccess, as on Grace-Blackwell), any
 * host memory; the buffers must be 16-byte aligned for this.  Other buffers
 * are copied through the workspace.  Copies are enqueued on the handle's
 * stream, inputs before the step and the output after it.  Like every call
 * it is asynchronous: out_host holds the output once the stream has passed
 * the step (md_sync, or a synchronisation of the stream), and the input
 * buffers must stay unchanged until then.  Layouts as md_decode_step:
 *   q_host                  bf16 [batch][L][Hq][D]   (host)
 *   k_new_host, v_new_host  bf16 [batch][L][Hkv][D]  (host)
 *   new_region_host         [batch]                  (host)
 *   out_host                bf16 [batch][L][Hq][D]   (host, written)
 * Errors as md_decode_step; every argument check runs before any copy or
 * launch. */
md_status md_decode_step_host(md_ctx *ctx, int batch, const void *q_host, const void *k_new_host,
                              const void *v_new_host, const uint8_t *new_region_host,
                              void *out_host);

/* The same decode step, one layer per call, for a model that runs its other
 * per-layer work (MLP, norms) between the layers' attentions: the production
 * shape of the loop (Fig. 1: the decode engine appends KV and attends layer
 * by layer; Sec. III-C: the mass is gathered over all layers).  Call it for
 * layers 0, 1, ..., L-1 in order; after the call for layer L-1 the step is
 * complete and equivalent to md_decode_step.  Layer 0 advances the step
 * counter, takes new pages and starts the new tokens' state (it reads
 * new_region_host); every layer writes its own K/V row of the new tokens and
 * runs stage 1 for that layer only.  While a step is in progress, calls other
 * than the next layer return MD_ERR_STATE.
 *   q_dev                bf16 [batch][Hq][D]   (this layer)
 *   k_new_dev, v_new_dev bf16 [batch][Hkv][D]  (this layer)
 *   new_region_host      [batch]               (host; read at layer 0)
 *   out_dev              bf16 [batch][Hq][D]   (written) */
md_status md_decode_layer(md_ctx *ctx, int layer, int batch, const void *q_dev,
                          const void *k_new_dev, const void *v_new_dev,
                          const uint8_t *new_region_host, void *out_dev);

/* The observation step of Algorithm 1 for sequences [0, batch): stages 2-4.
 * If decode steps ran since the last call, Abar_i = (attention mass summed
 * over those k steps, layers and query heads) / (k L Hq), then Eq. 2, Eq. 3
 * with tau = tau_scale / |K_t| (|K_t| = tokens cached now); if none ran, the
 * EWMA and the clocks are left as they are.  Then Eq. 4 and Eq. 5 (pinned
 * pages and each sequence's last page, the one being written, score +inf),
 * and, for every sequence holding more pages than budget_pages_host[b]
 * (partial last page included), eviction of the lowest-S_p evictable pages
 * (ties: lower logical page index first), stable compaction of its block-table
 * row, and a push of the freed physical ids onto the free stack in
 * (sequence, logical page) order.
 *   budget_pages_host [batch]            (host)
 *   n_evicted_host    [batch] or NULL    (host, written before return: the
 *                                         counts come from the host mirror)
 *   evicted_ids_dev   [batch][max_pages_per_seq] or NULL (device, written:
 *                     freed physical ids in logical order, -1 padded)
 * Returns MD_WARN_OVER_BUDGET when pinned pages keep a sequence above its
 * budget. */
md_status md_evict(md_ctx *ctx, int batch, const int32_t *budget_pages_host,
                   int32_t *n_evicted_host, int32_t *evicted_ids_dev);

/* Waits for the handle's stream and returns the sticky device status. */
md_status md_sync(md_ctx *ctx);

md_status md_destroy(md_ctx *ctx);

/* ---- inspection, test and checkpoint support -------------------------- */

enum {
  MD_STATE_BLOCK_TABLE = 0, /* int32 [max_batch][max_pages_per_seq] physical ids     */
  MD_STATE_PAGE_SCORE = 1,  /* fp32  [max_batch][max_pages_per_seq] S_p (last evict)  */
  MD_STATE_TOKEN_PRIO = 2,  /* fp32  [num_phys_pages*page_size] s_i per physical slot */
  MD_STATE_A = 3,           /* fp32  [slots] a_i                                      */
  MD_STATE_T_REF = 4,       /* int32 [slots] t_ref_i                                  */
  MD_STATE_AHAT = 5,        /* fp32  [slots] Abar_i of the last observation           */
  MD_STATE_FREE = 6,        /* int32 [num_phys_pages] free stack (top: md_query)      */
  MD_STATE_REGION = 7,      /* uint8 [slots] region label                             */
  MD_STATE_WINDOW = 8,      /* fp32  [slots] attention mass of folded window steps    */
  MD_STATE_MASS = 9,        /* u64   [slots] attention mass of the last decode step,
                               summed over layers and query heads, in fixed point
                               (2^48 = 1.0); cleared when an evict or the next
                               step folds it                                  */
  MD_STATE_POOL = 10,       /* bf16  [L][num_phys_pages][Hkv][2][page_size][D] K/V    */
  MD_STATE_T_INS = 11,      /* int32 [slots] insertion step                           */
  MD_STATE_PAGE_FILL = 12,  /* uint8 [max_batch][max_pages_per_seq] tokens per page   */
  MD_STATE_SEQ_TOKENS = 13, /* int32 [max_batch] tokens per sequence (device count)   */
  MD_STATE_CALIB = 14       /* bytes: the calibration histogram, u64 [8][MD_CALIB_BUCKETS]
                               fixed-point mass sums (2^32 = 1.0), then u32 [8][MD_CALIB_BUCKETS]
                               counts; part of a checkpoint                            */
};

/* Device-to-device copy of one state array into dst_dev (bytes must equal the
 * array's size), enqueued on the stream. */
md_status md_get_state(md_ctx *ctx, int what, void *dst_dev, size_t bytes);

/* Overwrites one state array from src_dev (test support: lets a parity test
 * put the oracle's choice back where floating-point ties allowed the GPU
 * another valid one).  Only BLOCK_TABLE, FREE, A, T_REF, PAGE_FILL and
 * SEQ_TOKENS; the caller keeps them consistent with the host mirror's counts. */
md_status md_set_state(md_ctx *ctx, int what, const void *src_dev, size_t bytes);

enum {
  MD_QUERY_TOKENS = 0,   /* cached tokens of sequence seq            */
  MD_QUERY_PAGES = 1,    /* resident pages of sequence seq           */
  MD_QUERY_FREE_TOP = 2, /* free-stack height                        */
  MD_QUERY_STEP = 3,     /* current decode step t                    */
  MD_QUERY_WINDOW = 4,   /* decode steps since the last observation  */
  MD_QUERY_PINNED_PAGES = 5 /* pages of seq holding a pinned token   */
};
md_status md_query(const md_ctx *ctx, int what, int seq, int64_t *out);

/* Checkpoint of everything but the page pool's contents: device state into
 * dst_dev (md_state_bytes() device bytes) and the host mirror into host_blob
 * (host bytes).  Only between observation windows (MD_ERR_STATE otherwise).
 * md_load_state restores both, and clears any step mass the live state had
 * pending; the pool must still hold the saved pages. */
md_status md_state_bytes(const md_ctx *ctx, size_t *device_bytes, size_t *host_bytes);
md_status md_save_state(md_ctx *ctx, void *dst_dev, void *host_blob);
md_status md_load_state(md_ctx *ctx, const void *src_dev, const void *host_blob);

/* Per-stage GPU time, from CUDA events recorded around each launch while
 * enabled.  Stages: 0 append, 1 attention (stage 1), 2 window fold,
 * 3 score + page reduce (stages 2-3), 4 select + compact (stage 4).
 * md_profile_read synchronises the stream and returns, for each stage, the
 * summed milliseconds and the number of launches since enabling.  Each event
 * pair keeps consecutive kernels from overlapping (about 2 us per event on a
 * GB300), so profiled steps are slower than unprofiled ones: time whole
 * steps with profiling off. */
md_status md_profile_enable(md_ctx *ctx, int enable);
md_status md_profile_read(md_ctx *ctx, double *ms_per_stage, int64_t *launches_per_stage,
                          int n_stages);

/* Test and tuning support.
 *   MD_DEBUG_SPIN_LIMIT_NS    limit of each device-side wait (default 2e9)
 *   MD_DEBUG_EXTRA_ARRIVALS   extra arrivals the attention exchange waits for
 *                             on its next launch (a wait nothing completes;
 *                             the kernel then reports MD_ERR_DEVICE_TIMEOUT)
 *   MD_DEBUG_GRID_LIMIT       cap on the attention kernel's persistent CTAs
 *                             (0 = all that fit on the device; otherwise at
 *                             least MD_MAX_CHUNKS, so that all chunks of an
 *                             item fit in one round of the grid)
 *   MD_DEBUG_UNIT_OVERHEAD    per-unit cost, in KiB of K/V streamed, that the
 *                             attention work planner adds to each chunk
 *                             (default 112; 0..65536)
 *   MD_DEBUG_FORCE_CHUNKS     chunks per (sequence, layer, KV head) item
 *                             (0 = planned; otherwise clamped to the limits)
 *   MD_DEBUG_COMBINE_OVERHEAD cost, in KiB of K/V streamed by one CTA, that
 *                             the planner adds to a split giving any item
 *                             several chunks (default 192; 0..65536)
 *   MD_DEBUG_ZERO_COPY        1 (default): md_decode_step_host uses the K/V
 *                             and output buffers in place where the device
 *                             reaches them; 0: it copies every buffer
 *                             through the workspace */
enum {
  MD_DEBUG_SPIN_LIMIT_NS = 0,
  MD_DEBUG_EXTRA_ARRIVALS = 1,
  MD_DEBUG_GRID_LIMIT = 2,
  MD_DEBUG_UNIT_OVERHEAD = 3,
  MD_DEBUG_FORCE_CHUNKS = 4,
  MD_DEBUG_COMBINE_OVERHEAD = 5,
  MD_DEBUG_ZERO_COPY = 6
};
md_status md_debug_set(md_ctx *ctx, int key, int64_t value);

/* Text of the last error on this handle ("" if none). */
const char *md_last_error(const md_ctx *ctx);

/* ---- calibration by-product (Sec. IV-B, Eqs. 6-7) --------------------- */

/* While enabled, every observation step (md_evict after decode steps) adds
 * each cached token's observed mass Abar_i to a histogram indexed by its
 * region and its age bucket floor((t - t_ins) / MD_CALIB_BUCKET_WIDTH), ages
 * 0 .. MD_CALIB_BUCKETS * width - 1 (older tokens are not counted): the data
 * behind the paper's per-region lifetime curves (Fig. 3).  Enabling clears
 * the histogram.  Sums are kept in fixed point (resolution 2^-32 per token),
 * so the histogram is deterministic. */
md_status md_calib_enable(md_ctx *ctx, int enable);

/* Copies the histogram out: mass_sum[r][b] (sum of Abar), count[r][b]
 * (observations), r < MD_NUM_REGIONS, b < MD_CALIB_BUCKETS (host arrays).
 * Synchronises the handle's stream. */
md_status md_calib_read(md_ctx *ctx, double *mass_sum, int64_t *count);

/* Eq. 6 fit, host arithmetic only: per region, over the buckets with at least
 * min_count observations and a positive mean, weighted least squares of
 * log(mean mass) against the bucket's centre age (bucket_width * b +
 * bucket_width / 2) with the observation counts as weights (the count-weighted
 * fit of Sec. IV-B).  rate_out[r] = lambda_hat_r (NaN with fewer than two
 * buckets), half_life_out[r] = ln 2 / lambda_hat_r (Eq. 7; +inf if
 * lambda_hat_r <= 0).  Arrays are [MD_NUM_REGIONS][n_buckets] in,
 * [MD_NUM_REGIONS] out. */
md_status md_calib_fit(const double *mass_sum, const int64_t *count, int n_buckets,
                       int bucket_width, int64_t min_count, double *rate_out,
                       double *half_life_out);

/* ---- stage 1 for callers that cannot allocate device memory ----------- */

/* The paper has no counterpart to this call.  It exists for callers that
 * cannot call cudaMalloc or any allocating routine: code running where the
 * allocator is owned by someone else (a serving engine or framework that
 * hands out only the tensors it allocated), code that must not allocate
 * once it is running, or embedders whose memory budget is fixed up front.
 * Those callers cannot provide md_decode_step's workspace.
 *
 * It runs stage 1 alone -- paged GQA decode attention over every cached
 * token plus each token's attention mass per (layer, KV head) -- over a paged
 * cache the caller already owns, with md_decode_step's kernel (an instance
 * that writes the masses as rows instead of adding them into one sum per
 * token) and its arithmetic.
 * The kernel's scratch memory (score rows, split partials, arrival counters,
 * status words) lives in one fixed 24 MiB device array inside the library,
 * which every GPU that loads the library holds until the process exits.
 * Nothing is allocated by this call.
 *
 *   kv_pool_dev      bf16 [L][num_phys_pages][Hkv][2][page_size][128]: for
 *                    each (layer, page, KV head) the page's K rows then its V
 *                    rows (md_decode_step's pool layout; 16-byte aligned)
 *   block_table_dev  int32 [batch][max_pages_per_seq] physical page ids
 *   n_tokens_host    [batch] cached tokens per sequence (host), each >= 1 and
 *                    at most max_pages_per_seq * page_size
 *   q_dev            bf16 [batch][L][Hq][128]
 *   out_dev          bf16 [batch][L][Hq][128] (written)
 *   mass_dev         fp32 [L*Hkv][num_phys_pages*page_size] (written at the
 *                    slots of cached tokens: sum over the KV head's query heads
 *                    of their softmax weight on the token)
 *   stream           cudaStream_t
 *
 * Limits: the work must fit the 24 MiB array.  Each (sequence, layer, KV
 * head) is split into C chunks of at most 1,024 tokens (C <= MD_MAX_CHUNKS),
 * as few as keep every CTA of the grid busy.  The array holds one arrival
 * counter per item, two rows of chunk scores (32 bytes per token) per CTA of
 * the launched grid, and, when C > 1, C partials of 4,352 bytes per item.
 * In practice: any batch whose sequences all hold at most 1,024 tokens (one
 * chunk per item, no partials) fits; so does, for instance, 16 sequences of
 * 3,000 tokens over 16 layers and 2 KV heads (C = 4, about 23.5 MiB).  Work
 * that fits no split (for instance 32 sequences of 1,700 tokens over 36
 * layers and 2 KV heads) is rejected with MD_ERR_CAPACITY before anything is
 * launched, and so is a split whose C exceeds the CTAs the device holds at
 * once (all chunks of an item must run in one round of the persistent
 * grid); bad arguments with MD_ERR_INVALID_ARG.
 *
 * The first call on a device, with that device current, looks up the
 * array's device address (cudaGetSymbolAddress), the kernel's resident CTAs
 * (occupancy query; it also sets the kernel's shared-memory limit) and the
 * driver's tensor-map encoder, and keeps them for the process.
 * Every call on a device shares the same array and clears its counters and
 * status words on the stream before the kernel; calls whose GPU work overlaps
 * (other streams, other threads) race on the array and must be serialised by
 * the caller.  The call is asynchronous and cannot report a device-side wait
 * timeout; it returns MD_OK once the work is enqueued. */
md_status md_attend_mass_noalloc(const void *kv_pool_dev, const int32_t *block_table_dev,
                                 const int32_t *n_tokens_host, const void *q_dev, void *out_dev,
                                 float *mass_dev, int batch, int num_layers, int num_q_heads,
                                 int num_kv_heads, int page_size, int max_pages_per_seq,
                                 int num_phys_pages, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* MEMDECAY_H */
