/* Internal declarations of libmemdecay: workspace layout, launch parameters
 * (passed by value; per-sequence counts come from the exact host mirror) and
 * the launchers of the four kernels. */
#ifndef MD_INTERNAL_H
#define MD_INTERNAL_H

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/memdecay.h"

namespace md {

constexpr int D = MD_HEAD_DIM;
constexpr int GP = MD_MAX_GROUP;            // query heads per KV head, padded
constexpr int PARTIAL_FLOATS = 1088;        // m[8] l[8] O[8][128], padded to 256 B
constexpr int MAX_GRID = 512;               // persistent attention CTAs (>= 2 x SM count)

enum DevStatus { ST_CODE = 0, ST_ABORT = 1, ST_DIAG = 2, ST_WORDS = 8 };

/* A decode step's attention mass per token, summed over layers and query
 * heads, is accumulated in fixed point: u64 with MASS_FRAC_BITS fraction
 * bits.  Integer adds make the sum independent of the order in which the
 * (layer, KV head) items finish.  One token receives at most 1 from each
 * query head, so num_layers * num_q_heads < MASS_MAX_HEADS keeps the sum
 * below 2^64. */
constexpr int MASS_FRAC_BITS = 48;
constexpr float MASS_SCALE = 281474976710656.0f;        // 2^48
constexpr float MASS_UNIT = 3.5527136788005009e-15f;    // 2^-48
constexpr long long MASS_MAX_HEADS = 65536;
constexpr int CALIB_BUCKETS = MD_CALIB_BUCKETS;      // age buckets per region
constexpr int CALIB_WIDTH = MD_CALIB_BUCKET_WIDTH;   // decode steps per bucket

struct RegionTable {
  float base[8];
  float half_life[8];
  int pinned[8];
};

/* Byte offsets of every array inside the caller's workspace. */
struct Layout {
  size_t pool, block_table, page_score, free_stack, region, a, t_ref, t_ins, window, ahat, prio, mass_acc,
      scratch, partials, counters, evict_list, staging_regions, staging_steps, staging_slots, status,
      calib, page_fill, seq_tokens, io_q, io_k, io_v, io_out, total;
  size_t slots, n_items;
  int scratch_tokens, chunk_stride;
};

size_t compute_layout(const md_config &c, Layout *lay);

/* ------------------------------------------------------------- append --- */
struct AppendParams {
  uint16_t *pool;
  int32_t *block_table;
  const int32_t *free_stack;
  uint8_t *region;
  float *a, *window, *ahat, *prio;
  int32_t *t_ref, *t_ins;
  const uint16_t *k_src, *v_src;
  long long sb, sl, sh, si;              // element strides of the source (seq, layer, head, token)
  const uint8_t *regions_dev;            // per token (prefill) or null
  const int32_t *steps_dev;              // per token (prefill) or null
  const int32_t *slots_dev;              // per token slot in the sequence (prefill) or null
  uint8_t *page_fill;                    // [max_batch][P_max] tokens per page
  int32_t *seq_tokens;                   // [max_batch] tokens per sequence
  int L, Hkv, ps, P_phys, P_max;         // L: layers written by this launch
  int l0;                                // first pool layer written
  int init_state;                        // 1: start token state, record new pages
  int lookup_only;                       // 1: pages already in the block table
  int n_seqs, n_per_seq, seq0, insert_step;
  int tok0[MD_MAX_BATCH];                // slot of the first token (slots_dev == null)
  int pages_before[MD_MAX_BATCH];        // pages of the sequence before this append
  int pop_base[MD_MAX_BATCH];            // free-stack index of the first page taken
  uint8_t regions_param[MD_MAX_BATCH];   // decode: region of each new token
};
cudaError_t launch_append(const AppendParams &p, cudaStream_t s);

/* ---------------------------------------------------------- attention --- */
struct AttnParams {
  const uint16_t *q;
  uint16_t *out;
  const int32_t *block_table;
  const uint8_t *page_fill;  // [max_batch][P_max] tokens per page, or null: pages are
                             // full up to n_tokens
  unsigned long long *mass_acc;   // [slots] fixed-point mass of the step, or null:
  float *mass;                    // [L*Hkv][slots] one fp32 row per (layer, KV head)
  float *scratch;      // [grid][2][scratch_tokens][8]
  float *partials;     // [items][chunk_stride][PARTIAL_FLOATS]
  int *counters;       // [items]
  int *status;         // sticky device status words
  int L, Hq, Hkv, G, ps, P_phys, P_max;   // L: layers of the model
  int l0, L_launch;    // layers [l0, l0 + L_launch) attended by this launch
  int q_layers;        // layers held by the q / out tensors (L or 1)
  long long slots;
  int scratch_tokens;  // scratch row capacity per CTA slot (tokens)
  int chunk_stride;    // partial slots reserved per item
  float scale_log2;    // log2(e) / sqrt(D)
  long long spin_limit_ns;
  int extra_arrivals;
  int n_seqs, total_units;
  int units_per_seq;   // > 0: every sequence has this many units (no search)
  int n_tokens[MD_MAX_BATCH];
  int n_pages[MD_MAX_BATCH];
  int chunks[MD_MAX_BATCH];
  int unit_start[MD_MAX_BATCH + 1];
};
cudaError_t launch_attention(const AttnParams &p, const CUtensorMap &tmap, int grid,
                             cudaStream_t s);
int attention_grid_limit(int ps);     // CTAs resident at once (0 on error)
cudaError_t attention_prepare(int ps); // one-time function attributes

/* --------------------------------------------------- fold / score ------- */
struct ScoreParams {
  unsigned long long *mass_acc;    // [slots] fixed-point mass of the pending step (read, zeroed)
  float *window, *a, *ahat, *prio, *page_score;
  int32_t *t_ref;
  const int32_t *t_ins;
  const uint8_t *region;
  const int32_t *block_table;
  const uint8_t *page_fill;        // [max_batch][P_max] tokens per page
  const int32_t *seq_tokens;       // [max_batch] |K_t| per sequence
  unsigned long long *calib_sum;   // [8][CALIB_BUCKETS] observed mass, fixed point 2^-32
  unsigned int *calib_cnt;         // [8][CALIB_BUCKETS] observations
  int calib_on;
  long long slots;
  int ps, P_max;
  int fold_only;         // 1: window += the pending step's mass and nothing else
  int observe, mass_pending;
  float norm;            // window steps * L * Hq
  int t;
  float rho, gamma, tau_scale, alpha;
  int score_mode, page_reduce, keep_prio;
  unsigned long long random_seed;
  RegionTable reg;
  int n_seqs, total_pages;
  int n_tokens[MD_MAX_BATCH];
  int n_pages[MD_MAX_BATCH];
  int page_start[MD_MAX_BATCH + 1];
};
cudaError_t launch_score(const ScoreParams &p, cudaStream_t s);

/* ------------------------------------------------------------- select --- */
struct SelectParams {
  const float *page_score;
  int32_t *block_table;
  int32_t *free_stack;
  int32_t *evict_list;    // [max_batch][P_max] internal
  int32_t *user_evicted;  // optional [n_seqs][P_max]
  uint8_t *page_fill;     // [max_batch][P_max], compacted with the block table
  int32_t *seq_tokens;    // [max_batch], less the evicted pages' tokens
  int *status;
  int P_max, n_seqs, top;
  int n_pages[MD_MAX_BATCH];
  int n_evict[MD_MAX_BATCH];
  int push_off[MD_MAX_BATCH];
};
cudaError_t launch_select(const SelectParams &p, cudaStream_t s);

/* Launch of a kernel taking one parameter struct, with programmatic stream
 * serialization (the kernel calls pdl_wait() before touching global memory). */
template <class P>
cudaError_t launch_pdl(void (*kernel)(P), int grid, int threads, int smem, cudaStream_t s, const P &p) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, p);
}

/* --------------------------------------------------------------- init --- */
cudaError_t launch_init(int32_t *free_stack, int P_phys, int *status, int *counters,
                        size_t n_items, cudaStream_t s);

}  // namespace md

#endif
