/* Host side of libmemdecay: the C ABI of include/memdecay.h.
 *
 * The handle keeps an exact host mirror of the cache's bookkeeping (tokens
 * and pages per sequence, pages holding a pinned token, the free-stack
 * height, the decode step and the observation window).  Region labels are
 * given on the host, so the number of evictable pages of every sequence is
 * known here and the eviction counts, the free-stack offsets and the attention
 * work split are computed without reading anything back from the GPU.  The
 * kernels get these numbers by value in their launch parameters. */
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "md_internal.h"

#define MD_API extern "C" __attribute__((visibility("default")))

using namespace md;

namespace {

constexpr int N_STAGES = 5;
constexpr int STAGE_APPEND = 0, STAGE_ATTN = 1, STAGE_FOLD = 2, STAGE_SCORE = 3,
              STAGE_SELECT = 4;

struct ProfRec {
  int stage;
  cudaEvent_t a, b;
};

struct HostMirror {
  int64_t t = 0;
  int window_steps = 0, window_batch = 0;
  int mass_pending = 0, mass_batch = 0;
  int64_t free_top = 0;
  int layer_next = 0;     // md_decode_layer: next layer expected (0 = none in progress)
  int layer_batch = 0;
};

}  // namespace

struct md_ctx {
  md_config cfg;
  Layout lay;
  uint8_t *ws = nullptr;
  cudaStream_t stream = nullptr;
  CUtensorMap tmap;
  int grid_limit = 0;
  RegionTable reg;
  HostMirror m;
  std::vector<int64_t> n_tokens;           // tokens per sequence (exact while tokens_exact)
  std::vector<int> n_pages, pinned_pages;
  std::vector<int> tail_fill, tail_region;  // the page being written
  std::vector<uint8_t> tail_pinned, tokens_exact;
  bool poisoned = false;
  std::string err;
  long long spin_limit_ns = 2000000000LL;
  int extra_arrivals = 0;
  int grid_cap = 0;          // 0: every CTA that fits
  int unit_overhead_kib = 112;   // planner: per-unit cost, as KiB of K/V streamed
  int combine_overhead_kib = 192;   // planner: cost of a split into several chunks per item
  int force_chunks = 0;      // planner: 0 = choose
  /* the planner's last choice of pages per chunk, reused while its inputs
   * (batch, layers, knobs, pages per sequence) repeat */
  std::vector<int> plan_pages;
  int plan_batch = -1, plan_layers = -1, plan_T = 0, plan_G = 0;
  int plan_knobs[5] = {-1, -1, -1, -1, -1};
  bool calib_on = false;     // calibration histogram being gathered
  int pageable_access = 0;   // the device reads and writes pageable host memory coherently
  int zero_copy = 1;         // md_decode_step_host: new K/V and output used in place when reachable
  bool prof = false;
  std::vector<cudaEvent_t> ev_pool;
  std::vector<ProfRec> pending;
  double prof_ms[N_STAGES] = {0};
  int64_t prof_n[N_STAGES] = {0};
  std::vector<uint8_t> staging_host;
};

namespace {

md_status fail(md_ctx *c, md_status s, const char *fmt, ...) __attribute__((format(printf, 3, 4)));
md_status fail(md_ctx *c, md_status s, const char *fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return s;
}

md_status cuda_fail(md_ctx *c, cudaError_t e, const char *what) {
  if (c) {
    c->err = std::string(what) + ": " + cudaGetErrorString(e);
    c->poisoned = true;
  }
  return MD_ERR_CUDA;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

const char *check_config(const md_config &c) {
  if (c.num_layers < 1 || c.num_layers > 255) return "num_layers must be in [1, 255]";
  if (c.num_kv_heads < 1 || c.num_q_heads < c.num_kv_heads) return "bad head counts";
  if ((long long)c.num_layers * c.num_q_heads >= MASS_MAX_HEADS)
    return "num_layers * num_q_heads must stay below 65,536";
  if (c.num_q_heads % c.num_kv_heads) return "num_q_heads must be a multiple of num_kv_heads";
  if (c.num_q_heads / c.num_kv_heads > MD_MAX_GROUP) return "GQA group above 8 query heads";
  if (c.head_dim != MD_HEAD_DIM) return "head_dim must be 128";
  if (c.page_size != 16 && c.page_size != 32) return "page_size must be 16 or 32";
  if (c.max_batch < 1 || c.max_batch > MD_MAX_BATCH) return "max_batch must be in [1, 256]";
  if (c.max_pages_per_seq < 1 ||
      (long long)c.max_pages_per_seq * c.page_size >
          (long long)MD_MAX_CHUNKS * MD_MAX_CHUNK_TOKENS)
    return "max_pages_per_seq out of range";
  if (c.num_phys_pages < 1) return "num_phys_pages must be positive";
  const long long rows =
      (long long)c.num_layers * c.num_phys_pages * c.num_kv_heads * 2 * c.page_size;
  if (rows >= (1LL << 31)) return "page pool too large (rows of K/V must stay below 2^31)";
  if ((long long)c.num_phys_pages * c.page_size >= (1LL << 31)) return "too many token slots";
  if (!(c.rho >= 0.f && c.rho <= 1.f) || !(c.gamma >= 0.f) || !isfinite(c.gamma))
    return "rho must be in [0,1] and gamma >= 0";
  if (!(c.tau_scale >= 0.f) || !isfinite(c.tau_scale)) return "tau_scale must be >= 0";
  if (!(c.attn_weight >= 0.f) || !isfinite(c.attn_weight)) return "attn_weight must be >= 0";
  if (c.score_mode < 0 || c.score_mode > 4) return "score_mode must be in [0, 4]";
  if (c.page_reduce != 0 && c.page_reduce != 1) return "page_reduce must be 0 or 1";
  return nullptr;
}

void prof_begin(md_ctx *c, cudaEvent_t *a) {
  *a = nullptr;
  if (!c->prof) return;
  if (c->ev_pool.empty()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return;
    c->ev_pool.push_back(e);
  }
  *a = c->ev_pool.back();
  c->ev_pool.pop_back();
  cudaEventRecord(*a, c->stream);
}

void prof_end(md_ctx *c, int stage, cudaEvent_t a) {
  if (!c->prof || !a) return;
  cudaEvent_t b;
  if (c->ev_pool.empty()) {
    if (cudaEventCreate(&b) != cudaSuccess) {
      c->ev_pool.push_back(a);
      return;
    }
  } else {
    b = c->ev_pool.back();
    c->ev_pool.pop_back();
  }
  cudaEventRecord(b, c->stream);
  c->pending.push_back({stage, a, b});
}

template <class T>
T *ptr(md_ctx *c, size_t off) {
  return (T *)(c->ws + off);
}

/* Pages of sequence b that can be evicted: everything but pinned pages and
 * the page being written (the last one). */
int evictable_pages(const md_ctx *c, int b) {
  const int P = c->n_pages[b];
  if (P == 0) return 0;
  return P - c->pinned_pages[b] - (c->tail_pinned[b] ? 0 : 1);
}

/* Whether a token of region r opens a fresh page: no page yet, the tail page
 * full, or (region-aligned allocation) a region different from the tail's. */
bool opens_page(const md_ctx *c, int b, int r) {
  return c->n_pages[b] == 0 || c->tail_fill[b] == c->cfg.page_size ||
         (c->cfg.region_aligned_pages && c->tail_region[b] != r);
}

/* Slot (page * page_size + offset, in logical page order) the next token of
 * region r goes to. */
int next_slot(const md_ctx *c, int b, int r) {
  const int ps = c->cfg.page_size;
  return opens_page(c, b, r) ? c->n_pages[b] * ps : (c->n_pages[b] - 1) * ps + c->tail_fill[b];
}

/* Mirror bookkeeping for one appended token of region r. */
void mirror_token(md_ctx *c, int b, int r) {
  if (opens_page(c, b, r)) {
    c->n_pages[b] += 1;
    c->tail_fill[b] = 0;
    c->tail_pinned[b] = 0;
  }
  c->tail_fill[b] += 1;
  c->tail_region[b] = r;
  if (c->reg.pinned[r] && !c->tail_pinned[b]) {
    c->pinned_pages[b] += 1;
    c->tail_pinned[b] = 1;
  }
  c->n_tokens[b] += 1;
}

int64_t cached_tokens(const md_ctx *c) {
  int64_t s = 0;
  for (auto v : c->n_pages) s += v;
  return s;
}

/* Window fold: add the pending step's mass (summed over layers and heads)
 * into the window accumulator of every token that was attended in that step,
 * and clear the step's accumulator. */
md_status launch_fold(md_ctx *c) {
  ScoreParams sp;
  memset(&sp, 0, sizeof(sp));
  sp.mass_acc = ptr<unsigned long long>(c, c->lay.mass_acc);
  sp.window = ptr<float>(c, c->lay.window);
  sp.region = ptr<uint8_t>(c, c->lay.region);
  sp.block_table = ptr<int32_t>(c, c->lay.block_table);
  /* with contiguous pages the host's exact counts describe every page; the
   * device fills and counts are read only with region-aligned pages */
  if (c->cfg.region_aligned_pages) {
    sp.page_fill = ptr<uint8_t>(c, c->lay.page_fill);
    sp.seq_tokens = ptr<int32_t>(c, c->lay.seq_tokens);
  }
  sp.slots = (long long)c->lay.slots;
  sp.ps = c->cfg.page_size;
  sp.P_max = c->cfg.max_pages_per_seq;
  sp.fold_only = 1;
  sp.n_seqs = c->m.mass_batch;
  int tot = 0;
  for (int b = 0; b < sp.n_seqs; ++b) {
    sp.n_tokens[b] = (int)c->n_tokens[b];
    sp.n_pages[b] = c->n_pages[b];
    sp.page_start[b] = tot;
    tot += c->n_pages[b];
  }
  sp.page_start[sp.n_seqs] = tot;
  sp.total_pages = tot;
  cudaEvent_t e0;
  prof_begin(c, &e0);
  cudaError_t err = launch_score(sp, c->stream);
  prof_end(c, STAGE_FOLD, e0);
  if (err != cudaSuccess) return cuda_fail(c, err, "fold launch");
  c->m.mass_pending = 0;
  return MD_OK;
}

/* Round-aligned schedules.  The persistent grid takes units in rounds of G
 * consecutive unit ids.  A round that ends inside an item leaves the
 * finishers of that item's earlier chunks waiting for chunks of the next
 * round, which delays those CTAs' next units and, through the items they
 * share, their neighbours'.  Over a long launch the delays are absorbed; with
 * a few rounds per launch (a layer-by-layer call) they reach its end: at
 * config 4's full trace layer by layer, 344.7 us per layer against 327.2 us
 * with no such boundary.
 *
 * A split of every sequence into C chunks, with G a multiple of C and the
 * unit count a multiple of G, has no such boundary and gives every CTA the
 * same work, where the plain split's last round may be partly empty.  Costs
 * are CTA-time in pages (HBM is shared, so the time of a launch that keeps
 * it saturated follows the CTAs' summed busy time): the aligned split's
 * streamed pages plus per-unit overheads, against the plain split's makespan
 * times its grid, with a penalty of 0.4 / rounds when its rounds end inside
 * items (fitted to the measurement above).  Among aligned splits with
 * G >= 0.84 glim (fewer CTAs would not keep HBM saturated) the largest G,
 * then the fewest units, is taken when cheaper.  A plain split of one round
 * is kept: such a launch is too short to be HBM-bound and its time is the
 * largest unit's.  Returns the plain split (G = 0) otherwise. */
struct Aligned {
  int T, G;
};

Aligned aligned_schedule(const md_ctx *c, int batch, int items, int Pmax, int T0, double makespan0,
                         long long glim, double ov, double cov, double l2_budget) {
  const int ps = c->cfg.page_size;
  const int cmax = c->lay.chunk_stride;
  const int max_chunk_pages = std::max(1, c->lay.scratch_tokens / ps);
  double pages = 0.0;
  int active = 0;
  for (int b = 0; b < batch; ++b) {
    pages += (double)items * c->n_pages[b];
    active += c->n_pages[b] > 0;
  }
  /* the plain split: units, rounds, round boundaries inside an item */
  std::vector<long long> start(batch + 1, 0);
  std::vector<int> ch(batch, 0);
  for (int b = 0; b < batch; ++b) {
    const int P = c->n_pages[b];
    ch[b] = P > 0 ? std::min(std::min((P + T0 - 1) / T0, cmax), P) : 0;
    start[b + 1] = start[b] + (long long)items * ch[b];
  }
  const long long U0 = start[batch];
  if (U0 == 0 || active == 0) return {T0, 0};
  const long long G0 = std::max(1LL, std::min(U0, glim));
  const long long rounds = (U0 + G0 - 1) / G0;
  if (rounds < 2) return {T0, 0};
  int inside = 0;
  for (long long k = 1, b = 0; k < rounds; ++k) {
    const long long x = k * G0;
    while (start[b + 1] <= x) ++b;
    if ((x - start[b]) % ch[b] != 0) ++inside;
  }
  /* makespan0 already holds the plain split's combine cost (cov, in
   * pages of one CTA's time) when it splits items */
  double cost0 = makespan0 * (double)G0;
  if (inside > 0) cost0 *= 1.0 + 0.4 / (double)rounds;
  /* aligned splits */
  const long long itot = (long long)active * items;
  Aligned best{T0, 0};
  long long bestG = 0;
  double bestCost = cost0;
  for (int C = 1; C <= cmax; ++C) {
    const int T = (Pmax + C - 1) / C;
    if (T > max_chunk_pages) continue;
    bool uniform = true;
    for (int b = 0; b < batch && uniform; ++b) {
      const int P = c->n_pages[b];
      if (P > 0) uniform = std::min(std::min((P + T - 1) / T, cmax), P) == C;
    }
    if (!uniform) continue;
    long long m = glim / C;
    while (m > 0 && itot % m) --m;
    const long long G = m * C;
    if (G <= 0 || (double)G < 0.84 * (double)glim) continue;
    if ((double)G * 2 * T * ps * GP * 4 > l2_budget) continue;
    const double cost = pages + ov * (double)(itot * C) + (C > 1 ? cov * (double)G : 0.0);
    if (cost >= cost0) continue;
    if (G > bestG || (G == bestG && cost < bestCost)) {
      bestG = G;
      bestCost = cost;
      best = {T, (int)G};
    }
  }
  return best;
}

/* Split every (sequence, layer, KV head) item's pages into chunks for the
 * persistent grid, which takes units round-robin (unit u on CTA u mod G).
 * Each candidate split is costed by its exact makespan under that schedule:
 * a sequence's units are one contiguous run of unit ids, so every CTA gets
 * floor(n_b / G) of them plus one more on a cyclic CTA interval, and a
 * difference array gives all CTA loads in O(batch + G).  A unit costs its
 * pages plus a fixed per-unit overhead (Q load, merge, publish, ramp),
 * expressed as K/V bytes streamed.  A split that gives some item several
 * chunks also pays once for the cross-CTA combine (publishing partials,
 * waiting for the item's other chunks, combining them): at a few hundred
 * tokens per item a single chunk per item is faster than any split.  At most MD_MAX_CHUNK_TOKENS tokens per
 * chunk; the live raw-score scratch must stay inside L2.  A round-aligned
 * schedule (aligned_schedule) may then replace the split and the grid. */
void plan_attention(md_ctx *c, int batch, int layers, AttnParams &ap, int *grid) {
  const int ps = c->cfg.page_size;
  const int items = layers * c->cfg.num_kv_heads;
  int Pmax = 1;
  for (int b = 0; b < batch; ++b) Pmax = std::max(Pmax, c->n_pages[b]);
  const int max_chunk_pages = std::max(1, c->lay.scratch_tokens / ps);
  const int cmax = c->lay.chunk_stride;
  const long long glim =
      c->grid_cap > 0 ? std::min<long long>(c->grid_cap, c->grid_limit) : c->grid_limit;
  const double page_kib = ps * 512.0 / 1024.0;   // K+V of one (layer, KV head) page
  const double ov = c->unit_overhead_kib / page_kib;
  const double cov = c->combine_overhead_kib / page_kib;
  const int knobs[5] = {(int)glim, c->unit_overhead_kib, c->force_chunks, c->lay.scratch_tokens,
                        c->combine_overhead_kib};
  bool same = c->plan_batch == batch && c->plan_layers == layers &&
              std::equal(knobs, knobs + 5, c->plan_knobs);
  for (int b = 0; same && b < batch; ++b) same = c->plan_pages[b] == c->n_pages[b];
  double best = 1e300;
  int bestT = same ? c->plan_T : 0;
  int bestG = same ? c->plan_G : 0;   // 0: min(units, glim)
  double diff[MAX_GRID + 1];
  /* Every CTA keeps the raw scores of two units in L2 (evict_last) until the
   * finisher has read them; keep that set well inside L2 or its lines spill. */
  const double l2_budget = 46.0 * (1 << 20);
  for (int pass = 0; pass < 2 && bestT == 0; ++pass)
  for (int C = 1, Tprev = 0; C <= cmax; ++C) {
    const int T = (Pmax + C - 1) / C;
    if (c->force_chunks > 0) {
      const int need = (Pmax + max_chunk_pages - 1) / max_chunk_pages;
      if (C != std::min(cmax, std::max(c->force_chunks, need))) continue;
    } else {
      if (T == Tprev) continue;   // the same split as the previous candidate
      Tprev = T;
    }
    if (T > max_chunk_pages) continue;
    if (pass == 0 && (double)glim * 2 * T * ps * GP * 4 > l2_budget) continue;
    long long U = 0;
    for (int b = 0; b < batch; ++b) {
      const int P = c->n_pages[b];
      if (P > 0) U += (long long)items * std::min(std::min((P + T - 1) / T, cmax), P);
    }
    if (U == 0) continue;
    const int G = (int)std::max(1LL, std::min<long long>(U, glim));
    for (int g = 0; g <= G; ++g) diff[g] = 0.0;
    double base = 0.0;
    bool split = false;
    long long start = 0;
    for (int b = 0; b < batch; ++b) {
      const int P = c->n_pages[b];
      if (P == 0) continue;
      const int ch = std::min(std::min((P + T - 1) / T, cmax), P);
      split |= ch > 1;
      const long long n = (long long)items * ch;
      const double sz = (double)P / ch + ov;
      base += (double)(n / G) * sz;
      const int r = (int)(n % G), s0 = (int)(start % G);
      if (r > 0) {
        diff[s0] += sz;
        if (s0 + r <= G) {
          diff[s0 + r] -= sz;
        } else {
          diff[G] -= sz;
          diff[0] += sz;
          diff[s0 + r - G] -= sz;
        }
      }
      start += n;
    }
    double run = 0.0, peak = 0.0;
    for (int g = 0; g < G; ++g) {
      run += diff[g];
      peak = std::max(peak, run);
    }
    const double cost = base + peak + (split ? cov : 0.0);   // the combine: once per launch
    if (cost < best - 1e-9) {
      best = cost;
      bestT = T;
    }
  }
  if (bestT == 0) bestT = max_chunk_pages;
  if (!same && c->force_chunks == 0 && c->grid_cap == 0) {
    const Aligned a = aligned_schedule(c, batch, items, Pmax, bestT, best, glim, ov, cov, l2_budget);
    bestT = a.T;
    bestG = a.G;
  }
  if (!same) {
    c->plan_G = bestG;
    c->plan_batch = batch;
    c->plan_layers = layers;
    std::copy(knobs, knobs + 5, c->plan_knobs);
    c->plan_pages.assign(c->n_pages.begin(), c->n_pages.begin() + batch);
    c->plan_T = bestT;
  }
  long long U = 0;
  for (int b = 0; b < batch; ++b) {
    const int P = c->n_pages[b];
    int ch = 0;
    if (P > 0) ch = std::min(std::min((P + bestT - 1) / bestT, cmax), P);
    ap.chunks[b] = ch;
    ap.unit_start[b] = (int)U;
    ap.n_pages[b] = P;
    ap.n_tokens[b] = (int)c->n_tokens[b];
    U += (long long)items * ch;
  }
  ap.unit_start[batch] = (int)U;
  ap.total_units = (int)U;
  ap.n_seqs = batch;
  ap.units_per_seq = batch > 0 ? (int)(U / batch) : 0;
  for (int b = 0; b < batch && ap.units_per_seq > 0; ++b)
    if (ap.unit_start[b + 1] - ap.unit_start[b] != ap.units_per_seq) ap.units_per_seq = 0;
  *grid = bestG > 0 ? bestG : (int)std::max(1LL, std::min<long long>(U, glim));
}

bool valid_region(int r) { return r >= 0 && r < MD_NUM_REGIONS; }

}  // namespace

/* ------------------------------------------------------------ layout ---- */
size_t md::compute_layout(const md_config &c, Layout *lay) {
  Layout L;
  memset(&L, 0, sizeof(L));
  const size_t ps = c.page_size;
  L.slots = (size_t)c.num_phys_pages * ps;
  L.n_items = (size_t)c.max_batch * c.num_layers * c.num_kv_heads;
  L.scratch_tokens =
      (int)std::min<long long>(MD_MAX_CHUNK_TOKENS, (long long)c.max_pages_per_seq * ps);
  L.scratch_tokens = (L.scratch_tokens + 15) / 16 * 16;
  L.chunk_stride = std::min(MD_MAX_CHUNKS, c.max_pages_per_seq);
  size_t off = 0;
  auto take = [&](size_t bytes, size_t align) {
    off = align_up(off, align);
    size_t o = off;
    off += bytes;
    return o;
  };
  L.status = take(ST_WORDS * 4 * 4, 256);
  L.pool = take((size_t)c.num_layers * c.num_phys_pages * c.num_kv_heads * 2 * ps * D * 2, 1024);
  L.block_table = take((size_t)c.max_batch * c.max_pages_per_seq * 4, 256);
  L.page_score = take((size_t)c.max_batch * c.max_pages_per_seq * 4, 256);
  L.free_stack = take((size_t)c.num_phys_pages * 4, 256);
  L.region = take(L.slots, 256);
  L.a = take(L.slots * 4, 256);
  L.t_ref = take(L.slots * 4, 256);
  L.t_ins = take(L.slots * 4, 256);
  L.window = take(L.slots * 4, 256);
  L.ahat = take(L.slots * 4, 256);
  L.prio = take(L.slots * 4, 256);
  L.mass_acc = take(L.slots * 8, 256);
  L.scratch = take((size_t)MAX_GRID * 2 * L.scratch_tokens * GP * 4, 256);
  L.partials = take(L.n_items * L.chunk_stride * PARTIAL_FLOATS * 4, 256);
  L.counters = take(L.n_items * 4, 256);
  L.evict_list = take((size_t)c.max_batch * c.max_pages_per_seq * 4, 256);
  L.staging_regions = take((size_t)c.max_pages_per_seq * ps, 256);
  L.staging_steps = take((size_t)c.max_pages_per_seq * ps * 4, 256);
  L.staging_slots = take((size_t)c.max_pages_per_seq * ps * 4, 256);
  L.page_fill = take((size_t)c.max_batch * c.max_pages_per_seq, 256);
  L.seq_tokens = take((size_t)c.max_batch * 4, 256);
  L.calib = take((size_t)8 * CALIB_BUCKETS * (8 + 4), 256);
  /* device copies of one step's tensors for md_decode_step_host */
  const size_t q_bytes = (size_t)c.max_batch * c.num_layers * c.num_q_heads * D * 2;
  const size_t kv_bytes = (size_t)c.max_batch * c.num_layers * c.num_kv_heads * D * 2;
  L.io_q = take(q_bytes, 256);
  L.io_k = take(kv_bytes, 256);
  L.io_v = take(kv_bytes, 256);
  L.io_out = take(q_bytes, 256);
  L.total = align_up(off, 256);
  if (lay) *lay = L;
  return L.total;
}

/* ------------------------------------------------------------- C ABI ---- */
MD_API size_t md_workspace_size(const md_config *cfg) {
  if (!cfg || check_config(*cfg)) return 0;
  return compute_layout(*cfg, nullptr);
}

MD_API md_status md_create(const md_config *cfg, md_ctx **out) {
  if (!cfg || !out) return MD_ERR_INVALID_ARG;
  *out = nullptr;
  if (check_config(*cfg)) return MD_ERR_INVALID_ARG;
  Layout lay;
  const size_t need = compute_layout(*cfg, &lay);
  if (!cfg->workspace || ((uintptr_t)cfg->workspace & 1023) || cfg->workspace_bytes < need)
    return MD_ERR_WORKSPACE;
  md_ctx *c = new md_ctx();
  c->cfg = *cfg;
  c->lay = lay;
  c->ws = (uint8_t *)cfg->workspace;
  c->stream = (cudaStream_t)cfg->stream;
  const int B = cfg->max_batch;
  c->n_tokens.assign(B, 0);
  c->n_pages.assign(B, 0);
  c->pinned_pages.assign(B, 0);
  c->tail_pinned.assign(B, 0);
  c->tail_fill.assign(B, 0);
  c->tail_region.assign(B, -1);
  c->tokens_exact.assign(B, 1);
  for (int r = 0; r < 8; ++r) {
    c->reg.base[r] = 0.f;
    c->reg.half_life[r] = INFINITY;
    c->reg.pinned[r] = 0;
  }
  c->m.free_top = cfg->num_phys_pages;

  cudaError_t e = attention_prepare(cfg->page_size);
  if (e != cudaSuccess) {
    delete c;
    return MD_ERR_CUDA;
  }
  {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&v, cudaDevAttrPageableMemoryAccess, dev) == cudaSuccess)
      c->pageable_access = v;
    cudaGetLastError();
  }
  c->grid_limit = attention_grid_limit(cfg->page_size);
  if (c->grid_limit <= 0) {
    delete c;
    return MD_ERR_CUDA;
  }
  if (c->grid_limit < MD_MAX_CHUNKS) {   // an item's chunks must fit in one round
    delete c;
    return MD_ERR_CAPACITY;
  }
  /* TMA descriptor over the pool viewed as [rows][128] bf16, rows = (layer,
   * page, KV head, K|V, token); one box = one page's K and V rows x 64 dims,
   * 128-byte swizzled. */
  void *fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
    delete c;
    return MD_ERR_CUDA;
  }
  typedef CUresult (*EncodeFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                               const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                               const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                               CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
  const cuuint64_t rows = (cuuint64_t)cfg->num_layers * cfg->num_phys_pages *
                          cfg->num_kv_heads * 2 * cfg->page_size;
  cuuint64_t dims[2] = {(cuuint64_t)D, rows};
  cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)(2 * cfg->page_size)};
  cuuint32_t estr[2] = {1, 1};
  CUresult cr = ((EncodeFn)fn)(&c->tmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->ws + lay.pool,
                               dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) {
    delete c;
    return MD_ERR_CUDA;
  }
  e = cudaMemsetAsync(c->ws, 0, need, c->stream);
  if (e == cudaSuccess)
    e = launch_init(ptr<int32_t>(c, lay.free_stack), cfg->num_phys_pages, ptr<int>(c, lay.status),
                    ptr<int>(c, lay.counters), lay.n_items, c->stream);
  if (e != cudaSuccess) {
    delete c;
    return MD_ERR_CUDA;
  }
  *out = c;
  return MD_OK;
}

MD_API md_status md_set_region_params(md_ctx *c, int region, float base, float half_life,
                                      int pinned) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (!valid_region(region)) return fail(c, MD_ERR_INVALID_ARG, "region %d out of range", region);
  if (!(base >= 0.f) || !isfinite(base))
    return fail(c, MD_ERR_INVALID_ARG, "base priority must be finite and >= 0");
  if (!(half_life > 0.f)) return fail(c, MD_ERR_INVALID_ARG, "half-life must be > 0 (or +inf)");
  const int pin = pinned ? 1 : 0;
  if (pin != c->reg.pinned[region] && cached_tokens(c) > 0)
    return fail(c, MD_ERR_STATE, "pinned flag can only change while the cache is empty");
  c->reg.base[region] = base;
  c->reg.half_life[region] = half_life;
  c->reg.pinned[region] = pin;
  return MD_OK;
}

MD_API md_status md_append_tokens(md_ctx *c, int seq, int n, const uint8_t *regions_host,
                                  const int32_t *steps_host, const void *k_dev,
                                  const void *v_dev) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (c->poisoned) return fail(c, MD_ERR_STATE, "handle unusable after an earlier error");
  if (c->m.layer_next != 0) return fail(c, MD_ERR_STATE, "a layer-by-layer step is in progress");
  const md_config &cf = c->cfg;
  if (seq < 0 || seq >= cf.max_batch) return fail(c, MD_ERR_INVALID_ARG, "seq out of range");
  if (n < 0) return fail(c, MD_ERR_INVALID_ARG, "negative token count");
  if (n == 0) return MD_OK;
  if (!regions_host || !k_dev || !v_dev) return fail(c, MD_ERR_INVALID_ARG, "null pointer");
  for (int i = 0; i < n; ++i)
    if (!valid_region(regions_host[i])) return fail(c, MD_ERR_INVALID_ARG, "bad region label");
  if (steps_host)
    for (int i = 0; i < n; ++i)
      if (steps_host[i] > c->m.t) return fail(c, MD_ERR_INVALID_ARG, "insertion step in the future");
  const int ps = cf.page_size;
  /* where the tokens go: the same page-opening rule as the mirror */
  std::vector<int32_t> slots(n);
  long long pages_after = c->n_pages[seq];
  {
    int fill = c->tail_fill[seq], treg = c->tail_region[seq];
    for (int i = 0; i < n; ++i) {
      const int r = regions_host[i];
      if (pages_after == 0 || fill == ps || (cf.region_aligned_pages && treg != r)) {
        ++pages_after;
        fill = 0;
      }
      slots[i] = (int32_t)((pages_after - 1) * ps + fill);
      ++fill;
      treg = r;
    }
  }
  const long long new_pages = pages_after - c->n_pages[seq];
  if (pages_after > cf.max_pages_per_seq)
    return fail(c, MD_ERR_CAPACITY, "sequence %d would need %lld pages (max %d)", seq,
                pages_after, cf.max_pages_per_seq);
  if (new_pages > c->m.free_top)
    return fail(c, MD_ERR_CAPACITY, "page pool exhausted (%lld free, %lld needed)",
                (long long)c->m.free_top, new_pages);
  if (c->m.mass_pending) {
    md_status st = launch_fold(c);
    if (st != MD_OK) return st;
  }
  cudaError_t e = cudaMemcpyAsync(c->ws + c->lay.staging_regions, regions_host, (size_t)n,
                                  cudaMemcpyHostToDevice, c->stream);
  if (e == cudaSuccess && steps_host)
    e = cudaMemcpyAsync(c->ws + c->lay.staging_steps, steps_host, (size_t)n * 4,
                        cudaMemcpyHostToDevice, c->stream);
  if (e == cudaSuccess && cf.region_aligned_pages)
    e = cudaMemcpyAsync(c->ws + c->lay.staging_slots, slots.data(), (size_t)n * 4,
                        cudaMemcpyHostToDevice, c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "staging copy");
  AppendParams ap;
  memset(&ap, 0, sizeof(ap));
  ap.pool = ptr<uint16_t>(c, c->lay.pool);
  ap.block_table = ptr<int32_t>(c, c->lay.block_table);
  ap.free_stack = ptr<int32_t>(c, c->lay.free_stack);
  ap.region = ptr<uint8_t>(c, c->lay.region);
  ap.a = ptr<float>(c, c->lay.a);
  ap.window = ptr<float>(c, c->lay.window);
  ap.ahat = ptr<float>(c, c->lay.ahat);
  ap.prio = ptr<float>(c, c->lay.prio);
  ap.t_ref = ptr<int32_t>(c, c->lay.t_ref);
  ap.t_ins = ptr<int32_t>(c, c->lay.t_ins);
  ap.page_fill = ptr<uint8_t>(c, c->lay.page_fill);
  ap.seq_tokens = ptr<int32_t>(c, c->lay.seq_tokens);
  ap.slots_dev = cf.region_aligned_pages ? ptr<int32_t>(c, c->lay.staging_slots) : nullptr;
  ap.k_src = (const uint16_t *)k_dev;
  ap.v_src = (const uint16_t *)v_dev;
  ap.sb = 0;
  ap.sl = (long long)cf.num_kv_heads * n * D;
  ap.sh = (long long)n * D;
  ap.si = D;
  ap.regions_dev = ptr<uint8_t>(c, c->lay.staging_regions);
  ap.steps_dev = steps_host ? ptr<int32_t>(c, c->lay.staging_steps) : nullptr;
  ap.L = cf.num_layers;
  ap.Hkv = cf.num_kv_heads;
  ap.ps = ps;
  ap.P_phys = cf.num_phys_pages;
  ap.P_max = cf.max_pages_per_seq;
  ap.l0 = 0;
  ap.init_state = 1;
  ap.lookup_only = 0;
  ap.n_seqs = 1;
  ap.n_per_seq = n;
  ap.seq0 = seq;
  ap.insert_step = (int)c->m.t;
  ap.tok0[0] = slots[0];
  ap.pages_before[0] = c->n_pages[seq];
  ap.pop_base[0] = (int)(c->m.free_top - 1);
  cudaEvent_t e0;
  prof_begin(c, &e0);
  e = launch_append(ap, c->stream);
  prof_end(c, STAGE_APPEND, e0);
  if (e != cudaSuccess) return cuda_fail(c, e, "append launch");
  for (int i = 0; i < n; ++i) mirror_token(c, seq, regions_host[i]);
  c->m.free_top -= new_pages;
  return MD_OK;
}

namespace {

/* Checks shared by md_decode_step and layer 0 of md_decode_layer. */
md_status check_step(md_ctx *c, int batch, const uint8_t *new_region_host) {
  const md_config &cf = c->cfg;
  if (batch < 1 || batch > cf.max_batch) return fail(c, MD_ERR_INVALID_ARG, "batch out of range");
  if (!new_region_host) return fail(c, MD_ERR_INVALID_ARG, "null pointer");
  if (c->m.window_steps > 0 && batch != c->m.window_batch)
    return fail(c, MD_ERR_INVALID_ARG, "batch changed inside an observation window");
  const int ps = cf.page_size;
  long long need_total = 0;
  for (int b = 0; b < batch; ++b) {
    if (!valid_region(new_region_host[b])) return fail(c, MD_ERR_INVALID_ARG, "bad region label");
    const int need = opens_page(c, b, new_region_host[b]) ? 1 : 0;
    if (c->n_pages[b] + need > cf.max_pages_per_seq)
      return fail(c, MD_ERR_CAPACITY, "sequence %d block table full", b);
    need_total += need;
  }
  if (need_total > c->m.free_top) return fail(c, MD_ERR_CAPACITY, "page pool exhausted");
  if (c->m.t + 1 >= (1LL << 31)) return fail(c, MD_ERR_STATE, "step counter overflow");
  return MD_OK;
}

void fill_append_common(md_ctx *c, AppendParams &ap) {
  const md_config &cf = c->cfg;
  memset(&ap, 0, sizeof(ap));
  ap.pool = ptr<uint16_t>(c, c->lay.pool);
  ap.block_table = ptr<int32_t>(c, c->lay.block_table);
  ap.free_stack = ptr<int32_t>(c, c->lay.free_stack);
  ap.region = ptr<uint8_t>(c, c->lay.region);
  ap.a = ptr<float>(c, c->lay.a);
  ap.window = ptr<float>(c, c->lay.window);
  ap.ahat = ptr<float>(c, c->lay.ahat);
  ap.prio = ptr<float>(c, c->lay.prio);
  ap.t_ref = ptr<int32_t>(c, c->lay.t_ref);
  ap.t_ins = ptr<int32_t>(c, c->lay.t_ins);
  ap.page_fill = ptr<uint8_t>(c, c->lay.page_fill);
  ap.seq_tokens = ptr<int32_t>(c, c->lay.seq_tokens);
  ap.Hkv = cf.num_kv_heads;
  ap.ps = cf.page_size;
  ap.P_phys = cf.num_phys_pages;
  ap.P_max = cf.max_pages_per_seq;
  ap.n_per_seq = 1;
  ap.seq0 = 0;
}

/* Start of a decode step: advance t, take the new pages, append the new
 * tokens' K/V for layers [l0, l0 + L) and start their state. */
md_status begin_step(md_ctx *c, int batch, int l0, int L, long long sb, long long sl,
                     const void *k_new, const void *v_new, const uint8_t *new_region_host) {
  const int ps = c->cfg.page_size;
  if (c->m.mass_pending) {
    md_status st = launch_fold(c);
    if (st != MD_OK) return st;
  }
  c->m.t += 1;
  AppendParams ap;
  fill_append_common(c, ap);
  ap.k_src = (const uint16_t *)k_new;
  ap.v_src = (const uint16_t *)v_new;
  ap.sb = sb;
  ap.sl = sl;
  ap.sh = D;
  ap.si = 0;
  ap.L = L;
  ap.l0 = l0;
  ap.init_state = 1;
  ap.lookup_only = 0;
  ap.n_seqs = batch;
  ap.insert_step = (int)c->m.t;
  long long popped = 0;
  for (int b = 0; b < batch; ++b) {
    ap.tok0[b] = next_slot(c, b, new_region_host[b]);
    ap.pages_before[b] = c->n_pages[b];
    ap.pop_base[b] = (int)(c->m.free_top - 1 - popped);
    ap.regions_param[b] = new_region_host[b];
    if (opens_page(c, b, new_region_host[b])) popped += 1;
  }
  cudaEvent_t e0;
  prof_begin(c, &e0);
  cudaError_t e = launch_append(ap, c->stream);
  prof_end(c, STAGE_APPEND, e0);
  if (e != cudaSuccess) return cuda_fail(c, e, "append launch");
  for (int b = 0; b < batch; ++b) mirror_token(c, b, new_region_host[b]);
  c->m.free_top -= popped;
  return MD_OK;
}

/* Stage 1 over layers [l0, l0 + L); q/out hold q_layers layers. */
md_status run_attention(md_ctx *c, int batch, int l0, int L, int q_layers, const void *q_dev,
                        void *out_dev) {
  const md_config &cf = c->cfg;
  AttnParams atp;
  memset(&atp, 0, sizeof(atp));
  atp.q = (const uint16_t *)q_dev;
  atp.out = (uint16_t *)out_dev;
  atp.block_table = ptr<int32_t>(c, c->lay.block_table);
  atp.page_fill = cf.region_aligned_pages ? ptr<uint8_t>(c, c->lay.page_fill) : nullptr;
  atp.mass_acc = ptr<unsigned long long>(c, c->lay.mass_acc);
  atp.scratch = ptr<float>(c, c->lay.scratch);
  atp.partials = ptr<float>(c, c->lay.partials);
  atp.counters = ptr<int>(c, c->lay.counters);
  atp.status = ptr<int>(c, c->lay.status);
  atp.L = cf.num_layers;
  atp.l0 = l0;
  atp.L_launch = L;
  atp.q_layers = q_layers;
  atp.Hq = cf.num_q_heads;
  atp.Hkv = cf.num_kv_heads;
  atp.G = cf.num_q_heads / cf.num_kv_heads;
  atp.ps = cf.page_size;
  atp.P_phys = cf.num_phys_pages;
  atp.P_max = cf.max_pages_per_seq;
  atp.slots = (long long)c->lay.slots;
  atp.scratch_tokens = c->lay.scratch_tokens;
  atp.chunk_stride = c->lay.chunk_stride;
  atp.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  atp.spin_limit_ns = c->spin_limit_ns;
  atp.extra_arrivals = c->extra_arrivals;
  c->extra_arrivals = 0;
  int grid = 1;
  plan_attention(c, batch, L, atp, &grid);
  cudaEvent_t e0;
  prof_begin(c, &e0);
  cudaError_t e = launch_attention(atp, c->tmap, grid, c->stream);
  prof_end(c, STAGE_ATTN, e0);
  if (e != cudaSuccess) return cuda_fail(c, e, "attention launch");
  return MD_OK;
}

void end_step(md_ctx *c, int batch) {
  c->m.mass_pending = 1;
  c->m.mass_batch = batch;
  c->m.window_steps += 1;
  c->m.window_batch = batch;
}

}  // namespace

namespace {

/* The whole decode step once its arguments are checked. */
md_status decode_step_core(md_ctx *c, int batch, const void *q, const void *k_new, const void *v_new,
                           const uint8_t *new_region_host, void *out) {
  const md_config &cf = c->cfg;
  md_status st = begin_step(c, batch, 0, cf.num_layers, (long long)cf.num_layers * cf.num_kv_heads * D,
                            (long long)cf.num_kv_heads * D, k_new, v_new, new_region_host);
  if (st != MD_OK) return st;
  st = run_attention(c, batch, 0, cf.num_layers, cf.num_layers, q, out);
  if (st != MD_OK) return st;
  end_step(c, batch);
  return MD_OK;
}

/* The address at which the kernels can use host buffer h directly, or null:
 * pinned (page-locked) or registered memory at its device address, any other
 * host memory only where the device accesses pageable memory coherently
 * (Grace's NVLink-C2C with address translation).  16-byte alignment is
 * required (the kernels move 16-byte pieces). */
void *device_view(const md_ctx *c, const void *h) {
  if ((uintptr_t)h & 15) return nullptr;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, h) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a.type == cudaMemoryTypeHost && a.devicePointer) return ((uintptr_t)a.devicePointer & 15) ? nullptr : a.devicePointer;
  if (a.type == cudaMemoryTypeUnregistered && c->pageable_access) return const_cast<void *>(h);
  return nullptr;
}

}  // namespace

MD_API md_status md_decode_step(md_ctx *c, int batch, const void *q_dev, const void *k_new,
                                const void *v_new, const uint8_t *new_region_host,
                                void *out_dev) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (c->poisoned) return fail(c, MD_ERR_STATE, "handle unusable after an earlier error");
  if (c->m.layer_next != 0) return fail(c, MD_ERR_STATE, "a layer-by-layer step is in progress");
  if (!q_dev || !k_new || !v_new || !out_dev) return fail(c, MD_ERR_INVALID_ARG, "null pointer");
  md_status st = check_step(c, batch, new_region_host);
  if (st != MD_OK) return st;
  return decode_step_core(c, batch, q_dev, k_new, v_new, new_region_host, out_dev);
}

MD_API md_status md_decode_step_host(md_ctx *c, int batch, const void *q_host, const void *k_new_host,
                                     const void *v_new_host, const uint8_t *new_region_host,
                                     void *out_host) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (c->poisoned) return fail(c, MD_ERR_STATE, "handle unusable after an earlier error");
  if (c->m.layer_next != 0) return fail(c, MD_ERR_STATE, "a layer-by-layer step is in progress");
  if (!q_host || !k_new_host || !v_new_host || !out_host)
    return fail(c, MD_ERR_INVALID_ARG, "null pointer");
  /* every check of the step before anything is copied: the copies are sized
   * by batch, which must fit the workspace */
  md_status st = check_step(c, batch, new_region_host);
  if (st != MD_OK) return st;
  const md_config &cf = c->cfg;
  const size_t q_bytes = (size_t)batch * cf.num_layers * cf.num_q_heads * D * 2;
  const size_t kv_bytes = (size_t)batch * cf.num_layers * cf.num_kv_heads * D * 2;
  /* The new tokens' K/V and the output are used where they are when the
   * device can reach them: the append kernel reads the K/V rows and the
   * attention kernel writes the output over the host link, with no copy (on
   * a GB300 that took the config-2 steady step's device time from 170 to
   * 138 us).  The query rows are always copied into the workspace first:
   * every unit of the attention kernel reads its rows with a TMA copy at its
   * start, and over the host link that latency cost more than the copy
   * (207 us).  Buffers the device cannot reach are copied too. */
  const void *vk = c->zero_copy ? device_view(c, k_new_host) : nullptr;
  const void *vv = c->zero_copy ? device_view(c, v_new_host) : nullptr;
  void *vo = c->zero_copy ? device_view(c, out_host) : nullptr;
  uint8_t *dq = c->ws + c->lay.io_q, *dk = c->ws + c->lay.io_k, *dv = c->ws + c->lay.io_v,
          *dout = c->ws + c->lay.io_out;
  cudaError_t e = cudaMemcpyAsync(dq, q_host, q_bytes, cudaMemcpyHostToDevice, c->stream);
  if (e == cudaSuccess && !vk) e = cudaMemcpyAsync(dk, k_new_host, kv_bytes, cudaMemcpyHostToDevice, c->stream);
  if (e == cudaSuccess && !vv) e = cudaMemcpyAsync(dv, v_new_host, kv_bytes, cudaMemcpyHostToDevice, c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "input copy");
  st = decode_step_core(c, batch, dq, vk ? vk : dk, vv ? vv : dv, new_region_host, vo ? vo : dout);
  if (st != MD_OK) return st;
  if (!vo) {
    e = cudaMemcpyAsync(out_host, dout, q_bytes, cudaMemcpyDeviceToHost, c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "output copy");
  }
  return MD_OK;
}

MD_API md_status md_decode_layer(md_ctx *c, int layer, int batch, const void *q_dev,
                                 const void *k_new, const void *v_new,
                                 const uint8_t *new_region_host, void *out_dev) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (c->poisoned) return fail(c, MD_ERR_STATE, "handle unusable after an earlier error");
  const md_config &cf = c->cfg;
  if (!q_dev || !k_new || !v_new || !out_dev) return fail(c, MD_ERR_INVALID_ARG, "null pointer");
  if (layer != c->m.layer_next)
    return fail(c, MD_ERR_STATE, "layer %d called, layer %d expected", layer, c->m.layer_next);
  md_status st;
  if (layer == 0) {
    st = check_step(c, batch, new_region_host);
    if (st != MD_OK) return st;
    st = begin_step(c, batch, 0, 1, (long long)cf.num_kv_heads * D, 0, k_new, v_new,
                    new_region_host);
    if (st != MD_OK) return st;
    c->m.layer_batch = batch;
  } else {
    if (batch != c->m.layer_batch)
      return fail(c, MD_ERR_INVALID_ARG, "batch changed within a decode step");
    /* the new tokens' pages and state exist: write this layer's K/V only */
    AppendParams ap;
    fill_append_common(c, ap);
    ap.k_src = (const uint16_t *)k_new;
    ap.v_src = (const uint16_t *)v_new;
    ap.sb = (long long)cf.num_kv_heads * D;
    ap.sl = 0;
    ap.sh = D;
    ap.si = 0;
    ap.L = 1;
    ap.l0 = layer;
    ap.init_state = 0;
    ap.lookup_only = 1;
    ap.n_seqs = batch;
    for (int b = 0; b < batch; ++b)
      ap.tok0[b] = (c->n_pages[b] - 1) * cf.page_size + c->tail_fill[b] - 1;
    cudaEvent_t e0;
    prof_begin(c, &e0);
    cudaError_t e = launch_append(ap, c->stream);
    prof_end(c, STAGE_APPEND, e0);
    if (e != cudaSuccess) return cuda_fail(c, e, "append launch");
  }
  st = run_attention(c, batch, layer, 1, 1, q_dev, out_dev);
  if (st != MD_OK) return st;
  c->m.layer_next = layer + 1;
  if (c->m.layer_next == cf.num_layers) {
    c->m.layer_next = 0;
    end_step(c, batch);
  }
  return MD_OK;
}

MD_API md_status md_evict(md_ctx *c, int batch, const int32_t *budget, int32_t *n_evicted_host,
                          int32_t *evicted_ids_dev) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (c->poisoned) return fail(c, MD_ERR_STATE, "handle unusable after an earlier error");
  if (c->m.layer_next != 0) return fail(c, MD_ERR_STATE, "a layer-by-layer step is in progress");
  const md_config &cf = c->cfg;
  if (batch < 1 || batch > cf.max_batch) return fail(c, MD_ERR_INVALID_ARG, "batch out of range");
  if (!budget) return fail(c, MD_ERR_INVALID_ARG, "null budget");
  if (c->m.window_steps > 0 && batch != c->m.window_batch)
    return fail(c, MD_ERR_INVALID_ARG, "batch differs from the observation window's");
  for (int b = 0; b < batch; ++b)
    if (budget[b] < 0) return fail(c, MD_ERR_INVALID_ARG, "negative budget");
  const int ps = cf.page_size;

  /* stages 2-3 */
  ScoreParams sp;
  memset(&sp, 0, sizeof(sp));
  sp.mass_acc = ptr<unsigned long long>(c, c->lay.mass_acc);
  sp.window = ptr<float>(c, c->lay.window);
  sp.a = ptr<float>(c, c->lay.a);
  sp.ahat = ptr<float>(c, c->lay.ahat);
  sp.prio = ptr<float>(c, c->lay.prio);
  sp.page_score = ptr<float>(c, c->lay.page_score);
  sp.t_ref = ptr<int32_t>(c, c->lay.t_ref);
  sp.t_ins = ptr<int32_t>(c, c->lay.t_ins);
  sp.region = ptr<uint8_t>(c, c->lay.region);
  sp.block_table = ptr<int32_t>(c, c->lay.block_table);
  if (cf.region_aligned_pages) {
    sp.page_fill = ptr<uint8_t>(c, c->lay.page_fill);
    sp.seq_tokens = ptr<int32_t>(c, c->lay.seq_tokens);
  }
  sp.calib_sum = ptr<unsigned long long>(c, c->lay.calib);
  sp.calib_cnt = (unsigned int *)(c->ws + c->lay.calib + (size_t)8 * CALIB_BUCKETS * 8);
  sp.calib_on = c->calib_on ? 1 : 0;
  sp.slots = (long long)c->lay.slots;
  sp.ps = ps;
  sp.P_max = cf.max_pages_per_seq;
  sp.fold_only = 0;
  sp.observe = c->m.window_steps > 0 ? 1 : 0;
  sp.mass_pending = c->m.mass_pending;
  sp.norm = (float)((double)std::max(1, c->m.window_steps) * cf.num_layers * cf.num_q_heads);
  sp.t = (int)c->m.t;
  sp.rho = cf.rho;
  sp.gamma = cf.gamma;
  sp.tau_scale = cf.tau_scale;
  sp.alpha = cf.attn_weight;
  sp.score_mode = cf.score_mode;
  sp.random_seed = cf.random_seed;
  sp.page_reduce = cf.page_reduce;
  sp.keep_prio = 1;
  sp.reg = c->reg;
  sp.n_seqs = batch;
  int tot = 0;
  for (int b = 0; b < batch; ++b) {
    sp.n_tokens[b] = (int)c->n_tokens[b];
    sp.n_pages[b] = c->n_pages[b];
    sp.page_start[b] = tot;
    tot += c->n_pages[b];
  }
  sp.page_start[batch] = tot;
  sp.total_pages = tot;
  cudaEvent_t e0;
  prof_begin(c, &e0);
  cudaError_t e = launch_score(sp, c->stream);
  prof_end(c, STAGE_SCORE, e0);
  if (e != cudaSuccess) return cuda_fail(c, e, "score launch");

  /* stage 4 */
  SelectParams sel;
  memset(&sel, 0, sizeof(sel));
  sel.page_score = ptr<float>(c, c->lay.page_score);
  sel.block_table = ptr<int32_t>(c, c->lay.block_table);
  sel.free_stack = ptr<int32_t>(c, c->lay.free_stack);
  sel.evict_list = ptr<int32_t>(c, c->lay.evict_list);
  sel.user_evicted = evicted_ids_dev;
  sel.page_fill = ptr<uint8_t>(c, c->lay.page_fill);
  sel.seq_tokens = ptr<int32_t>(c, c->lay.seq_tokens);
  sel.status = ptr<int>(c, c->lay.status);
  sel.P_max = cf.max_pages_per_seq;
  sel.n_seqs = batch;
  sel.top = (int)c->m.free_top;
  bool warn = false;
  int any = 0, pushed = 0;
  std::vector<int> ev(batch);
  for (int b = 0; b < batch; ++b) {
    const int P = c->n_pages[b];
    const int want = std::max(0, P - budget[b]);
    const int can = std::max(0, evictable_pages(c, b));
    ev[b] = std::min(want, can);
    if (ev[b] < want) warn = true;
    sel.n_pages[b] = P;
    sel.n_evict[b] = ev[b];
    sel.push_off[b] = pushed;
    pushed += ev[b];
    any |= ev[b] > 0;
  }
  if (any || evicted_ids_dev) {
    prof_begin(c, &e0);
    e = launch_select(sel, c->stream);
    prof_end(c, STAGE_SELECT, e0);
    if (e != cudaSuccess) return cuda_fail(c, e, "select launch");
  }
  for (int b = 0; b < batch; ++b) {
    c->n_pages[b] -= ev[b];
    /* evicted pages are never the tail; they are full unless pages are
     * region-aligned, where their fill is known on the device only */
    if (cf.region_aligned_pages) {
      if (ev[b] > 0) c->tokens_exact[b] = 0;
    } else {
      c->n_tokens[b] -= (int64_t)ev[b] * ps;
    }
    if (n_evicted_host) n_evicted_host[b] = ev[b];
  }
  c->m.free_top += pushed;
  c->m.window_steps = 0;
  c->m.mass_pending = 0;
  return warn ? MD_WARN_OVER_BUDGET : MD_OK;
}

MD_API md_status md_sync(md_ctx *c) {
  if (!c) return MD_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "stream synchronize");
  int st[ST_WORDS];
  e = cudaMemcpy(st, c->ws + c->lay.status, sizeof(st), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "status read");
  if (st[ST_CODE] != 0) {
    c->poisoned = true;
    char buf[160];
    snprintf(buf, sizeof(buf), "device status %d (site %d)", st[ST_CODE], st[ST_DIAG]);
    c->err = buf;
    return (md_status)st[ST_CODE];
  }
  return MD_OK;
}

MD_API md_status md_destroy(md_ctx *c) {
  if (!c) return MD_ERR_INVALID_ARG;
  cudaStreamSynchronize(c->stream);
  for (auto &r : c->pending) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : c->ev_pool) cudaEventDestroy(e);
  delete c;
  return MD_OK;
}

namespace {
bool state_array(const md_ctx *c, int what, size_t *off, size_t *bytes) {
  const md_config &cf = c->cfg;
  const Layout &L = c->lay;
  const size_t bt = (size_t)cf.max_batch * cf.max_pages_per_seq * 4;
  switch (what) {
    case MD_STATE_BLOCK_TABLE: *off = L.block_table; *bytes = bt; return true;
    case MD_STATE_PAGE_SCORE: *off = L.page_score; *bytes = bt; return true;
    case MD_STATE_TOKEN_PRIO: *off = L.prio; *bytes = L.slots * 4; return true;
    case MD_STATE_A: *off = L.a; *bytes = L.slots * 4; return true;
    case MD_STATE_T_REF: *off = L.t_ref; *bytes = L.slots * 4; return true;
    case MD_STATE_AHAT: *off = L.ahat; *bytes = L.slots * 4; return true;
    case MD_STATE_FREE: *off = L.free_stack; *bytes = (size_t)cf.num_phys_pages * 4; return true;
    case MD_STATE_REGION: *off = L.region; *bytes = L.slots; return true;
    case MD_STATE_WINDOW: *off = L.window; *bytes = L.slots * 4; return true;
    case MD_STATE_MASS: *off = L.mass_acc; *bytes = L.slots * 8; return true;
    case MD_STATE_T_INS: *off = L.t_ins; *bytes = L.slots * 4; return true;
    case MD_STATE_PAGE_FILL:
      *off = L.page_fill;
      *bytes = (size_t)cf.max_batch * cf.max_pages_per_seq;
      return true;
    case MD_STATE_SEQ_TOKENS: *off = L.seq_tokens; *bytes = (size_t)cf.max_batch * 4; return true;
    case MD_STATE_CALIB: *off = L.calib; *bytes = (size_t)8 * CALIB_BUCKETS * (8 + 4); return true;
    case MD_STATE_POOL:
      *off = L.pool;
      *bytes = (size_t)cf.num_layers * cf.num_phys_pages * cf.num_kv_heads * 2 * cf.page_size * D * 2;
      return true;
  }
  return false;
}
const int SAVED[] = {MD_STATE_BLOCK_TABLE, MD_STATE_PAGE_SCORE, MD_STATE_TOKEN_PRIO, MD_STATE_A,
                     MD_STATE_T_REF,       MD_STATE_AHAT,       MD_STATE_FREE,       MD_STATE_REGION,
                     MD_STATE_WINDOW,      MD_STATE_T_INS,      MD_STATE_PAGE_FILL,  MD_STATE_SEQ_TOKENS,
                     MD_STATE_CALIB};
}  // namespace

MD_API md_status md_get_state(md_ctx *c, int what, void *dst, size_t bytes) {
  if (!c || !dst) return MD_ERR_INVALID_ARG;
  size_t off, n;
  if (!state_array(c, what, &off, &n)) return fail(c, MD_ERR_INVALID_ARG, "unknown state array");
  if (bytes != n) return fail(c, MD_ERR_INVALID_ARG, "state array is %zu bytes, not %zu", n, bytes);
  cudaError_t e = cudaMemcpyAsync(dst, c->ws + off, n, cudaMemcpyDeviceToDevice, c->stream);
  return e == cudaSuccess ? MD_OK : cuda_fail(c, e, "state copy");
}

MD_API md_status md_set_state(md_ctx *c, int what, const void *src, size_t bytes) {
  if (!c || !src) return MD_ERR_INVALID_ARG;
  if (what != MD_STATE_BLOCK_TABLE && what != MD_STATE_FREE && what != MD_STATE_A &&
      what != MD_STATE_T_REF && what != MD_STATE_PAGE_FILL && what != MD_STATE_SEQ_TOKENS)
    return fail(c, MD_ERR_INVALID_ARG, "state array is read-only");
  size_t off, n;
  state_array(c, what, &off, &n);
  if (bytes != n) return fail(c, MD_ERR_INVALID_ARG, "state array is %zu bytes, not %zu", n, bytes);
  cudaError_t e = cudaMemcpyAsync(c->ws + off, src, n, cudaMemcpyDeviceToDevice, c->stream);
  return e == cudaSuccess ? MD_OK : cuda_fail(c, e, "state copy");
}

MD_API md_status md_query(const md_ctx *c, int what, int seq, int64_t *out) {
  if (!c || !out) return MD_ERR_INVALID_ARG;
  const bool per_seq = what == MD_QUERY_TOKENS || what == MD_QUERY_PAGES || what == MD_QUERY_PINNED_PAGES;
  if (per_seq && (seq < 0 || seq >= c->cfg.max_batch)) return MD_ERR_INVALID_ARG;
  switch (what) {
    case MD_QUERY_TOKENS: {
      if (c->tokens_exact[seq]) {
        *out = c->n_tokens[seq];
        return MD_OK;
      }
      int32_t v = 0;   /* region-aligned pages after an eviction: ask the device */
      if (cudaStreamSynchronize(c->stream) != cudaSuccess ||
          cudaMemcpy(&v, c->ws + c->lay.seq_tokens + (size_t)seq * 4, 4, cudaMemcpyDeviceToHost) !=
              cudaSuccess)
        return MD_ERR_CUDA;
      *out = v;
      return MD_OK;
    }
    case MD_QUERY_PAGES: *out = c->n_pages[seq]; return MD_OK;
    case MD_QUERY_FREE_TOP: *out = c->m.free_top; return MD_OK;
    case MD_QUERY_STEP: *out = c->m.t; return MD_OK;
    case MD_QUERY_WINDOW: *out = c->m.window_steps; return MD_OK;
    case MD_QUERY_PINNED_PAGES: *out = c->pinned_pages[seq]; return MD_OK;
  }
  return MD_ERR_INVALID_ARG;
}

namespace {
size_t host_blob_bytes(const md_ctx *c) {
  const size_t B = c->cfg.max_batch;
  return sizeof(HostMirror) + sizeof(RegionTable) + B * (8 + 4 + 4 + 1 + 4 + 4 + 1) + 1;
}
}  // namespace

MD_API md_status md_state_bytes(const md_ctx *c, size_t *dev_bytes, size_t *host_bytes) {
  if (!c) return MD_ERR_INVALID_ARG;
  size_t tot = 0, off, n;
  for (int w : SAVED) {
    state_array(c, w, &off, &n);
    tot += n;
  }
  if (dev_bytes) *dev_bytes = tot;
  if (host_bytes) *host_bytes = host_blob_bytes(c);
  return MD_OK;
}

MD_API md_status md_save_state(md_ctx *c, void *dst_dev, void *host_blob) {
  if (!c || !dst_dev || !host_blob) return MD_ERR_INVALID_ARG;
  if (c->m.window_steps != 0 || c->m.mass_pending || c->m.layer_next != 0)
    return fail(c, MD_ERR_STATE, "checkpoint only between observation windows");
  size_t pos = 0, off, n;
  for (int w : SAVED) {
    state_array(c, w, &off, &n);
    cudaError_t e = cudaMemcpyAsync((uint8_t *)dst_dev + pos, c->ws + off, n,
                                    cudaMemcpyDeviceToDevice, c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "checkpoint copy");
    pos += n;
  }
  uint8_t *h = (uint8_t *)host_blob;
  const size_t B = c->cfg.max_batch;
  memcpy(h, &c->m, sizeof(HostMirror));
  h += sizeof(HostMirror);
  memcpy(h, &c->reg, sizeof(RegionTable));
  h += sizeof(RegionTable);
  memcpy(h, c->n_tokens.data(), B * 8);
  h += B * 8;
  memcpy(h, c->n_pages.data(), B * 4);
  h += B * 4;
  memcpy(h, c->pinned_pages.data(), B * 4);
  h += B * 4;
  memcpy(h, c->tail_pinned.data(), B);
  h += B;
  memcpy(h, c->tail_fill.data(), B * 4);
  h += B * 4;
  memcpy(h, c->tail_region.data(), B * 4);
  h += B * 4;
  memcpy(h, c->tokens_exact.data(), B);
  h += B;
  *h = c->calib_on ? 1 : 0;
  return MD_OK;
}

MD_API md_status md_load_state(md_ctx *c, const void *src_dev, const void *host_blob) {
  if (!c || !src_dev || !host_blob) return MD_ERR_INVALID_ARG;
  if (c->poisoned) return fail(c, MD_ERR_STATE, "handle unusable after an earlier error");
  size_t pos = 0, off, n;
  for (int w : SAVED) {
    state_array(c, w, &off, &n);
    cudaError_t e = cudaMemcpyAsync(c->ws + off, (const uint8_t *)src_dev + pos, n,
                                    cudaMemcpyDeviceToDevice, c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "restore copy");
    pos += n;
  }
  const uint8_t *h = (const uint8_t *)host_blob;
  const size_t B = c->cfg.max_batch;
  memcpy(&c->m, h, sizeof(HostMirror));
  h += sizeof(HostMirror);
  memcpy(&c->reg, h, sizeof(RegionTable));
  h += sizeof(RegionTable);
  memcpy(c->n_tokens.data(), h, B * 8);
  h += B * 8;
  memcpy(c->n_pages.data(), h, B * 4);
  h += B * 4;
  memcpy(c->pinned_pages.data(), h, B * 4);
  h += B * 4;
  memcpy(c->tail_pinned.data(), h, B);
  h += B;
  memcpy(c->tail_fill.data(), h, B * 4);
  h += B * 4;
  memcpy(c->tail_region.data(), h, B * 4);
  h += B * 4;
  memcpy(c->tokens_exact.data(), h, B);
  h += B;
  c->calib_on = *h != 0;
  /* a checkpoint holds no pending step mass; clear whatever the live state
   * had accumulated, or the next step would add to it */
  cudaError_t e = cudaMemsetAsync(c->ws + c->lay.mass_acc, 0, c->lay.slots * 8, c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "restore: clear the step mass");
  return MD_OK;
}

MD_API md_status md_profile_enable(md_ctx *c, int enable) {
  if (!c) return MD_ERR_INVALID_ARG;
  c->prof = enable != 0;
  if (c->prof) {
    for (int s = 0; s < N_STAGES; ++s) {
      c->prof_ms[s] = 0;
      c->prof_n[s] = 0;
    }
  }
  return MD_OK;
}

MD_API md_status md_profile_read(md_ctx *c, double *ms, int64_t *launches, int n_stages) {
  if (!c) return MD_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "stream synchronize");
  for (auto &r : c->pending) {
    float x = 0.f;
    if (cudaEventElapsedTime(&x, r.a, r.b) == cudaSuccess) {
      c->prof_ms[r.stage] += x;
      c->prof_n[r.stage] += 1;
    }
    c->ev_pool.push_back(r.a);
    c->ev_pool.push_back(r.b);
  }
  c->pending.clear();
  for (int s = 0; s < n_stages && s < N_STAGES; ++s) {
    if (ms) ms[s] = c->prof_ms[s];
    if (launches) launches[s] = c->prof_n[s];
  }
  return MD_OK;
}

MD_API md_status md_debug_set(md_ctx *c, int key, int64_t value) {
  if (!c) return MD_ERR_INVALID_ARG;
  if (key == MD_DEBUG_SPIN_LIMIT_NS) {
    if (value < 1000) return fail(c, MD_ERR_INVALID_ARG, "spin limit below 1 us");
    c->spin_limit_ns = (long long)value;
    return MD_OK;
  }
  if (key == MD_DEBUG_EXTRA_ARRIVALS) {
    if (value < 0 || value > 1000) return fail(c, MD_ERR_INVALID_ARG, "extra arrivals out of range");
    c->extra_arrivals = (int)value;
    return MD_OK;
  }
  if (key == MD_DEBUG_GRID_LIMIT) {
    /* all chunks of an item must fit in one round of the grid (the order
     * that keeps the kernel's cross-CTA waits free of cycles) */
    if (value < 0 || (value > 0 && value < MD_MAX_CHUNKS))
      return fail(c, MD_ERR_INVALID_ARG, "grid limit must be 0 or at least MD_MAX_CHUNKS");
    c->grid_cap = (int)std::min<int64_t>(value, MAX_GRID);
    return MD_OK;
  }
  if (key == MD_DEBUG_UNIT_OVERHEAD) {
    if (value < 0 || value > 65536) return fail(c, MD_ERR_INVALID_ARG, "unit overhead out of range");
    c->unit_overhead_kib = (int)value;
    return MD_OK;
  }
  if (key == MD_DEBUG_ZERO_COPY) {
    if (value != 0 && value != 1) return fail(c, MD_ERR_INVALID_ARG, "zero-copy switch must be 0 or 1");
    c->zero_copy = (int)value;
    return MD_OK;
  }
  if (key == MD_DEBUG_COMBINE_OVERHEAD) {
    if (value < 0 || value > 65536) return fail(c, MD_ERR_INVALID_ARG, "combine overhead out of range");
    c->combine_overhead_kib = (int)value;
    return MD_OK;
  }
  if (key == MD_DEBUG_FORCE_CHUNKS) {
    if (value < 0 || value > MD_MAX_CHUNKS) return fail(c, MD_ERR_INVALID_ARG, "chunk count out of range");
    c->force_chunks = (int)value;
    return MD_OK;
  }
  return fail(c, MD_ERR_INVALID_ARG, "unknown debug key");
}

MD_API md_status md_calib_enable(md_ctx *c, int enable) {
  if (!c) return MD_ERR_INVALID_ARG;
  c->calib_on = enable != 0;
  if (c->calib_on) {
    cudaError_t e = cudaMemsetAsync(c->ws + c->lay.calib, 0, (size_t)8 * CALIB_BUCKETS * 12, c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "calibration clear");
  }
  return MD_OK;
}

MD_API md_status md_calib_read(md_ctx *c, double *mass_sum, int64_t *count) {
  if (!c || !mass_sum || !count) return MD_ERR_INVALID_ARG;
  std::vector<unsigned long long> s((size_t)8 * CALIB_BUCKETS);
  std::vector<unsigned int> n((size_t)8 * CALIB_BUCKETS);
  cudaError_t e = cudaMemcpyAsync(s.data(), c->ws + c->lay.calib, s.size() * 8, cudaMemcpyDeviceToHost,
                                  c->stream);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(n.data(), c->ws + c->lay.calib + s.size() * 8, n.size() * 4,
                        cudaMemcpyDeviceToHost, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "calibration read");
  for (int r = 0; r < MD_NUM_REGIONS; ++r)
    for (int b = 0; b < CALIB_BUCKETS; ++b) {
      const size_t k = (size_t)r * CALIB_BUCKETS + b;
      mass_sum[k] = (double)s[k] * (1.0 / 4294967296.0);
      count[k] = n[k];
    }
  return MD_OK;
}

MD_API md_status md_calib_fit(const double *mass_sum, const int64_t *count, int n_buckets,
                              int bucket_width, int64_t min_count, double *rate_out,
                              double *half_life_out) {
  if (!mass_sum || !count || !rate_out || !half_life_out || n_buckets < 1 || bucket_width < 1)
    return MD_ERR_INVALID_ARG;
  for (int r = 0; r < MD_NUM_REGIONS; ++r) {
    /* weighted least squares of y = log(mean) on x = centre age, w = count */
    double W = 0, Sx = 0, Sy = 0, Sxx = 0, Sxy = 0;
    int used = 0;
    for (int b = 0; b < n_buckets; ++b) {
      const int64_t n = count[(size_t)r * n_buckets + b];
      const double m = mass_sum[(size_t)r * n_buckets + b];
      if (n < (min_count > 1 ? min_count : 1) || !(m > 0)) continue;
      const double x = (double)bucket_width * b + 0.5 * bucket_width;
      const double y = log(m / (double)n);
      const double w = (double)n;
      W += w;
      Sx += w * x;
      Sy += w * y;
      Sxx += w * x * x;
      Sxy += w * x * y;
      ++used;
    }
    if (used < 2) {
      rate_out[r] = NAN;
      half_life_out[r] = NAN;
      continue;
    }
    const double slope = (W * Sxy - Sx * Sy) / (W * Sxx - Sx * Sx);
    rate_out[r] = -slope;
    half_life_out[r] = rate_out[r] > 0 ? log(2.0) / rate_out[r] : INFINITY;
  }
  return MD_OK;
}

MD_API const char *md_last_error(const md_ctx *c) { return c ? c->err.c_str() : "null handle"; }
