/* Stages 0, 2, 3, 4 of the MemDecay step and the workspace initialiser.
 *
 *   append   write new tokens' K/V into the page pool (taking fresh pages
 *            from the free stack) and start each token's state: region label,
 *            t_ref = insertion step, a = 0 (Sec. III-A; Fig. 1 "append KV").
 *   score    per page, one lane per token: Abar from the window accumulator
 *            and the step's mass summed over layers and heads (Sec. III-C;
 *            a fixed-point accumulator the attention kernel fills), the EWMA
 *            (Eq. 2), the refresh test Abar >= tau_scale/|K_t| (Eq. 3), the
 *            retention score (Eq. 4, lambda = ln2 / half-life, Eq. 7) and the
 *            page score by a shuffle reduction over the page's lanes (Eq. 5;
 *            pinned pages and the page being written score +inf).  With
 *            fold_only it only adds the step's mass into the window accumulator.
 *   select   one CTA per sequence: radix select (4 passes of 8-bit digits
 *            over order-preserving uint32 keys, ties by logical page index)
 *            of the e lowest evictable pages, stable compaction of the block
 *            table row, push of the freed ids onto the free stack
 *            (Sec. III-D, Algorithm 1: lowest S_p first; a selection, not a
 *            sort or a heap). */
#include <float.h>

#include "md_internal.h"
#include "md_ptx.cuh"

namespace md {

/* ---------------------------------------------------------------- init --- */
__global__ void init_kernel(int32_t *free_stack, int P_phys, int *status, int *counters,
                            size_t n_items) {
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < (size_t)P_phys; i += stride)
    free_stack[i] = P_phys - 1 - (int)i;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_items; i += stride)
    counters[i] = 0;
  if (blockIdx.x == 0 && threadIdx.x < ST_WORDS) status[threadIdx.x] = 0;
}

cudaError_t launch_init(int32_t *free_stack, int P_phys, int *status, int *counters,
                        size_t n_items, cudaStream_t s) {
  init_kernel<<<304, 256, 0, s>>>(free_stack, P_phys, status, counters, n_items);
  return cudaGetLastError();
}

/* -------------------------------------------------------------- append --- */
/* One thread per 16-byte piece of a token's K or V row in one (layer, head). */
__global__ void append_kernel(const __grid_constant__ AppendParams p) {
  pdl_wait();
  pdl_trigger();
  const long long per_token = (long long)p.L * p.Hkv * 2 * 16;
  const long long total = (long long)p.n_seqs * p.n_per_seq * per_token;
  for (long long w = (long long)blockIdx.x * blockDim.x + threadIdx.x; w < total;
       w += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(w & 15);
    long long r = w >> 4;
    const int kv = (int)(r & 1);
    r >>= 1;
    const int h = (int)(r % p.Hkv);
    r /= p.Hkv;
    const int l = (int)(r % p.L);
    r /= p.L;
    const int i = (int)(r % p.n_per_seq);
    const int j = (int)(r / p.n_per_seq);
    const int seq = p.seq0 + j;
    const int tok = p.slots_dev ? p.slots_dev[i] : p.tok0[j] + i;   // slot in the sequence
    const int pg = tok / p.ps, off = tok - pg * p.ps;
    const int pages_before = p.lookup_only ? 0x7fffffff : p.pages_before[j];
    int phys;
    if (pg < pages_before)
      phys = p.block_table[(size_t)seq * p.P_max + pg];
    else
      phys = p.free_stack[p.pop_base[j] - (pg - pages_before)];

    const uint16_t *src = (kv == 0 ? p.k_src : p.v_src) + (long long)j * p.sb +
                          (long long)l * p.sl + (long long)h * p.sh + (long long)i * p.si;
    uint16_t *dst = p.pool +
                    ((((size_t)(p.l0 + l) * p.P_phys + phys) * p.Hkv + h) * 2 + kv) * (size_t)p.ps * D +
                    (size_t)off * D;
    ((uint4 *)dst)[c] = ((const uint4 *)src)[c];

    if (p.init_state && c == 0 && kv == 0 && h == 0 && l == 0) {
      const size_t slot = (size_t)phys * p.ps + off;
      p.region[slot] = p.regions_dev ? p.regions_dev[i] : p.regions_param[j];
      p.t_ref[slot] = p.steps_dev ? p.steps_dev[i] : p.insert_step;
      p.t_ins[slot] = p.t_ref[slot];
      p.a[slot] = 0.f;
      p.window[slot] = 0.f;
      p.ahat[slot] = 0.f;
      p.prio[slot] = 0.f;
      if (off == 0 && pg >= pages_before) p.block_table[(size_t)seq * p.P_max + pg] = phys;
      /* the last token this append puts on a page sets the page's fill */
      const int next = (i + 1 < p.n_per_seq) ? (p.slots_dev ? p.slots_dev[i + 1] : tok + 1) : -1;
      if (next < 0 || next / p.ps != pg) p.page_fill[(size_t)seq * p.P_max + pg] = (uint8_t)(off + 1);
      if (i == 0) p.seq_tokens[seq] += p.n_per_seq;
    }
  }
}

cudaError_t launch_append(const AppendParams &p, cudaStream_t s) {
  const long long total = (long long)p.n_seqs * p.n_per_seq * p.L * p.Hkv * 32;
  if (total == 0) return cudaSuccess;
  long long blocks = (total + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  return launch_pdl(append_kernel, (int)blocks, 256, 0, s, p);
}

/* ------------------------------------------------------ score / fold ----- */
__device__ __forceinline__ int find_seq(const int *start, int n, int x) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (start[mid] <= x) lo = mid; else hi = mid - 1;
  }
  return lo;
}

/* Uniform draw in [0, 1) for the random-baseline score: the SplitMix64
 * finaliser (Steele, Lea and Flood, 2014) of (seed, step, slot); the top 24
 * bits scaled by 2^-24 are exact in fp32. */
__device__ __forceinline__ float random_draw(unsigned long long seed, int t, size_t slot) {
  unsigned long long z = (seed * 0x9E3779B97F4A7C15ull) ^ ((unsigned long long)(unsigned)t << 40) ^
                         (unsigned long long)slot;
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  z ^= z >> 31;
  return (float)(z >> 40) * 5.9604644775390625e-08f;
}

/* A tile is 32/PS consecutive pages, one lane per token slot, one warp per
 * tile; the loop count is uniform across the block so the segmented shuffle
 * reductions see every lane.  A token's step mass is one fixed-point
 * accumulator (the attention kernel adds every (layer, KV head) into it):
 * read and zeroed here, loaded together with the token's state.  The
 * launcher sizes the grid to one wave of resident blocks. */
template <int PS>
__global__ void __launch_bounds__(256, 6) score_kernel(const __grid_constant__ ScoreParams p) {
  pdl_wait();
  pdl_trigger();
  constexpr int PPW = 32 / PS;
  /* calibration histogram of this block (Sec. IV-B, Eq. 6's input): observed
   * mass in fixed point, so integer atomics keep the sums order-independent */
  __shared__ unsigned long long h_sum[8 * CALIB_BUCKETS];
  __shared__ unsigned int h_cnt[8 * CALIB_BUCKETS];
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const int tiles = (p.total_pages + PPW - 1) / PPW;
  const bool need_mass = p.fold_only || (p.observe && p.mass_pending);
  const float INF = INFINITY;
  const bool calib = p.calib_on && p.observe && !p.fold_only;
  if (calib) {
    for (int k = threadIdx.x; k < 8 * CALIB_BUCKETS; k += blockDim.x) {
      h_sum[k] = 0ull;
      h_cnt[k] = 0u;
    }
    __syncthreads();
  }
  for (int t0 = blockIdx.x * 8; t0 < tiles; t0 += gridDim.x * 8) {
    const int base = (t0 + wib) * PPW;
    const int gp = base + lane / PS;
    const int off = lane % PS;
    const bool page_ok = gp < p.total_pages;
    int b = 0, pg = 0, P = 0;
    bool valid = false;
    size_t slot = 0;
    if (page_ok) {
      b = find_seq(p.page_start, p.n_seqs, gp);
      pg = gp - p.page_start[b];
      P = p.n_pages[b];
      valid = p.page_fill ? off < p.page_fill[(size_t)b * p.P_max + pg]
                          : pg * PS + off < p.n_tokens[b];
      slot = (size_t)p.block_table[(size_t)b * p.P_max + pg] * PS + off;
    }
    /* the token's state and its step mass, all loads independent */
    int reg = 0, tr = 0, tins = 0, ntok = 1;
    float a = 0.f, w = 0.f;
    unsigned long long macc = 0ull;
    if (valid) {
      if (need_mass) macc = __ldcs(p.mass_acc + slot);
      if (p.fold_only) {
        w = p.window[slot];
      } else {
        reg = p.region[slot];
        a = p.a[slot];
        tr = p.t_ref[slot];
        if (p.observe) w = p.window[slot];
        if (p.observe || p.score_mode == 2) ntok = p.seq_tokens ? p.seq_tokens[b] : p.n_tokens[b];
        if (calib || p.score_mode == 3) tins = p.t_ins[slot];
      }
    }
    /* the sum over layers and query heads, rounded once to fp32 */
    const float msum = __ull2float_rn(macc) * MASS_UNIT;
    if (valid && need_mass) p.mass_acc[slot] = 0ull;
    float s = 0.f;
    int pinned = 0;
    if (valid) {
      if (p.fold_only) {
        p.window[slot] = w + msum;
      } else {
        if (p.observe) {
          if (p.mass_pending) w += msum;
          const float abar = __fdiv_rn(w, p.norm);                    // Sec. III-C
          a = p.rho * a + p.gamma * abar;                             // Eq. 2
          const float tau = __fdiv_rn(p.tau_scale, (float)ntok);
          if (abar >= tau) tr = p.t;                                  // Eq. 3
          p.window[slot] = 0.f;
          p.ahat[slot] = abar;
          p.a[slot] = a;
          p.t_ref[slot] = tr;
          if (calib) {
            const int age = p.t - tins;
            const int bkt = age >= 0 ? age / CALIB_WIDTH : -1;
            if (bkt >= 0 && bkt < CALIB_BUCKETS) {
              atomicAdd(&h_sum[reg * CALIB_BUCKETS + bkt], __float2ull_rn(abar * 4294967296.0f));
              atomicAdd(&h_cnt[reg * CALIB_BUCKETS + bkt], 1u);
            }
          }
        }
        const float x = __fdiv_rn((float)(p.t - tr), p.reg.half_life[reg]);
        const float d = exp2f(-x);                                    // Eqs. 4, 7
        switch (p.score_mode) {
          case 0: s = p.reg.base[reg] * d + p.alpha * a; break;       // Eq. 4
          case 1: s = (p.reg.base[reg] + p.alpha * a) * d; break;
          case 2: s = p.reg.base[reg] * d + p.alpha * a * (float)ntok; break;
          case 3: s = (float)tins; break;                             // recency
          default: s = random_draw(p.random_seed, p.t, slot); break;   // random
        }
        pinned = p.reg.pinned[reg];
        if (pinned) s = INF;
        if (p.keep_prio) p.prio[slot] = s;
      }
    }
    if (!p.fold_only) {
      float sum = (valid && !pinned) ? s : 0.f;
      float mx = (valid && !pinned) ? s : -INF;
      int anyp = (valid && pinned) ? 1 : 0;
      int cnt = valid ? 1 : 0;
#pragma unroll
      for (int o = PS / 2; o > 0; o >>= 1) {
        sum += __shfl_xor_sync(0xffffffffu, sum, o, PS);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o, PS));
        anyp |= __shfl_xor_sync(0xffffffffu, anyp, o, PS);
        cnt += __shfl_xor_sync(0xffffffffu, cnt, o, PS);
      }
      if (page_ok && off == 0) {
        float S;
        if (anyp || pg == P - 1) S = INF;                            // pinning, tail
        else S = (p.page_reduce == 0) ? __fdiv_rn(sum, (float)cnt) : mx;   // Eq. 5
        p.page_score[(size_t)b * p.P_max + pg] = S;
      }
    }
  }
  if (calib) {
    __syncthreads();
    for (int k = threadIdx.x; k < 8 * CALIB_BUCKETS; k += blockDim.x)
      if (h_cnt[k]) {
        atomicAdd(&p.calib_sum[k], h_sum[k]);
        atomicAdd(&p.calib_cnt[k], h_cnt[k]);
      }
  }
}

/* Blocks of the score kernel that are resident at once on the current device
 * (SMs x blocks per SM from the occupancy of the instance).  The kernel gives
 * every block an equal share of the pages, so a grid larger than one wave
 * would leave the second wave's blocks as a tail. */
template <int PS>
static int score_grid_cap() {
  static int cached[64];   // per device ordinal; a racy first fill writes the same value
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152 * 4;
  if (cached[dev] > 0) return cached[dev];
  int sms = 0, per_sm = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<PS>, 256, 0) != cudaSuccess ||
      sms <= 0 || per_sm <= 0)
    return 152 * 4;
  cached[dev] = sms * per_sm;
  return cached[dev];
}

cudaError_t launch_score(const ScoreParams &p, cudaStream_t s) {
  if (p.total_pages == 0) return cudaSuccess;
  const int ppb = 256 / p.ps;   // pages per block and iteration: one warp per tile
  const int cap = p.ps == 16 ? score_grid_cap<16>() : score_grid_cap<32>();
  long long blocks = (p.total_pages + ppb - 1) / ppb;
  if (blocks > cap) blocks = cap;
  if (p.ps == 16) return launch_pdl(score_kernel<16>, (int)blocks, 256, 0, s, p);
  return launch_pdl(score_kernel<32>, (int)blocks, 256, 0, s, p);
}

/* -------------------------------------------------------------- select --- */
constexpr int SEL_THREADS = 1024;
constexpr uint32_t KEY_PINNED = 0xFFFFFFFFu;

/* Order-preserving map of fp32 onto uint32 (larger float -> larger key). */
__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

/* Block-wide exclusive scan of one int per thread; returns the prefix and
 * writes the block total to *total. */
__device__ __forceinline__ int block_exclusive_scan(int v, int *warp_sums, int *total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[wid] = x;
  __syncthreads();
  if (wid == 0) {
    const int nw = blockDim.x >> 5;
    int s = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < nw) warp_sums[lane] = s;   // inclusive sums of warps
  }
  __syncthreads();
  const int before = (wid > 0 ? warp_sums[wid - 1] : 0) + x - v;
  *total = warp_sums[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(SEL_THREADS) select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ uint32_t sm[];
  uint32_t *keys = sm;                               // [P_max]
  int32_t *phys = (int32_t *)(sm + p.P_max);         // [P_max]
  uint8_t *fills = (uint8_t *)(sm + 2 * (size_t)p.P_max);   // [P_max]
  __shared__ int hist[256];
  __shared__ int warp_sums[32];
  __shared__ uint32_t s_prefix;
  __shared__ int s_k, s_bad, s_gone, s_cnt;

  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  const int P = p.n_pages[b];
  const int e = p.n_evict[b];
  int32_t *row = p.block_table + (size_t)b * p.P_max;
  int32_t *uout = p.user_evicted ? p.user_evicted + (size_t)b * p.P_max : nullptr;
  if (e == 0) {
    if (uout)
      for (int i = threadIdx.x; i < p.P_max; i += blockDim.x) uout[i] = -1;
    return;
  }
  const float *sc = p.page_score + (size_t)b * p.P_max;
  uint8_t *frow = p.page_fill + (size_t)b * p.P_max;
  for (int i = threadIdx.x; i < P; i += blockDim.x) {
    const float S = sc[i];
    keys[i] = (S == INFINITY) ? KEY_PINNED : order_key(S);
    phys[i] = row[i];
    fills[i] = frow[i];
  }
  if (threadIdx.x == 0) { s_prefix = 0u; s_k = e; s_bad = 0; s_gone = 0; s_cnt = 0; }
  __syncthreads();

  /* radix select of the e-th smallest evictable key, most significant digit
   * first.  It stops early once the digit's bucket holds exactly the keys
   * still to be taken: then every key below the bucket and every key in it
   * is evicted, the same set the remaining passes would pick. */
  uint32_t mask = 0u;
  bool whole_bucket = false;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    const uint32_t prefix = s_prefix;
    for (int i = threadIdx.x; i < P; i += blockDim.x) {
      const uint32_t k = keys[i];
      if (k != KEY_PINNED && (k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      /* the digit holding the k-th smallest remaining key: one warp, eight
       * bins per lane; the lane whose cumulative range (excl, incl] holds k
       * walks its bins (the same digit and residual a serial scan finds) */
      const int lane = threadIdx.x;
      const int k = s_k;
      int c[8], sum = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = hist[lane * 8 + j];
        sum += c[j];
      }
      int incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int excl = incl - sum;
      const bool mine = excl < k && k <= incl;
      if (__ballot_sync(0xffffffffu, mine) == 0u) {
        if (lane == 0) s_bad = 1;         // fewer evictable pages than e
      } else if (mine) {
        int cum = excl, digit = lane * 8;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (cum + c[j] >= k) { digit = lane * 8 + j; break; }
          cum += c[j];
        }
        s_prefix = prefix | ((uint32_t)digit << shift);
        s_k = k - cum;
        s_cnt = hist[digit];
      }
    }
    __syncthreads();
    if (s_bad) {
      if (threadIdx.x == 0) atomicCAS(&p.status[ST_CODE], 0, (int)MD_ERR_STATE);
      return;
    }
    mask |= 0xFFu << shift;
    if (pass < 3 && s_k == s_cnt) {   // the same value in every thread
      whole_bucket = true;
      break;
    }
  }
  /* key of the e-th smallest evictable page and how many pages with key == T
   * are evicted; for a whole bucket, T is the bucket's largest key and every
   * page equal to it goes */
  const uint32_t T = whole_bucket ? (s_prefix | ~mask) : s_prefix;
  const int take_eq = whole_bucket ? P : s_k;

  /* evict: key < T, or key == T among the first take_eq in logical order;
   * compact kept pages in order; list the evicted ones in logical order */
  int carry_eq = 0, carry_ev = 0, gone = 0;
  const int base_push = p.top + p.push_off[b];
  for (int t0 = 0; t0 < P; t0 += blockDim.x) {
    const int i = t0 + threadIdx.x;
    const bool in = i < P;
    const uint32_t k = in ? keys[i] : KEY_PINNED;
    const int eq = (in && k == T) ? 1 : 0;
    int tot_eq;
    const int rank_eq = carry_eq + block_exclusive_scan(eq, warp_sums, &tot_eq);
    const int ev = (in && k != KEY_PINNED && (k < T || (eq && rank_eq < take_eq))) ? 1 : 0;
    int tot_ev;
    const int idx_ev = carry_ev + block_exclusive_scan(ev, warp_sums, &tot_ev);
    if (in) {
      const int id = phys[i];
      if (ev) {
        p.evict_list[(size_t)b * p.P_max + idx_ev] = id;
        p.free_stack[base_push + idx_ev] = id;
        if (uout) uout[idx_ev] = id;
        gone += fills[i];
      } else {
        row[i - idx_ev] = id;
        frow[i - idx_ev] = fills[i];
      }
    }
    carry_eq += tot_eq;
    carry_ev += tot_ev;
  }
  if (gone) atomicAdd(&s_gone, gone);
  __syncthreads();
  if (threadIdx.x == 0) p.seq_tokens[b] -= s_gone;
  for (int i = P - e + threadIdx.x; i < P; i += blockDim.x) {
    row[i] = -1;
    frow[i] = 0;
  }
  if (uout)
    for (int i = e + threadIdx.x; i < p.P_max; i += blockDim.x) uout[i] = -1;
}

cudaError_t launch_select(const SelectParams &p, cudaStream_t s) {
  if (p.n_seqs == 0) return cudaSuccess;
  /* one thread per page of the longest sequence (whole warps, at least 128,
   * at most SEL_THREADS): fewer warps make the passes' barriers cheaper */
  int pmax = 0;
  for (int b = 0; b < p.n_seqs; ++b) pmax = p.n_pages[b] > pmax ? p.n_pages[b] : pmax;
  int threads = (pmax + 31) / 32 * 32;
  threads = threads < 128 ? 128 : (threads > SEL_THREADS ? SEL_THREADS : threads);
  const size_t smem = (size_t)p.P_max * 9;
  /* raise the kernel's dynamic shared-memory limit only when a larger table
   * needs it (a host call per launch costs more than the kernel at small
   * sizes); per device ordinal, a racy first fill sets the same value */
  static int granted[64];
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= 64 || granted[dev] < (int)smem) {
    err = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    if (dev >= 0 && dev < 64) granted[dev] = (int)smem;
  }
  return launch_pdl(select_kernel, p.n_seqs, threads, (int)smem, s, p);
}

}  // namespace md
