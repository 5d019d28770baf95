/* Stage 1: paged GQA decode attention that also yields every cached token's
 * attention mass (Sec. III-C: Abar_i, the attention a token receives averaged
 * over heads and layers, is what MemDecay observes).
 *
 * Work unit: (sequence b, layer l, KV head kvh, chunk j of the sequence's
 * pages).  The chunks of one (b, l, kvh) item split its pages (flash-decoding
 * style) so that ~all 152 SMs stream K/V at once.  Two persistent cooperative
 * CTAs per SM; CTA c walks the units c, c+grid, c+2*grid, ...
 *
 * Per CTA: warp 0 is the producer.  One elected lane issues, per page, two
 * TMA tile loads (cp.async.bulk.tensor, 128-byte swizzle, L2 evict_first) of
 * the page's K and V rows into a ring of shared-memory stages with mbarrier
 * completion.  Warps 1..NCW consume pages round-robin by the CTA-wide page
 * index i (warp i % NCW, stage i % R), so each warp owns R / NCW stages: the
 * warps may run up to a unit apart and no wait is ever more than one phase
 * ahead:
 *   S^T[16 tokens x 8 heads] = K[16 x 128] . Q^T    (mma.sync m16n8k16 bf16)
 *   online softmax per head (exp2 domain), raw scores kept in scratch
 *   O^T[128 x 8] += V^T[128 x 16] . P^T             (P^T via movmatrix.trans)
 * GQA makes both products real dense tiles: the G <= 8 query heads of one KV
 * head share every K/V byte read, so K/V are read from HBM once per step.
 *
 * Exact mass without re-reading K: a token's mass is sum_h exp(s_hi - m_h)/Z_h
 * with the item's global (m_h, Z_h).  A unit publishes its partial (m, Z, O)
 * and bumps the item's arrival counter.  The last warp of the CTA, the
 * finisher, then takes the unit over while the consumers stream the next
 * one: it waits, bounded by %globaltimer, for all chunks of the item,
 * combines the partials (its slice of the output O) and turns the stored
 * scores into masses.  Each token's mass is added at L2 into its physical
 * slot's fixed-point accumulator (an integer add, so the sum over layers and
 * KV heads does not depend on the order in which items finish); the
 * no-allocation entry point writes one fp32 row per (layer, KV head)
 * instead.  Raw scores live in two slots per CTA; the consumers reuse a slot only
 * after the finisher has released it (mbarrier hand-off both ways), so a
 * unit's finish overlaps the streaming of the next one.  All waits are
 * bounded; on expiry the kernel records MD_ERR_DEVICE_TIMEOUT, raises an abort
 * flag every CTA polls, drains its in-flight copies and returns.  No float
 * atomics: results are bit-identical run to run. */
#include <cuda_bf16.h>
#include <float.h>

#include "md_internal.h"
#include "md_ptx.cuh"

namespace md {

template <int PS, int NCW>
struct AttnShape {
  static constexpr int NT = PS / 16;                 // 16-token tiles per page
  static constexpr int HALF_BYTES = 2 * PS * 128;    // 64 columns of K and V rows
  static constexpr int STAGE_BYTES = 2 * HALF_BYTES; // one page of one (layer, KV head)
  static constexpr int R = (PS == 16) ? 8 : 4;       // ring stages (64 KiB per CTA)
  static_assert(R % NCW == 0, "every consumer warp owns R / NCW stages");
  static constexpr int RING_BYTES = R * STAGE_BYTES;
  static constexpr int CTAS_PER_SM = 2;
  static constexpr int THREADS = 32 * (NCW + 2);     // producer, NCW consumers, finisher
  static constexpr int Q_BYTES = GP * D * 2;         // one unit's query heads
  static constexpr int MAX_UNIT_PAGES = MD_MAX_CHUNK_TOKENS / PS;
  static constexpr int MERGE_FLOATS = NCW * (24 + GP * D);
  static constexpr int FIN_FLOATS = 16 + 3 * MD_MAX_CHUNKS * GP;
  static constexpr int OBUF_FLOATS = GP * D + MD_MAX_CHUNKS;   // C slices of ceil(G*D/C)
  static constexpr size_t SMEM = 1024 + RING_BYTES + 2 * Q_BYTES + (2 * R + 10) * 8 +
                                 4 * MERGE_FLOATS + 4 * FIN_FLOATS + 8 * MAX_UNIT_PAGES +
                                 4 * OBUF_FLOATS + 4 * R + 64;
};

struct Unit {
  int b, l, kvh, j, C, p0, p1, X;
};

__device__ __forceinline__ Unit decode_unit(const AttnParams &p, int u) {
  int lo = 0, hi = p.n_seqs - 1;
  if (p.units_per_seq > 0) {          // every sequence has the same number of units
    lo = u / p.units_per_seq;
  } else {
    while (lo < hi) {
      int mid = (lo + hi + 1) >> 1;
      if (p.unit_start[mid] <= u) lo = mid; else hi = mid - 1;
    }
  }
  Unit un;
  un.b = lo;
  un.C = p.chunks[lo];
  int rem = u - p.unit_start[lo];
  int item = rem / un.C;
  un.j = rem - item * un.C;
  const int ll = item / p.Hkv;
  un.kvh = item - ll * p.Hkv;
  un.l = p.l0 + ll;
  int P = p.n_pages[lo];
  un.p0 = (int)(((long long)un.j * P) / un.C);
  un.p1 = (int)(((long long)(un.j + 1) * P) / un.C);
  un.X = (lo * p.L + un.l) * p.Hkv + un.kvh;
  return un;
}

/* Physical ids (and, with region-aligned pages, fills) of pages [from,
 * min(from + 8, to)) of unit x; returns how many.  The loads are
 * independent, so all of them are in flight at once. */
template <bool ALIGNED>
__device__ __forceinline__ int load_batch(const AttnParams &p, const Unit &x, int from, int to, int (&ph)[8],
                                          int (&fl)[8]) {
  const int cnt = min(8, to - from);
  const int32_t *bt = p.block_table + (size_t)x.b * p.P_max;
#pragma unroll
  for (int k = 0; k < 8; ++k) ph[k] = k < cnt ? bt[from + k] : 0;
  if (ALIGNED) {
    const uint8_t *fr = p.page_fill + (size_t)x.b * p.P_max;
#pragma unroll
    for (int k = 0; k < 8; ++k) fl[k] = k < cnt ? fr[from + k] : 0;
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) fl[k] = 0;
  }
  return cnt;
}

__device__ __forceinline__ void raise_status(const AttnParams &p, int code, int diag) {
  atomicCAS(&p.status[ST_CODE], 0, code);
  atomicExch(&p.status[ST_DIAG], diag);
  atomicExch(&p.status[ST_ABORT], 1);
}

/* Bounded wait on an mbarrier phase; false on abort or timeout. */
__device__ __noinline__ bool wait_phase(uint32_t bar, uint32_t parity, const AttnParams &p,
                                        int diag, bool honour_abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = globaltimer();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (honour_abort && ld_volatile(&p.status[ST_ABORT])) return false;
    if (globaltimer() - t0 > p.spin_limit_ns) {
      raise_status(p, MD_ERR_DEVICE_TIMEOUT, diag);
      return false;
    }
  }
}

/* Address of the 16-byte chunk holding (row, d..d+7) of a stage stored as two
 * 64-column halves of 128-byte rows with the TMA 128-byte swizzle. */
template <int PS>
__device__ __forceinline__ uint32_t swz(uint32_t stage, int row, int d) {
  const int half = d >> 6;
  const int chunk = (d & 63) >> 3;
  return stage + half * (2 * PS * 128) + row * 128 + ((chunk ^ (row & 7)) << 4);
}

/* Shared memory of the end-of-unit pass. */
struct FinSmem {
  float *fin;     // [16]: head max, then 1/Z
  float *pm, *pl; // [MD_MAX_CHUNKS][8] partial maxima and sums
  float *fac;     // [MD_MAX_CHUNKS][8] combine factors
  float *obuf;    // staged partial O slices
  int *sphys;     // [unit pages] physical page ids
  int *sfill;     // [unit pages] tokens per page (region-aligned pages)
  int *okflag;    // the bounded wait's outcome, for every thread
};

template <int NT>
__device__ __forceinline__ void fin_sync() {
  if (NT == 32) __syncwarp();
  else named_barrier(1, NT);
}

/* The unit's physical page ids (and, with region-aligned pages, their fills)
 * into shared memory, loaded in batches. */
template <bool ALIGNED, int NT>
__device__ __forceinline__ void load_page_ids(const AttnParams &p, const Unit &pv, int tid,
                                              const FinSmem &f) {
  const int npg = pv.p1 - pv.p0;
  const int32_t *bt = p.block_table + (size_t)pv.b * p.P_max;
  for (int q0 = 0; q0 < npg; q0 += NT * 4) {
    int ph[4], fl[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int q = q0 + r * NT + tid;
      ph[r] = fl[r] = 0;
      if (q < npg) {
        ph[r] = bt[pv.p0 + q];
        if (ALIGNED) fl[r] = p.page_fill[(size_t)pv.b * p.P_max + pv.p0 + q];
      }
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int q = q0 + r * NT + tid;
      if (q < npg) {
        f.sphys[q] = ph[r];
        if (ALIGNED) f.sfill[q] = fl[r];
      }
    }
  }
}

/* Token masses of a unit from its stored raw scores and the item's per-head
 * (max, 1/Z) in f.fin: mass_i = sum_h exp2(s_hi - max_h) / Z_h, added in
 * fixed point to the token's slot of the step's accumulator (kept in L2
 * with evict_last: every (layer, KV head) adds to the same slots), or
 * written to the (layer, KV head) row at that slot.  Four tokens per thread
 * in flight (a batch's loads are issued before any store). */
template <int PS, bool ALIGNED, int NT, bool ROWS>
__device__ __forceinline__ void mass_pass(const AttnParams &p, const Unit &pv, int slot, int tid,
                                          const FinSmem &f) {
  const int G = p.G;
  const int npg = pv.p1 - pv.p0;
  const float *scr = p.scratch + ((size_t)blockIdx.x * 2 + slot) * p.scratch_tokens * GP;
  const int ntok = npg * PS;
  unsigned long long *acc = p.mass_acc;
  float *mrow = ROWS ? p.mass + (size_t)(pv.l * p.Hkv + pv.kvh) * p.slots : nullptr;
  const uint64_t acc_pol = policy_evict_last();
  float fm[GP], fz[GP];
#pragma unroll
  for (int h = 0; h < GP; ++h) {
    fm[h] = f.fin[h];
    fz[h] = (h < G) ? f.fin[8 + h] : 0.f;
  }
  /* contiguous pages: the valid tokens are a prefix of the unit; with
   * region-aligned pages every page has its own fill */
  const int nvalid = ALIGNED ? ntok : min(ntok, p.n_tokens[pv.b] - pv.p0 * PS);
  constexpr int NB = 4;
  for (int tk0 = 0; tk0 < nvalid; tk0 += NT * NB) {
    float4 s0[NB], s1[NB];
#pragma unroll
    for (int r = 0; r < NB; ++r) {
      const int tk = tk0 + r * NT + tid;
      if (tk < nvalid) {
        s0[r] = __ldcg((const float4 *)(scr + (size_t)tk * GP));
        s1[r] = __ldcg((const float4 *)(scr + (size_t)tk * GP + 4));
      }
    }
#pragma unroll
    for (int r = 0; r < NB; ++r) {
      const int tk = tk0 + r * NT + tid;
      if (tk >= nvalid) continue;
      if (ALIGNED && (tk % PS) >= f.sfill[tk / PS]) continue;
      float m = exp2f(s0[r].x - fm[0]) * fz[0] + exp2f(s0[r].y - fm[1]) * fz[1] +
                exp2f(s0[r].z - fm[2]) * fz[2] + exp2f(s0[r].w - fm[3]) * fz[3];
      m += exp2f(s1[r].x - fm[4]) * fz[4] + exp2f(s1[r].y - fm[5]) * fz[5] +
           exp2f(s1[r].z - fm[6]) * fz[6] + exp2f(s1[r].w - fm[7]) * fz[7];
      const size_t slot_i = (size_t)f.sphys[tk / PS] * PS + (tk % PS);
      if (ROWS)
        mrow[slot_i] = m;
      else
        red_add_u64_hint(acc + slot_i, __float2ull_rn(m * MASS_SCALE), acc_pol);
    }
  }
}

/* The end of a unit: wait (bounded) for all C chunks of its (sequence, layer,
 * KV head) item, combine their partials (m, Z, O) into this chunk's slice of
 * the output O and the item's per-head (max, 1/Z), turn the unit's stored
 * scores into token masses sum_h exp2(s_hi - max_h) / Z_h (Sec. III-C), then
 * count the chunk as finished.  Run by NT threads, tid < NT: the finisher
 * warp, or all consumer warps for a CTA's last unit.  Returns false, the same
 * for every thread, on abort or timeout.  Loads are issued in batches before
 * the dependent stores, so a pass costs a few L2 round trips. */
template <int PS, bool ALIGNED, int NT, int OBUF_FLOATS, bool ROWS>
__device__ __forceinline__ bool finish_unit(const AttnParams &p, const Unit &pv, int slot, int tid,
                                            const FinSmem &f) {
  const float NEG_INF = -INFINITY;
  const int G = p.G;
  const int C = pv.C;
  /* the unit's page ids (no wait needed) */
  load_page_ids<ALIGNED, NT>(p, pv, tid, f);
  /* all chunks of the item published */
  if (tid == 0) {
    int okw = 1;
    const int target = C + p.extra_arrivals;
    if (ld_acquire_gpu(&p.counters[pv.X]) < target) {
      const long long t0 = globaltimer();
      while (ld_acquire_gpu(&p.counters[pv.X]) < target) {
        if (ld_volatile(&p.status[ST_ABORT])) { okw = 0; break; }
        if (globaltimer() - t0 > p.spin_limit_ns) {
          raise_status(p, MD_ERR_DEVICE_TIMEOUT, 3);
          okw = 0;
          break;
        }
        __nanosleep(64);
      }
    }
    *f.okflag = okw;
  }
  fin_sync<NT>();
  if (!*f.okflag) return false;
  const float *base = p.partials + (size_t)pv.X * p.chunk_stride * PARTIAL_FLOATS;
  for (int i0 = 0; i0 < C * GP; i0 += NT * 8) {
    float vm[8], vl[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const int idx = i0 + r * NT + tid;
      vm[r] = vl[r] = 0.f;
      if (idx < C * GP) {
        const float *pj = base + (size_t)(idx >> 3) * PARTIAL_FLOATS;
        vm[r] = __ldcg(pj + (idx & 7));
        vl[r] = __ldcg(pj + 8 + (idx & 7));
      }
    }
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const int idx = i0 + r * NT + tid;
      if (idx < C * GP) {
        f.pm[idx] = vm[r];
        f.pl[idx] = vl[r];
      }
    }
  }
  fin_sync<NT>();
  if (tid < 32) {
    /* per head: global max and normaliser over the C chunks */
    const int h = tid & 7, part = tid >> 3;
    float M = NEG_INF;
    for (int j = part; j < C; j += 4) M = fmaxf(M, f.pm[j * GP + h]);
    M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 8));
    M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 16));
    const float Mr = (M == NEG_INF) ? 0.f : M;
    float Z = 0.f;
    for (int j = part; j < C; j += 4) Z += exp2f(f.pm[j * GP + h] - Mr) * f.pl[j * GP + h];
    Z += __shfl_xor_sync(0xffffffffu, Z, 8);
    Z += __shfl_xor_sync(0xffffffffu, Z, 16);
    if (part == 0) {
      f.fin[h] = Mr;
      f.fin[8 + h] = Z > 0.f ? 1.f / Z : 0.f;
    }
  }
  fin_sync<NT>();
  for (int idx = tid; idx < C * GP; idx += NT)
    f.fac[idx] = exp2f(f.pm[idx] - f.fin[idx & 7]) * f.fin[8 + (idx & 7)];
  /* this chunk's slice [lo, hi) of the item's output O[h][d] (h < G): the C
   * partial slices are staged in shared memory with independent loads (one
   * batch, all in flight), then each thread sums its elements' chunks in
   * chunk order */
  const int E = G * D;
  const int lo = (int)(((long long)pv.j * E) / C);
  const int hi = (int)(((long long)(pv.j + 1) * E) / C);
  const int SE = hi - lo;
  const int n_all = C * SE;   // <= E + C - 1 < OBUF_FLOATS
  {
    constexpr int NBO = (OBUF_FLOATS + NT - 1) / NT;
    float v[NBO];
#pragma unroll
    for (int r = 0; r < NBO; ++r) {
      const int n = r * NT + tid;
      v[r] = 0.f;
      if (n < n_all) {
        const int j = n / SE;
        v[r] = __ldcg(base + (size_t)j * PARTIAL_FLOATS + 16 + lo + (n - j * SE));
      }
    }
#pragma unroll
    for (int r = 0; r < NBO; ++r) {
      const int n = r * NT + tid;
      if (n < n_all) f.obuf[n] = v[r];
    }
  }
  fin_sync<NT>();
  {
    uint16_t *orow = p.out + (((size_t)pv.b * p.q_layers + (pv.l - p.l0)) * p.Hq + (size_t)pv.kvh * G) * D;
    for (int e = lo + tid; e < hi; e += NT) {
      const int h = e >> 7;
      float acc = 0.f;
      for (int j = 0; j < C; ++j) acc += f.fac[j * GP + h] * f.obuf[j * SE + (e - lo)];
      __nv_bfloat16 bv = __float2bfloat16_rn(acc);
      orow[e] = *(uint16_t *)&bv;
    }
  }
  mass_pass<PS, ALIGNED, NT, ROWS>(p, pv, slot, tid, f);
  fin_sync<NT>();
  if (tid == 0) {
    const int old = atomicAdd(&p.counters[pv.X], 1);
    if (old == 2 * C - 1) atomicExch(&p.counters[pv.X], 0);
  }
  return true;
}

/* Merge the NCW consumer warps' running softmax states of a unit (per head:
 * max, sum, O^T) into the chunk's partial (m, Z, O) and publish it: write the
 * partial, then one gpu-scope fence (cumulative over the threads' writes,
 * which the sync orders before thread 0) and the item's arrival count.  Run
 * by NT threads, tid < NT. */
template <int NCW, int NT>
__device__ __forceinline__ void merge_publish(const AttnParams &p, const Unit &un, int tid,
                                              const float *wm, const float *wl, float *wf,
                                              const float *wO) {
  const float NEG_INF = -INFINITY;
  float *part = p.partials + ((size_t)un.X * p.chunk_stride + un.j) * PARTIAL_FLOATS;
  if (tid < GP) {
    float M = NEG_INF;
    for (int w = 0; w < NCW; ++w) M = fmaxf(M, wm[w * 8 + tid]);
    const float Mr = (M == NEG_INF) ? 0.f : M;
    float Lsum = 0.f;
    for (int w = 0; w < NCW; ++w) {
      const float f = exp2f(wm[w * 8 + tid] - Mr);
      wf[w * 8 + tid] = f;
      Lsum += f * wl[w * 8 + tid];
    }
    part[tid] = M;
    part[8 + tid] = Lsum;
  }
  fin_sync<NT>();
  for (int e = tid; e < GP * D; e += NT) {
    const int h = e >> 7;
    float acc = 0.f;
#pragma unroll
    for (int w = 0; w < NCW; ++w) acc += wf[w * 8 + h] * wO[(size_t)w * GP * D + e];
    part[16 + e] = acc;
  }
  fin_sync<NT>();
  if (tid == 0) {
    __threadfence();
    atomicAdd(&p.counters[un.X], 1);
  }
}

/* The end of a unit that is its item's only chunk (C == 1): the merge of
 * the warps' states is already the item's softmax, so there is no partial,
 * no counter and no combine.  Writes the per-head (max, 1/Z) to f.fin and
 * the item's output O, with the same arithmetic (and so the same bits) as
 * merge_publish followed by finish_unit's combine.  Ends with a sync, after
 * which the merge buffers are free. */
template <int NCW, int NT>
__device__ __forceinline__ void merge_single(const AttnParams &p, const Unit &un, int tid,
                                             const float *wm, const float *wl, float *wf,
                                             const float *wO, const FinSmem &f) {
  const float NEG_INF = -INFINITY;
  if (tid < GP) {
    float M = NEG_INF;
    for (int w = 0; w < NCW; ++w) M = fmaxf(M, wm[w * 8 + tid]);
    const float Mr = (M == NEG_INF) ? 0.f : M;
    float Lsum = 0.f;
    for (int w = 0; w < NCW; ++w) {
      const float fw = exp2f(wm[w * 8 + tid] - Mr);
      wf[w * 8 + tid] = fw;
      Lsum += fw * wl[w * 8 + tid];
    }
    f.fin[tid] = Mr;
    f.fin[8 + tid] = Lsum > 0.f ? 1.f / Lsum : 0.f;
  }
  fin_sync<NT>();
  const int E = p.G * D;
  uint16_t *orow = p.out + (((size_t)un.b * p.q_layers + (un.l - p.l0)) * p.Hq + (size_t)un.kvh * p.G) * D;
  for (int e = tid; e < E; e += NT) {
    const int h = e >> 7;
    float acc = 0.f;
#pragma unroll
    for (int w = 0; w < NCW; ++w) acc += wf[w * 8 + h] * wO[(size_t)w * GP * D + e];
    acc = f.fin[8 + h] * acc;
    __nv_bfloat16 bv = __float2bfloat16_rn(acc);
    orow[e] = *(uint16_t *)&bv;
  }
  fin_sync<NT>();
}

/* The whole end of a single-chunk unit: the page ids, the merge straight
 * into (max, 1/Z) and the output, the release of the merge buffers (mdone,
 * when given: the finisher's hand-off), the token masses. */
template <int PS, bool ALIGNED, int NCW, int NT, bool ROWS>
__device__ __forceinline__ void single_end(const AttnParams &p, const Unit &un, int slot, int tid,
                                        const float *wm, const float *wl, float *wf,
                                        const float *wO, const FinSmem &f, uint32_t mdone) {
  load_page_ids<ALIGNED, NT>(p, un, tid, f);
  merge_single<NCW, NT>(p, un, tid, wm, wl, wf, wO, f);
  if (mdone != 0 && tid == 0) mbar_arrive(mdone);   // merge buffers free again
  mass_pass<PS, ALIGNED, NT, ROWS>(p, un, slot, tid, f);
  fin_sync<NT>();
}

/* ALIGNED: pages carry their own fill (region-aligned allocation); otherwise
 * every page but the last is full and the fills follow from n_tokens.  ROWS:
 * the masses go to one fp32 row per (layer, KV head) (the no-allocation entry
 * point) instead of the step's fixed-point accumulator; a compile-time choice,
 * since this end-of-unit code runs once per unit and is often fetched cold. */
template <int PS, int NCW, bool ALIGNED, bool ROWS>
__global__ void __launch_bounds__(AttnShape<PS, NCW>::THREADS, AttnShape<PS, NCW>::CTAS_PER_SM)
    attn_mass_kernel(const __grid_constant__ AttnParams p,
                     const __grid_constant__ CUtensorMap tmap) {
  using S = AttnShape<PS, NCW>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t *ring = smem;
  uint8_t *sQ = ring + S::RING_BYTES;                   // [2][8 heads][128] bf16
  uint64_t *full = (uint64_t *)(sQ + 2 * S::Q_BYTES);
  uint64_t *empty = full + S::R;
  uint64_t *qfull = empty + S::R;                       // [2]
  uint64_t *qempty = qfull + 2;                         // [2]
  uint64_t *cdone = qempty + 2;    // [2] score slot written, unit published
  uint64_t *fdone = cdone + 2;     // [2] score slot read by the finisher
  uint64_t *mdone = fdone + 2;     // [1] merge buffers read by the finisher
  float *wm = (float *)(mdone + 2);           // [NCW][8] per-warp running max
  float *wl = wm + NCW * 8;                   // [NCW][8] per-warp running sum
  float *wf = wl + NCW * 8;                   // [NCW][8] per-warp merge factor
  float *wO = wf + NCW * 8;                   // [NCW][8][128] per-warp O^T
  float *fin = wm + S::MERGE_FLOATS;          // [16]: head max, then 1/Z
  float *pm = fin + 16;                       // [MD_MAX_CHUNKS][8] partial maxima
  float *pl = pm + MD_MAX_CHUNKS * GP;        // [MD_MAX_CHUNKS][8] partial sums
  float *fac = pl + MD_MAX_CHUNKS * GP;       // [MD_MAX_CHUNKS][8] combine factors
  int *sphys = (int *)(fac + MD_MAX_CHUNKS * GP);   // [MAX_UNIT_PAGES] page ids
  int *sfill = sphys + S::MAX_UNIT_PAGES;            // [MAX_UNIT_PAGES] tokens per page
  float *obuf = (float *)(sfill + S::MAX_UNIT_PAGES);   // [OBUF_FLOATS] staged O slices
  int *fillbuf = (int *)(obuf + S::OBUF_FLOATS);         // [R] fill of the page in each stage
  int *flag = fillbuf + S::R;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t ring_u32 = smem_u32(ring);
  const uint32_t sQ_u32 = smem_u32(sQ);
  const int G = p.G;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::R; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&qfull[s]), 1);
      mbar_init(smem_u32(&qempty[s]), NCW);
      mbar_init(smem_u32(&cdone[s]), NCW);   // every consumer warp, once per unit
      mbar_init(smem_u32(&fdone[s]), 1);
    }
    mbar_init(smem_u32(&mdone[0]), 1);
    flag[0] = flag[1] = flag[2] = 0;
    fence_barrier_init();
  }
  __syncthreads();
  /* The kernel ahead in the stream (the step's append) writes the new
   * token's K/V into each sequence's last page, that page's block-table
   * entry and fill, and the new token's state.  Every thread waits for it
   * before its first global access, except the producer's issuing lane,
   * which first starts its first unit's copies that append cannot touch
   * (the query rows and the pages before the sequence's last one). */
  const bool issuer = warp == 0 && lane == 0;
  if (!issuer) {
    pdl_wait();
    pdl_trigger();
  }

  if (warp == 0) {
    /* ------------------------------------------------------- producer ---- */
    /* One thread issues every copy (a single active lane keeps this warp off
     * the issue slots the consumers need); page ids are loaded eight at a
     * time so no copy waits on a dependent load. */
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      tma_prefetch_desc(&tmap);
      /* the i-th page this CTA streams goes to stage i % R, consumed by warp
       * i % NCW: R is a multiple of NCW, so every stage belongs to one warp */
      int i = 0, nu = 0;
      bool ok = true;
      /* The CTA's pages as one stream of batches of up to 8 pages (never
       * across a unit); the page ids (and fills) of the next batch are loaded
       * before the current batch's copies are issued, so their latency hides
       * behind the waits for free stages instead of emptying the ring. */
      int u = blockIdx.x;
      Unit un{};
      int pb = 0, cnt = 0;
      int ph[8], fl[8];
      if (u < p.total_units) {
        un = decode_unit(p, u);
        /* before the wait: the first unit's query rows (the caller's) and,
         * when the unit is its item's only chunk, its pages below the
         * sequence's last one, at most one per stage (measured on a GB300:
         * 3 us off a 24 us step with single-chunk items; with split items the
         * early pages made the launch 2 us longer, so they wait there) */
        mbar_arrive_expect_tx(smem_u32(&qfull[0]), G * D * 2);
        bulk_load(sQ_u32, p.q + (((size_t)un.b * p.q_layers + (un.l - p.l0)) * p.Hq + (size_t)un.kvh * G) * D,
                  G * D * 2, smem_u32(&qfull[0]));
        nu = 1;
        const int early_end = un.C == 1 ? min(min(un.p1, un.p0 + S::R), p.n_pages[un.b] - 1) : un.p0;
        for (pb = un.p0; pb < early_end; pb += 8) {
          cnt = load_batch<ALIGNED>(p, un, pb, early_end, ph, fl);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            if (k >= cnt) break;
            const int s = i;   // i < R: every stage is still empty
            const int row = (((un.l * p.P_phys + ph[k]) * p.Hkv + un.kvh) * 2) * PS;
            const uint32_t st = ring_u32 + s * S::STAGE_BYTES;
            if (ALIGNED) fillbuf[s] = fl[k];
            mbar_arrive_expect_tx(smem_u32(&full[s]), S::STAGE_BYTES);
            tma_load_2d(st, &tmap, 0, row, smem_u32(&full[s]), pol);
            tma_load_2d(st + S::HALF_BYTES, &tmap, 64, row, smem_u32(&full[s]), pol);
            ++i;
          }
        }
        pb = un.p0 + i;
      }
      pdl_wait();
      pdl_trigger();
      if (u < p.total_units) cnt = pb < un.p1 ? load_batch<ALIGNED>(p, un, pb, un.p1, ph, fl) : 0;
      while (u < p.total_units && ok) {
        Unit nx = un;
        int npb = pb + 8, nxu = u, cntn = 0;
        int phn[8] = {0, 0, 0, 0, 0, 0, 0, 0}, fln[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        if (npb >= un.p1) {
          nxu = u + gridDim.x;
          if (nxu < p.total_units) {
            nx = decode_unit(p, nxu);
            npb = nx.p0;
          }
        }
        if (nxu < p.total_units) cntn = load_batch<ALIGNED>(p, nx, npb, nx.p1, phn, fln);
        if (pb == un.p0 && u != (int)blockIdx.x) {   // the first unit's rows went out before the wait
          /* the unit's G query rows: one bulk copy into a double-buffered slot */
          const int qs = nu & 1;
          if (nu >= 2) {
            if (!wait_phase(smem_u32(&qempty[qs]), ((nu >> 1) - 1) & 1, p, 5, true)) {
              ok = false;
              break;
            }
            /* the consumers read the slot through the generic proxy; the bulk
             * copy writes it through the async proxy */
            fence_proxy_async_smem();
          }
          mbar_arrive_expect_tx(smem_u32(&qfull[qs]), G * D * 2);
          bulk_load(sQ_u32 + qs * S::Q_BYTES,
                    p.q + (((size_t)un.b * p.q_layers + (un.l - p.l0)) * p.Hq + (size_t)un.kvh * G) * D,
                    G * D * 2, smem_u32(&qfull[qs]));
          ++nu;
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (k >= cnt) break;
          const int s = i % S::R;
          if (i >= S::R) {
            if (!wait_phase(smem_u32(&empty[s]), ((i / S::R) - 1) & 1, p, 1, true)) {
              ok = false;
              break;
            }
            /* the stage's last reads (ldmatrix, generic proxy) must be
             * ordered before the TMA refill (async proxy): without this
             * fence a refill can overwrite V rows still being read */
            fence_proxy_async_smem();
          }
          const int row = (((un.l * p.P_phys + ph[k]) * p.Hkv + un.kvh) * 2) * PS;
          const uint32_t st = ring_u32 + s * S::STAGE_BYTES;
          if (ALIGNED) fillbuf[s] = fl[k];   // published by the arrive below
          mbar_arrive_expect_tx(smem_u32(&full[s]), S::STAGE_BYTES);
          tma_load_2d(st, &tmap, 0, row, smem_u32(&full[s]), pol);
          tma_load_2d(st + S::HALF_BYTES, &tmap, 64, row, smem_u32(&full[s]), pol);
          ++i;
        }
        un = nx;
        pb = npb;
        u = nxu;
        cnt = cntn;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          ph[k] = phn[k];
          fl[k] = fln[k];
        }
      }
      /* No copy may still be writing this CTA's shared memory when it exits:
       * wait for the last copy issued into every stage. */
      for (int k = (i > S::R ? i - S::R : 0); k < i; ++k)
        wait_phase(smem_u32(&full[k % S::R]), (k / S::R) & 1, p, 2, false);
      for (int k = (nu > 2 ? nu - 2 : 0); k < nu; ++k)
        wait_phase(smem_u32(&qfull[k & 1]), (k >> 1) & 1, p, 6, false);
    }
    return;
  }

  const FinSmem fs{fin, pm, pl, fac, obuf, sphys, sfill, &flag[2]};

  if (warp == NCW + 1) {
    /* ------------------------------------------------------- finisher ---- */
    /* The end of every unit but the CTA's last, one warp, while the
     * consumers stream the next unit: merge the warps' states and publish
     * the chunk's partial, release the merge buffers, finish the unit, then
     * release its score slot. */
    int k = 0;
    for (int u = blockIdx.x; u < p.total_units; u += gridDim.x, ++k) {
      if (u + (int)gridDim.x >= p.total_units) break;   // the consumers finish the last unit
      const Unit pv = decode_unit(p, u);
      const bool ok = wait_phase(smem_u32(&cdone[k & 1]), (k >> 1) & 1, p, 8, true);
      if (!__all_sync(0xffffffffu, ok)) break;
      if (pv.C == 1) {
        single_end<PS, ALIGNED, NCW, 32, ROWS>(p, pv, k & 1, lane, wm, wl, wf, wO, fs, smem_u32(&mdone[0]));
      } else {
        merge_publish<NCW, 32>(p, pv, lane, wm, wl, wf, wO);
        if (lane == 0) mbar_arrive(smem_u32(&mdone[0]));   // merge buffers free again
        if (!finish_unit<PS, ALIGNED, 32, S::OBUF_FLOATS, ROWS>(p, pv, k & 1, lane, fs)) break;
      }
      if (lane == 0) mbar_arrive(smem_u32(&fdone[k & 1]));   // slot and finish area free
    }
    return;
  }

  /* ------------------------------------------------------- consumers ----- */
  const int cw = warp - 1;
  const int ct = threadIdx.x - 32;
  const int NC = NCW * 32;
  const int g = lane >> 2, t = lane & 3;
  const bool hv0 = (2 * t) < G, hv1 = (2 * t + 1) < G;
  const uint64_t pol_keep = policy_evict_last();
  const float NEG_INF = -INFINITY;

  int i_base = 0, nunit = 0;   // pages streamed before this unit; units done
  bool aborted = false;        // this warp gave up a wait
  for (int u = blockIdx.x; u < p.total_units; u += gridDim.x) {
    const Unit un = decode_unit(p, u);
    const int npg = un.p1 - un.p0;
    const int slot = nunit & 1;
    float *scr = p.scratch + ((size_t)blockIdx.x * 2 + slot) * p.scratch_tokens * GP;

    /* Q^T fragments (B operand) from the prefetched rows: head g, dims
     * 16kk + {2t, 2t+1} and 16kk + 8 + {2t, 2t+1}; padded heads are zero. */
    uint32_t qf[8][2];
    {
      const int qs = nunit & 1;
      if (!wait_phase(smem_u32(&qfull[qs]), (nunit >> 1) & 1, p, 7, true)) aborted = true;
      const int mi = lane >> 3, rr = lane & 7;
      const uint32_t qb = sQ_u32 + qs * S::Q_BYTES + rr * (D * 2) + mi * 16;
#pragma unroll
      for (int kk = 0; kk < 8; kk += 2) {
        uint32_t r0, r1, r2, r3;
        ldmatrix_x4(qb + kk * 32, r0, r1, r2, r3);
        const bool gv = g < G;
        qf[kk][0] = gv ? r0 : 0u;
        qf[kk][1] = gv ? r1 : 0u;
        qf[kk + 1][0] = gv ? r2 : 0u;
        qf[kk + 1][1] = gv ? r3 : 0u;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&qempty[qs]));
    }
    /* the score slot is free once the finisher is done with the unit that
     * used it two units ago */
    if (nunit >= 2 && !aborted &&
        !wait_phase(smem_u32(&fdone[slot]), ((nunit >> 1) - 1) & 1, p, 9, true))
      aborted = true;
    aborted = __any_sync(0xffffffffu, aborted);   // one decision per warp
    float m0 = NEG_INF, m1 = NEG_INF, l0 = 0.f, l1 = 0.f;
    float o[8][4];
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    const int ntok_seq = p.n_tokens[un.b];
    const int mi = lane >> 3, rr = lane & 7;

    /* this warp's pages are those whose CTA-wide index gi = i_base + jp is
     * cw modulo NCW: they land only in this warp's own stages (gi % R), so a
     * wait is never more than one phase ahead of the copies however far the
     * warps drift apart, and a unit's extra pages rotate over the warps */
    const int j0 = ((cw - i_base) % NCW + NCW) % NCW;
    for (int jp = j0; jp < npg && !aborted; jp += NCW) {
      const int gi = i_base + jp;
      const int s = gi % S::R;
      if (!wait_phase(smem_u32(&full[s]), (gi / S::R) & 1, p, 4, true)) {
        aborted = true;
        break;
      }
      const uint32_t st = ring_u32 + s * S::STAGE_BYTES;
      const int fill = ALIGNED ? fillbuf[s] : ntok_seq - (un.p0 + jp) * PS;

      float acc[S::NT][4];
#pragma unroll
      for (int tt = 0; tt < S::NT; ++tt) acc[tt][0] = acc[tt][1] = acc[tt][2] = acc[tt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
#pragma unroll
        for (int tt = 0; tt < S::NT; ++tt) {
          uint32_t a0, a1, a2, a3;
          ldmatrix_x4(swz<PS>(st, tt * 16 + (mi & 1) * 8 + rr, kk * 16 + (mi >> 1) * 8), a0, a1,
                      a2, a3);
          mma_bf16(acc[tt], a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
        }
      }
      /* scale to the exp2 domain, mask padded heads / unwritten tail slots,
       * keep the raw scores for the mass pass */
      float mx0 = NEG_INF, mx1 = NEG_INF;
#pragma unroll
      for (int tt = 0; tt < S::NT; ++tt) {
        const int ta = tt * 16 + g, tb = ta + 8;
        const bool va = ta < fill, vb = tb < fill;
        acc[tt][0] = (va && hv0) ? acc[tt][0] * p.scale_log2 : NEG_INF;
        acc[tt][1] = (va && hv1) ? acc[tt][1] * p.scale_log2 : NEG_INF;
        acc[tt][2] = (vb && hv0) ? acc[tt][2] * p.scale_log2 : NEG_INF;
        acc[tt][3] = (vb && hv1) ? acc[tt][3] * p.scale_log2 : NEG_INF;
        st_v2_hint(scr + (size_t)(jp * PS + ta) * GP + 2 * t, acc[tt][0], acc[tt][1], pol_keep);
        st_v2_hint(scr + (size_t)(jp * PS + tb) * GP + 2 * t, acc[tt][2], acc[tt][3], pol_keep);
        mx0 = fmaxf(mx0, fmaxf(acc[tt][0], acc[tt][2]));
        mx1 = fmaxf(mx1, fmaxf(acc[tt][1], acc[tt][3]));
      }
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
      }
      const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);
      const float r0 = (n0 == NEG_INF) ? 0.f : n0, r1 = (n1 == NEG_INF) ? 0.f : n1;
      const float al0 = exp2f(m0 - r0), al1 = exp2f(m1 - r1);
      m0 = n0;
      m1 = n1;
      l0 *= al0;
      l1 *= al1;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        o[mt][0] *= al0;
        o[mt][1] *= al1;
        o[mt][2] *= al0;
        o[mt][3] *= al1;
      }
#pragma unroll
      for (int tt = 0; tt < S::NT; ++tt) {
        const float p00 = exp2f(acc[tt][0] - r0), p01 = exp2f(acc[tt][1] - r1);
        const float p10 = exp2f(acc[tt][2] - r0), p11 = exp2f(acc[tt][3] - r1);
        l0 += p00 + p10;
        l1 += p01 + p11;
        const uint32_t b0 = movmatrix_trans(pack_bf16(p00, p01));
        const uint32_t b1 = movmatrix_trans(pack_bf16(p10, p11));
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          uint32_t a0, a1, a2, a3;
          ldmatrix_x4_trans(swz<PS>(st, PS + tt * 16 + (mi >> 1) * 8 + rr, mt * 16 + (mi & 1) * 8),
                            a0, a1, a2, a3);
          mma_bf16(o[mt], a0, a1, a2, a3, b0, b1);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[s]));
    }

    /* ---- the unit's end: this warp's softmax state goes to the merge ---- */
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, off);
      l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    aborted = __any_sync(0xffffffffu, aborted);
    const bool last = u + (int)gridDim.x >= p.total_units;
    /* the merge buffers hold the previous unit's states until the finisher
     * has read them; on the CTA's last unit the finisher must be done with
     * everything (its finish area is used below) */
    if (!aborted && nunit >= 1) {
      const bool okw = last ? wait_phase(smem_u32(&fdone[(nunit - 1) & 1]), ((nunit - 1) >> 1) & 1, p, 9, true)
                            : wait_phase(smem_u32(&mdone[0]), (nunit - 1) & 1, p, 10, true);
      if (!okw) aborted = true;
      aborted = __any_sync(0xffffffffu, aborted);
    }
    if (!aborted) {
      if (g == 0) {
        wm[cw * 8 + 2 * t] = m0;
        wm[cw * 8 + 2 * t + 1] = m1;
        wl[cw * 8 + 2 * t] = l0;
        wl[cw * 8 + 2 * t + 1] = l1;
      }
      float *wo = wO + (size_t)cw * GP * D;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        wo[(2 * t) * D + 16 * mt + g] = o[mt][0];
        wo[(2 * t + 1) * D + 16 * mt + g] = o[mt][1];
        wo[(2 * t) * D + 16 * mt + g + 8] = o[mt][2];
        wo[(2 * t + 1) * D + 16 * mt + g + 8] = o[mt][3];
      }
    }
    if (!last) {
      /* hand the unit to the finisher and go on at once; a warp that gave
       * up a wait runs on without waiting to the last unit's barrier */
      __syncwarp();
      if (!aborted && lane == 0) mbar_arrive(smem_u32(&cdone[slot]));
      i_base += npg;
      ++nunit;
      continue;
    }
    /* the CTA's last unit: nothing is left to overlap with, so all consumer
     * warps merge, publish and finish it */
    if (aborted) flag[0] = 1;
    named_barrier(1, NC);
    if (flag[0]) break;
    if (un.C == 1) {
      single_end<PS, ALIGNED, NCW, NCW * 32, ROWS>(p, un, slot, ct, wm, wl, wf, wO, fs, 0u);
      break;
    }
    merge_publish<NCW, NCW * 32>(p, un, ct, wm, wl, wf, wO);
    if (ct == 0) flag[1] = ld_volatile(&p.status[ST_ABORT]);
    named_barrier(1, NC);
    if (flag[1]) break;
    finish_unit<PS, ALIGNED, NCW * 32, S::OBUF_FLOATS, ROWS>(p, un, slot, ct, fs);
    break;
  }
}

template <int PS, int NCW, bool AL, bool ROWS>
static cudaError_t prepare_impl() {
  return cudaFuncSetAttribute(attn_mass_kernel<PS, NCW, AL, ROWS>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)AttnShape<PS, NCW>::SMEM);
}

/* The instances of one page size: the step's (contiguous or region-aligned
 * pages) and the no-allocation entry point's (contiguous pages, mass rows). */
template <int PS, int NCW>
static cudaError_t prepare_all() {
  cudaError_t e = prepare_impl<PS, NCW, false, false>();
  if (e == cudaSuccess) e = prepare_impl<PS, NCW, true, false>();
  if (e == cudaSuccess) e = prepare_impl<PS, NCW, false, true>();
  return e;
}

template <int PS, int NCW>
static int grid_limit_impl() {
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (prepare_all<PS, NCW>() != cudaSuccess) return 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attn_mass_kernel<PS, NCW, false, false>,
                                                    AttnShape<PS, NCW>::THREADS,
                                                    AttnShape<PS, NCW>::SMEM) != cudaSuccess)
    return 0;
  int g = sms * per_sm;
  return g > MAX_GRID ? MAX_GRID : g;
}

template <int PS, int NCW, bool AL, bool ROWS>
static cudaError_t launch_impl(const AttnParams &p, const CUtensorMap &tmap, int grid,
                               cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(AttnShape<PS, NCW>::THREADS);
  cfg.dynamicSmemBytes = AttnShape<PS, NCW>::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, attn_mass_kernel<PS, NCW, AL, ROWS>, p, tmap);
}

constexpr int NCW_DEFAULT = 4;

cudaError_t attention_prepare(int ps) {
  return ps == 16 ? prepare_all<16, NCW_DEFAULT>() : prepare_all<32, NCW_DEFAULT>();
}

int attention_grid_limit(int ps) {
  return ps == 16 ? grid_limit_impl<16, NCW_DEFAULT>() : grid_limit_impl<32, NCW_DEFAULT>();
}

cudaError_t launch_attention(const AttnParams &p, const CUtensorMap &tmap, int grid,
                             cudaStream_t s) {
  if (p.total_units == 0) return cudaSuccess;
  if (!p.mass_acc) {   // mass rows: the no-allocation entry point, contiguous pages
    if (p.page_fill) return cudaErrorInvalidValue;
    return p.ps == 16 ? launch_impl<16, NCW_DEFAULT, false, true>(p, tmap, grid, s)
                      : launch_impl<32, NCW_DEFAULT, false, true>(p, tmap, grid, s);
  }
  if (p.page_fill)
    return p.ps == 16 ? launch_impl<16, NCW_DEFAULT, true, false>(p, tmap, grid, s)
                      : launch_impl<32, NCW_DEFAULT, true, false>(p, tmap, grid, s);
  return p.ps == 16 ? launch_impl<16, NCW_DEFAULT, false, false>(p, tmap, grid, s)
                    : launch_impl<32, NCW_DEFAULT, false, false>(p, tmap, grid, s);
}

}  // namespace md

/* ------------------------------------------------------------------------ */
/* Stage 1 without any device allocation.                                   */
/*                                                                          */
/* The attention kernel above needs scratch memory besides its inputs and   */
/* outputs: per-CTA rows of raw scores, the split partials (m, Z, O) of     */
/* every (sequence, layer, KV head) item and one arrival counter per item.  */
/* md_decode_step finds them in the caller's workspace.  This variant finds */
/* them in the fixed array below instead, for callers that cannot allocate  */
/* device memory at all (see md_attend_mass_noalloc in memdecay.h).         */
/* ------------------------------------------------------------------------ */

namespace md {

constexpr size_t NOALLOC_BYTES = (size_t)24 << 20;     // 24 MiB, every device that loads us
constexpr int NOALLOC_TOKENS = 1024;                   // tokens per chunk at most
constexpr size_t NOALLOC_STATUS_BYTES = 256;

static __device__ __align__(256) uint8_t g_noalloc_scratch[NOALLOC_BYTES];

}  // namespace md

#include <math.h>
#include <string.h>

#include <mutex>

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

/* What a call needs from its device, found by the first call on that device
 * (with the device current) and kept for the process: the device address of
 * g_noalloc_scratch and the attention CTAs resident at once, for pages of 16
 * and of 32 tokens (the latter also sets the kernel's shared-memory limit). */
struct NoallocDevice {
  void *base = nullptr;
  int grid_limit[2] = {0, 0};
};
constexpr int NOALLOC_MAX_DEVICES = 128;
std::mutex g_noalloc_mu;
NoallocDevice g_noalloc_dev[NOALLOC_MAX_DEVICES];
EncodeTiledFn g_encode = nullptr;

cudaError_t noalloc_device(int ps, void **base, int *grid_limit, EncodeTiledFn *encode) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= NOALLOC_MAX_DEVICES) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  NoallocDevice &d = g_noalloc_dev[dev];
  if (!d.base) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, md::g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    d.base = p;
  }
  int &gl = d.grid_limit[ps == 32 ? 1 : 0];
  if (gl <= 0) {
    gl = md::attention_grid_limit(ps);
    if (gl <= 0) return cudaErrorUnknown;
  }
  if (!g_encode) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorUnknown;
    g_encode = (EncodeTiledFn)fn;
  }
  *base = d.base;
  *grid_limit = gl;
  *encode = g_encode;
  return cudaSuccess;
}

/* One candidate split of every (sequence, layer, KV head) item into C chunks
 * and the bytes of the fixed array it occupies: status words, one arrival
 * counter per item, two score rows of the chunk's tokens per CTA of the grid
 * that will be launched, and (only when some item has several chunks) C
 * partials per item. */
struct NoallocPlan {
  int C, T, grid, scratch_tokens;
  long long units;
  size_t counters_bytes, scores_bytes, partial_bytes;
};

NoallocPlan noalloc_plan(int C, int Pmax, int ps, const int *n_pages, int batch, long long items_per_seq,
                         int grid_limit) {
  NoallocPlan pl;
  pl.C = C;
  pl.T = (Pmax + C - 1) / C;
  pl.scratch_tokens = (pl.T * ps + 15) / 16 * 16;
  pl.units = 0;
  bool multi = false;
  for (int b = 0; b < batch; ++b) {
    int ch = (n_pages[b] + pl.T - 1) / pl.T;
    if (ch > C) ch = C;
    if (ch > n_pages[b]) ch = n_pages[b];
    multi |= ch > 1;
    pl.units += items_per_seq * ch;
  }
  pl.grid = (int)(pl.units < grid_limit ? pl.units : grid_limit);
  if (pl.grid < 1) pl.grid = 1;
  const long long items = items_per_seq * batch;
  pl.counters_bytes = (size_t)((items * 4 + 255) / 256 * 256);
  pl.scores_bytes = (size_t)pl.grid * 2 * pl.scratch_tokens * md::GP * 4;
  pl.partial_bytes = multi ? (size_t)items * C * md::PARTIAL_FLOATS * 4 : 0;
  return pl;
}

bool noalloc_fits(const NoallocPlan &pl) {
  return md::NOALLOC_STATUS_BYTES + pl.counters_bytes + pl.scores_bytes + pl.partial_bytes <=
         md::NOALLOC_BYTES;
}

}  // namespace

extern "C" __attribute__((visibility("default"))) md_status md_attend_mass_noalloc(
    const void *kv_pool_dev, const int32_t *block_table_dev, const int32_t *n_tokens_host,
    const void *q_dev, void *out_dev, float *mass_dev, int batch, int num_layers,
    int num_q_heads, int num_kv_heads, int page_size, int max_pages_per_seq, int num_phys_pages,
    void *stream) {
  using namespace md;
  if (!kv_pool_dev || !block_table_dev || !n_tokens_host || !q_dev || !out_dev || !mass_dev)
    return MD_ERR_INVALID_ARG;
  if (batch < 1 || batch > MD_MAX_BATCH || num_layers < 1 || num_layers > 255 ||
      num_kv_heads < 1 || num_q_heads < num_kv_heads || num_q_heads % num_kv_heads ||
      num_q_heads / num_kv_heads > MD_MAX_GROUP || (page_size != 16 && page_size != 32) ||
      max_pages_per_seq < 1 || num_phys_pages < 1)
    return MD_ERR_INVALID_ARG;
  if ((uintptr_t)kv_pool_dev & 15) return MD_ERR_INVALID_ARG;
  const long long rows = (long long)num_layers * num_phys_pages * num_kv_heads * 2 * page_size;
  if (rows >= (1LL << 31)) return MD_ERR_INVALID_ARG;
  const int ps = page_size;
  for (int b = 0; b < batch; ++b)
    if (n_tokens_host[b] < 1 || (long long)n_tokens_host[b] > (long long)max_pages_per_seq * ps)
      return MD_ERR_INVALID_ARG;

  void *base = nullptr;
  int grid_limit = 0;
  EncodeTiledFn encode = nullptr;
  if (noalloc_device(ps, &base, &grid_limit, &encode) != cudaSuccess) return MD_ERR_CUDA;

  AttnParams ap;
  memset(&ap, 0, sizeof(ap));
  int Pmax = 1;
  for (int b = 0; b < batch; ++b) {
    const int P = (n_tokens_host[b] + ps - 1) / ps;
    ap.n_pages[b] = P;
    ap.n_tokens[b] = n_tokens_host[b];
    if (P > Pmax) Pmax = P;
  }
  /* the split: chunks of at most NOALLOC_TOKENS tokens and at most
   * MD_MAX_CHUNKS per item, as few as fill the grid, among those that fit
   * the fixed array (the most that fit if none fills it).  Every chunk of an
   * item must fit in one round of the grid (a finisher waits only for chunks
   * placed before its own next unit), so C may not exceed the grid. */
  const long long items_per_seq = (long long)num_layers * num_kv_heads;
  const int cap_pages = NOALLOC_TOKENS / ps;
  const int need = (Pmax + cap_pages - 1) / cap_pages;
  const int cmax = Pmax < MD_MAX_CHUNKS ? Pmax : MD_MAX_CHUNKS;
  NoallocPlan best;
  best.C = 0;
  for (int C = need; C <= cmax; ++C) {
    const NoallocPlan pl = noalloc_plan(C, Pmax, ps, ap.n_pages, batch, items_per_seq, grid_limit);
    if (C > pl.grid || !noalloc_fits(pl)) continue;
    best = pl;
    if (pl.units >= grid_limit) break;
  }
  if (best.C == 0) return MD_ERR_CAPACITY;
  long long U = 0;
  for (int b = 0; b < batch; ++b) {
    int ch = (ap.n_pages[b] + best.T - 1) / best.T;
    if (ch > best.C) ch = best.C;
    if (ch > ap.n_pages[b]) ch = ap.n_pages[b];
    ap.chunks[b] = ch;
    ap.unit_start[b] = (int)U;
    U += items_per_seq * ch;
  }
  ap.unit_start[batch] = (int)U;
  ap.total_units = (int)U;
  ap.n_seqs = batch;
  ap.units_per_seq = (int)(U / batch);
  for (int b = 0; b < batch && ap.units_per_seq > 0; ++b)
    if (ap.unit_start[b + 1] - ap.unit_start[b] != ap.units_per_seq) ap.units_per_seq = 0;

  uint8_t *s8 = (uint8_t *)base;
  ap.status = (int *)s8;
  ap.counters = (int *)(s8 + NOALLOC_STATUS_BYTES);
  ap.scratch = (float *)(s8 + NOALLOC_STATUS_BYTES + best.counters_bytes);
  ap.partials = (float *)(s8 + NOALLOC_STATUS_BYTES + best.counters_bytes + best.scores_bytes);
  ap.q = (const uint16_t *)q_dev;
  ap.out = (uint16_t *)out_dev;
  ap.block_table = block_table_dev;
  ap.mass = mass_dev;
  ap.L = num_layers;
  ap.l0 = 0;
  ap.L_launch = num_layers;
  ap.q_layers = num_layers;
  ap.Hq = num_q_heads;
  ap.Hkv = num_kv_heads;
  ap.G = num_q_heads / num_kv_heads;
  ap.ps = ps;
  ap.P_phys = num_phys_pages;
  ap.P_max = max_pages_per_seq;
  ap.slots = (long long)num_phys_pages * ps;
  ap.scratch_tokens = best.scratch_tokens;
  ap.chunk_stride = best.C;
  ap.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  ap.spin_limit_ns = 2000000000LL;
  ap.extra_arrivals = 0;

  CUtensorMap tmap;
  cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)(2 * ps)};
  cuuint32_t estr[2] = {1, 1};
  if (encode(&tmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void *)kv_pool_dev, dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return MD_ERR_INVALID_ARG;

  /* the array keeps the previous call's contents: counters and status words
   * must start at zero */
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaMemsetAsync(s8, 0, NOALLOC_STATUS_BYTES + best.counters_bytes, st);
  if (e != cudaSuccess) return MD_ERR_CUDA;
  e = launch_attention(ap, tmap, best.grid, st);
  return e == cudaSuccess ? MD_OK : MD_ERR_CUDA;
}
