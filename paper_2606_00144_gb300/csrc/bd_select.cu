// KV-budget selection (Sec. 3.4 TopKChunks; Algorithm 2, sparsify) in two kernels (three
// in self mode, where window_lse_kernel first computes the window rows' normalisers, see
// its own comment below):
//
// score_kernel  (tcgen05)  score[k] = sum_{h in group, w < W, k <= p_w} exp2(s_{h,w,k} log2e/sqrt(d)
//               - lse_{h,w} log2e) for every middle key k.  Keys sit on the M side of the
//               UMMA (128 keys per tile = the 128 TMEM lanes) and the group's window query
//               rows on N, so every epilogue thread owns one key and reduces its own TMEM
//               row: no cross-thread reduction.  Persistent CTAs (one per SM):
//                 warp 0   producer: K tiles by TMA (128-byte swizzle, 4-stage ring) and the
//                          unit's window queries into a double-buffered swizzled Q tile;
//                          the first stages' K tiles (context rows) stream before the
//                          grid-dependency wait, the queries (which bd_advance may have
//                          just rewritten) and the later tiles after it;
//                 warp 1   one lane issues tcgen05.mma into four fp32 TMEM accumulators
//                          (two when the window rows need more columns) and commits to
//                          the smem/TMEM barriers;
//                 warps 2-17 epilogue (four groups of 4, every fourth tile): tcgen05.ld,
//                          packed f32x2 FMA, ex2 (MUFU), packed row sums, coalesced store.
// top-B         one CTA per (sequence, KV head): a linear histogram between the min and
//               max score finds the bin holding the k-th largest; that bin's few items are
//               ranked exactly by (score desc, position asc) (4-pass radix select on the
//               fp32 bits when the bin is crowded); then an ascending compaction (warp
//               ballots + block scan) with sinks and recents.  Four kernels of that
//               method: topk_rows_kernel (token level, up to 16K middle positions, every
//               score in registers), topk_rows_chunk_kernel (chunk level, up to 16K chunks,
//               every chunk score in registers), topk_token_kernel (token level, up to 32K,
//               scores in shared memory) and topk_kernel (longer middles of either level).
#include <algorithm>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

constexpr int kSKeys = 128;          // keys per tile (UMMA M)
constexpr int kSThreads = 576;       // producer, MMA, 4 x 4 epilogue warps
constexpr int kMaxAcc = 4;           // TMEM accumulators (<= 512 columns)
constexpr int kSQOffset = 12288;     // shared-memory offset of the window-query tiles
constexpr int kTopkThreads = 1024;
constexpr int kTopkSmemBytes = 200 * 1024;   // item values staged in shared memory up to this size
constexpr int kBins = 4096;                   // linear histogram bins of the value range
constexpr int kBinCandMax = 2048;             // items of the boundary bin ranked exactly

struct ScoreParams {
  const __nv_bfloat16* q_win;   // [units * nq_rows][D]
  const float* lse_win;         // [units * nq_rows] natural log
  float* score;                 // [units][n_mid_pad]
  int* status;
  int nq_rows, nq_pad, window, t_ctx, n_sink, mid_end, n_mid_pad;
  int tiles_per_unit, total_tiles, tiles_per_cta;
  int acc_stride;               // TMEM columns between accumulators
  int n_acc;                    // accumulators: tile i uses i % n_acc; epilogue group i % 4
  uint32_t tmem_cols;
  float scale_log2;
  const int32_t* seq_lens;      // per-sequence context lengths [batch] or null (all t_ctx)
  int h_kv;
  int window_ready;             // BD_SELECT_WINDOW_READY: the queries may load before the dependency wait
};

// RAGGED: per-sequence lengths (the tile layout is built on the device); a separate
// instance, since the uniform kernel measured 6 us slower with the ragged branches inlined.
template <int D, int STAGES, int NQB, bool RAGGED>
__global__ void __launch_bounds__(kSThreads, 1) score_kernel(const ScoreParams p,
                                                             const __grid_constant__ CUtensorMap kmap,
                                                             const __grid_constant__ CUtensorMap qmap) {
  constexpr uint32_t KHALF = kSKeys * 128;         // one 64-column half of a K tile
  constexpr uint32_t KTILE = kSKeys * D * 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty_bar = full_bar + STAGES;
  uint64_t* tfull_bar = empty_bar + STAGES;        // [kMaxAcc]
  uint64_t* tempty_bar = tfull_bar + kMaxAcc;      // [kMaxAcc]
  uint64_t* qfull_bar = tempty_bar + kMaxAcc;
  uint64_t* qempty_bar = qfull_bar + 2;
  uint64_t* drain_bar = qempty_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t qbytes = (uint32_t)p.nq_pad * D * 2;
  uint8_t* qbuf = smem + kSQOffset;                            // NQB x qbytes
  uint8_t* kstage = qbuf + NQB * qbytes;                       // STAGES x KTILE (1024-aligned)

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_acc = p.n_acc;
  const int n_units = p.total_tiles / p.tiles_per_unit;
  // per-sequence lengths: every CTA lays out the units' middle tiles itself (prefix table
  // after the K stages; the lengths may come from the preceding kernel, so after the
  // dependency wait) and cuts the tile list over the actual tiles
  int* spref = reinterpret_cast<int*>(kstage + STAGES * KTILE);   // [units + 1]
  int total = p.total_tiles, tpc = p.tiles_per_cta;
  if (RAGGED) {
    // with BD_SELECT_WINDOW_READY the lengths were settled before the kernel just before
    // this one too, so the layout (and the streaming) need not wait for it
    if (!p.window_ready) grid_dependency_wait();
    int* wtot = reinterpret_cast<int*>(smem + 1024);
    const int per = (n_units + kSThreads - 1) / kSThreads;
    const int u0 = min(n_units, tid * per), u1 = min(n_units, u0 + per);
    const int tail = p.t_ctx - p.mid_end;            // recent positions
    auto tiles_of = [&](int u) {
      const int t_u = unit_context(p.seq_lens, u, p.h_kv, p.t_ctx, nullptr);
      return (max(0, t_u - tail - p.n_sink) + kSKeys - 1) / kSKeys;
    };
    int sum = 0;
    for (int u = u0; u < u1; ++u) sum += tiles_of(u);
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) wtot[warp] = incl;
    __syncthreads();
    int run = incl - sum;
    for (int w = 0; w < warp; ++w) run += wtot[w];
    for (int u = u0; u < u1; ++u) {
      spref[u] = run;
      run += tiles_of(u);
    }
    if (tid == kSThreads - 1) spref[n_units] = run;
    __syncthreads();
    total = spref[n_units];
    tpc = (total + (int)gridDim.x - 1) / (int)gridDim.x;
  }
  const int first = blockIdx.x * tpc;
  const int n = max(0, min(tpc, total - first));
  // (unit, tile within the unit's middle) of tile g of the list
  auto locate = [&](int g, int& unit, int& tt) {
    if (!RAGGED) {
      unit = g / p.tiles_per_unit;
      tt = g - unit * p.tiles_per_unit;
      return;
    }
    int lo = 0, hi = n_units - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (spref[mid] <= g) lo = mid;
      else hi = mid - 1;
    }
    unit = lo;
    tt = g - spref[lo];
  };
  auto last_of_unit = [&](int g, int unit) {
    return RAGGED ? g + 1 == spref[unit + 1] : (g + 1) % p.tiles_per_unit == 0;
  };

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int a = 0; a < kMaxAcc; ++a) {
      mbar_init(&tfull_bar[a], 1);
      mbar_init(&tempty_bar[a], 4);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&qfull_bar[i], 1);
      mbar_init(&qempty_bar[i], 1);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    allow_dependent_launch();
    if (lane == 0) {
      tma_prefetch_map(&kmap);
      tma_prefetch_map(&qmap);
    }
    // K tile i into its ring stage (lane 0; false once a wait gave up)
    int k_issued = 0;
    auto issue_k = [&](int i) -> bool {
      bool ok = true;
      if (lane == 0) {
        int unit, tt;
        locate(first + i, unit, tt);
        const int s = i % STAGES;
        if (i >= STAGES) ok = mbar_wait(&empty_bar[s], ((i / STAGES) & 1) ^ 1, p.status, abort_flag);
        if (ok) {
          uint8_t* st = kstage + s * KTILE;
          mbar_arrive_expect_tx(&full_bar[s], KTILE);
          const int key0 = p.n_sink + kSKeys * tt;
#pragma unroll
          for (int h = 0; h < D / 64; ++h) tma_load_3d(st + h * KHALF, &kmap, &full_bar[s], 64 * h, key0, unit);
          k_issued = i + 1;
        }
      }
      return __shfl_sync(0xffffffffu, ok, 0);
    };
    // the first stages' K tiles (context rows, which the kernel just before never writes)
    // stream before the grid-dependency wait; the window queries may come from that kernel
    // (bd_advance rewrites them in place), so they load after it, unless the caller says
    // they were written earlier (then queries and tiles interleave from the start)
    const int pre = p.window_ready ? 0 : min(n, STAGES);
    for (int i = 0; i < pre; ++i) issue_k(i);
    if (!p.window_ready) {
      if (n > 0) {   // the first unit's queries on their way into L2 meanwhile
        int u0, t0;
        locate(first, u0, t0);
        prefetch_lines_l2(p.q_win + (size_t)u0 * p.nq_rows * D, (size_t)p.nq_rows * D * 2, lane, 32);
      }
      grid_dependency_wait();
    }
    int cur_unit = -1, qcount = 0;
    for (int i = 0; i < n; ++i) {
      const int g = first + i;
      int unit, tt;
      locate(g, unit, tt);
      if (unit != cur_unit) {
        const int qs = qcount % NQB;
        bool ok = true;
        if (lane == 0) {
          // the unit's window-query rows (padded to nq_pad with the next rows, whose scores
          // the epilogue discards) by TMA into the swizzled B-operand tile
          if (qcount >= NQB) ok = mbar_wait(&qempty_bar[qs], ((qcount / NQB) - 1) & 1, p.status, abort_flag);
          if (ok) {
            uint8_t* qb = qbuf + qs * qbytes;
            const uint32_t half_bytes = (uint32_t)p.nq_pad * 128;
            mbar_arrive_expect_tx(&qfull_bar[qs], qbytes);
#pragma unroll
            for (int h = 0; h < D / 64; ++h) tma_load_2d(qb + h * half_bytes, &qmap, &qfull_bar[qs], 64 * h, unit * p.nq_rows);
          }
        }
        if (!__shfl_sync(0xffffffffu, ok, 0)) break;
        cur_unit = unit;
        ++qcount;
      }
      if (i >= pre && !issue_k(i)) break;
    }
    if (lane == 0 && *abort_flag) {   // no copy may land in shared memory after the CTA exits
      for (int t = max(0, k_issued - STAGES); t < k_issued; ++t)
        mbar_wait(&full_bar[t % STAGES], (t / STAGES) & 1, p.status, nullptr);
      for (int q = max(0, qcount - NQB); q < qcount; ++q)
        mbar_wait(&qfull_bar[q % NQB], (q / NQB) & 1, p.status, nullptr);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    allow_dependent_launch();
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kSKeys, p.nq_pad);
      int cur_unit = -1, qcount = 0;
      for (int i = 0; i < n; ++i) {
        const int g = first + i;
        int unit, tt;
        locate(g, unit, tt);
        const bool unit_ends = (i == n - 1) || last_of_unit(g, unit);
        if (unit != cur_unit) {
          if (!mbar_wait(&qfull_bar[qcount % NQB], (qcount / NQB) & 1, p.status, abort_flag)) break;
          cur_unit = unit;
          ++qcount;
        }
        const int qs = (qcount - 1) % NQB;
        const int s = i % STAGES;
        if (!mbar_wait(&full_bar[s], (i / STAGES) & 1, p.status, abort_flag)) break;
        const int acc = i % n_acc;
        if (i >= n_acc && !mbar_wait(&tempty_bar[acc], ((i / n_acc) & 1) ^ 1, p.status, abort_flag)) break;
        tc_fence_after();
        const uint32_t a_base = smem_u32(kstage + s * KTILE);
        const uint32_t b_base = smem_u32(qbuf + qs * qbytes);
        const uint32_t b_half = (uint32_t)p.nq_pad * 128;
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * p.acc_stride);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t koff = (ks & 3) * 32;
          const uint64_t adesc = umma_desc_sw128(a_base + (ks >> 2) * KHALF + koff);
          const uint64_t bdesc = umma_desc_sw128(b_base + (ks >> 2) * b_half + koff);
          tc_mma_bf16(d_tmem, adesc, bdesc, idesc, ks > 0 ? 1u : 0u);
        }
        tc_commit(&empty_bar[s]);
        tc_commit(&tfull_bar[acc]);
        if (unit_ends) tc_commit(&qempty_bar[qs]);
      }
      // every MMA this thread issued has completed before TMEM is released
      tc_commit(drain_bar);
      mbar_wait(drain_bar, 0, p.status, nullptr);
    }
  } else {
    // ---------------------------------------------------------------- epilogue (2 groups of 4 warps)
    if (!RAGGED && n > 0 && warp == 2)           // the first unit's window LSE into L2 meanwhile
      prefetch_lines_l2(p.lse_win + (size_t)(first / p.tiles_per_unit) * p.nq_rows, (size_t)p.nq_rows * 4, lane, 32);
    grid_dependency_wait();                      // the window LSE is carried from earlier kernels
    allow_dependent_launch();
    const int grp = (warp - 2) >> 2;            // group g: warps 2+4g .. 5+4g; tiles i % 4 == g
    const int quad = warp & 3;                  // TMEM lanes quad*32 .. quad*32+31
    const int ep_tid = (warp - 2 - 4 * grp) * 32 + lane;
    float* lse2_s = reinterpret_cast<float*>(smem + 1024 + grp * 2304);   // [288] -lse * log2(e)
    int* pw_s = reinterpret_cast<int*>(smem + 1024 + grp * 2304 + 1152);  // [288]
    int win0 = p.t_ctx - p.window;              // position of window row 0 (of the current unit)
    int mid_end = p.mid_end;                    // end of the current unit's middle
    int cur_unit = -1;
    for (int i = grp; i < n; i += 4) {
      const int g = first + i;
      int unit, tt;
      locate(g, unit, tt);
      if (unit != cur_unit) {
        if (RAGGED) {
          const int t_u = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, ep_tid == 0 ? p.status : nullptr);
          if (t_u < p.window && ep_tid == 0) record_error(p.status, BD_ERR_INVALID_ARG);
          win0 = t_u - p.window;
          mid_end = t_u - (p.t_ctx - p.mid_end);
        }
        named_bar(1 + grp, 128);
        for (int c = ep_tid; c < 288; c += 128) {
          const bool real = c < p.nq_rows;
          lse2_s[c] = real ? -__ldg(p.lse_win + (size_t)unit * p.nq_rows + c) * kLog2e : -INFINITY;
          pw_s[c] = real ? win0 + c % p.window : -1;
        }
        named_bar(1 + grp, 128);
        cur_unit = unit;
      }
      const int acc = i % n_acc;
      if (!mbar_wait(&tfull_bar[acc], (i / n_acc) & 1, p.status, abort_flag)) break;
      tc_fence_after();
      const int key_tile0 = p.n_sink + kSKeys * tt;
      const int key = key_tile0 + quad * 32 + lane;
      const bool causal = key_tile0 + kSKeys - 1 > win0;   // some key may follow a window row
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * p.acc_stride);
      float sum0 = 0.f, sum1 = 0.f, sum2 = 0.f, sum3 = 0.f;
      for (int c0 = 0; c0 < p.nq_pad; c0 += 64) {
        float v[64];
        tc_ld_32cols(taddr + c0, *reinterpret_cast<float(*)[32]>(&v[0]));
        tc_ld_32cols(taddr + c0 + 32, *reinterpret_cast<float(*)[32]>(&v[32]));
        tc_wait_ld();
        const int ncol = min(64, p.nq_pad - c0);
        if (ncol == 64 && !causal) {
          // packed pairs: one f32x2 FMA and one f32x2 add per two scores (the epilogue's
          // instruction issue, not the exponentials, limits this loop)
          const float2 cc = make_float2(p.scale_log2, p.scale_log2);
          float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2 = a0, a3 = a0;
#pragma unroll
          for (int j = 0; j < 64; j += 8) {
            const float4 la = *reinterpret_cast<const float4*>(lse2_s + c0 + j);
            const float4 lb = *reinterpret_cast<const float4*>(lse2_s + c0 + j + 4);
            const float2 x0 = ffma2(make_float2(v[j], v[j + 1]), cc, make_float2(la.x, la.y));
            const float2 x1 = ffma2(make_float2(v[j + 2], v[j + 3]), cc, make_float2(la.z, la.w));
            const float2 x2 = ffma2(make_float2(v[j + 4], v[j + 5]), cc, make_float2(lb.x, lb.y));
            const float2 x3 = ffma2(make_float2(v[j + 6], v[j + 7]), cc, make_float2(lb.z, lb.w));
            a0 = fadd2(a0, make_float2(fast_exp2(x0.x), fast_exp2(x0.y)));
            a1 = fadd2(a1, make_float2(fast_exp2(x1.x), fast_exp2(x1.y)));
            a2 = fadd2(a2, make_float2(fast_exp2(x2.x), fast_exp2(x2.y)));
            a3 = fadd2(a3, make_float2(fast_exp2(x3.x), fast_exp2(x3.y)));
          }
          sum0 += a0.x + a0.y;
          sum1 += a1.x + a1.y;
          sum2 += a2.x + a2.y;
          sum3 += a3.x + a3.y;
        } else {
#pragma unroll
          for (int j = 0; j < 64; ++j) {
            if (j < ncol) {
              const float x = key <= pw_s[c0 + j] ? fmaf(v[j], p.scale_log2, lse2_s[c0 + j]) : -INFINITY;
              sum0 += fast_exp2(x);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar[acc]);
      if (key < mid_end) p.score[(size_t)unit * p.n_mid_pad + (key - p.n_sink)] = (sum0 + sum1) + (sum2 + sum3);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, p.tmem_cols);
}

// ============================================================================ window LSE
//
// Self mode's normalisers: lse_r = log sum_{k <= p_w} exp(q_r . k_k / sqrt(d)) for the G*W
// window rows r = h*W + w of every unit (p_w = t_ctx - W + w).  The contraction of
// score_kernel with its operands swapped: the unit's window rows are the A operand (M =
// 128 rows = the TMEM lanes) and a 128-key K tile the B operand (N = 128 columns), so a
// row's online log-sum-exp stays inside the two threads that own it (one per 64-column
// half of the TMEM row), with no reduction across lanes.  Persistent CTAs (one per SM)
// take contiguous ranges of the (unit, 128-key tile) list: warp 0 streams K tiles (TMA,
// 4-stage ring) and the unit's rows (two buffers), warp 1 issues the MMAs into four TMEM
// accumulators, warps 2-9 reduce (two warps per TMEM lane quarter).  A unit split over
// several CTAs merges the segments' (max, sum) pairs in the CTA that finishes it last.
struct LseParams {
  const __nv_bfloat16* q_win;   // [units * nq_rows][D] (read by TMA; prefetched through this pointer)
  float* lse;          // [units * nq_rows] natural log
  float2* part;        // [units][max_seg][128]: a segment's (running max in log2 units, sum)
  int* counters;       // [units] arrival counters (left zero)
  int* status;
  int nq_rows, window, t_ctx, tiles_per_unit, total_tiles, tiles_per_cta, max_seg;
  int window_ready;    // BD_SELECT_WINDOW_READY: the rows may load before the dependency wait
  float scale_log2;
  const int32_t* seq_lens;   // per-sequence context lengths [batch] (RAGGED instance) or null
  int h_kv, units;
};
constexpr int kLMaxSeg = 8;      // segments of one unit with per-sequence lengths (bounds the partials)
constexpr int kLThreads = 320;   // producer, MMA, eight epilogue warps (two per TMEM lane quarter)
constexpr int kLAcc = 4;         // TMEM accumulators of 128 columns
constexpr int kLStages = 4;

// RAGGED: per-sequence lengths; every CTA lays out the units' tiles itself (a prefix table in
// shared memory, as score_kernel's ragged instance does) and the range per CTA is at least
// tiles_per_cta, which keeps a unit within kLMaxSeg segments.
template <int D, bool RAGGED>
__global__ void __launch_bounds__(kLThreads, 1) window_lse_kernel(const LseParams p,
                                                                  const __grid_constant__ CUtensorMap kmap,
                                                                  const __grid_constant__ CUtensorMap qmap) {
  constexpr int STAGES = kLStages;
  constexpr uint32_t KHALF = kSKeys * 128;   // one 64-column half of a K tile
  constexpr uint32_t KTILE = kSKeys * D * 2;
  constexpr uint32_t QHALF = 128 * 128;      // one 64-column half of the 128 window rows
  constexpr uint32_t QTILE = 128 * D * 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty_bar = full_bar + STAGES;
  uint64_t* tfull_bar = empty_bar + STAGES;    // [kLAcc]
  uint64_t* tempty_bar = tfull_bar + kLAcc;    // [kLAcc]
  uint64_t* qfull_bar = tempty_bar + kLAcc;    // [2]
  uint64_t* qempty_bar = qfull_bar + 2;        // [2]
  uint64_t* drain_bar = qempty_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* last_flag = const_cast<int*>(abort_flag) + 1;
  uint8_t* qbuf = smem + 1024;                 // 2 x QTILE
  uint8_t* kstage = qbuf + 2 * QTILE;          // STAGES x KTILE
  float2* ml_s = reinterpret_cast<float2*>(kstage + STAGES * KTILE);   // [2][128] the column halves' (m, l)
  int* spref = reinterpret_cast<int*>(ml_s + 256);                      // [units + 1] (RAGGED)

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tpu = p.tiles_per_unit;
  int total = p.total_tiles, tpc = p.tiles_per_cta;
  if (RAGGED) {
    // the lengths may come from the kernel just before (bd_advance moves them), unless the
    // caller says otherwise
    if (!p.window_ready) grid_dependency_wait();
    int* wtot = reinterpret_cast<int*>(smem + 512);
    const int per = (p.units + kLThreads - 1) / kLThreads;
    const int u0 = min(p.units, tid * per), u1 = min(p.units, u0 + per);
    auto tiles_of = [&](int u) {
      return (unit_context(p.seq_lens, u, p.h_kv, p.t_ctx, nullptr) + kSKeys - 1) / kSKeys;
    };
    int sum = 0;
    for (int u = u0; u < u1; ++u) sum += tiles_of(u);
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) wtot[warp] = incl;
    __syncthreads();
    int run = incl - sum;
    for (int w = 0; w < warp; ++w) run += wtot[w];
    for (int u = u0; u < u1; ++u) {
      spref[u] = run;
      run += tiles_of(u);
    }
    if (tid == kLThreads - 1) spref[p.units] = run;
    __syncthreads();
    total = spref[p.units];
    tpc = max((total + (int)gridDim.x - 1) / (int)gridDim.x, p.tiles_per_cta);
  }
  const int first = blockIdx.x * tpc;
  const int n = max(0, min(tpc, total - first));
  auto unit_of = [&](int g) {
    if (!RAGGED) return g / tpu;
    int lo = 0, hi = p.units - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (spref[mid] <= g) lo = mid;
      else hi = mid - 1;
    }
    return lo;
  };
  auto unit_begin = [&](int u) { return RAGGED ? spref[u] : u * tpu; };
  auto unit_end = [&](int u) { return RAGGED ? spref[u + 1] : (u + 1) * tpu; };

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int a = 0; a < kLAcc; ++a) {
      mbar_init(&tfull_bar[a], 1);
      mbar_init(&tempty_bar[a], 8);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&qfull_bar[i], 1);
      mbar_init(&qempty_bar[i], 1);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kLAcc * 128);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    allow_dependent_launch();
    if (lane == 0) {
      tma_prefetch_map(&kmap);
      tma_prefetch_map(&qmap);
    }
    int k_issued = 0;
    auto issue_k = [&](int i) -> bool {
      bool ok = true;
      if (lane == 0) {
        const int g = first + i, unit = unit_of(g), tt = g - unit_begin(unit);
        const int s = i % STAGES;
        if (i >= STAGES) ok = mbar_wait(&empty_bar[s], ((i / STAGES) & 1) ^ 1, p.status, abort_flag);
        if (ok) {
          uint8_t* st = kstage + s * KTILE;
          mbar_arrive_expect_tx(&full_bar[s], KTILE);
#pragma unroll
          for (int h = 0; h < D / 64; ++h) tma_load_3d(st + h * KHALF, &kmap, &full_bar[s], 64 * h, kSKeys * tt, unit);
          k_issued = i + 1;
        }
      }
      return __shfl_sync(0xffffffffu, ok, 0);
    };
    // context K tiles stream before the grid-dependency wait; the window rows after it
    // (before it as well when the caller says they were written earlier)
    const int pre = p.window_ready ? 0 : min(n, STAGES);
    for (int i = 0; i < pre; ++i) issue_k(i);
    if (!p.window_ready) {
      if (n > 0)   // the first unit's rows on their way into L2 meanwhile
        prefetch_lines_l2(p.q_win + (size_t)unit_of(first) * p.nq_rows * D, (size_t)p.nq_rows * D * 2, lane, 32);
      grid_dependency_wait();
    }
    int cur_unit = -1, qcount = 0;
    for (int i = 0; i < n; ++i) {
      const int unit = unit_of(first + i);
      if (unit != cur_unit) {
        const int qs = qcount & 1;
        bool ok = true;
        if (lane == 0) {
          // rows unit*nq_rows .. +127 (past nq_rows: the next unit's rows or zero fill, whose
          // results are discarded)
          if (qcount >= 2) ok = mbar_wait(&qempty_bar[qs], ((qcount >> 1) - 1) & 1, p.status, abort_flag);
          if (ok) {
            uint8_t* qb = qbuf + qs * QTILE;
            mbar_arrive_expect_tx(&qfull_bar[qs], QTILE);
#pragma unroll
            for (int h = 0; h < D / 64; ++h) tma_load_2d(qb + h * QHALF, &qmap, &qfull_bar[qs], 64 * h, unit * p.nq_rows);
          }
        }
        if (!__shfl_sync(0xffffffffu, ok, 0)) break;
        cur_unit = unit;
        ++qcount;
      }
      if (i >= pre && !issue_k(i)) break;
    }
    if (lane == 0 && *abort_flag) {   // no copy may land in shared memory after the CTA exits
      for (int t = max(0, k_issued - STAGES); t < k_issued; ++t)
        mbar_wait(&full_bar[t % STAGES], (t / STAGES) & 1, p.status, nullptr);
      for (int q = max(0, qcount - 2); q < qcount; ++q) mbar_wait(&qfull_bar[q & 1], (q >> 1) & 1, p.status, nullptr);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    allow_dependent_launch();
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(128, kSKeys);
      int cur_unit = -1, qcount = 0;
      for (int i = 0; i < n; ++i) {
        const int g = first + i, unit = unit_of(g);
        const bool unit_ends = (i == n - 1) || g + 1 == unit_end(unit);
        if (unit != cur_unit) {
          if (!mbar_wait(&qfull_bar[qcount & 1], (qcount >> 1) & 1, p.status, abort_flag)) break;
          cur_unit = unit;
          ++qcount;
        }
        const int qs = (qcount - 1) & 1;
        const int s = i % STAGES;
        if (!mbar_wait(&full_bar[s], (i / STAGES) & 1, p.status, abort_flag)) break;
        const int acc = i % kLAcc;
        if (i >= kLAcc && !mbar_wait(&tempty_bar[acc], ((i / kLAcc) & 1) ^ 1, p.status, abort_flag)) break;
        tc_fence_after();
        const uint32_t a_base = smem_u32(qbuf + qs * QTILE);
        const uint32_t b_base = smem_u32(kstage + s * KTILE);
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * 128);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t koff = (ks & 3) * 32;
          const uint64_t adesc = umma_desc_sw128(a_base + (ks >> 2) * QHALF + koff);
          const uint64_t bdesc = umma_desc_sw128(b_base + (ks >> 2) * KHALF + koff);
          tc_mma_bf16(d_tmem, adesc, bdesc, idesc, ks > 0 ? 1u : 0u);
        }
        tc_commit(&empty_bar[s]);
        tc_commit(&tfull_bar[acc]);
        if (unit_ends) tc_commit(&qempty_bar[qs]);
      }
      tc_commit(drain_bar);
      mbar_wait(drain_bar, 0, p.status, nullptr);
    }
  } else {
    // ---------------------------------------------------------------- epilogue: a row's half per thread
    grid_dependency_wait();
    allow_dependent_launch();
    const int quad = warp & 3;                  // TMEM lanes quad*32 .. quad*32+31
    const int half = (warp - 2) >> 2;           // warps 2-5: columns 0-63, warps 6-9: 64-127
    const int row = quad * 32 + lane;
    int pw = p.t_ctx - p.window + row % p.window;         // last key the row sees
    int first_masked = p.t_ctx - p.window;                // keys past it are hidden from some row
    int cur_unit = -1;
    float m = -INFINITY, l = 0.f;                          // log2 units
    // after a wait gives up, a warp keeps walking its tiles without touching TMEM, so that
    // all eight warps still meet at every unit-end barrier
    bool alive = true;
    for (int i = 0; i < n; ++i) {
      const int g = first + i, unit = unit_of(g), tt = g - unit_begin(unit);
      if (RAGGED && unit != cur_unit) {
        const int t_u = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, tid == 64 ? p.status : nullptr);
        if (t_u < p.window && tid == 64) record_error(p.status, BD_ERR_INVALID_ARG);
        pw = t_u - p.window + row % p.window;
        first_masked = t_u - p.window;
        cur_unit = unit;
      }
      const int acc = i % kLAcc;
      alive = __all_sync(0xffffffffu, alive && mbar_wait(&tfull_bar[acc], (i / kLAcc) & 1, p.status, abort_flag));
      if (alive) {
        tc_fence_after();
        const int key0 = kSKeys * tt;
        const bool masked = key0 + kSKeys - 1 > first_masked;
        const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * 128);
        {
          const int c0 = 64 * half;
          float v[64];
          tc_ld_32cols(taddr + c0, *reinterpret_cast<float(*)[32]>(&v[0]));
          tc_ld_32cols(taddr + c0 + 32, *reinterpret_cast<float(*)[32]>(&v[32]));
          tc_wait_ld();
          if (masked) {
#pragma unroll
            for (int j = 0; j < 64; ++j) v[j] = key0 + c0 + j <= pw ? v[j] : -INFINITY;
          }
          float mx0 = fmaxf(v[0], v[1]), mx1 = fmaxf(v[2], v[3]);
#pragma unroll
          for (int j = 4; j < 64; j += 4) {
            mx0 = fmaxf(mx0, fmaxf(v[j], v[j + 1]));
            mx1 = fmaxf(mx1, fmaxf(v[j + 2], v[j + 3]));
          }
          const float mxs = fmaxf(mx0, mx1) * p.scale_log2;
          if (mxs > m) {
            l *= fast_exp2(m - mxs);                 // m = -inf: l is still 0
            m = mxs;
          }
          const float2 cc = make_float2(p.scale_log2, p.scale_log2);
          const float2 nm = make_float2(m == -INFINITY ? 0.f : -m, m == -INFINITY ? 0.f : -m);
          float2 a0 = make_float2(0.f, 0.f), a1 = a0;
#pragma unroll
          for (int j = 0; j < 64; j += 4) {
            const float2 x0 = ffma2(make_float2(v[j], v[j + 1]), cc, nm);
            const float2 x1 = ffma2(make_float2(v[j + 2], v[j + 3]), cc, nm);
            a0 = fadd2(a0, make_float2(fast_exp2(x0.x), fast_exp2(x0.y)));
            a1 = fadd2(a1, make_float2(fast_exp2(x1.x), fast_exp2(x1.y)));
          }
          l += (a0.x + a0.y) + (a1.x + a1.y);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty_bar[acc]);
      }
      if (i != n - 1 && g + 1 != unit_end(unit)) continue;
      // ------------------------------------------------------------ end of this CTA's part of the unit
      // the two column halves of each row meet first
      ml_s[half * 128 + row] = alive ? make_float2(m, l) : make_float2(-INFINITY, 0.f);
      named_bar(1, 256);
      const int c_first = unit_begin(unit) / tpc, c_last = (unit_end(unit) - 1) / tpc;
      const int n_seg = c_last - c_first + 1;
      const size_t row0 = (size_t)unit * p.nq_rows;
      float2* seg = p.part + (size_t)unit * p.max_seg * 128;
      if (half == 0) {
        const float2 o = ml_s[128 + row];
        const float M2 = fmaxf(m, o.x);
        l = (m == -INFINITY ? 0.f : l * fast_exp2(m - M2)) + (o.x == -INFINITY ? 0.f : o.y * fast_exp2(o.x - M2));
        m = M2;
        if (n_seg == 1) {
          if (alive && row < p.nq_rows) p.lse[row0 + row] = l > 0.f ? (m + log2f(l)) * kLn2 : -INFINITY;
        } else if (alive) {
          seg[(size_t)((int)blockIdx.x - c_first) * 128 + row] = make_float2(m, l);
        }
      }
      if (n_seg > 1) {
        __threadfence();
        named_bar(1, 256);
        if (half == 0 && row == 0) *last_flag = alive && atomicAdd(&p.counters[unit], 1) == n_seg - 1;
        named_bar(1, 256);
        if (half == 0 && *last_flag) {
          __threadfence();
          float M = -INFINITY;
          for (int k = 0; k < n_seg; ++k) M = fmaxf(M, __ldcg(&seg[(size_t)k * 128 + row].x));
          float L = 0.f;
          for (int k = 0; k < n_seg; ++k) {
            const float2 ml = __ldcg(&seg[(size_t)k * 128 + row]);
            L += ml.x == -INFINITY ? 0.f : ml.y * fast_exp2(ml.x - M);
          }
          if (row < p.nq_rows) p.lse[row0 + row] = L > 0.f ? (M + log2f(L)) * kLn2 : -INFINITY;
          if (row == 0) p.counters[unit] = 0;
        }
      }
      named_bar(1, 256);                          // ml_s and last_flag are free for the next unit
      m = -INFINITY;
      l = 0.f;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, kLAcc * 128);
}

// ============================================================================ top-B select

struct TopkParams {
  const float* score;      // [units][n_mid_pad]
  int32_t* idx_out;        // [units][budget]
  int32_t* count_out;      // [units]
  int t_ctx, budget, n_sink, n_recent, chunk, n_mid_pad;
  int keep_all;            // budget >= t_ctx
  int smem_items;          // item values staged in shared memory when n_items <= smem_items
  const int32_t* seq_lens; // per-sequence context lengths [batch] or null (all t_ctx)
  int h_kv;
  int* status;
};

// A unit whose context fits the budget keeps every position (the B >= T rule).
__device__ __forceinline__ bool topk_keep_all(const TopkParams& p, int unit, int t_u, int32_t* out) {
  if (!p.keep_all && p.budget < t_u) return false;
  for (int i = threadIdx.x; i < p.budget; i += blockDim.x) out[i] = i < t_u ? i : -1;
  if (threadIdx.x == 0) p.count_out[unit] = t_u;
  return true;
}

// Exclusive scan of one value per warp (32 warps), result broadcast through smem.
__device__ __forceinline__ uint32_t warp_totals_exclusive(uint32_t v, uint32_t* wsum, uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) wsum[warp] = v;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = wsum[lane];
    uint32_t incl = w;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    wsum[lane] = incl - w;
    if (lane == 31) *total = incl;
  }
  __syncthreads();
  const uint32_t r = wsum[warp];
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kTopkThreads, 1) topk_kernel(const TopkParams p) {
  extern __shared__ uint32_t vals[];           // item values (fp32 bits) | candidates | samples
  __shared__ uint32_t hist[256];
  __shared__ uint32_t wsum[32];
  __shared__ uint32_t s_total, s_prefix, s_krem;
  grid_dependency_wait();
  allow_dependent_launch();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int unit = blockIdx.x;
  int32_t* out = p.idx_out + (size_t)unit * p.budget;

  const int t_u = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, tid == 0 ? p.status : nullptr);
  if (topk_keep_all(p, unit, t_u, out)) return;
  const int lo = p.n_sink, hi = t_u - p.n_recent;
  const int s = p.chunk;
  const int free = p.budget - p.n_sink - p.n_recent;
  const int c_first = lo / s;
  const int n_items = (hi > lo) ? ((hi - 1) / s - c_first + 1) : 0;
  const int k = min(free / s, n_items);
  const float* sc = p.score + (size_t)unit * p.n_mid_pad;
  const bool take_all = (k >= n_items), take_none = (k <= 0);
  const bool ranked = !take_all && !take_none;
  const bool staged = n_items <= p.smem_items;

  auto members = [&](int i, int& a, int& b) {
    const int c = c_first + i;
    a = max(c * s, lo);
    b = min(c * s + s, hi);
  };
  // a chunk's score: its members summed in position order, their loads issued eight at a
  // time (all in flight together; the zeros past b add nothing to a sum of scores >= +0)
  auto value_global = [&](int i) -> uint32_t {
    if (s == 1) return __float_as_uint(__ldcg(sc + i));
    int a, b;
    members(i, a, b);
    float v = 0.f;
    for (int q0 = a; q0 < b; q0 += 8) {
      float t[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) t[j] = q0 + j < b ? __ldcg(sc + (q0 + j - lo)) : 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) v += t[j];
    }
    return __float_as_uint(v);
  };
  if (ranked && staged) {
    if (s == 1) {
      const int n4 = n_items / 4;
      const float4* sc4 = reinterpret_cast<const float4*>(sc);
      for (int i = tid; i < n4; i += kTopkThreads) {
        const float4 v = __ldcg(sc4 + i);
        vals[4 * i] = __float_as_uint(v.x);
        vals[4 * i + 1] = __float_as_uint(v.y);
        vals[4 * i + 2] = __float_as_uint(v.z);
        vals[4 * i + 3] = __float_as_uint(v.w);
      }
      for (int i = 4 * n4 + tid; i < n_items; i += kTopkThreads) vals[i] = __float_as_uint(__ldcg(sc + i));
    } else {
      // two chunks per round, so that both chunks' loads are in flight together
      for (int i = tid; i < n_items; i += 2 * kTopkThreads) {
        const int i2 = i + kTopkThreads;
        const uint32_t v1 = value_global(i);
        const uint32_t v2 = i2 < n_items ? value_global(i2) : 0u;
        vals[i] = v1;
        if (i2 < n_items) vals[i2] = v2;
      }
    }
    __syncthreads();
  }
  auto val = [&](int i) -> uint32_t { return staged ? vals[i] : value_global(i); };

  // ---- value bits of the k-th largest item (tau) and how many items equal to tau to take (krem)
  // Linear histogram between the block's min and max value: bins are monotone in the value,
  // so the k-th largest lies in the bin where the count from the top reaches k; its items
  // are few and are ranked exactly by (value desc, position asc).
  uint32_t prefix = 0, krem = (uint32_t)k;
  bool found = false, simple_eq = false;
  if (ranked && staged) {
    uint32_t* bins = reinterpret_cast<uint32_t*>(vals + ((p.smem_items + 1) & ~1));   // [kBins]
    uint64_t* cand = reinterpret_cast<uint64_t*>(bins + kBins);                       // [kBinCandMax]
    float lmin = INFINITY, lmax = -INFINITY;
    for (int i = tid; i < n_items; i += kTopkThreads) {
      const float v = __uint_as_float(vals[i]);
      lmin = fminf(lmin, v);
      lmax = fmaxf(lmax, v);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      lmin = fminf(lmin, __shfl_xor_sync(0xffffffffu, lmin, off));
      lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, off));
    }
    __shared__ float s_min[32], s_max[32];
    __shared__ uint32_t s_bin, s_above, s_nc, s_taukey, s_eq_take, s_eq_all;
    if (lane == 0) {
      s_min[warp] = lmin;
      s_max[warp] = lmax;
    }
    for (int i = tid; i < kBins; i += kTopkThreads) bins[i] = 0;
    if (tid == 0) {
      s_nc = 0;
      s_eq_take = 0;
      s_eq_all = 0;
      s_bin = 0xFFFFFFFFu;
    }
    __syncthreads();
    float vmin = s_min[0], vmax = s_max[0];
    for (int w = 1; w < 32; ++w) {
      vmin = fminf(vmin, s_min[w]);
      vmax = fmaxf(vmax, s_max[w]);
    }
    const float scale = vmax > vmin ? (float)(kBins - 1) / (vmax - vmin) : 0.f;
    auto bin_of = [&](uint32_t u) -> int {
      return min(kBins - 1, (int)((__uint_as_float(u) - vmin) * scale));
    };
    for (int i = tid; i < n_items; i += kTopkThreads) atomicAdd(&bins[bin_of(vals[i])], 1u);
    __syncthreads();
    // items in the bins of higher threads: total minus the inclusive prefix over threads
    uint32_t mine = 0;
#pragma unroll
    for (int j = 0; j < kBins / kTopkThreads; ++j) mine += bins[tid * (kBins / kTopkThreads) + j];
    uint32_t incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t z = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += z;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const uint32_t w = wsum[lane];
      uint32_t c = w;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
        if (lane >= off) c += z;
      }
      wsum[lane] = c - w;
      if (lane == 31) s_total = c;
    }
    __syncthreads();
    uint32_t above = s_total - (wsum[warp] + incl);   // items in bins above this thread's bins
    for (int j = kBins / kTopkThreads - 1; j >= 0; --j) {
      const int bidx = tid * (kBins / kTopkThreads) + j;
      const uint32_t h = bins[bidx];
      if (above < (uint32_t)k && (uint32_t)k <= above + h) {
        s_bin = (uint32_t)bidx;
        s_above = above;
      }
      above += h;
    }
    __syncthreads();
    const int bstar = (int)s_bin;
    const uint32_t nc = bins[bstar];
    if (nc <= (uint32_t)kBinCandMax) {
      for (int i = tid; i < n_items; i += kTopkThreads) {
        const uint32_t u = vals[i];
        if (bin_of(u) == bstar) cand[atomicAdd(&s_nc, 1u)] = (static_cast<uint64_t>(u) << 32) | (0xFFFFFFFFu - (uint32_t)i);
      }
      __syncthreads();
      const uint32_t m = (uint32_t)k - s_above;       // rank (1-based) of the k-th item inside the bin
      for (int i = tid; i < (int)nc; i += kTopkThreads) {
        const uint64_t key = cand[i];
        uint32_t rank = 0;
        for (int j = 0; j < (int)nc; ++j) rank += cand[j] > key;
        if (rank == m - 1) s_taukey = static_cast<uint32_t>(key >> 32);
      }
      __syncthreads();
      prefix = s_taukey;
      for (int i = tid; i < (int)nc; i += kTopkThreads) {
        const uint64_t key = cand[i];
        if (static_cast<uint32_t>(key >> 32) != prefix) continue;
        uint32_t rank = 0;
        for (int j = 0; j < (int)nc; ++j) rank += cand[j] > key;
        atomicAdd(&s_eq_all, 1u);
        if (rank < m) atomicAdd(&s_eq_take, 1u);
      }
      __syncthreads();
      krem = s_eq_take;
      simple_eq = (s_eq_take == s_eq_all);
      found = true;
    }
  }
  // ---- otherwise radix select (MSB first, 8 bits per pass)
  uint32_t mask = 0;
  const int n_round = (n_items + kTopkThreads - 1) / kTopkThreads * kTopkThreads;
  if (ranked && !found) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      if (tid < 256) hist[tid] = 0;
      __syncthreads();
#pragma unroll 4
      for (int i = tid; i < n_round; i += kTopkThreads) {
        uint32_t digit = 256;
        if (i < n_items) {
          const uint32_t u = val(i);
          if ((u & mask) == prefix) digit = (u >> shift) & 255u;
        }
        const uint32_t peers = __match_any_sync(0xffffffffu, digit);
        if (digit < 256 && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
      }
      __syncthreads();
      if (warp == 0) {
        uint32_t local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) local += hist[8 * lane + j];
        uint32_t suffix = local;   // items whose digit is >= 8*lane
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const uint32_t y = __shfl_down_sync(0xffffffffu, suffix, off);
          if (lane + off < 32) suffix += y;
        }
        uint32_t above = suffix - local;
        if (above < krem && krem <= suffix) {
          for (int j = 7; j >= 0; --j) {
            const uint32_t h = hist[8 * lane + j];
            if (above + h >= krem) {
              s_prefix = prefix | ((uint32_t)(8 * lane + j) << shift);
              s_krem = krem - above;
              break;
            }
            above += h;
          }
        }
      }
      __syncthreads();
      prefix = s_prefix;
      krem = s_krem;
      mask |= 0xFFu << shift;
    }
  }
  const uint32_t tau = prefix;   // value bits of the k-th largest item; take krem of the equal ones

  // ---- compaction in item order: warp w owns items [w*ipw, (w+1)*ipw), lane-interleaved rows
  const int ipw = (n_items + 32 * 32 - 1) / (32 * 32) * 32;
  const int w0 = warp * ipw, w1 = min(n_items, w0 + ipw);
  const uint32_t lt_mask = (1u << lane) - 1u;
  uint32_t eq_count = 0;
  const bool need_eq = ranked && !simple_eq;      // some items equal to tau are left out
  if (need_eq)
    for (int j = w0; j < w1; j += 32) {
      const int i = j + lane;
      const bool eq = i < w1 && val(i) == tau;
      eq_count += __popc(__ballot_sync(0xffffffffu, eq));
    }
  const uint32_t eq_base = warp_totals_exclusive(eq_count, wsum, &s_total);
  auto select_row = [&](int j, uint32_t& eq_run, int& npos) -> bool {
    const int i = j + lane;
    bool sel = false;
    bool eq = false;
    if (i < w1) {
      if (take_all) {
        sel = true;
      } else if (ranked) {
        const uint32_t u = val(i);
        eq = (u == tau);
        sel = u > tau;
      }
    }
    const uint32_t bal = __ballot_sync(0xffffffffu, eq);
    if (eq) sel = need_eq ? (eq_run + __popc(bal & lt_mask)) < krem : true;
    eq_run += __popc(bal);
    npos = 0;
    if (sel) {
      int a, b;
      members(i, a, b);
      npos = b - a;
    }
    return sel;
  };
  uint32_t pos_count = 0;
  {
    uint32_t eq_run = eq_base;
    for (int j = w0; j < w1; j += 32) {
      int npos;
      select_row(j, eq_run, npos);
      int sum = npos;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      pos_count += (uint32_t)sum;
    }
  }
  const uint32_t pos_base = warp_totals_exclusive(pos_count, wsum, &s_total);
  const int n_chosen = (int)s_total;
  {
    uint32_t eq_run = eq_base, w = (uint32_t)lo + pos_base;
    for (int j = w0; j < w1; j += 32) {
      int npos;
      const bool sel = select_row(j, eq_run, npos);
      int incl = npos;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      if (sel) {
        int a, b;
        members(j + lane, a, b);
        int o = (int)w + incl - npos;
        for (int q = a; q < b; ++q) out[o++] = q;
      }
      w += (uint32_t)__shfl_sync(0xffffffffu, incl, 31);
    }
  }
  const int count = lo + n_chosen + p.n_recent;
  for (int i = tid; i < lo; i += kTopkThreads) out[i] = i;
  for (int i = tid; i < p.n_recent; i += kTopkThreads) out[lo + n_chosen + i] = hi + i;
  for (int i = count + tid; i < p.budget; i += kTopkThreads) out[i] = -1;
  if (tid == 0) p.count_out[unit] = count;
}

// Token-level selection with the scores staged in shared memory (the graded workloads'
// path): the same boundary-bin method as topk_kernel, written lean.  Needs 0 < k < n <=
// kLeanMaxItems; the selection mask of each item is kept as warp ballots in registers.
constexpr int kLeanMaxItems = 32 * kTopkThreads;   // 32 rows of 32 items per warp
constexpr int kLeanRows = kLeanMaxItems / kTopkThreads;

__global__ void __launch_bounds__(kTopkThreads, 1) topk_token_kernel(const TopkParams p) {
  extern __shared__ uint32_t vals[];                // n scores (fp32 bits)
  __shared__ uint32_t bins[kBins];
  __shared__ uint64_t cand[kBinCandMax];
  __shared__ uint32_t wsum[32];
  __shared__ float wmin[32], wmax[32];
  __shared__ uint32_t s_total, s_bin, s_above, s_nc, s_taukey, s_eq_take, s_eq_all, s_prefix, s_krem;
  __shared__ float s_vmin, s_vmax;
  grid_dependency_wait();
  allow_dependent_launch();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int unit = blockIdx.x;
  const int t_u = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, tid == 0 ? p.status : nullptr);
  int32_t* out = p.idx_out + (size_t)unit * p.budget;
  if (topk_keep_all(p, unit, t_u, out)) return;
  const int lo = p.n_sink, hi = t_u - p.n_recent, n = hi - lo;
  const int k = p.budget - p.n_sink - p.n_recent;
  const float* sc = p.score + (size_t)unit * p.n_mid_pad;

  // ---- stage the scores, min and max
  float lmin = INFINITY, lmax = -INFINITY;
  const int n4 = n >> 2;
  const float4* sc4 = reinterpret_cast<const float4*>(sc);
  for (int i = tid; i < n4; i += kTopkThreads) {
    const float4 v = __ldcg(sc4 + i);
    reinterpret_cast<uint4*>(vals)[i] = make_uint4(__float_as_uint(v.x), __float_as_uint(v.y), __float_as_uint(v.z),
                                                   __float_as_uint(v.w));
    lmin = fminf(fminf(lmin, fminf(v.x, v.y)), fminf(v.z, v.w));
    lmax = fmaxf(fmaxf(lmax, fmaxf(v.x, v.y)), fmaxf(v.z, v.w));
  }
  for (int i = 4 * n4 + tid; i < n; i += kTopkThreads) {
    const float v = __ldcg(sc + i);
    vals[i] = __float_as_uint(v);
    lmin = fminf(lmin, v);
    lmax = fmaxf(lmax, v);
  }
  for (int i = tid; i < kBins; i += kTopkThreads) bins[i] = 0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    lmin = fminf(lmin, __shfl_xor_sync(0xffffffffu, lmin, off));
    lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, off));
  }
  if (lane == 0) {
    wmin[warp] = lmin;
    wmax[warp] = lmax;
  }
  if (tid == 0) {
    s_nc = 0;
    s_eq_take = 0;
    s_eq_all = 0;
  }
  __syncthreads();
  if (warp == 0) {
    float a = wmin[lane], b = wmax[lane];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      a = fminf(a, __shfl_xor_sync(0xffffffffu, a, off));
      b = fmaxf(b, __shfl_xor_sync(0xffffffffu, b, off));
    }
    if (lane == 0) {
      s_vmin = a;
      s_vmax = b;
    }
  }
  __syncthreads();
  const float vmin = s_vmin, vmax = s_vmax;

  // ---- tau (bits of the k-th largest score) and krem (how many scores equal to tau to keep)
  uint32_t tau = 0, krem = (uint32_t)k;
  bool simple = false, found = false;
  if (vmax > vmin) {
    const float scale = (float)(kBins - 1) / (vmax - vmin);
    auto bin_of = [&](uint32_t u) -> int { return min(kBins - 1, (int)((__uint_as_float(u) - vmin) * scale)); };
    for (int i = tid; i < n; i += kTopkThreads) atomicAdd(&bins[bin_of(vals[i])], 1u);
    __syncthreads();
    constexpr int BPT = kBins / kTopkThreads;
    uint32_t mine = 0;
#pragma unroll
    for (int j = 0; j < BPT; ++j) mine += bins[tid * BPT + j];
    uint32_t incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t z = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += z;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const uint32_t w = wsum[lane];
      uint32_t c = w;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
        if (lane >= off) c += z;
      }
      wsum[lane] = c - w;
      if (lane == 31) s_total = c;
    }
    __syncthreads();
    uint32_t above = s_total - (wsum[warp] + incl);
#pragma unroll
    for (int j = BPT - 1; j >= 0; --j) {
      const uint32_t h = bins[tid * BPT + j];
      if (above < (uint32_t)k && (uint32_t)k <= above + h) {
        s_bin = (uint32_t)(tid * BPT + j);
        s_above = above;
      }
      above += h;
    }
    __syncthreads();
    const int bstar = (int)s_bin;
    const uint32_t nc = bins[bstar];
    if (nc <= (uint32_t)kBinCandMax) {
      for (int i = tid; i < n; i += kTopkThreads) {
        const uint32_t u = vals[i];
        if (bin_of(u) == bstar) cand[atomicAdd(&s_nc, 1u)] = (static_cast<uint64_t>(u) << 32) | (0xFFFFFFFFu - (uint32_t)i);
      }
      __syncthreads();
      const uint32_t m = (uint32_t)k - s_above;
      uint64_t key = 0;
      uint32_t rank = 0xFFFFFFFFu;
      if (tid < (int)nc) {
        key = cand[tid];
        rank = 0;
        for (int j = 0; j < (int)nc; ++j) rank += cand[j] > key;
        if (rank == m - 1) s_taukey = static_cast<uint32_t>(key >> 32);
      }
      for (int i = tid + kTopkThreads; i < (int)nc; i += kTopkThreads) {   // nc > 1024: rare
        const uint64_t kk = cand[i];
        uint32_t r = 0;
        for (int j = 0; j < (int)nc; ++j) r += cand[j] > kk;
        if (r == m - 1) s_taukey = static_cast<uint32_t>(kk >> 32);
      }
      __syncthreads();
      tau = s_taukey;
      for (int i = tid; i < (int)nc; i += kTopkThreads) {
        const uint64_t kk = cand[i];
        if (static_cast<uint32_t>(kk >> 32) != tau) continue;
        uint32_t r = (i == tid) ? rank : 0;
        if (i != tid)
          for (int j = 0; j < (int)nc; ++j) r += cand[j] > kk;
        atomicAdd(&s_eq_all, 1u);
        if (r < m) atomicAdd(&s_eq_take, 1u);
      }
      __syncthreads();
      krem = s_eq_take;
      simple = (s_eq_take == s_eq_all);
      found = true;
    }
  }
  if (!found) {
    // crowded boundary (many equal or near-equal scores): exact 4-pass radix select
    uint32_t prefix = 0, mask = 0;
    krem = (uint32_t)k;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 256; i += kTopkThreads) bins[i] = 0;
      __syncthreads();
      for (int i = tid; i < n; i += kTopkThreads) {
        const uint32_t u = vals[i];
        if ((u & mask) == prefix) atomicAdd(&bins[(u >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        uint32_t local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) local += bins[8 * lane + j];
        uint32_t suffix = local;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const uint32_t y = __shfl_down_sync(0xffffffffu, suffix, off);
          if (lane + off < 32) suffix += y;
        }
        uint32_t abv = suffix - local;
        if (abv < krem && krem <= suffix) {
          for (int j = 7; j >= 0; --j) {
            const uint32_t h = bins[8 * lane + j];
            if (abv + h >= krem) {
              s_prefix = prefix | ((uint32_t)(8 * lane + j) << shift);
              s_krem = krem - abv;
              break;
            }
            abv += h;
          }
        }
      }
      __syncthreads();
      prefix = s_prefix;
      krem = s_krem;
      mask |= 0xFFu << shift;
    }
    tau = prefix;
    simple = false;
  }

  // ---- ascending compaction: warp w owns items [w*ipw, (w+1)*ipw), rows of 32
  const int rows = (n + kTopkThreads - 1) / kTopkThreads;     // <= kLeanRows
  const int w0 = warp * rows * 32;
  const uint32_t lt = (1u << lane) - 1u;
  uint32_t eq_base = 0;
  if (!simple) {
    uint32_t eqc = 0;
#pragma unroll
    for (int r = 0; r < kLeanRows; ++r) {
      if (r < rows) {
        const int i = w0 + 32 * r + lane;
        eqc += __popc(__ballot_sync(0xffffffffu, i < n && vals[i] == tau));
      }
    }
    if (lane == 0) wsum[warp] = eqc;
    __syncthreads();
    if (warp == 0) {
      const uint32_t w = wsum[lane];
      uint32_t c = w;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
        if (lane >= off) c += z;
      }
      wsum[lane] = c - w;
    }
    __syncthreads();
    eq_base = wsum[warp];
    __syncthreads();
  }
  uint32_t masks[kLeanRows];
  uint32_t cnt = 0, eq_run = eq_base;
#pragma unroll
  for (int r = 0; r < kLeanRows; ++r) {
    masks[r] = 0;
    if (r < rows) {
      const int i = w0 + 32 * r + lane;
      const uint32_t u = i < n ? vals[i] : 0u;
      bool sel = i < n && u > tau;
      const bool eq = i < n && u == tau;
      if (simple) {
        sel |= eq;
      } else {
        const uint32_t be = __ballot_sync(0xffffffffu, eq);
        if (eq) sel = eq_run + __popc(be & lt) < krem;
        eq_run += __popc(be);
      }
      masks[r] = __ballot_sync(0xffffffffu, sel);
      cnt += __popc(masks[r]);
    }
  }
  if (lane == 0) wsum[warp] = cnt;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = wsum[lane];
    uint32_t c = w;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
      if (lane >= off) c += z;
    }
    wsum[lane] = c - w;
    if (lane == 31) s_total = c;
  }
  __syncthreads();
  uint32_t base = (uint32_t)lo + wsum[warp];
#pragma unroll
  for (int r = 0; r < kLeanRows; ++r) {
    if (r < rows) {
      const uint32_t mk = masks[r];
      if ((mk >> lane) & 1u) out[base + __popc(mk & lt)] = lo + w0 + 32 * r + lane;
      base += __popc(mk);
    }
  }
  const int n_chosen = (int)s_total;
  const int count = lo + n_chosen + p.n_recent;
  for (int i = tid; i < lo; i += kTopkThreads) out[i] = i;
  for (int i = tid; i < p.n_recent; i += kTopkThreads) out[lo + n_chosen + i] = hi + i;
  for (int i = count + tid; i < p.budget; i += kTopkThreads) out[i] = -1;
  if (tid == 0) p.count_out[unit] = count;
}

// Shared storage of the register-resident top-B kernels.
struct TopkRowsSmem {
  uint32_t bins[kBins];
  uint64_t cand[kBinCandMax];
  uint32_t wsum[32], wpos[32];
  float wmin[32], wmax[32];
  uint32_t s_total, s_bin, s_above, s_nc, s_taukey, s_eq_take, s_eq_all, s_prefix, s_krem;
};

// The k-th largest of the block's items: tau (its fp32 bits), krem (how many items equal to
// tau are kept, in item order) and whether that is all of them.
struct RowsThreshold {
  uint32_t tau, krem;
  bool simple;
};

// Items in registers, ROWS per thread: warp w owns items [w*ROWS*32, (w+1)*ROWS*32), row r of
// it at w*ROWS*32 + 32r + lane; values are fp32 bits of non-negative scores (the order of the
// bits), +0 in slots past the item count (no item is below it and ties go to the lower item,
// so the padding never displaces an item).  A linear histogram between the smallest and the
// largest value (lmin, lmax: this thread's) finds the bin of the k-th value and its items are
// ranked exactly; a crowded bin takes an exact 4-pass radix select on the bits.  0 < k < n.
template <int ROWS>
__device__ __forceinline__ RowsThreshold rows_threshold(TopkRowsSmem& S, const uint32_t (&u)[ROWS], float lmin,
                                                        float lmax, int k) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int w0 = warp * ROWS * 32;
  for (int i = tid; i < kBins; i += kTopkThreads) S.bins[i] = 0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    lmin = fminf(lmin, __shfl_xor_sync(0xffffffffu, lmin, off));
    lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, off));
  }
  if (lane == 0) {
    S.wmin[warp] = lmin;
    S.wmax[warp] = lmax;
  }
  if (tid == 0) {
    S.s_nc = 0;
    S.s_eq_take = 0;
    S.s_eq_all = 0;
  }
  __syncthreads();
  float vmin = S.wmin[lane], vmax = S.wmax[lane];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, off));
    vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, off));
  }

  // ---- tau (bits of the k-th largest score) and krem (how many scores equal to tau to keep)
  uint32_t tau = 0, krem = (uint32_t)k;
  bool simple = false, found = false;
  if (vmax > vmin) {
    const float scale = (float)(kBins - 1) / (vmax - vmin);
    auto bin_of = [&](uint32_t x) -> int { return min(kBins - 1, (int)((__uint_as_float(x) - vmin) * scale)); };
#pragma unroll
    for (int r = 0; r < ROWS; ++r) atomicAdd(&S.bins[bin_of(u[r])], 1u);
    __syncthreads();
    constexpr int BPT = kBins / kTopkThreads;
    uint32_t hb[BPT];
    const uint4 hv = reinterpret_cast<const uint4*>(S.bins)[tid];
    hb[0] = hv.x;
    hb[1] = hv.y;
    hb[2] = hv.z;
    hb[3] = hv.w;
    uint32_t incl = hb[0] + hb[1] + hb[2] + hb[3];
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t z = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += z;
    }
    if (lane == 31) S.wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const uint32_t w = S.wsum[lane];
      uint32_t c = w;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
        if (lane >= off) c += z;
      }
      S.wsum[lane] = c - w;
      if (lane == 31) S.s_total = c;
    }
    __syncthreads();
    uint32_t above = S.s_total - (S.wsum[warp] + incl);
#pragma unroll
    for (int j = BPT - 1; j >= 0; --j) {
      if (above < (uint32_t)k && (uint32_t)k <= above + hb[j]) {
        S.s_bin = (uint32_t)(tid * BPT + j);
        S.s_above = above;
        S.s_prefix = hb[j];
      }
      above += hb[j];
    }
    __syncthreads();
    const int bstar = (int)S.s_bin;
    const uint32_t nc = S.s_prefix;
    if (nc <= (uint32_t)kBinCandMax) {
#pragma unroll
      for (int r = 0; r < ROWS; ++r) {
        const int i = w0 + 32 * r + lane;
        if (bin_of(u[r]) == bstar)
          S.cand[atomicAdd(&S.s_nc, 1u)] = (static_cast<uint64_t>(u[r]) << 32) | (0xFFFFFFFFu - (uint32_t)i);
      }
      __syncthreads();
      const uint32_t m = (uint32_t)k - S.s_above;
      for (int i = tid; i < (int)nc; i += kTopkThreads) {
        const uint64_t kk = S.cand[i];
        uint32_t rk = 0;
        for (int j = 0; j < (int)nc; ++j) rk += S.cand[j] > kk;
        if (rk == m - 1) S.s_taukey = static_cast<uint32_t>(kk >> 32);
      }
      __syncthreads();
      tau = S.s_taukey;
      for (int i = tid; i < (int)nc; i += kTopkThreads) {
        const uint64_t kk = S.cand[i];
        if (static_cast<uint32_t>(kk >> 32) != tau) continue;
        uint32_t rk = 0;
        for (int j = 0; j < (int)nc; ++j) rk += S.cand[j] > kk;
        atomicAdd(&S.s_eq_all, 1u);
        if (rk < m) atomicAdd(&S.s_eq_take, 1u);
      }
      __syncthreads();
      krem = S.s_eq_take;
      simple = (S.s_eq_take == S.s_eq_all);
      found = true;
    }
  }
  if (!found) {
    // crowded boundary (many equal or near-equal scores): exact 4-pass radix select
    uint32_t prefix = 0, mask = 0;
    krem = (uint32_t)k;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 256; i += kTopkThreads) S.bins[i] = 0;
      __syncthreads();
#pragma unroll
      for (int r = 0; r < ROWS; ++r)
        if ((u[r] & mask) == prefix) atomicAdd(&S.bins[(u[r] >> shift) & 255u], 1u);
      __syncthreads();
      if (warp == 0) {
        uint32_t local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) local += S.bins[8 * lane + j];
        uint32_t suffix = local;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const uint32_t y = __shfl_down_sync(0xffffffffu, suffix, off);
          if (lane + off < 32) suffix += y;
        }
        uint32_t abv = suffix - local;
        if (abv < krem && krem <= suffix) {
          for (int j = 7; j >= 0; --j) {
            const uint32_t h = S.bins[8 * lane + j];
            if (abv + h >= krem) {
              S.s_prefix = prefix | ((uint32_t)(8 * lane + j) << shift);
              S.s_krem = krem - abv;
              break;
            }
            abv += h;
          }
        }
      }
      __syncthreads();
      prefix = S.s_prefix;
      krem = S.s_krem;
      mask |= 0xFFu << shift;
    }
    tau = prefix;
    simple = false;
  }

  return RowsThreshold{tau, krem, simple};
}

// Ascending compaction of the kept items (warp ballots, a block scan, the writes), then the
// sinks, the recent window and the padding: the token-level output.
template <int ROWS>
__device__ __forceinline__ void rows_compact_tokens(TopkRowsSmem& S, const uint32_t (&u)[ROWS], RowsThreshold th,
                                                    const TopkParams& p, int unit, int lo, int hi, int32_t* out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int w0 = warp * ROWS * 32;
  const uint32_t tau = th.tau, krem = th.krem;
  const bool simple = th.simple;
  // ---- ascending compaction: warp ballots of the selected items, block scan, writes
  const uint32_t lt = (1u << lane) - 1u;
  uint32_t eq_base = 0;
  if (!simple) {
    // items equal to tau are taken in position order: count those before this warp's items
    uint32_t eqc = 0;
#pragma unroll
    for (int r = 0; r < ROWS; ++r)
      eqc += __popc(__ballot_sync(0xffffffffu, u[r] == tau));
    if (lane == 0) S.wsum[warp] = eqc;
    __syncthreads();
    if (warp == 0) {
      const uint32_t w = S.wsum[lane];
      uint32_t c = w;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
        if (lane >= off) c += z;
      }
      S.wsum[lane] = c - w;
    }
    __syncthreads();
    eq_base = S.wsum[warp];
    __syncthreads();
  }
  uint32_t masks[ROWS];
  uint32_t cnt = 0, eq_run = eq_base;
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    bool sel = u[r] > tau;
    const bool eq = u[r] == tau;
    if (simple) {
      sel |= eq;
    } else {
      const uint32_t be = __ballot_sync(0xffffffffu, eq);
      if (eq) sel = eq_run + __popc(be & lt) < krem;
      eq_run += __popc(be);
    }
    masks[r] = __ballot_sync(0xffffffffu, sel);
    cnt += __popc(masks[r]);
  }
  if (lane == 0) S.wsum[warp] = cnt;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = S.wsum[lane];
    uint32_t c = w;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t z = __shfl_up_sync(0xffffffffu, c, off);
      if (lane >= off) c += z;
    }
    S.wsum[lane] = c - w;
    if (lane == 31) S.s_total = c;
  }
  __syncthreads();
  uint32_t base = (uint32_t)lo + S.wsum[warp];
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    const uint32_t mk = masks[r];
    if (mk == 0u) continue;                        // warp-uniform: most rows hold no kept item
    if ((mk >> lane) & 1u) out[base + __popc(mk & lt)] = lo + w0 + 32 * r + lane;
    base += __popc(mk);
  }
  const int n_chosen = (int)S.s_total;
  const int count = lo + n_chosen + p.n_recent;
  for (int i = tid; i < lo; i += kTopkThreads) out[i] = i;
  for (int i = tid; i < p.n_recent; i += kTopkThreads) out[lo + n_chosen + i] = hi + i;
  for (int i = count + tid; i < p.budget; i += kTopkThreads) out[i] = -1;
  if (tid == 0) p.count_out[unit] = count;
}

// Token-level selection with every score held in registers (up to 16 per thread), the count
// a template parameter so every pass is straight-line code.  Needs 0 < k < n <= ROWS * kTopkThreads.
template <int ROWS>
__global__ void __launch_bounds__(kTopkThreads, 1) topk_rows_kernel(const TopkParams p) {
  __shared__ TopkRowsSmem S;
  // the unit's scores on their way into L2 while the score kernel finishes (its K stream
  // has pushed the early ones out to DRAM by now)
  prefetch_lines_l2(p.score + (size_t)blockIdx.x * p.n_mid_pad, (size_t)p.n_mid_pad * 4, threadIdx.x, kTopkThreads);
  grid_dependency_wait();
  allow_dependent_launch();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int unit = blockIdx.x;
  const int t_u = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, tid == 0 ? p.status : nullptr);
  int32_t* out = p.idx_out + (size_t)unit * p.budget;
  if (topk_keep_all(p, unit, t_u, out)) return;
  const int lo = p.n_sink, hi = t_u - p.n_recent, n = hi - lo;
  const int k = p.budget - p.n_sink - p.n_recent;
  const float* sc = p.score + (size_t)unit * p.n_mid_pad;
  const int w0 = warp * ROWS * 32;
  uint32_t u[ROWS];
  float lmin = INFINITY, lmax = -INFINITY;
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    const int i = w0 + 32 * r + lane;
    const float v = i < n ? __ldcg(sc + i) : 0.f;
    u[r] = __float_as_uint(v);
    lmin = fminf(lmin, v);
    lmax = fmaxf(lmax, v);
  }
  rows_compact_tokens<ROWS>(S, u, rows_threshold<ROWS>(S, u, lmin, lmax, k), p, unit, lo, hi, out);
}

// Chunk-level selection (chunk = s > 1, the paper's policy) with every chunk's score in
// registers.  Chunk c covers positions [c s, c s + s) clipped to the middle [lo, hi), so the
// first and the last may hold fewer, and scores the sum of its members' scores in position
// order; the top k = floor(free / s) chunks (ties to the lower chunk) by rows_threshold are
// written member by member in position order.  Items are the chunks, n_items <= ROWS *
// kTopkThreads; a unit with no chunk to rank keeps all of them or none.
template <int ROWS>
__global__ void __launch_bounds__(kTopkThreads, 1) topk_rows_chunk_kernel(const TopkParams p) {
  __shared__ TopkRowsSmem S;
  prefetch_lines_l2(p.score + (size_t)blockIdx.x * p.n_mid_pad, (size_t)p.n_mid_pad * 4, threadIdx.x, kTopkThreads);
  grid_dependency_wait();
  allow_dependent_launch();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int unit = blockIdx.x;
  const int t_u = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, tid == 0 ? p.status : nullptr);
  int32_t* out = p.idx_out + (size_t)unit * p.budget;
  if (topk_keep_all(p, unit, t_u, out)) return;
  const int lo = p.n_sink, hi = t_u - p.n_recent, s = p.chunk;
  const int c_first = lo / s;
  const int n_items = hi > lo ? (hi - 1) / s - c_first + 1 : 0;
  const int k = min((p.budget - p.n_sink - p.n_recent) / s, n_items);
  const bool take_all = k >= n_items, ranked = k > 0 && !take_all;
  const float* sc = p.score + (size_t)unit * p.n_mid_pad;
  const int w0 = warp * ROWS * 32;
  auto members = [&](int i, int& a, int& b) {
    const int c = c_first + i;
    a = max(c * s, lo);
    b = min(c * s + s, hi);
  };

  // ---- chunk scores: members summed in position order, their loads eight at a time (four
  // rows' chunks in flight together; the zeros past b add nothing to scores >= +0)
  constexpr int RB = ROWS < 4 ? ROWS : 4;
  uint32_t u[ROWS];
  float lmin = INFINITY, lmax = -INFINITY;
#pragma unroll
  for (int r0 = 0; r0 < ROWS; r0 += RB) {
    int ma[RB], mb[RB];
    float v[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int i = w0 + 32 * (r0 + r) + lane;
      ma[r] = 0;
      mb[r] = 0;
      if (i < n_items) members(i, ma[r], mb[r]);
      v[r] = 0.f;
    }
    for (int q0 = 0; q0 < s; q0 += 8) {
      float t[RB][8];
#pragma unroll
      for (int r = 0; r < RB; ++r)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int q = ma[r] + q0 + j;
          t[r][j] = q < mb[r] ? __ldcg(sc + (q - lo)) : 0.f;
        }
#pragma unroll
      for (int r = 0; r < RB; ++r)
#pragma unroll
        for (int j = 0; j < 8; ++j) v[r] += t[r][j];
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      u[r0 + r] = __float_as_uint(v[r]);            // +0 past n_items
      lmin = fminf(lmin, v[r]);
      lmax = fmaxf(lmax, v[r]);
    }
  }
  RowsThreshold th{0u, 0u, true};
  if (ranked) th = rows_threshold<ROWS>(S, u, lmin, lmax, k);

  // ---- kept chunks, their members in position order
  const uint32_t lt = (1u << lane) - 1u;
  uint32_t eq_base = 0;
  if (ranked && !th.simple) {   // chunks equal to tau are taken in chunk order: those before this warp
    uint32_t eqc = 0;
#pragma unroll
    for (int r = 0; r < ROWS; ++r) eqc += __popc(__ballot_sync(0xffffffffu, w0 + 32 * r + lane < n_items && u[r] == th.tau));
    if (lane == 0) S.wsum[warp] = eqc;
    __syncthreads();
    eq_base = __reduce_add_sync(0xffffffffu, lane < warp ? S.wsum[lane] : 0u);
    __syncthreads();
  }
  bool sel[ROWS];
  int incl[ROWS], rowoff[ROWS];
  int warp_pos = 0;
  uint32_t eq_run = eq_base;
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    const bool real = w0 + 32 * r + lane < n_items;
    bool sl = real && (take_all || (ranked && u[r] > th.tau));
    const bool eq = real && ranked && u[r] == th.tau;
    const uint32_t be = __ballot_sync(0xffffffffu, eq);
    if (eq) sl = th.simple || eq_run + __popc(be & lt) < th.krem;
    eq_run += __popc(be);
    sel[r] = sl;
    int a = 0, b = 0;
    if (real) members(w0 + 32 * r + lane, a, b);
    const int m = sl ? b - a : 0;
    int c = m;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, c, off);
      if (lane >= off) c += y;
    }
    incl[r] = c;
    rowoff[r] = warp_pos;
    warp_pos += __shfl_sync(0xffffffffu, c, 31);
  }
  if (lane == 0) S.wpos[warp] = (uint32_t)warp_pos;
  __syncthreads();
  const int base = lo + (int)__reduce_add_sync(0xffffffffu, lane < warp ? S.wpos[lane] : 0u);
  const int n_chosen = (int)__reduce_add_sync(0xffffffffu, S.wpos[lane]);
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    if (sel[r]) {
      int a, b;
      members(w0 + 32 * r + lane, a, b);
      int o = base + rowoff[r] + incl[r] - (b - a);
      for (int q = a; q < b; ++q) out[o++] = q;
    }
  }
  const int count = lo + n_chosen + p.n_recent;
  for (int i = tid; i < lo; i += kTopkThreads) out[i] = i;
  for (int i = tid; i < p.n_recent; i += kTopkThreads) out[lo + n_chosen + i] = hi + i;
  for (int i = count + tid; i < p.budget; i += kTopkThreads) out[i] = -1;
  if (tid == 0) p.count_out[unit] = count;
}

// ============================================================================ host side

namespace {
struct ScoreKernel {
  void* fn;
  int stages, nqb;
};
// Two window-query buffers (a unit switch inside a CTA's range does not stall) and four
// K stages when they fit, else one Q buffer and as many stages as fit (measured: a fifth
// stage does not speed the kernel up).
ScoreKernel score_fn(int d, int nq_pad, bool ragged) {
  const size_t qbytes = (size_t)nq_pad * d * 2;
  const size_t kt = (size_t)kSKeys * d * 2;
  const size_t budget = 227 * 1024 - 1024 - kSQOffset;
  int stages = 4, nqb = 2;
  if (2 * qbytes + 4 * kt > budget) {
    nqb = 1;
    if (qbytes + 5 * kt <= budget) stages = 5;
  }
#define BD_SK(DD, ST, NB)                                                                              \
  if (d == DD && stages == ST && nqb == NB)                                                              \
    return {ragged ? reinterpret_cast<void*>(&score_kernel<DD, ST, NB, true>)                            \
                   : reinterpret_cast<void*>(&score_kernel<DD, ST, NB, false>), ST, NB};
  BD_SK(64, 5, 1) BD_SK(64, 4, 2) BD_SK(64, 4, 1) BD_SK(128, 5, 1) BD_SK(128, 4, 2) BD_SK(128, 4, 1)
#undef BD_SK
  return {nullptr, 0, 0};
}

uint32_t pow2_at_least(uint32_t x) {
  uint32_t r = 32;
  while (r < x) r <<= 1;
  return r;
}
}  // namespace

bool select_plan(const bd_shape& s, int window, int budget, int n_sink, int n_recent, int chunk,
                 SelectPlan* plan) {
  *plan = SelectPlan{};
  const int group = s.h_q / s.h_kv;
  const int units = s.batch * s.h_kv;
  plan->keep_all = budget >= s.t_ctx;
  plan->nq_rows = group * window;
  plan->nq_pad = (int)align_up(plan->nq_rows, 16);
  plan->n_mid = std::max(0, s.t_ctx - n_sink - n_recent);
  plan->n_mid_pad = (int)align_up(std::max(plan->n_mid, 1), 4);
  const int free = budget - n_sink - n_recent;
  plan->need_scores = !plan->keep_all && plan->n_mid > 0 && free / chunk > 0;
  if (plan->nq_pad > 256) return false;
  const ScoreKernel sk = score_fn(s.head_dim, plan->nq_pad, s.seq_lens != nullptr);
  if (!sk.fn) return false;
  plan->tiles_per_unit = (plan->n_mid + kSKeys - 1) / kSKeys;
  plan->total_tiles = plan->tiles_per_unit * units;
  plan->grid = std::max(1, std::min(plan->total_tiles, current_sm_count()));
  plan->tiles_per_cta = (plan->total_tiles + plan->grid - 1) / plan->grid;
  plan->grid = std::max(1, (plan->total_tiles + plan->tiles_per_cta - 1) / plan->tiles_per_cta);
  plan->stages = sk.stages;
  plan->nqb = sk.nqb;
  const uint32_t acc_stride = (uint32_t)align_up(plan->nq_pad, 32);
  plan->n_acc = 4u * acc_stride <= 512u ? 4 : 2;
  plan->tmem_cols = pow2_at_least((uint32_t)plan->n_acc * acc_stride);
  plan->smem_bytes = 1024 + kSQOffset + (size_t)sk.nqb * plan->nq_pad * s.head_dim * 2 +
                     (size_t)sk.stages * kSKeys * s.head_dim * 2;
  if (s.seq_lens) {   // the units' tile table of per-sequence lengths
    plan->smem_bytes += align_up((size_t)(units + 1) * 4, 16);
    if (plan->smem_bytes > 227 * 1024) return false;
  }
  plan->score_bytes = plan->need_scores ? align_up((size_t)units * plan->n_mid_pad * 4, 256) : 0;
  plan->lse_bytes = align_up((size_t)s.batch * s.h_q * window * 4, 256);
  // self mode's window LSE (carry mode does not need it): window_lse_kernel on the tensor
  // cores for up to 128 window rows per KV head (with per-sequence lengths a unit spans at
  // most kLMaxSeg CTA ranges), else the lse-only verify kernel
  plan->lse_tc = plan->nq_rows <= 128 && (long)units * plan->nq_rows >= 128;
  if (plan->lse_tc) {
    const int tpu = (s.t_ctx + kSKeys - 1) / kSKeys;
    const long total = (long)units * tpu;
    if (total >= (1L << 31)) return false;
    int grid = (int)std::max<long>(1, std::min<long>(total, current_sm_count()));
    int tpc = (int)((total + grid - 1) / grid);
    int max_seg = 1;
    if (s.seq_lens) {
      // the lengths are read on the device: every SM gets a CTA, and the range per CTA is
      // bounded below so that a unit of tpu tiles spans at most kLMaxSeg ranges
      grid = current_sm_count();
      tpc = (tpu + kLMaxSeg - 2) / (kLMaxSeg - 1);
      max_seg = kLMaxSeg;
    } else {
      grid = (int)((total + tpc - 1) / tpc);
      for (long u = 0; u < units; ++u)
        max_seg = std::max(max_seg, (int)((u * tpu + tpu - 1) / tpc - (u * tpu) / tpc + 1));
    }
    plan->lse_tiles_per_unit = tpu;
    plan->lse_total_tiles = (int)total;
    plan->lse_tiles_per_cta = tpc;
    plan->lse_grid = grid;
    plan->lse_max_seg = max_seg;
    plan->lse_smem_bytes = 2048 + (size_t)2 * 128 * s.head_dim * 2 + (size_t)kLStages * kSKeys * s.head_dim * 2 +
                           2 * 128 * sizeof(float2) + (s.seq_lens ? align_up((size_t)(units + 1) * 4, 16) : 0);
    plan->lse_part_bytes = max_seg > 1 ? align_up((size_t)units * max_seg * 128 * sizeof(float2), 256) : 0;
    // a units' table too large for shared memory: the lse-only verify kernel below instead
    plan->lse_tc = plan->lse_smem_bytes <= 227 * 1024;
  }
  if (plan->lse_tc) {
    plan->self_mode = true;
  } else {
    bd_shape ls = s;
    ls.t_ctx = s.t_ctx - window;
    plan->self_mode = verify_plan(ls, window, false, &plan->lse_plan);
  }
  return true;
}

size_t select_region_bytes(const bd_shape& s, const SelectPlan& plan) {
  if (!plan.self_mode) return plan.score_bytes;
  bd_shape ls = s;
  ls.t_ctx = s.t_ctx - plan.nq_rows / std::max(1, s.h_q / s.h_kv);
  return plan.score_bytes + plan.lse_bytes +
         (plan.lse_tc ? plan.lse_part_bytes : verify_partials_bytes(ls, plan.lse_plan));
}

cudaError_t launch_select(const bd_shape& s, const SelectPlan& plan, const void* k_cache,
                          const void* q_window, const float* window_lse, int window, int budget,
                          int n_sink, int n_recent, int chunk, unsigned flags, int32_t* idx_out, int32_t* count_out,
                          void* ws_region, int* counters, int* status, cudaStream_t stream) {
  const int units = s.batch * s.h_kv;
  uint8_t* region = static_cast<uint8_t*>(ws_region);
  float* score = reinterpret_cast<float*>(region);
  cudaError_t err;
  if (plan.need_scores) {
    const float* lse = window_lse;
    if (lse == nullptr) {   // self mode: window LSE over [0, p_w]
      float* lse_buf = reinterpret_cast<float*>(region + plan.score_bytes);
      if (plan.lse_tc) {
        CUtensorMap lkmap, lqmap;
        err = make_cache_map(&lkmap, k_cache, units, s.t_cap, s.t_ctx, s.head_dim, kSKeys);
        if (err != cudaSuccess) return err;
        err = make_rows_map(&lqmap, q_window, (long long)units * plan.nq_rows, s.head_dim, 128);
        if (err != cudaSuccess) return err;
        LseParams lp;
        lp.q_win = static_cast<const __nv_bfloat16*>(q_window);
        lp.lse = lse_buf;
        lp.part = reinterpret_cast<float2*>(region + plan.score_bytes + plan.lse_bytes);
        lp.counters = counters;
        lp.status = status;
        lp.nq_rows = plan.nq_rows;
        lp.window = window;
        lp.t_ctx = s.t_ctx;
        lp.tiles_per_unit = plan.lse_tiles_per_unit;
        lp.total_tiles = plan.lse_total_tiles;
        lp.tiles_per_cta = plan.lse_tiles_per_cta;
        lp.max_seg = plan.lse_max_seg;
        lp.window_ready = (flags & BD_SELECT_WINDOW_READY) ? 1 : 0;
        lp.seq_lens = s.seq_lens;
        lp.h_kv = s.h_kv;
        lp.units = units;
        lp.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
        void* lfn = s.seq_lens ? (s.head_dim == 64 ? reinterpret_cast<void*>(&window_lse_kernel<64, true>)
                                                   : reinterpret_cast<void*>(&window_lse_kernel<128, true>))
                               : (s.head_dim == 64 ? reinterpret_cast<void*>(&window_lse_kernel<64, false>)
                                                   : reinterpret_cast<void*>(&window_lse_kernel<128, false>));
        err = cudaFuncSetAttribute(lfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.lse_smem_bytes);
        if (err != cudaSuccess) return err;
        void* largs[] = {&lp, &lkmap, &lqmap};
        err = launch_kernel(lfn, dim3(plan.lse_grid), dim3(kLThreads), plan.lse_smem_bytes, stream, largs, 0);
      } else {
        bd_shape ls = s;
        ls.t_ctx = s.t_ctx - window;
        err = launch_verify(ls, plan.lse_plan, window, q_window, k_cache, nullptr, nullptr, lse_buf,
                            region + plan.score_bytes + plan.lse_bytes, counters, status, stream, -window);
      }
      if (err != cudaSuccess) return err;
      lse = lse_buf;
    }
    CUtensorMap kmap, qmap;
    err = make_cache_map(&kmap, k_cache, units, s.t_cap, s.t_ctx, s.head_dim, kSKeys);
    if (err != cudaSuccess) return err;
    err = make_rows_map(&qmap, q_window, (long long)units * plan.nq_rows, s.head_dim, plan.nq_pad);
    if (err != cudaSuccess) return err;
    ScoreParams p;
    p.q_win = static_cast<const __nv_bfloat16*>(q_window);
    p.lse_win = lse;
    p.score = score;
    p.status = status;
    p.nq_rows = plan.nq_rows;
    p.nq_pad = plan.nq_pad;
    p.window = window;
    p.t_ctx = s.t_ctx;
    p.n_sink = n_sink;
    p.mid_end = s.t_ctx - n_recent;
    p.n_mid_pad = plan.n_mid_pad;
    p.tiles_per_unit = plan.tiles_per_unit;
    p.total_tiles = plan.total_tiles;
    p.tiles_per_cta = plan.tiles_per_cta;
    p.acc_stride = (int)align_up(plan.nq_pad, 32);
    p.n_acc = plan.n_acc;
    p.tmem_cols = plan.tmem_cols;
    p.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
    p.seq_lens = s.seq_lens;
    p.h_kv = s.h_kv;
    p.window_ready = (flags & BD_SELECT_WINDOW_READY) ? 1 : 0;
    void* fn = score_fn(s.head_dim, plan.nq_pad, s.seq_lens != nullptr).fn;
    err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem_bytes);
    if (err != cudaSuccess) return err;
    void* args[] = {&p, &kmap, &qmap};
    err = launch_kernel(fn, dim3(plan.grid), dim3(kSThreads), plan.smem_bytes, stream, args, 0);
    if (err != cudaSuccess) return err;
  }
  TopkParams tp;
  tp.score = score;
  tp.idx_out = idx_out;
  tp.count_out = count_out;
  tp.t_ctx = s.t_ctx;
  tp.budget = budget;
  tp.n_sink = n_sink;
  tp.n_recent = n_recent;
  tp.chunk = chunk;
  tp.n_mid_pad = plan.n_mid_pad;
  tp.keep_all = plan.keep_all ? 1 : 0;
  tp.seq_lens = s.seq_lens;
  tp.h_kv = s.h_kv;
  tp.status = status;
  void* targs[] = {&tp};
  const int free = budget - n_sink - n_recent;
  if (!plan.keep_all && plan.need_scores && chunk == 1 && free < plan.n_mid && plan.n_mid <= 16 * kTopkThreads) {
    const int rows = (plan.n_mid + kTopkThreads - 1) / kTopkThreads;
    void* fn = rows <= 1   ? reinterpret_cast<void*>(&topk_rows_kernel<1>)
               : rows <= 2 ? reinterpret_cast<void*>(&topk_rows_kernel<2>)
               : rows <= 4 ? reinterpret_cast<void*>(&topk_rows_kernel<4>)
               : rows <= 8 ? reinterpret_cast<void*>(&topk_rows_kernel<8>)
                           : reinterpret_cast<void*>(&topk_rows_kernel<16>);
    return launch_kernel(fn, dim3(units), dim3(kTopkThreads), 0, stream, targs, 0);
  }
  if (!plan.keep_all && plan.need_scores && chunk == 1 && plan.n_mid <= kLeanMaxItems && free < plan.n_mid) {
    const size_t smem = (size_t)align_up(plan.n_mid, 4) * 4;
    void* fn = reinterpret_cast<void*>(&topk_token_kernel);
    err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    return launch_kernel(fn, dim3(units), dim3(kTopkThreads), smem, stream, targs, 0);
  }
  if (!plan.keep_all && plan.need_scores && chunk > 1) {
    // chunks of the longest middle: the register kernel while it holds them
    const int lo = n_sink, hi = s.t_ctx - n_recent;
    const int n_items = hi > lo ? (hi - 1) / chunk - lo / chunk + 1 : 0;
    if (n_items <= 16 * kTopkThreads) {
      const int rows = std::max(1, (n_items + kTopkThreads - 1) / kTopkThreads);
      void* fn = rows <= 1   ? reinterpret_cast<void*>(&topk_rows_chunk_kernel<1>)
                 : rows <= 2 ? reinterpret_cast<void*>(&topk_rows_chunk_kernel<2>)
                 : rows <= 4 ? reinterpret_cast<void*>(&topk_rows_chunk_kernel<4>)
                 : rows <= 8 ? reinterpret_cast<void*>(&topk_rows_chunk_kernel<8>)
                             : reinterpret_cast<void*>(&topk_rows_chunk_kernel<16>);
      return launch_kernel(fn, dim3(units), dim3(kTopkThreads), 0, stream, targs, 0);
    }
  }
  const int extra = kBins * 4 + kBinCandMax * 8 + 16;      // histogram + boundary-bin candidates
  const int max_items = (kTopkSmemBytes - extra) / 4;
  const int n_items = plan.n_mid;                     // upper bound for chunk mode as well
  tp.smem_items = std::min(n_items, max_items);
  const size_t smem = (size_t)((tp.smem_items + 1) & ~1) * 4 + extra;
  err = cudaFuncSetAttribute(reinterpret_cast<void*>(&topk_kernel), cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
  if (err != cudaSuccess) return err;
  return launch_kernel(reinterpret_cast<void*>(&topk_kernel), dim3(units), dim3(kTopkThreads), smem, stream, targs,
                       0);
}

}  // namespace bd
