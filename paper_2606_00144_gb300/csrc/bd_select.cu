// KV-budget selection (Sec. 3.4 TopKChunks; Algorithm 2, sparsify) in two kernels:
//
// score_kernel  (tcgen05)  score[k] = sum_{h in group, w < W, k <= p_w} exp2(s_{h,w,k} log2e/sqrt(d)
//               - lse_{h,w} log2e) for every middle key k.  Keys sit on the M side of the
//               UMMA (128 keys per tile = the 128 TMEM lanes) and the group's window query
//               rows on N, so every epilogue thread owns one key and reduces its own TMEM
//               row: no cross-thread reduction.  Persistent CTAs (one per SM):
//                 warp 0   producer: K tiles by TMA (128-byte swizzle, 4-stage ring) and the
//                          unit's window queries into a double-buffered swizzled Q tile;
//                 warp 1   one lane issues tcgen05.mma into a double-buffered fp32 TMEM
//                          accumulator and commits to the smem/TMEM barriers;
//                 warps 2-5 epilogue: tcgen05.ld, ex2 (MUFU), row sums, coalesced store.
// topk_kernel   one CTA per (sequence, KV head): 4-pass MSB radix select on the fp32 score
//               bits (warp-aggregated shared histograms), lower-index tie break by a block
//               scan over the equal keys, ascending compaction with sinks and recents.
#include <algorithm>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

constexpr int kSKeys = 128;          // keys per tile (UMMA M)
constexpr int kSThreads = 192;       // producer, MMA, 4 epilogue warps
constexpr int kTopkThreads = 1024;

struct ScoreParams {
  const __nv_bfloat16* q_win;   // [units * nq_rows][D]
  const float* lse_win;         // [units * nq_rows] natural log
  float* score;                 // [units][n_mid_pad]
  int* status;
  int nq_rows, nq_pad, window, t_ctx, n_sink, mid_end, n_mid_pad;
  int tiles_per_unit, total_tiles, tiles_per_cta;
  int acc_stride;               // TMEM columns between the two accumulators
  uint32_t tmem_cols;
  float scale_log2;
};

template <int D, int STAGES>
__global__ void __launch_bounds__(kSThreads, 1) score_kernel(const ScoreParams p,
                                                             const __grid_constant__ CUtensorMap kmap) {
  constexpr uint32_t KHALF = kSKeys * 128;         // one 64-column half of a K tile
  constexpr uint32_t KTILE = kSKeys * D * 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty_bar = full_bar + STAGES;
  uint64_t* tfull_bar = empty_bar + STAGES;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint64_t* qfull_bar = tempty_bar + 2;
  uint64_t* qempty_bar = qfull_bar + 2;
  uint64_t* drain_bar = qempty_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* lse2_s = reinterpret_cast<float*>(smem + 1024);     // [288]
  int* pw_s = reinterpret_cast<int*>(smem + 2304);            // [288]
  const uint32_t qbytes = (uint32_t)p.nq_pad * D * 2;
  uint8_t* qbuf = smem + 4096;                                 // 2 x qbytes
  uint8_t* kstage = qbuf + 2 * qbytes;                         // STAGES x KTILE (1024-aligned)

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int first = blockIdx.x * p.tiles_per_cta;
  const int n = max(0, min(p.tiles_per_cta, p.total_tiles - first));

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], 4);
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
    if (lane == 0) tma_prefetch_map(&kmap);
    int cur_unit = -1, qcount = 0;
    for (int i = 0; i < n; ++i) {
      const int g = first + i;
      const int unit = g / p.tiles_per_unit, tt = g % p.tiles_per_unit;
      if (unit != cur_unit) {
        const int qs = qcount & 1;
        bool ok = true;
        if (qcount >= 2) ok = mbar_wait(&qempty_bar[qs], ((qcount >> 1) - 1) & 1, p.status, abort_flag);
        if (!__all_sync(0xffffffffu, ok)) break;
        uint8_t* qb = qbuf + qs * qbytes;
        const __nv_bfloat16* src = p.q_win + (size_t)unit * p.nq_rows * D;
        const uint32_t half_bytes = (uint32_t)p.nq_pad * 128;
        for (int c = lane; c < p.nq_pad * (D / 8); c += 32) {
          const int r = c / (D / 8), ch = c % (D / 8);
          uint4 val = make_uint4(0u, 0u, 0u, 0u);
          if (r < p.nq_rows) val = __ldg(reinterpret_cast<const uint4*>(src + (size_t)r * D + ch * 8));
          *reinterpret_cast<uint4*>(qb + sw128_offset(r, ch * 8, half_bytes)) = val;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&qfull_bar[qs]);
        cur_unit = unit;
        ++qcount;
      }
      bool ok = true;
      if (lane == 0) {
        const int s = i % STAGES;
        if (i >= STAGES) ok = mbar_wait(&empty_bar[s], ((i / STAGES) & 1) ^ 1, p.status, abort_flag);
        if (ok) {
          uint8_t* st = kstage + s * KTILE;
          mbar_arrive_expect_tx(&full_bar[s], KTILE);
          const int key0 = p.n_sink + kSKeys * tt;
#pragma unroll
          for (int h = 0; h < D / 64; ++h) tma_load_3d(st + h * KHALF, &kmap, &full_bar[s], 64 * h, key0, unit);
        }
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kSKeys, p.nq_pad);
      int cur_unit = -1, qcount = 0;
      for (int i = 0; i < n; ++i) {
        const int g = first + i;
        const int unit = g / p.tiles_per_unit;
        const bool last_of_unit = (i == n - 1) || ((g + 1) / p.tiles_per_unit != unit);
        if (unit != cur_unit) {
          if (!mbar_wait(&qfull_bar[qcount & 1], (qcount >> 1) & 1, p.status, abort_flag)) break;
          cur_unit = unit;
          ++qcount;
        }
        const int qs = (qcount - 1) & 1;
        const int s = i % STAGES;
        if (!mbar_wait(&full_bar[s], (i / STAGES) & 1, p.status, abort_flag)) break;
        const int acc = i & 1;
        if (i >= 2 && !mbar_wait(&tempty_bar[acc], ((i >> 1) & 1) ^ 1, p.status, abort_flag)) break;
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
        if (last_of_unit) tc_commit(&qempty_bar[qs]);
      }
      // every MMA this thread issued has completed before TMEM is released
      tc_commit(drain_bar);
      mbar_wait(drain_bar, 0, p.status, nullptr);
    }
  } else {
    // ---------------------------------------------------------------- epilogue (warps 2..5)
    const int quad = warp & 3;                  // TMEM lanes quad*32 .. quad*32+31
    const int ep_tid = tid - 64;
    const int win0 = p.t_ctx - p.window;        // position of window row 0
    int cur_unit = -1;
    for (int i = 0; i < n; ++i) {
      const int g = first + i;
      const int unit = g / p.tiles_per_unit, tt = g % p.tiles_per_unit;
      if (unit != cur_unit) {
        named_bar(1, 128);
        for (int c = ep_tid; c < 288; c += 128) {
          const bool real = c < p.nq_rows;
          lse2_s[c] = real ? __ldg(p.lse_win + (size_t)unit * p.nq_rows + c) * kLog2e : INFINITY;
          pw_s[c] = real ? win0 + c % p.window : -1;
        }
        named_bar(1, 128);
        cur_unit = unit;
      }
      const int acc = i & 1;
      if (!mbar_wait(&tfull_bar[acc], (i >> 1) & 1, p.status, abort_flag)) break;
      tc_fence_after();
      const int key_tile0 = p.n_sink + kSKeys * tt;
      const int key = key_tile0 + quad * 32 + lane;
      const bool causal = key_tile0 + kSKeys - 1 > win0;   // some key may follow a window row
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(acc * p.acc_stride);
      float sum = 0.f;
      for (int c0 = 0; c0 < p.nq_pad; c0 += 32) {
        float v[32];
        tc_ld_32cols(taddr + c0, v);
        tc_wait_ld();
        const int ncol = min(32, p.nq_pad - c0);
        if (ncol == 32 && !causal) {
#pragma unroll
          for (int j = 0; j < 32; ++j) sum += fast_exp2(fmaf(v[j], p.scale_log2, -lse2_s[c0 + j]));
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            if (j < ncol) {
              const float x = key <= pw_s[c0 + j] ? fmaf(v[j], p.scale_log2, -lse2_s[c0 + j]) : -INFINITY;
              sum += fast_exp2(x);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar[acc]);
      if (key < p.mid_end) p.score[(size_t)unit * p.n_mid_pad + (key - p.n_sink)] = sum;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, p.tmem_cols);
}

// ============================================================================ top-B select

struct TopkParams {
  const float* score;      // [units][n_mid_pad]
  int32_t* idx_out;        // [units][budget]
  int32_t* count_out;      // [units]
  int t_ctx, budget, n_sink, n_recent, chunk, n_mid_pad;
  int keep_all;            // budget >= t_ctx
};

__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_sums, uint32_t* total) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t w = lane < (int)(blockDim.x >> 5) ? warp_sums[lane] : 0u;
    uint32_t incl = w;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    warp_sums[lane] = incl - w;               // exclusive prefix of warp totals
    if (lane == 31) *total = incl;
  }
  __syncthreads();
  const uint32_t r = warp_sums[warp] + x - v;
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kTopkThreads) topk_kernel(const TopkParams p) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t warp_sums[32];
  __shared__ uint32_t s_total, s_prefix, s_krem;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int unit = blockIdx.x;
  int32_t* out = p.idx_out + (size_t)unit * p.budget;

  if (p.keep_all) {
    for (int i = tid; i < p.budget; i += kTopkThreads) out[i] = i < p.t_ctx ? i : -1;
    if (tid == 0) p.count_out[unit] = p.t_ctx;
    return;
  }
  const int lo = p.n_sink, hi = p.t_ctx - p.n_recent;
  const int s = p.chunk;
  const int free = p.budget - p.n_sink - p.n_recent;
  const int c_first = lo / s;
  const int n_items = (hi > lo) ? ((hi - 1) / s - c_first + 1) : 0;
  const int k = min(free / s, n_items);
  const float* sc = p.score + (size_t)unit * p.n_mid_pad;

  auto item_value = [&](int i) -> uint32_t {
    if (s == 1) return __float_as_uint(__ldcg(sc + i));
    const int c = c_first + i;
    const int a = max(c * s, lo), b = min(c * s + s, hi);
    float v = 0.f;
    for (int q = a; q < b; ++q) v += __ldcg(sc + (q - lo));
    return __float_as_uint(v);
  };
  auto item_members = [&](int i, int& a, int& b) {
    const int c = c_first + i;
    a = max(c * s, lo);
    b = min(c * s + s, hi);
  };

  // ---- radix select: value bits of the k-th largest item, and how many equal ones to take
  uint32_t prefix = 0, mask = 0, krem = (uint32_t)k;
  const bool take_all = (k >= n_items), take_none = (k <= 0);
  if (!take_all && !take_none) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 256; i += kTopkThreads) hist[i] = 0;
      __syncthreads();
      for (int base = 0; base < n_items; base += kTopkThreads) {
        const int i = base + tid;
        uint32_t digit = 256;
        if (i < n_items) {
          const uint32_t u = item_value(i);
          if ((u & mask) == prefix) digit = (u >> shift) & 255u;
        }
        const uint32_t peers = __match_any_sync(0xffffffffu, digit);
        if (digit < 256 && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
      }
      __syncthreads();
      if (warp == 0) {
        // lane l owns digits 8l .. 8l+7; count of items with a larger digit than lane l's range
        uint32_t local = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) local += hist[8 * lane + j];
        uint32_t suffix = local;   // inclusive suffix sum over lanes >= lane
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
      __syncthreads();
    }
  }
  const uint32_t tau = prefix;

  // ---- compaction in item order (contiguous ranges per thread keep the output ascending)
  const int per = (n_items + kTopkThreads - 1) / kTopkThreads;
  const int i0 = min(n_items, tid * per), i1 = min(n_items, i0 + per);
  uint32_t eq_local = 0;
  if (!take_all && !take_none)
    for (int i = i0; i < i1; ++i) eq_local += (item_value(i) == tau);
  const uint32_t eq_base = block_exclusive_scan(eq_local, warp_sums, &s_total);
  auto selected = [&](int i, uint32_t& eq_seen) -> bool {
    if (take_all) return true;
    if (take_none) return false;
    const uint32_t u = item_value(i);
    if (u > tau) return true;
    if (u == tau) return (eq_base + eq_seen++) < krem;
    return false;
  };
  uint32_t npos_local = 0;
  {
    uint32_t eq_seen = 0;
    for (int i = i0; i < i1; ++i)
      if (selected(i, eq_seen)) {
        int a, b;
        item_members(i, a, b);
        npos_local += (uint32_t)(b - a);
      }
  }
  const uint32_t pos_base = block_exclusive_scan(npos_local, warp_sums, &s_total);
  const uint32_t n_chosen = s_total;
  {
    uint32_t eq_seen = 0, w = (uint32_t)lo + pos_base;
    for (int i = i0; i < i1; ++i)
      if (selected(i, eq_seen)) {
        int a, b;
        item_members(i, a, b);
        for (int q = a; q < b; ++q) out[w++] = q;
      }
  }
  const int count = lo + (int)n_chosen + p.n_recent;
  for (int i = tid; i < lo; i += kTopkThreads) out[i] = i;
  for (int i = tid; i < p.n_recent; i += kTopkThreads) out[lo + n_chosen + i] = hi + i;
  for (int i = count + tid; i < p.budget; i += kTopkThreads) out[i] = -1;
  if (tid == 0) p.count_out[unit] = count;
}

// ============================================================================ host side

namespace {
constexpr int kSStages = 4;
void* score_fn(int d) {
  if (d == 64) return reinterpret_cast<void*>(&score_kernel<64, kSStages>);
  if (d == 128) return reinterpret_cast<void*>(&score_kernel<128, kSStages>);
  return nullptr;
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
  if (plan->nq_pad > 256 || !score_fn(s.head_dim)) return false;
  plan->tiles_per_unit = (plan->n_mid + kSKeys - 1) / kSKeys;
  plan->total_tiles = plan->tiles_per_unit * units;
  plan->grid = std::max(1, std::min(plan->total_tiles, current_sm_count()));
  plan->tiles_per_cta = (plan->total_tiles + plan->grid - 1) / plan->grid;
  plan->grid = std::max(1, (plan->total_tiles + plan->tiles_per_cta - 1) / plan->tiles_per_cta);
  plan->stages = kSStages;
  plan->tmem_cols = pow2_at_least(2u * (uint32_t)align_up(plan->nq_pad, 32));
  plan->smem_bytes = 1024 + 4096 + 2 * (size_t)plan->nq_pad * s.head_dim * 2 +
                     (size_t)kSStages * kSKeys * s.head_dim * 2;
  plan->score_bytes = plan->need_scores ? align_up((size_t)units * plan->n_mid_pad * 4, 256) : 0;
  plan->lse_bytes = align_up((size_t)s.batch * s.h_q * window * 4, 256);
  bd_shape ls = s;
  ls.t_ctx = s.t_ctx - window;
  if (!verify_plan(ls, window, false, &plan->lse_plan)) return false;
  return true;
}

size_t select_region_bytes(const bd_shape& s, const SelectPlan& plan) {
  bd_shape ls = s;
  return plan.score_bytes + plan.lse_bytes + verify_partials_bytes(ls, plan.lse_plan);
}

cudaError_t launch_select(const bd_shape& s, const SelectPlan& plan, const void* k_cache,
                          const void* q_window, const float* window_lse, int window, int budget,
                          int n_sink, int n_recent, int chunk, int32_t* idx_out, int32_t* count_out,
                          void* ws_region, int* counters, int* status, cudaStream_t stream) {
  const int units = s.batch * s.h_kv;
  uint8_t* region = static_cast<uint8_t*>(ws_region);
  float* score = reinterpret_cast<float*>(region);
  cudaError_t err;
  if (plan.need_scores) {
    const float* lse = window_lse;
    if (lse == nullptr) {   // self mode: window LSE over [0, p_w] through the verify kernel
      float* lse_buf = reinterpret_cast<float*>(region + plan.score_bytes);
      bd_shape ls = s;
      ls.t_ctx = s.t_ctx - window;
      err = launch_verify(ls, plan.lse_plan, window, q_window, k_cache, nullptr, nullptr, lse_buf,
                          region + plan.score_bytes + plan.lse_bytes, counters, status, stream);
      if (err != cudaSuccess) return err;
      lse = lse_buf;
    }
    CUtensorMap kmap;
    err = make_cache_map(&kmap, k_cache, units, s.t_cap, s.t_ctx, s.head_dim, kSKeys);
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
    p.tmem_cols = plan.tmem_cols;
    p.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
    void* fn = score_fn(s.head_dim);
    err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem_bytes);
    if (err != cudaSuccess) return err;
    void* args[] = {&p, &kmap};
    err = cudaLaunchKernel(fn, dim3(plan.grid), dim3(kSThreads), args, plan.smem_bytes, stream);
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
  topk_kernel<<<units, kTopkThreads, 0, stream>>>(tp);
  return cudaGetLastError();
}

}  // namespace bd
