// Drafter decode pass over the sparse view (Algorithm 2, Draft): one query per head,
// keys = the selected rows idx[0:count] plus the drafted rows t_ctx .. t_ctx+step_j.
//
// Memory-bound gather (4 flop per byte): the G query heads of a GQA group share every
// gathered row, so one CTA serves one (sequence, KV head) unit and one slice of its entry
// list.  Rows are gathered with 16-byte cp.async into padded shared-memory tiles (K
// first, V behind it so its latency overlaps the QK^T), scores and softmax run in fp32 on
// CUDA cores with warp-shuffle reductions, and a slice longer than one tile is folded in
// with an online softmax.  Each CTA writes a normalised partial; the last CTA of a unit
// merges them (log-sum-exp) into the bf16 output.
#include <algorithm>
#include <mutex>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

constexpr int kDRows = 64;        // rows per shared-memory tile
constexpr int kDThreads = 128;

struct DraftParams {
  const __nv_bfloat16* q;      // [units * G][D]
  const __nv_bfloat16* k;      // [units][t_cap][D]
  const __nv_bfloat16* v;
  const int32_t* idx;          // [units][budget]
  const int32_t* count;        // [units]
  __nv_bfloat16* o;            // [units * G][D]
  float* lse;                  // [units * G] or null
  float* o_part;               // [n_split][units * G][D]
  float* lse_part;             // [n_split][units * G]
  int* counters;
  int* status;
  int units, budget, step_j, t_ctx, t_cap, n_split, rows_per_split;
  float scale_log2;
};

template <int D, int G>
__global__ void __launch_bounds__(kDThreads) draft_kernel(const DraftParams p) {
  constexpr int PITCH = D + 8;                 // bf16 per tile row (16-byte pad: conflict-free)
  constexpr int TPR = kDThreads / kDRows;      // threads per row in the score phase
  constexpr int DP = D / 2;                    // bf16 pairs per row
  constexpr int RG = kDThreads / DP;           // row groups in the PV phase
  __shared__ __align__(16) __nv_bfloat16 ks[kDRows * PITCH];
  __shared__ __align__(16) __nv_bfloat16 vs[kDRows * PITCH];
  __shared__ float qf[G * D];
  __shared__ float sc[kDRows * G];
  __shared__ int rowpos[kDRows];
  __shared__ float m_run[G], l_run[G], alpha_s[G];
  __shared__ int last_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int split = blockIdx.x, unit = blockIdx.y;
  int cnt = p.count[unit];
  if (cnt < 0 || cnt > p.budget) {
    if (tid == 0) record_error(p.status, BD_ERR_INVALID_ARG);
    cnt = min(max(cnt, 0), p.budget);
  }
  const int n_entries = cnt + p.step_j + 1;
  const int e_begin = split * p.rows_per_split;
  const int e_end = min(e_begin + p.rows_per_split, n_entries);

  const __nv_bfloat16* qsrc = p.q + (size_t)unit * G * D;
  for (int i = tid; i < G * D; i += kDThreads) qf[i] = __bfloat162float(qsrc[i]);
  if (tid < G) {
    m_run[tid] = -INFINITY;
    l_run[tid] = 0.f;
  }
  const __nv_bfloat16* kunit = p.k + (size_t)unit * p.t_cap * D;
  const __nv_bfloat16* vunit = p.v + (size_t)unit * p.t_cap * D;
  const int32_t* iunit = p.idx + (size_t)unit * p.budget;

  float acc[G][2];
#pragma unroll
  for (int g = 0; g < G; ++g) acc[g][0] = acc[g][1] = 0.f;
  const int dp = tid % DP, rg = tid / DP;

  for (int e0 = e_begin; e0 < e_end; e0 += kDRows) {
    const int nrows = min(kDRows, e_end - e0);
    __syncthreads();                           // previous tile fully consumed
    if (tid < nrows) {
      const int e = e0 + tid;
      int pos;
      if (e < cnt) {
        pos = __ldg(iunit + e);
        if (pos < 0 || pos >= p.t_ctx) {
          record_error(p.status, BD_ERR_INVALID_ARG);
          pos = -1;
        }
      } else {
        pos = p.t_ctx + (e - cnt);
      }
      rowpos[tid] = pos;
    }
    __syncthreads();
    // gather K rows, then V rows (two cp.async groups)
    for (int c = tid; c < nrows * (D / 8); c += kDThreads) {
      const int r = c / (D / 8), ch = c % (D / 8);
      const int pos = max(rowpos[r], 0);
      cp_async16(ks + r * PITCH + ch * 8, kunit + (size_t)pos * D + ch * 8);
    }
    cp_async_commit();
    for (int c = tid; c < nrows * (D / 8); c += kDThreads) {
      const int r = c / (D / 8), ch = c % (D / 8);
      const int pos = max(rowpos[r], 0);
      cp_async16(vs + r * PITCH + ch * 8, vunit + (size_t)pos * D + ch * 8);
    }
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();

    // scores: TPR threads per row, interleaved 16-byte chunks
    {
      const int r = tid / TPR, part = tid % TPR;
      float s[G];
#pragma unroll
      for (int g = 0; g < G; ++g) s[g] = 0.f;
#pragma unroll 4
      for (int ch = part; ch < D / 8; ch += TPR) {
        const uint4 raw = *reinterpret_cast<const uint4*>(ks + r * PITCH + ch * 8);
        const __nv_bfloat162* kv2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 kf = __bfloat1622float2(kv2[j]);
#pragma unroll
          for (int g = 0; g < G; ++g) {
            s[g] = fmaf(qf[g * D + ch * 8 + 2 * j], kf.x, s[g]);
            s[g] = fmaf(qf[g * D + ch * 8 + 2 * j + 1], kf.y, s[g]);
          }
        }
      }
#pragma unroll
      for (int off = 1; off < TPR; off <<= 1)
#pragma unroll
        for (int g = 0; g < G; ++g) s[g] += __shfl_xor_sync(0xffffffffu, s[g], off);
      if (part == 0) {
        const bool ok = r < nrows && rowpos[r] >= 0;
#pragma unroll
        for (int g = 0; g < G; ++g) sc[r * G + g] = ok ? s[g] * p.scale_log2 : -INFINITY;
      }
    }
    __syncthreads();
    // softmax bookkeeping per head (one warp per head, heads strided over the 4 warps)
    for (int g = warp; g < G; g += kDThreads / 32) {
      float mx = -INFINITY;
      for (int r = lane; r < kDRows; r += 32) mx = fmaxf(mx, sc[r * G + g]);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float m_old = m_run[g];
      const float m_new = fmaxf(m_old, mx);
      const float m_use = m_new == -INFINITY ? 0.f : m_new;
      float sum = 0.f;
      for (int r = lane; r < kDRows; r += 32) {
        const float pr = fast_exp2(sc[r * G + g] - m_use);
        sc[r * G + g] = pr;
        sum += pr;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      __syncwarp();
      if (lane == 0) {
        const float al = fast_exp2(m_old - m_use);
        alpha_s[g] = al;
        l_run[g] = l_run[g] * al + sum;
        m_run[g] = m_new;
      }
    }
    cp_async_wait<0>();
    __syncthreads();
    // O += P V (fp32), thread = (bf16 pair dp, row group rg)
#pragma unroll
    for (int g = 0; g < G; ++g) {
      acc[g][0] *= alpha_s[g];
      acc[g][1] *= alpha_s[g];
    }
    for (int r = rg; r < nrows; r += RG) {
      const float2 vf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(vs + r * PITCH + 2 * dp));
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float pr = sc[r * G + g];
        acc[g][0] = fmaf(pr, vf.x, acc[g][0]);
        acc[g][1] = fmaf(pr, vf.y, acc[g][1]);
      }
    }
  }

  // reduce the row groups, normalise, write
  __syncthreads();
  float* red = reinterpret_cast<float*>(ks);   // [RG][G][D] floats (fits in the K tile)
#pragma unroll
  for (int g = 0; g < G; ++g) {
    red[(rg * G + g) * D + 2 * dp] = acc[g][0];
    red[(rg * G + g) * D + 2 * dp + 1] = acc[g][1];
  }
  __syncthreads();
  const bool direct = p.n_split == 1;
  for (int i = tid; i < G * D; i += kDThreads) {
    const int g = i / D, d = i % D;
    float a = 0.f;
    for (int j = 0; j < RG; ++j) a += red[(j * G + g) * D + d];
    const float l = l_run[g];
    const float o = l > 0.f ? a / l : 0.f;
    const size_t row = (size_t)unit * G + g;
    if (direct) {
      p.o[row * D + d] = __float2bfloat16_rn(o);
    } else {
      p.o_part[((size_t)split * p.units * G + row) * D + d] = o;
    }
  }
  if (tid < G) {
    const float l = l_run[tid];
    const float lse = l > 0.f ? (m_run[tid] + log2f(l)) * kLn2 : -INFINITY;
    const size_t row = (size_t)unit * G + tid;
    if (direct) {
      if (p.lse) p.lse[row] = lse;
    } else {
      p.lse_part[(size_t)split * p.units * G + row] = lse;
    }
  }
  if (direct) return;

  __threadfence();
  __syncthreads();
  if (tid == 0) last_flag = (atomicAdd(&p.counters[unit], 1) == p.n_split - 1);
  __syncthreads();
  if (last_flag) {
    __threadfence();
    const size_t row0 = (size_t)unit * G;
    float* w = reinterpret_cast<float*>(vs);   // n_split * G floats
    merge_partials<D>(p.o_part + row0 * D, p.lse_part + row0, p.n_split, G, (size_t)p.units * G * D,
                      (size_t)p.units * G, p.o + row0 * D, p.lse ? p.lse + row0 : nullptr,
                      [](int r) { return r; }, w, tid, kDThreads, 0);
    if (tid == 0) p.counters[unit] = 0;
  }
}

// ============================================================================ host side

namespace {
using DraftFn = void (*)(DraftParams);
DraftFn pick(int d, int g) {
#define BD_DK(DD, GG) \
  if (d == DD && g == GG) return &draft_kernel<DD, GG>;
  BD_DK(64, 1) BD_DK(64, 2) BD_DK(64, 4) BD_DK(64, 8)
  BD_DK(128, 1) BD_DK(128, 2) BD_DK(128, 4) BD_DK(128, 8)
#undef BD_DK
  return nullptr;
}
}  // namespace

// The last CTA's merge weights (n_split * G floats) live in the V tile.
static int max_split_for_merge(int d, int g) { return (kDRows * (d + 8) * 2) / (g * 4); }

bool draft_plan(const bd_shape& s, int budget, int n_steps, DraftPlan* plan) {
  const int g = s.h_q / s.h_kv;
  if (!pick(s.head_dim, g)) return false;
  const int units = s.batch * s.h_kv;
  const long entries = (long)budget + n_steps;
  const int cap = std::max(1, 4 * current_sm_count() / std::max(1, units));
  int n_split = (int)std::min<long>((entries + kDRows - 1) / kDRows, cap);
  n_split = std::min(std::max(n_split, 1), max_split_for_merge(s.head_dim, g));
  plan->n_entries_max = (int)entries;
  plan->rows_per_split = (int)((entries + n_split - 1) / n_split);
  plan->n_split = (int)((entries + plan->rows_per_split - 1) / plan->rows_per_split);
  return true;
}

size_t draft_partials_bytes(const bd_shape& s, const DraftPlan& plan) {
  if (plan.n_split <= 1) return 0;
  const size_t rows = (size_t)plan.n_split * s.batch * s.h_q;
  return align_up(rows * s.head_dim * 4, 256) + align_up(rows * 4, 256);
}

cudaError_t launch_draft(const bd_shape& s, const DraftPlan& plan, const void* q, const void* k_cache,
                         const void* v_cache, const int32_t* idx, const int32_t* count, int budget,
                         int step_j, void* o_out, float* lse_out, void* ws_region, int* counters,
                         int* status, cudaStream_t stream) {
  const int units = s.batch * s.h_kv;
  DraftParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.k = static_cast<const __nv_bfloat16*>(k_cache);
  p.v = static_cast<const __nv_bfloat16*>(v_cache);
  p.idx = idx;
  p.count = count;
  p.o = static_cast<__nv_bfloat16*>(o_out);
  p.lse = lse_out;
  const size_t rows = (size_t)plan.n_split * s.batch * s.h_q;
  p.o_part = static_cast<float*>(ws_region);
  p.lse_part = reinterpret_cast<float*>(static_cast<uint8_t*>(ws_region) + align_up(rows * s.head_dim * 4, 256));
  p.counters = counters;
  p.status = status;
  p.units = units;
  p.budget = budget;
  p.step_j = step_j;
  p.t_ctx = s.t_ctx;
  p.t_cap = s.t_cap;
  p.n_split = plan.n_split;
  p.rows_per_split = plan.rows_per_split;
  p.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
  DraftFn fn = pick(s.head_dim, s.h_q / s.h_kv);
  fn<<<dim3(plan.n_split, units), kDThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

// ============================================================================ allocation-free variant
//
// bd_draft_attn_static runs the same kernel as bd_draft_attn, but its scratch (status
// word, per-unit arrival counters, split partials) lives in this file-scope device array
// instead of a caller-provided workspace, for callers that cannot allocate device memory.
// The array is part of the library image: every GPU that loads the library holds it
// until the process exits.  All calls share it, so calls that overlap on the GPU race.

constexpr size_t kDraftStaticScratchBytes = size_t(4) << 20;   // 4 MiB
static __device__ __align__(256) unsigned char g_draft_scratch[kDraftStaticScratchBytes];

size_t draft_static_scratch_bytes() { return kDraftStaticScratchBytes; }

// Device address of g_draft_scratch on the current device.  In host code the symbol is
// only a host-side stand-in, so the address is looked up once per device, with that
// device current, and cached.
static cudaError_t draft_scratch_address(void** out) {
  static std::mutex mu;
  static void* addr[256] = {nullptr};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= 256) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    err = cudaGetSymbolAddress(&p, g_draft_scratch);
    if (err != cudaSuccess) return err;
    addr[dev] = p;
  }
  *out = addr[dev];
  return cudaSuccess;
}

cudaError_t launch_draft_static(const bd_shape& s, const DraftPlan& plan, const void* q, const void* k_cache,
                                const void* v_cache, const int32_t* idx, const int32_t* count, int budget,
                                int step_j, void* o_out, float* lse_out, cudaStream_t stream) {
  void* base = nullptr;
  cudaError_t err = draft_scratch_address(&base);
  if (err != cudaSuccess) return err;
  const int units = s.batch * s.h_kv;
  uint8_t* b = static_cast<uint8_t*>(base);
  // The array keeps whatever the previous call left: clear the status word and the
  // arrival counters (they must start at zero) before this call's kernel.
  err = cudaMemsetAsync(b, 0, ws_region_offset(units), stream);
  if (err != cudaSuccess) return err;
  return launch_draft(s, plan, q, k_cache, v_cache, idx, count, budget, step_j, o_out, lse_out,
                      b + ws_region_offset(units), reinterpret_cast<int*>(b + ws_counters_offset()),
                      reinterpret_cast<int*>(b), stream);
}

}  // namespace bd
