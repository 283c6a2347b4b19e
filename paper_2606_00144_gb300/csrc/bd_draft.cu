// Drafter decode pass over the sparse view (Algorithm 2, Draft): one query per head,
// keys = the selected rows idx[0:count] plus the drafted rows t_ctx .. t_ctx+step_j.
//
// Memory-bound gather (4 flop per byte) whose cost is latency, so the design minimises
// dependent round trips.  A thread-block cluster of up to 8 CTAs serves one (sequence,
// KV head) unit, each CTA one slice of its entry list:
//   1. count and the slice's indices are fetched together (indices speculatively, before
//      count is known);
//   2. rows (80 per CTA) are gathered with 16-byte cp.async straight into the 128-byte
//      swizzled layout (unused rows zero-filled) and the five warps run the mma.sync
//      sub-tile code shared with the verify kernel (bd_attn_warp.cuh), the G heads of the
//      GQA group forming one n8 query tile (two for groups of 9 to 16);
//   3. every CTA stores its normalised partial straight into the shared memory of the
//      cluster's rank-0 CTA (distributed shared memory); after one cluster barrier rank 0
//      merges them (log-sum-exp) from its own shared memory and writes the bf16 output:
//      no global partials, fences or atomics.
// Launched with programmatic dependent launch: the grid-dependency wait is the first thing
// a CTA does, except with BD_DRAFT_VIEW_READY, where the selected rows (and the unit's
// context length) are read and gathered first and only the queries and the drafted rows
// after the wait.  The next kernel may be scheduled as soon as every CTA has passed it.
#include <cooperative_groups.h>

#include <algorithm>
#include <mutex>

#include "bd_attn_warp.cuh"
#include "bd_common.cuh"
#include "bd_internal.h"

namespace cg = cooperative_groups;

namespace bd {

constexpr int kDRows = 80;        // rows per shared-memory tile: 5 sub-tiles of 16, one per warp
constexpr int kDWarps = kDRows / 16;
constexpr int kDThreads = 32 * kDWarps;
constexpr int kDMaxCluster = 8;   // CTAs per (sequence, KV head): the portable cluster size

struct DraftParams {
  const __nv_bfloat16* q;      // [units * g][D]
  const __nv_bfloat16* k;      // [units][t_cap][D]
  const __nv_bfloat16* v;
  const int32_t* idx;          // [units][budget]
  const int32_t* count;        // [units]
  __nv_bfloat16* o;            // [units * g][D]
  float* lse;                  // [units * g] or null
  int g;                       // query heads of a KV head (<= the kernel's G; the rest are padding)
  int* status;
  const int32_t* seq_lens;      // per-sequence context lengths [batch] or null (all t_ctx)
  int h_kv;
  int budget, step_j, t_ctx, t_cap, n_split, rows_per_split;
  int n_stage;                 // 1, or 2 when a CTA gathers more than one tile (double buffer)
  int pos_slots;               // rows_per_split rounded up to whole tiles (row positions in shared memory)
  unsigned flags;              // BD_DRAFT_VIEW_READY: gather the selected rows before the dependency wait
  float scale_log2;
};

template <int D, int G>
struct DraftSmem {
  static constexpr int NQC = 8 * ((G + 7) / 8);   // query columns: the group in n8 tiles
  static constexpr uint32_t TILE_BYTES = kDRows * D * 2;
  static constexpr uint32_t STAGE_BYTES = 2 * TILE_BYTES;                 // K and V
  static constexpr size_t kMerge = (size_t)(3 * kDWarps * NQC) * 4 + (size_t)kDWarps * NQC * (D + 4) * 4;
  // one CTA's partial in rank 0: G rows of D floats, then G lse padded to 16 bytes
  static constexpr int kSlot = G * D + ((G + 3) & ~3);
  // stages (the warp-merge scratch reuses them) | rowpos [pos_slots] (the row of every
  // entry of the CTA's slice) | partials of the cluster's CTAs [C][kSlot] (rank 0 only)
  static size_t bytes(int n_stage, int cluster, int pos_slots) {
    const size_t stages = std::max<size_t>((size_t)n_stage * STAGE_BYTES, kMerge);
    return 1024 + stages + (size_t)pos_slots * 4 + (size_t)cluster * kSlot * 4 + 16;
  }
};

template <int D, int G>
__global__ void __launch_bounds__(kDThreads) draft_kernel(const DraftParams p) {
  using L = DraftSmem<D, G>;
  constexpr int NT = (G + 7) / 8, NQC = L::NQC;   // the group's query heads in n8 tiles
  constexpr uint32_t HALF_BYTES = kDRows * 128;
  constexpr int CH = D / 8;                    // 16-byte chunks per row
  const bool early = (p.flags & BD_DRAFT_VIEW_READY) != 0;
  // the pass's queries (read after the wait below) on their way into L2 meanwhile
  prefetch_lines_l2(p.q + (size_t)blockIdx.y * p.g * D, (size_t)p.g * D * 2, threadIdx.x, kDThreads);
  if (!early) {
    grid_dependency_wait();
    allow_dependent_launch();
  }

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  constexpr size_t kMergeBytes = L::kMerge;
  const size_t stage_bytes = (size_t)p.n_stage * L::STAGE_BYTES > kMergeBytes ? (size_t)p.n_stage * L::STAGE_BYTES
                                                                               : kMergeBytes;
  uint8_t* stage = smem;                                                  // n_stage x (K, V)
  int* rowpos = reinterpret_cast<int*>(smem + stage_bytes);               // [pos_slots]
  float* parts = reinterpret_cast<float*>(rowpos + p.pos_slots);          // [C][kSlot]
  float* m_s = reinterpret_cast<float*>(stage);                           // warp-merge scratch
  float* l_s = m_s + kDWarps * NQC;
  float* f_s = l_s + kDWarps * NQC;
  float* o_s = f_s + kDWarps * NQC;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int split = blockIdx.x, unit = blockIdx.y;
  const int32_t* iunit = p.idx + (size_t)unit * p.budget;
  // announce this CTA has started; the matching wait precedes the first remote store
  if (p.n_split > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  const int e_begin = split * p.rows_per_split;
  // count and the first tile's indices in flight together
  int idx_pref = -1;
  if (tid < kDRows) {
    const int e = e_begin + tid;
    if (e < p.budget && tid < p.rows_per_split) idx_pref = __ldg(iunit + e);
  }
  int cnt = __ldg(p.count + unit);
  if (cnt < 0 || cnt > p.budget) {
    if (tid == 0) record_error(p.status, BD_ERR_INVALID_ARG);
    cnt = min(max(cnt, 0), p.budget);
  }
  // the unit's context length (like idx and count, written before the preceding kernel
  // when the view is ready, so it may be read before the dependency wait)
  const int t_unit = unit_context(p.seq_lens, unit, p.h_kv, p.t_ctx, tid == 0 ? p.status : nullptr);
  const int n_entries = cnt + p.step_j + 1;
  const int e_end = min(e_begin + p.rows_per_split, n_entries);
  const int n_tiles = e_end > e_begin ? (e_end - e_begin + kDRows - 1) / kDRows : 0;
  const __nv_bfloat16* kunit = p.k + (size_t)unit * p.t_cap * D;
  const __nv_bfloat16* vunit = p.v + (size_t)unit * p.t_cap * D;

  auto position = [&](int e, int idx_value) -> int {
    if (e >= cnt) return t_unit + (e - cnt);             // a drafted row
    if (idx_value < 0 || idx_value >= t_unit) {
      record_error(p.status, BD_ERR_INVALID_ARG);
      return -1;                                         // skipped
    }
    return idx_value;
  };
  // the row of every entry of the slice, up front: tile 0 from the prefetched indices, the
  // later tiles' loads all in flight together (no index round trip between tiles)
  auto set_all_rows = [&]() {
    if (tid < kDRows) {
      const int e = e_begin + tid;
      rowpos[tid] = e < e_end ? position(e, idx_pref) : -1;
    }
    for (int e = e_begin + kDRows + tid; e < e_end; e += kDThreads)
      rowpos[e - e_begin] = position(e, e < cnt ? __ldg(iunit + e) : 0);
  };
  // part 0: context rows (and zero fill), part 1: drafted rows (t_ctx and later), part 2: all
  auto gather = [&](int tile, int b, int part) {
    const int nrows = min(kDRows, e_end - (e_begin + tile * kDRows));
    uint8_t* kt = stage + b * L::STAGE_BYTES;
    uint8_t* vt = kt + L::TILE_BYTES;
    for (int c = tid; c < kDRows * CH; c += kDThreads) {
      const int r = c / CH, ch = c % CH;
      const int pos = rowpos[tile * kDRows + r];
      const bool live = r < nrows && pos >= 0;   // others zero-filled (0 * garbage could be NaN in P V)
      const bool drafted = live && pos >= t_unit;
      if ((part == 0 && drafted) || (part == 1 && !drafted)) continue;
      const uint32_t off = sw128_offset(r, ch * 8, HALF_BYTES);
      const size_t src = live ? (size_t)pos * D + ch * 8 : 0;   // slots past the slice are not initialised
      cp_async16_zfill(kt + off, kunit + src, live);
      cp_async16_zfill(vt + off, vunit + src, live);
    }
    cp_async_commit();
  };

  const bool dbuf = p.n_stage == 2;
  if (n_tiles > 0) {
    set_all_rows();
    __syncthreads();
    gather(0, 0, early ? 0 : 2);
  }
  if (early) {   // the selection and the context rows are already in flight
    grid_dependency_wait();
    allow_dependent_launch();
    if (n_tiles > 0) gather(0, 0, 1);
  }
  uint32_t bq[NT][D / 16][2];
  WarpAttn<D, NT, true>::load_q(bq, p.q + (size_t)unit * p.g * D, p.g, 0, lane);
  WarpAttn<D, NT, true> wa;
  wa.init();
  for (int t = 0; t < n_tiles; ++t) {
    const int b = dbuf ? (t & 1) : 0;
    if (dbuf && t + 1 < n_tiles) {
      gather(t + 1, (t + 1) & 1, 2);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int nrows = min(kDRows, e_end - (e_begin + t * kDRows));
    const uint32_t kbase = smem_u32(stage + b * L::STAGE_BYTES);
    const int* rp = rowpos + t * kDRows;
    if (16 * warp < nrows) {
      const int kb = 16 * warp;
      wa.step(kbase, kbase + L::TILE_BYTES, HALF_BYTES, kb, bq, p.scale_log2, lane, [&](int ko, int, int) {
        const int r = kb + ko;
        return r < nrows && rp[r] >= 0;
      });
    }
    __syncthreads();                              // buffer b is free again
    if (!dbuf && t + 1 < n_tiles) gather(t + 1, 0, 2);
  }
  wa.finish_rows();
  wa.store(m_s, l_s, o_s, warp, NQC, 0, lane);
  __syncthreads();
  const size_t row0 = (size_t)unit * p.g;
  if (p.n_split == 1) {
    merge_warps_flat<D, kDWarps, true>(m_s, l_s, o_s, NQC, p.g, p.lse ? p.lse + row0 : nullptr, p.o + row0 * D, tid,
                                       kDThreads);
    return;
  }
  // ---------------------------------------------------------------- cluster merge (DSMEM)
  constexpr int SLOT = L::kSlot;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = p.n_split;
  const int rank = (int)cluster.block_rank();
  float* slot = cluster.map_shared_rank(parts, 0) + (size_t)rank * SLOT;   // in rank 0
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");          // every CTA is running
  merge_warps_flat<D, kDWarps, false>(m_s, l_s, o_s, NQC, G, slot + G * D, slot, tid, kDThreads);
  cluster.sync();                                  // all partials have landed in rank 0
  if (rank != 0) return;
  // each thread: four output columns of one head, its merge weights derived in place
  for (int i = tid; i < p.g * (D / 4); i += kDThreads) {
    const int g = i / (D / 4), d = (i % (D / 4)) * 4;
    float lr[kDMaxCluster];
    float mx = -INFINITY;
#pragma unroll
    for (int r = 0; r < kDMaxCluster; ++r) {
      lr[r] = r < C ? parts[r * SLOT + G * D + g] : -INFINITY;
      mx = fmaxf(mx, lr[r]);
    }
    float tot = 0.f;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int r = 0; r < kDMaxCluster; ++r) {
      if (r < C) {
        const float w = mx == -INFINITY ? 0.f : fast_exp2((lr[r] - mx) * kLog2e);
        const float4 v = *reinterpret_cast<const float4*>(parts + r * SLOT + g * D + d);
        tot += w;
        a.x += w * v.x;
        a.y += w * v.y;
        a.z += w * v.z;
        a.w += w * v.w;
      }
    }
    const float inv = tot > 0.f ? 1.f / tot : 0.f;
    uint2 packed;
    packed.x = pack_bf16x2(a.x * inv, a.y * inv);
    packed.y = pack_bf16x2(a.z * inv, a.w * inv);
    *reinterpret_cast<uint2*>(p.o + (row0 + g) * D + d) = packed;
    if (d == 0 && p.lse) p.lse[row0 + g] = mx == -INFINITY ? -INFINITY : mx + logf(tot);
  }
}

// ============================================================================ host side

namespace {
using DraftFn = void*;
DraftFn pick(int d, int g) {
#define BD_DK(DD, GG) \
  if (d == DD && g == GG) return reinterpret_cast<void*>(&draft_kernel<DD, GG>);
  BD_DK(64, 1) BD_DK(64, 2) BD_DK(64, 4) BD_DK(64, 8) BD_DK(64, 16)
  BD_DK(128, 1) BD_DK(128, 2) BD_DK(128, 4) BD_DK(128, 8) BD_DK(128, 16)
#undef BD_DK
  return nullptr;
}
size_t smem_bytes(int d, int g, int n_stage, int cluster, int pos_slots) {
#define BD_DS(DD, GG) \
  if (d == DD && g == GG) return DraftSmem<DD, GG>::bytes(n_stage, cluster, pos_slots);
  BD_DS(64, 1) BD_DS(64, 2) BD_DS(64, 4) BD_DS(64, 8) BD_DS(64, 16)
  BD_DS(128, 1) BD_DS(128, 2) BD_DS(128, 4) BD_DS(128, 8) BD_DS(128, 16)
#undef BD_DS
  return 0;
}
}  // namespace

// Tile buffers per CTA: double buffering (twice the tile memory, two CTAs per SM) where the
// grid still fits one wave at that occupancy, or where a CTA walks three tiles or more (a long
// loop gains more from overlapping its own gathers than from a single wave); a CTA of two
// tiles in a larger grid relies on its co-resident CTAs to hide its gathers.
static int draft_stages(const DraftPlan& plan, long units) {
  return (plan.rows_per_split > kDRows && units * plan.n_split <= 2L * current_sm_count()) ||
                 plan.rows_per_split > 2 * kDRows
             ? 2
             : 1;
}
// Entries of the CTA's row table: its slice rounded up to whole tiles.
static int draft_pos_slots(const DraftPlan& plan) { return (plan.rows_per_split + kDRows - 1) / kDRows * kDRows; }

// The kernel instance whose n8 query tiles hold a group of g query heads (g <= 16: one
// tile up to 8, two beyond).
int draft_group_instance(int g) { return g <= 1 ? 1 : g <= 2 ? 2 : g <= 4 ? 4 : g <= 8 ? 8 : 16; }

bool draft_plan(const bd_shape& s, int budget, int n_steps, DraftPlan* plan) {
  const int g = s.h_q / s.h_kv;
  if (g < 1 || g > 16 || !pick(s.head_dim, draft_group_instance(g))) return false;
  const long entries = (long)budget + n_steps;
  // one tile per CTA up to a cluster of 8, but no more CTAs than one wave holds at the
  // occupancy the slice's stage count gives (three single-stage or two double-buffered
  // CTAs per SM, draft_stages): a second wave would repeat the pass's whole latency chain
  const long units = (long)s.batch * s.h_kv;
  const long sms = current_sm_count();
  int n_split = (int)std::min<long>((entries + kDRows - 1) / kDRows, kDMaxCluster);
  for (; n_split > 1; --n_split) {
    const long rps = (entries + n_split - 1) / n_split, ctas = units * n_split;
    const bool dbuf = (rps > kDRows && ctas <= 2 * sms) || rps > 2 * kDRows;
    if (ctas <= (dbuf ? 2 : 3) * sms) break;
  }
  n_split = std::max(n_split, 1);
  const long rows_per_split = (entries + n_split - 1) / n_split;
  if (rows_per_split > (1L << 24)) return false;
  plan->rows_per_split = (int)rows_per_split;
  plan->n_split = n_split;
  // the row table of a CTA's slice sits in shared memory beside its tiles
  const int g_kernel = draft_group_instance(g);
  return smem_bytes(s.head_dim, g_kernel, draft_stages(*plan, units), n_split, draft_pos_slots(*plan)) <=
         227 * 1024;
}

size_t draft_partials_bytes(const bd_shape&, const DraftPlan&) { return 0; }   // merged in the cluster

cudaError_t launch_draft(const bd_shape& s, const DraftPlan& plan, const void* q, const void* k_cache,
                         const void* v_cache, const int32_t* idx, const int32_t* count, int budget,
                         int step_j, unsigned flags, void* o_out, float* lse_out, void* ws_region,
                         int* counters, int* status, cudaStream_t stream) {
  (void)ws_region;
  (void)counters;
  const int units = s.batch * s.h_kv;
  DraftParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.k = static_cast<const __nv_bfloat16*>(k_cache);
  p.v = static_cast<const __nv_bfloat16*>(v_cache);
  p.idx = idx;
  p.count = count;
  p.o = static_cast<__nv_bfloat16*>(o_out);
  p.lse = lse_out;
  p.status = status;
  p.budget = budget;
  p.step_j = step_j;
  p.t_ctx = s.t_ctx;
  p.seq_lens = s.seq_lens;
  p.h_kv = s.h_kv;
  p.t_cap = s.t_cap;
  p.n_split = plan.n_split;
  p.rows_per_split = plan.rows_per_split;
  p.n_stage = draft_stages(plan, units);
  p.pos_slots = draft_pos_slots(plan);
  p.flags = flags;
  p.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
  const int g = s.h_q / s.h_kv;
  const int g_kernel = draft_group_instance(g);
  p.g = g;
  void* fn = pick(s.head_dim, g_kernel);
  const size_t smem = smem_bytes(s.head_dim, g_kernel, p.n_stage, plan.n_split, p.pos_slots);
  if (smem > 227 * 1024) return cudaErrorInvalidValue;
  cudaError_t err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;

  void* args[] = {&p};
  return launch_kernel(fn, dim3(plan.n_split, units), dim3(kDThreads), smem, stream, args,
                       plan.n_split > 1 ? plan.n_split : 0);
}

// ============================================================================ allocation-free variant
//
// bd_draft_attn_static runs the same kernel as bd_draft_attn, but its scratch (status
// word and per-unit arrival counters; the split partials are merged inside each
// thread-block cluster and need none) lives in this file-scope device array
// instead of a caller-provided workspace, for callers that cannot allocate device memory.
// The array is part of the library image: every GPU that loads the library holds it
// until the process exits.  All calls share it, so calls that overlap on the GPU race.

constexpr size_t kDraftStaticScratchBytes = size_t(4) << 20;   // 4 MiB
static __device__ __align__(256) unsigned char g_draft_scratch[kDraftStaticScratchBytes];

size_t draft_static_scratch_bytes() { return kDraftStaticScratchBytes; }

// Device address of g_draft_scratch on the current device.  In host code the symbol is
// only a host-side stand-in, so the address is looked up once per device, with that
// device current, and cached.  A device reset (cudaDeviceReset) unloads the module and
// leaves the cached address stale: the entry point does not support calls after the
// reset of a device it has already been called on.
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
  // The array keeps whatever the previous call left: clear the arrival counters (they
  // must start at zero) before this call's kernel.  The status word keeps the errors of
  // earlier calls until draft_static_status reads it.
  err = cudaMemsetAsync(b + ws_counters_offset(), 0, ws_region_offset(units) - ws_counters_offset(), stream);
  if (err != cudaSuccess) return err;
  return launch_draft(s, plan, q, k_cache, v_cache, idx, count, budget, step_j, 0u, o_out, lse_out,
                      b + ws_region_offset(units), reinterpret_cast<int*>(b + ws_counters_offset()),
                      reinterpret_cast<int*>(b), stream);
}

// Reads and clears the array's status word on `stream` (after the calls queued on it).
cudaError_t draft_static_status(int* out, cudaStream_t stream) {
  void* base = nullptr;
  cudaError_t err = draft_scratch_address(&base);
  if (err != cudaSuccess) return err;
  int host = 0;
  err = cudaMemcpyAsync(&host, base, sizeof(int), cudaMemcpyDeviceToHost, stream);
  if (err != cudaSuccess) return err;
  err = cudaMemsetAsync(base, 0, sizeof(int), stream);
  if (err != cudaSuccess) return err;
  err = cudaStreamSynchronize(stream);
  if (err != cudaSuccess) return err;
  *out = host;
  return cudaSuccess;
}

}  // namespace bd
