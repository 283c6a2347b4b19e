// Verifier block attention (Algorithm 2, Verify) and the window-LSE pass of self-mode
// selection: n_q queries per head at positions t_ctx .. t_ctx+n_q-1 over keys
// [0, t_ctx + i] (causal inside the block).
//
// Persistent, stream-K scheduled: the (unit, 64-key tile) pairs of all (sequence, KV head)
// units form one list that is cut into contiguous ranges, one per CTA, of equal cost: each
// unit's tiles are preceded by a few virtual tiles that stand for the cost of starting a
// unit, so every SM streams about the same time whatever the batch.  A range covers one or
// two units; each piece of a unit ("segment") ends in a normalised partial (o, lse), and
// the last CTA to finish a unit merges its segments (log-sum-exp) into the final bf16
// output, staging the partials in shared memory with cp.async (one round trip).
//   warp 4      TMA producer: 64-key K (and V) tiles, 128-byte swizzle, 5-stage ring,
//               streaming straight across segment boundaries.  Context rows [0, t_ctx)
//               are streamed before the grid-dependency wait (they are not written by
//               the preceding kernel); the wait comes before the first tile that holds
//               the block's own rows (before the first load when per-sequence lengths
//               are given: any tile may then hold some sequence's block rows);
//   warps 0..3  consumers on mma.sync (bd_attn_warp.cuh): the GQA group's packed query
//               rows are the N side of S^T = K Q^T.
#include <algorithm>

#include "bd_attn_warp.cuh"
#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

constexpr int kVKeys = 64;            // keys per pipeline stage
constexpr int kVConsumers = 4;        // consumer warps
constexpr int kVThreads = 160;        // + one producer warp
constexpr int kVStages = 5;
constexpr int kVMaxSeg = 33;          // bound on the segments of one unit
constexpr int kVMaxRows = 96;         // query rows one CTA's consumer warps hold (with V)
constexpr int kVMaxChunks = 8;        // row chunks of one (sequence, KV head)

struct VerifyParams {
  const __nv_bfloat16* q;
  __nv_bfloat16* o;
  float* lse;
  float* o_part;       // [units][max_seg][nq_rows][D]
  float* lse_part;     // [units][max_seg][nq_rows]
  int* counters;       // [units]
  int* nseg;           // [units] segments of each unit (wide plans: read by verify_merge_kernel)
  int* status;
  const int32_t* seq_lens;  // per-sequence context lengths [batch] or null (all t_ctx)
  int h_kv;
  int len_offset;      // added to every length (the window LSE pass runs at T - W)
  int n_q, nq_rows, t_ctx, tiles_per_unit, total_tiles, max_seg;
  // Query rows of a (sequence, KV head) beyond what one CTA's warps hold are cut into
  // row_chunks chunks of nq_rows rows (the last may hold fewer): a "unit" below is one
  // (sequence, KV head, chunk), and a KV head's chunks are adjacent in the unit list, so
  // CTAs streaming the same keys run side by side (the second read hits L2).
  int rows_total;      // group * n_q
  int row_chunks;
  int seg_cost;        // virtual tiles charged for each unit a CTA starts (see verify_plan)
  int vtiles_per_cta;  // contiguous range of the virtual tile list per CTA
  float scale_log2;    // log2(e) / sqrt(D)
};

// The global tile list is cut into equal CTA ranges after every unit's tiles are preceded
// by `seg_cost` virtual tiles: a CTA whose range starts a unit (and so stops to merge one
// segment and load new queries) receives that many fewer real tiles.
// The CTA whose range holds real tile g.
__host__ __device__ __forceinline__ int tile_owner(int g, int tpu, int a, int vtpc) {
  const int u = g / tpu;
  return (u * (tpu + a) + a + (g - u * tpu)) / vtpc;
}

// The same layout seen per unit: unit u spans virtual tiles [vbase(u), vbase(u + 1)), its
// `a` virtual tiles first, then its real tiles 0 .. tiles(u) - 1; the list is cut into
// ranges of vtpc virtual tiles, one per CTA.  pref (shared memory, per-sequence lengths)
// holds vbase(u) for u = 0 .. units; null means every unit has tpu real tiles.
struct VerifyMap {
  const int* pref;
  int tpu, a, units, vtpc;
  __device__ __forceinline__ int vbase(int u) const { return pref ? pref[u] : u * (tpu + a); }
  __device__ __forceinline__ int tiles(int u) const { return vbase(u + 1) - vbase(u) - a; }
  __device__ __forceinline__ int unit_of(int v) const {   // the unit whose span holds v
    if (!pref) return v / (tpu + a);
    int lo = 0, hi = units - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (pref[mid] <= v) lo = mid;
      else hi = mid - 1;
    }
    return lo;
  }
  // real tiles of unit u inside the virtual range [v0, v1)
  __device__ __forceinline__ int first_tile(int u, int v0) const { return max(0, v0 - vbase(u) - a); }
  __device__ __forceinline__ int end_tile(int u, int v1) const { return min(tiles(u), v1 - vbase(u) - a); }
  __device__ __forceinline__ int owner(int u, int tile) const { return (vbase(u) + a + tile) / vtpc; }
};

template <int D, int NT, int WQ, bool WITH_V>
struct VerifySmem {
  static constexpr int WK = kVConsumers / WQ;
  static constexpr int NQC = 8 * NT * WQ;
  static constexpr uint32_t TILE_BYTES = kVKeys * D * 2;
  static constexpr uint32_t STAGE_BYTES = (WITH_V ? 2 : 1) * TILE_BYTES;
  static constexpr size_t kStages = (size_t)kVStages * STAGE_BYTES;
  static constexpr size_t kMerge = (size_t)(3 * WK * NQC) * 4 + (WITH_V ? (size_t)WK * NQC * (D + 4) * 4 : 0);
  static constexpr size_t kWeights = (size_t)kVMaxSeg * NQC * 4;
  // layout after the 1 KB barrier block: stages | merge scratch | merge weights
  static constexpr size_t kTotal = 1024 + 1024 + kStages + kMerge + kWeights;
};

// WIDE: the instance for plans whose units span more CTAs than the last one can merge in a
// single staged round trip (small and mid-size batches).  Every CTA only writes its
// segment's partial, the unit's first CTA its segment count, and verify_merge_kernel,
// launched right after, merges them with the whole GPU: a last-CTA merge of ten to twenty
// parts cost 10-16 us at the end of the kernel.  A separate instance, so that the common
// case's code (and register allocation) stays as it is.
template <int D, int NT, int WQ, bool WITH_V, bool WIDE>
__global__ void __launch_bounds__(kVThreads) verify_kernel(const VerifyParams p,
                                                           const __grid_constant__ CUtensorMap kmap,
                                                           const __grid_constant__ CUtensorMap vmap) {
  using L = VerifySmem<D, NT, WQ, WITH_V>;
  constexpr int WK = L::WK, SUBS = 4 / WK, NQC = L::NQC;
  constexpr uint32_t HALF_BYTES = kVKeys * 128;
  constexpr int STAGES = kVStages;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty_bar = full_bar + STAGES;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty_bar + STAGES);
  int* last_flag = const_cast<int*>(abort_flag) + 1;
  uint8_t* stage_base = smem + 1024;
  float* m_s = reinterpret_cast<float*>(stage_base + L::kStages);
  float* l_s = m_s + WK * NQC;
  float* f_s = l_s + WK * NQC;
  float* o_s = f_s + WK * NQC;
  float* w_s = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(m_s) + L::kMerge);
  int* pref = reinterpret_cast<int*>(reinterpret_cast<uint8_t*>(w_s) + L::kWeights);   // ragged: [units + 1]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_units = p.total_tiles / p.tiles_per_unit;
  VerifyMap map{nullptr, p.tiles_per_unit, p.seg_cost, n_units, p.vtiles_per_cta};
  if (p.seq_lens) {
    // per-sequence lengths: every CTA lays out the units' virtual tile spans itself (the
    // lengths may come from the preceding kernel, so after the dependency wait)
    grid_dependency_wait();
    int* wtot = reinterpret_cast<int*>(smem + 512);
    const int per = (n_units + kVThreads - 1) / kVThreads;
    const int u0 = min(n_units, tid * per), u1 = min(n_units, u0 + per);
    auto span = [&](int u) {
      const int t_u =
          max(0, unit_context(p.seq_lens, u / p.row_chunks, p.h_kv, p.t_ctx - p.len_offset, nullptr) + p.len_offset);
      return (t_u + p.n_q + kVKeys - 1) / kVKeys + p.seg_cost;
    };
    int sum = 0;
    for (int u = u0; u < u1; ++u) sum += span(u);
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
      pref[u] = run;
      run += span(u);
    }
    if (tid == kVThreads - 1) pref[n_units] = run;
    __syncthreads();
    map.pref = pref;
    map.vtpc = max((pref[n_units] + (int)gridDim.x - 1) / (int)gridDim.x, p.vtiles_per_cta);
  }
  const int v_total = map.vbase(n_units);
  const int v0 = min(v_total, (int)blockIdx.x * map.vtpc), v1 = min(v_total, v0 + map.vtpc);
  if (v0 >= v1) return;                           // whole CTA idle
  const int u_first = map.unit_of(v0), u_last = map.unit_of(v1 - 1);
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kVConsumers);
    }
    *abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();

  if (warp == kVConsumers) {
    // ------------------------------------------------------------------ producer
    allow_dependent_launch();
    if (lane == 0) {
      tma_prefetch_map(&kmap);
      if (WITH_V) tma_prefetch_map(&vmap);
      int issued = 0;
      // with per-sequence lengths any tile may hold some sequence's block rows (written by
      // the preceding kernels): the wait above came before the first load
      bool waited = p.seq_lens != nullptr;
      bool stop = false;
      for (int unit = u_first; unit <= u_last && !stop; ++unit) {
        const int tb = map.first_tile(unit, v0), te = map.end_tile(unit, v1);
        const int kv_unit = unit / p.row_chunks;
        for (int tile = tb; tile < te; ++tile) {
          const int t = issued;
          const int s = t % STAGES;
          if (t >= STAGES && !mbar_wait(&empty_bar[s], ((t / STAGES) & 1) ^ 1, p.status, abort_flag)) {
            stop = true;
            break;
          }
          const int key0 = tile * kVKeys;
          if (!waited && key0 + kVKeys > p.t_ctx) {    // this tile holds rows of the block itself
            grid_dependency_wait();
            waited = true;
          }
          uint8_t* st = stage_base + s * L::STAGE_BYTES;
          mbar_arrive_expect_tx(&full_bar[s], L::STAGE_BYTES);
#pragma unroll
          for (int h = 0; h < D / 64; ++h) tma_load_3d(st + h * HALF_BYTES, &kmap, &full_bar[s], 64 * h, key0, kv_unit);
          if (WITH_V) {
#pragma unroll
            for (int h = 0; h < D / 64; ++h)
              tma_load_3d(st + L::TILE_BYTES + h * HALF_BYTES, &vmap, &full_bar[s], 64 * h, key0, kv_unit);
          }
          issued = t + 1;
        }
      }
      if (*abort_flag) {   // never leave a copy in flight behind an aborted CTA
        for (int t = max(0, issued - STAGES); t < issued; ++t)
          mbar_wait(&full_bar[t % STAGES], (t / STAGES) & 1, p.status, nullptr);
      }
    }
    return;
  }

  // -------------------------------------------------------------------- consumers
  if (!p.seq_lens)   // the first unit's queries on their way into L2 while the predecessor finishes
    prefetch_lines_l2(p.q + ((size_t)(u_first / p.row_chunks) * p.rows_total + (u_first % p.row_chunks) * p.nq_rows) * D,
                      (size_t)p.nq_rows * D * 2, tid, kVConsumers * 32);
  grid_dependency_wait();                        // the queries come from the preceding kernels
  allow_dependent_launch();
  const int wq = warp % WQ, wk = warp / WQ;
  const int tig = lane & 3;
  const int nq = p.nq_rows;                      // rows per unit slot (the chunk size)
  constexpr int NCT = kVConsumers * 32;          // consumer threads
  int lim[NT][2];                                // last visible key of each of this thread's columns

  bool alive = true;   // false once this warp's wait gave up (the abort flag is then set)
  int t = 0;
  // the next unit of this range with real tiles here (past u_last: none)
  auto next_unit = [&](int u) {
    while (u <= u_last && map.first_tile(u, v0) >= map.end_tile(u, v1)) ++u;
    return u;
  };
  // the unit's queries: a chunk of rows of its KV head's block
  auto unit_q = [&](int u, uint32_t (&bq)[NT][D / 16][2]) {
    const int kv = u / p.row_chunks, base = (u - kv * p.row_chunks) * nq;
    WarpAttn<D, NT, WITH_V>::load_q(bq, p.q + ((size_t)kv * p.rows_total + base) * D, min(nq, p.rows_total - base),
                                    wq * NT, lane);
  };
  uint32_t bq[NT][D / 16][2];
  int unit = next_unit(u_first);
  if (unit <= u_last) unit_q(unit, bq);
  for (; unit <= u_last;) {
    const int tb = map.first_tile(unit, v0), te = map.end_tile(unit, v1);
    const int kv_unit = unit / p.row_chunks;
    const int row_base = (unit - kv_unit * p.row_chunks) * nq;   // first row of this chunk
    const int rows = min(nq, p.rows_total - row_base);
    const size_t row0 = (size_t)kv_unit * p.rows_total + row_base;   // its first row in q / o / lse
    const int t_unit =
        unit_context(p.seq_lens, kv_unit, p.h_kv, p.t_ctx - p.len_offset, tid == 0 ? p.status : nullptr) + p.len_offset;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int col = 8 * (wq * NT + nt) + 2 * tig + e;
        lim[nt][e] = col < rows ? t_unit + (row_base + col) % p.n_q : -1;
      }
    WarpAttn<D, NT, WITH_V> wa;
    wa.init();
    for (int tile = tb; tile < te && alive; ++tile, ++t) {
      const int s = t % STAGES;
      if (!mbar_wait(&full_bar[s], (t / STAGES) & 1, p.status, abort_flag)) {
        alive = false;
        break;
      }
      const uint32_t kbase = smem_u32(stage_base + s * L::STAGE_BYTES);
      const uint32_t vbase = kbase + L::TILE_BYTES;
      const int key_tile0 = tile * kVKeys;
#pragma unroll
      for (int sub = 0; sub < SUBS; ++sub) {
        const int kb = 16 * (wk + WK * sub);
        const int key_base = key_tile0 + kb;
        wa.step(kbase, vbase, HALF_BYTES, kb, bq, p.scale_log2, lane,
                [&](int ko, int nt, int e) { return key_base + ko <= lim[nt][e]; });
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[s]);
    }
    // the next unit's queries are requested now, so that they arrive while this segment
    // closes (its merge, partial write and arrival take several round trips to memory)
    const int next = next_unit(unit + 1);
    if (next <= u_last && alive) unit_q(next, bq);
    wa.finish_rows();

    // ---------------------------------------------------------------- end of a segment
    wa.store(m_s, l_s, o_s, wk, NQC, wq * NT, lane);
    named_bar(1, NCT);
    const int c = blockIdx.x;
    const int c_first = map.owner(unit, 0);
    const int c_last = map.owner(unit, map.tiles(unit) - 1);
    const int n_seg = c_last - c_first + 1;
    if (WIDE && c == c_first && tid == 0) p.nseg[unit] = n_seg;
    if (n_seg == 1) {
      merge_warps_and_store<D, WK, WITH_V>(m_s, l_s, f_s, o_s, NQC, rows, p.lse ? p.lse + row0 : nullptr,
                                           WITH_V ? static_cast<void*>(p.o + row0 * D) : nullptr, true, tid, NCT, 1);
    } else if constexpr (WIDE) {
      const size_t slot = (size_t)unit * p.max_seg + (c - c_first);
      merge_warps_and_store<D, WK, WITH_V>(m_s, l_s, f_s, o_s, NQC, rows, p.lse_part + slot * nq,
                                           WITH_V ? static_cast<void*>(p.o_part + slot * nq * D) : nullptr, false,
                                           tid, NCT, 1);
    } else {
      const size_t slot = (size_t)unit * p.max_seg + (c - c_first);
      merge_warps_and_store<D, WK, WITH_V>(m_s, l_s, f_s, o_s, NQC, rows, p.lse_part + slot * nq,
                                           WITH_V ? static_cast<void*>(p.o_part + slot * nq * D) : nullptr, false,
                                           tid, NCT, 1);
      __threadfence();
      named_bar(1, NCT);
      if (tid == 0) *last_flag = (atomicAdd(&p.counters[unit], 1) == n_seg - 1);
      named_bar(1, NCT);
      if (*last_flag) {
        __threadfence();
        const size_t base = (size_t)unit * p.max_seg;
        merge_partials<D>(p.o_part + base * nq * D, p.lse_part + base * nq, n_seg, rows, (size_t)nq * D, (size_t)nq,
                          WITH_V ? p.o + row0 * D : nullptr, p.lse ? p.lse + row0 : nullptr, [](int r) { return r; },
                          w_s, tid, NCT, 1, m_s, L::kMerge / 4);
        if (tid == 0) p.counters[unit] = 0;
      }
    }
    named_bar(1, NCT);                           // scratch free for the next segment
    // every consumer warp takes the same decision to stop after a timed-out wait
    if (tid == 0) last_flag[1] = *abort_flag;
    named_bar(1, NCT);
    if (last_flag[1]) break;
    unit = next;
  }
}

// Merge of the segments' partials for the wide plans: one CTA per (unit, output row); a
// unit whose segment count is 1 was written by the verify kernel itself.  Thread t takes
// four adjacent columns (t % (D/4)) of the segments s = t / (D/4) (mod 128 / (D/4)), so
// every part of the row is requested at once: the lse values, then the rows, two round
// trips to L2 in all; the groups' sums meet in shared memory.
template <int D>
__global__ void __launch_bounds__(128) verify_merge_kernel(const float* o_part, const float* lse_part,
                                                           const int* nseg, int max_seg, int nq, int rows_total,
                                                           int row_chunks, __nv_bfloat16* o, float* lse) {
  constexpr int Q = D / 4;                 // column quads per row
  constexpr int NG = 128 / Q;              // segment groups
  constexpr int PER = (kVMaxSeg + NG - 1) / NG;
  grid_dependency_wait();
  allow_dependent_launch();
  __shared__ float w[kVMaxSeg];
  __shared__ float4 part[NG][Q];
  const int unit = blockIdx.x, r = blockIdx.y, tid = threadIdx.x;
  const int kv_unit = unit / row_chunks, row_base = (unit - kv_unit * row_chunks) * nq;
  const int n = min(__ldcg(nseg + unit), kVMaxSeg);
  if (n <= 1 || row_base + r >= rows_total) return;
  const size_t orow = (size_t)kv_unit * rows_total + row_base + r;   // the output row
  const size_t base = (size_t)unit * max_seg;
  if (tid < 32) {
    const float l0 = tid < n ? __ldcg(lse_part + (base + tid) * nq + r) : -INFINITY;
    const float l1 = tid + 32 < n ? __ldcg(lse_part + (base + tid + 32) * nq + r) : -INFINITY;
    float mx = fmaxf(l0, l1);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    const float e0 = mx == -INFINITY ? 0.f : fast_exp2((l0 - mx) * kLog2e);
    const float e1 = mx == -INFINITY ? 0.f : fast_exp2((l1 - mx) * kLog2e);
    float tot = e0 + e1;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
    const float inv = tot > 0.f ? 1.f / tot : 0.f;
    if (tid < n) w[tid] = e0 * inv;
    if (tid + 32 < n) w[tid + 32] = e1 * inv;
    if (tid == 0 && lse) lse[orow] = mx == -INFINITY ? -INFINITY : mx + logf(tot);
  }
  if (o == nullptr) return;
  const int q = tid % Q, g = tid / Q;
  float4 v[PER];
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int sg = g + NG * k;
    v[k] = sg < n ? __ldcg(reinterpret_cast<const float4*>(o_part + ((base + sg) * nq + r) * D) + q)
                  : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  __syncthreads();                                  // the weights
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int sg = g + NG * k;
    const float wk = sg < n ? w[sg] : 0.f;
    if (wk != 0.f) {                                // an empty part never enters the sum
      acc.x += wk * v[k].x;
      acc.y += wk * v[k].y;
      acc.z += wk * v[k].z;
      acc.w += wk * v[k].w;
    }
  }
  part[g][q] = acc;
  __syncthreads();
  if (g == 0) {
#pragma unroll
    for (int h = 1; h < NG; ++h) {
      const float4 b = part[h][q];
      acc.x += b.x;
      acc.y += b.y;
      acc.z += b.z;
      acc.w += b.w;
    }
    uint2 packed;
    packed.x = pack_bf16x2(acc.x, acc.y);
    packed.y = pack_bf16x2(acc.z, acc.w);
    *reinterpret_cast<uint2*>(o + orow * D + 4 * q) = packed;
  }
}

// ============================================================================ host side

namespace {

struct Variant {
  int nt, wq;
};

Variant pick_variant(int nq_rows, bool with_v) {
  if (with_v) {
    if (nq_rows <= 8) return {1, 1};
    if (nq_rows <= 24) return {3, 1};
    if (nq_rows <= 48) return {3, 2};
    if (nq_rows <= 96) return {3, 4};
    return {0, 0};
  }
  if (nq_rows <= 32) return {4, 1};
  if (nq_rows <= 64) return {4, 2};
  if (nq_rows <= 128) return {4, 4};
  return {0, 0};
}

struct KernelInfo {
  void* fn;
  size_t smem;
  size_t merge_floats;   // the staging area a unit's last CTA merges the segments' partials in
};

template <int D, int NT, int WQ, bool WITH_V, bool WIDE>
KernelInfo info() {
  return {reinterpret_cast<void*>(&verify_kernel<D, NT, WQ, WITH_V, WIDE>), VerifySmem<D, NT, WQ, WITH_V>::kTotal,
          VerifySmem<D, NT, WQ, WITH_V>::kMerge / 4};
}

KernelInfo select_kernel(int d, int nt, int wq, bool with_v, bool wide) {
#define BD_VK(DD, N, W, V, X) \
  if (d == DD && nt == N && wq == W && with_v == V && wide == X) return info<DD, N, W, V, X>();
  BD_VK(64, 1, 1, true, false) BD_VK(64, 3, 1, true, false) BD_VK(64, 3, 2, true, false) BD_VK(64, 3, 4, true, false)
  BD_VK(128, 1, 1, true, false) BD_VK(128, 3, 1, true, false) BD_VK(128, 3, 2, true, false)
  BD_VK(128, 3, 4, true, false)
  BD_VK(64, 1, 1, true, true) BD_VK(64, 3, 1, true, true) BD_VK(64, 3, 2, true, true) BD_VK(64, 3, 4, true, true)
  BD_VK(128, 1, 1, true, true) BD_VK(128, 3, 1, true, true) BD_VK(128, 3, 2, true, true)
  BD_VK(128, 3, 4, true, true)
  BD_VK(64, 4, 1, false, false) BD_VK(64, 4, 2, false, false) BD_VK(64, 4, 4, false, false)
  BD_VK(128, 4, 1, false, false) BD_VK(128, 4, 2, false, false) BD_VK(128, 4, 4, false, false)
#undef BD_VK
  return {nullptr, 0, 0};
}

// Resident CTAs per SM of a kernel (cached per kernel and device).
int occupancy(const KernelInfo& k) {
  static thread_local void* last_fn = nullptr;
  static thread_local int last_dev = -1, last_occ = 1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (k.fn == last_fn && dev == last_dev) return last_occ;
  int occ = 1;
  cudaFuncSetAttribute(k.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)k.smem);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k.fn, kVThreads, k.smem) != cudaSuccess || occ < 1) occ = 1;
  (void)cudaGetLastError();
  last_fn = k.fn;
  last_dev = dev;
  last_occ = occ;
  return occ;
}

}  // namespace

bool verify_plan(const bd_shape& s, int n_q, bool with_v, VerifyPlan* plan) {
  const int group = s.h_q / s.h_kv;
  const long rows_total = (long)group * n_q;
  // more query rows than one CTA's warps hold (96 with V): chunks of equal size
  const int chunks = with_v && rows_total > kVMaxRows ? (int)((rows_total + kVMaxRows - 1) / kVMaxRows) : 1;
  if (chunks > kVMaxChunks) return false;
  const int nq_rows = (int)((rows_total + chunks - 1) / chunks);
  const Variant v = pick_variant(nq_rows, with_v);
  if (v.nt == 0) return false;
  const KernelInfo k = select_kernel(s.head_dim, v.nt, v.wq, with_v, false);
  if (!k.fn) return false;
  plan->nq_rows = nq_rows;
  plan->rows_total = (int)rows_total;
  plan->row_chunks = chunks;
  plan->nt = v.nt;
  plan->wq = v.wq;
  plan->with_v = with_v;
  plan->stages = kVStages;
  plan->smem_bytes = k.smem;
  const long n_keys = (long)s.t_ctx + n_q;
  plan->tiles_per_unit = (int)((n_keys + kVKeys - 1) / kVKeys);
  const long units = (long)s.batch * s.h_kv * chunks;
  const int tpu = plan->tiles_per_unit;
  const long total = units * tpu;
  const long ctas = std::max(1, current_sm_count() * occupancy(k));
  // A unit boundary inside a CTA's range (the segment's merge of the warps' partials, its
  // write, the arrival, the merge by the unit's last CTA) costs about 5 us of streaming time;
  // charge it as virtual tiles at the rate one CTA streams at when every SM streams
  // (~6.5 TB/s over all SMs).  Traced: with 3 us charged, the CTAs holding a boundary ended
  // their last tile ~5 us after the others; swept at 1-12 us, 5 us gave the shortest step.
  const double tile_bytes = (double)kVKeys * s.head_dim * 2 * (with_v ? 2 : 1);
  const double tile_us = tile_bytes / (6.5e6 / (double)std::max(1, current_sm_count()));
  const int a = (int)std::min(16.0, std::max(0.0, 5.0 / tile_us + 0.5));
  const long vtotal = units * (tpu + a);
  if (vtotal >= (1L << 31)) return false;
  long vtpc = (vtotal + ctas - 1) / ctas;
  vtpc = std::max<long>(vtpc, (tpu + a + kVMaxSeg - 2) / (kVMaxSeg - 1));   // <= kVMaxSeg segments
  plan->seg_cost = a;
  plan->tiles_per_cta = (int)vtpc;
  plan->total_tiles = (int)total;
  plan->grid = (int)((vtotal + vtpc - 1) / vtpc);
  int max_seg = 1;
  for (long u = 0; u < units; ++u) {
    const int c0 = tile_owner((int)(u * tpu), tpu, a, (int)vtpc);
    const int c1 = tile_owner((int)(u * tpu + tpu - 1), tpu, a, (int)vtpc);
    max_seg = std::max(max_seg, c1 - c0 + 1);
  }
  if (max_seg > kVMaxSeg) return false;
  plan->max_seg = max_seg;
  if (s.seq_lens) {
    // per-sequence lengths: the kernel cuts the ranges itself over the actual tiles, no
    // shorter than the bound that keeps every unit within kVMaxSeg segments; the units'
    // span table takes (units + 1) ints of shared memory
    plan->tiles_per_cta = (int)((tpu + a + kVMaxSeg - 2) / (kVMaxSeg - 1));
    plan->max_seg = kVMaxSeg;
    plan->smem_bytes += align_up((size_t)(units + 1) * 4, 16);
    if (plan->smem_bytes > 227 * 1024) return false;
  }
  // the unit's last CTA merges its segments in one staged round trip while they fit its
  // merge area; more segments take the chunked merge of the wide instance
  plan->wide = with_v && ((size_t)plan->max_seg * nq_rows * s.head_dim > k.merge_floats ||
                          (chunks > 1 && plan->max_seg > 1));   // the chunks' units have no arrival counters
  return true;
}

size_t verify_partials_bytes(const bd_shape& s, const VerifyPlan& plan) {
  if (plan.max_seg <= 1) return 0;
  const size_t units = (size_t)s.batch * s.h_kv * plan.row_chunks;
  const size_t rows = units * plan.max_seg * plan.nq_rows;
  return align_up(rows * s.head_dim * 4, 256) + align_up(rows * 4, 256) + (plan.wide ? align_up(units * 4, 256) : 0);
}

cudaError_t launch_verify(const bd_shape& s, const VerifyPlan& plan, int n_q, const void* q,
                          const void* k_cache, const void* v_cache, void* o_out, float* lse_out,
                          void* ws_region, int* counters, int* status, cudaStream_t stream, int len_offset) {
  const int units = s.batch * s.h_kv;
  CUtensorMap kmap, vmap;
  cudaError_t err = make_cache_map(&kmap, k_cache, units, s.t_cap, s.t_ctx + n_q, s.head_dim, kVKeys);
  if (err != cudaSuccess) return err;
  if (plan.with_v) {
    err = make_cache_map(&vmap, v_cache, units, s.t_cap, s.t_ctx + n_q, s.head_dim, kVKeys);
    if (err != cudaSuccess) return err;
  } else {
    vmap = kmap;
  }
  VerifyParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.o = static_cast<__nv_bfloat16*>(o_out);
  p.lse = lse_out;
  const size_t rows = (size_t)units * plan.row_chunks * plan.max_seg * plan.nq_rows;
  p.o_part = static_cast<float*>(ws_region);
  p.lse_part = reinterpret_cast<float*>(static_cast<uint8_t*>(ws_region) + align_up(rows * s.head_dim * 4, 256));
  p.counters = counters;
  p.nseg = reinterpret_cast<int*>(reinterpret_cast<uint8_t*>(p.lse_part) + align_up(rows * 4, 256));
  p.status = status;
  p.n_q = n_q;
  p.nq_rows = plan.nq_rows;
  p.rows_total = plan.rows_total;
  p.row_chunks = plan.row_chunks;
  p.t_ctx = s.t_ctx;
  p.seq_lens = s.seq_lens;
  p.h_kv = s.h_kv;
  p.len_offset = len_offset;
  p.tiles_per_unit = plan.tiles_per_unit;
  p.total_tiles = plan.total_tiles;
  p.seg_cost = plan.seg_cost;
  p.vtiles_per_cta = plan.tiles_per_cta;
  p.max_seg = plan.max_seg;
  p.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
  const KernelInfo k = select_kernel(s.head_dim, plan.nt, plan.wq, plan.with_v, plan.wide);
  err = cudaFuncSetAttribute(k.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem_bytes);
  if (err != cudaSuccess) return err;
  void* args[] = {&p, &kmap, &vmap};
  err = launch_kernel(k.fn, dim3(plan.grid), dim3(kVThreads), plan.smem_bytes, stream, args, 0);
  if (err != cudaSuccess || !plan.wide) return err;
  const float* op = p.o_part;
  const float* lp = p.lse_part;
  const int* ns = p.nseg;
  int max_seg = plan.max_seg, nq = plan.nq_rows, rows_total = plan.rows_total, chunks = plan.row_chunks;
  __nv_bfloat16* o = p.o;
  float* l = p.lse;
  void* margs[] = {&op, &lp, &ns, &max_seg, &nq, &rows_total, &chunks, &o, &l};
  void* mfn = s.head_dim == 64 ? reinterpret_cast<void*>(&verify_merge_kernel<64>)
                               : reinterpret_cast<void*>(&verify_merge_kernel<128>);
  return launch_kernel(mfn, dim3(units * plan.row_chunks, plan.nq_rows), dim3(128), 0, stream, margs, 0);
}

}  // namespace bd
