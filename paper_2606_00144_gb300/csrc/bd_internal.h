// Host-side plumbing shared by the translation units of libbudgetdraft: launch plans,
// workspace layout, tensor-map encoding and per-kernel launchers.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "budgetdraft.h"

namespace bd {

// ---------------------------------------------------------------------------- device facts
int current_sm_count();   // SMs of the current device (cached per device)

// Launch with programmatic dependent launch allowed (the kernel may be scheduled while
// its predecessor finishes; every kernel of this library waits on the grid dependency
// before touching its inputs) and, when cluster_x > 0, as clusters of cluster_x CTAs.
cudaError_t launch_kernel(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                          void** args, int cluster_x);

// ---------------------------------------------------------------------------- workspace
// [0, 256): status word; [256, 256 + units*4 rounded to 256): per-unit arrival counters;
// then the op-specific region.
size_t ws_counters_offset();
size_t ws_region_offset(int units);

// ---------------------------------------------------------------------------- verify
struct VerifyPlan {
  int nq_rows;          // query rows per unit (a chunk of the group * n_q rows of a KV head)
  int rows_total;       // group * n_q
  int row_chunks;       // chunks of a (sequence, KV head): units = batch * h_kv * row_chunks
  int nt, wq;           // n-tiles per warp, warp groups along queries
  int tiles_per_unit;   // 64-key tiles over [0, t_ctx + n_q)
  int total_tiles;      // over all units
  int tiles_per_cta;    // contiguous range of the virtual tile list per CTA
  int seg_cost;         // virtual tiles before each unit's tiles (the cost of starting a unit)
  int grid;
  int max_seg;          // most CTAs that share one unit
  int stages;
  size_t smem_bytes;
  bool with_v;
  bool wide;            // more segments per unit than one staged merge round holds
};
bool verify_plan(const bd_shape& s, int n_q, bool with_v, VerifyPlan* plan);
size_t verify_partials_bytes(const bd_shape& s, const VerifyPlan& plan);
// q/o/lse as in bd_verify_attn; ws_region points at the op region, counters/status into ws.
cudaError_t launch_verify(const bd_shape& s, const VerifyPlan& plan, int n_q, const void* q,
                          const void* k_cache, const void* v_cache, void* o_out, float* lse_out,
                          void* ws_region, int* counters, int* status, cudaStream_t stream,
                          int len_offset = 0);

// ---------------------------------------------------------------------------- draft
struct DraftPlan {
  int n_split;
  int rows_per_split;
};
bool draft_plan(const bd_shape& s, int budget, int n_steps, DraftPlan* plan);
size_t draft_partials_bytes(const bd_shape& s, const DraftPlan& plan);
cudaError_t launch_draft(const bd_shape& s, const DraftPlan& plan, const void* q, const void* k_cache,
                         const void* v_cache, const int32_t* idx, const int32_t* count, int budget,
                         int step_j, unsigned flags, void* o_out, float* lse_out, void* ws_region,
                         int* counters, int* status, cudaStream_t stream);

// Allocation-free variant: scratch in a file-scope device array of this many bytes.
size_t draft_static_scratch_bytes();
cudaError_t draft_static_status(int* out, cudaStream_t stream);
cudaError_t launch_draft_static(const bd_shape& s, const DraftPlan& plan, const void* q, const void* k_cache,
                                const void* v_cache, const int32_t* idx, const int32_t* count, int budget,
                                int step_j, void* o_out, float* lse_out, cudaStream_t stream);

// ---------------------------------------------------------------------------- select
struct SelectPlan {
  bool keep_all;        // budget >= t_ctx
  bool need_scores;     // some middle position (chunk) must be ranked
  int nq_rows, nq_pad;  // window query rows per KV head (padded to 16)
  int n_mid, n_mid_pad;
  int tiles_per_unit, total_tiles, grid, tiles_per_cta;
  int stages;           // K tiles in flight
  int nqb;              // window-query tile buffers
  int n_acc;            // TMEM accumulators
  uint32_t tmem_cols;
  size_t smem_bytes;
  size_t score_bytes, lse_bytes;
  VerifyPlan lse_plan;  // self mode: window LSE through the verify kernel (lse only)
  bool self_mode;       // the window LSE can be computed here (one of the two kernels below)
  bool lse_tc;          // self mode on window_lse_kernel (tcgen05) rather than the verify kernel
  int lse_tiles_per_unit, lse_total_tiles, lse_tiles_per_cta, lse_grid, lse_max_seg;
  size_t lse_smem_bytes, lse_part_bytes;
};
bool select_plan(const bd_shape& s, int window, int budget, int n_sink, int n_recent, int chunk,
                 SelectPlan* plan);
size_t select_region_bytes(const bd_shape& s, const SelectPlan& plan);
cudaError_t launch_select(const bd_shape& s, const SelectPlan& plan, const void* k_cache,
                          const void* q_window, const float* window_lse, int window, int budget,
                          int n_sink, int n_recent, int chunk, unsigned flags, int32_t* idx_out, int32_t* count_out,
                          void* ws_region, int* counters, int* status, cudaStream_t stream);

// ---------------------------------------------------------------------------- combine
// Largest part count of bd_combine: one row's merge weights (n_split floats) must fit the
// 48 KB of dynamic shared memory a launch gets without opting in.
constexpr int kCombineMaxSplit = 12288;
cudaError_t launch_combine(const float* o_part, const float* lse_part, int n_split, int rows,
                           int head_dim, void* o_out, float* lse_out, cudaStream_t stream);
int combine_rows_per_block(int n_split);
cudaError_t launch_wait_probe(int* status, long long limit_us, cudaStream_t stream);

// ---------------------------------------------------------------------------- acceptance
int argmax_cluster(int rows, int vocab);   // CTAs per row
cudaError_t launch_argmax(const void* logits, bool bf16, int rows, int vocab, int32_t* ids_out,
                          cudaStream_t stream);
cudaError_t launch_accept(int batch, int gamma, const int32_t* draft_tokens, const int32_t* verify_tokens,
                          int32_t* n_accept, int32_t* emit, cudaStream_t stream);
size_t advance_smem(int window, int head_dim);
cudaError_t launch_write_rows(const bd_shape& s, int n_rows, const void* k_rows, const void* v_rows, void* k_cache,
                              void* v_cache, cudaStream_t stream);
cudaError_t launch_advance(const bd_shape& s, int window, int n_q, const int32_t* n_accept, const void* q_verify,
                           const float* verify_lse, void* q_window, float* window_lse, int32_t* idx, int32_t* count,
                           int capacity, int32_t* advance_out, cudaStream_t stream);

// ---------------------------------------------------------------------------- TMA maps
// 3-D map over a [units, rows_total (stride t_cap), head_dim] bf16 cache: only rows
// [0, n_rows) of each unit are addressable (the rest reads as zero).  Box = 64 columns x
// box_rows rows x 1 unit, 128-byte swizzle.
cudaError_t make_cache_map(CUtensorMap* map, const void* base, int units, int t_cap, int n_rows,
                           int head_dim, int box_rows);
// 2-D map over a dense [n_rows, head_dim] bf16 matrix; box = 64 columns x box_rows rows,
// 128-byte swizzle; rows past n_rows read as zero.
cudaError_t make_rows_map(CUtensorMap* map, const void* base, long long n_rows, int head_dim, int box_rows);

}  // namespace bd
