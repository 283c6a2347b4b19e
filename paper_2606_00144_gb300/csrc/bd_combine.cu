// Standalone log-sum-exp merge of attention computed over disjoint key sets (bd_combine).
// The split-K paths of bd_draft_attn / bd_verify_attn run the same merge_partials code in
// their last-arriving CTA; this kernel serves callers that produce the parts themselves.
#include <algorithm>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

constexpr int kCThreads = 128;

template <int D>
__global__ void __launch_bounds__(kCThreads) combine_kernel(const float* o_part, const float* lse_part,
                                                            int n_split, int rows, int rows_per_block,
                                                            __nv_bfloat16* o_out, float* lse_out) {
  grid_dependency_wait();
  allow_dependent_launch();
  extern __shared__ float w_smem[];
  const int r0 = blockIdx.x * rows_per_block;
  const int nr = min(rows_per_block, rows - r0);
  merge_partials<D>(o_part + (size_t)r0 * D, lse_part + r0, n_split, nr, (size_t)rows * D, (size_t)rows,
                    o_out + (size_t)r0 * D, lse_out ? lse_out + r0 : nullptr, [](int r) { return r; }, w_smem,
                    threadIdx.x, kCThreads, 0);
}

int combine_rows_per_block(int n_split) {
  return std::max(1, std::min(16, 12288 / std::max(1, n_split)));
}

cudaError_t launch_combine(const float* o_part, const float* lse_part, int n_split, int rows, int head_dim,
                           void* o_out, float* lse_out, cudaStream_t stream) {
  const int rpb = combine_rows_per_block(n_split);
  const size_t smem = (size_t)n_split * rpb * sizeof(float);
  const dim3 grid((rows + rpb - 1) / rpb);
  __nv_bfloat16* o = static_cast<__nv_bfloat16*>(o_out);
  void* args[] = {&o_part, &lse_part, &n_split, &rows, const_cast<int*>(&rpb), &o, &lse_out};
  void* fn = head_dim == 64 ? reinterpret_cast<void*>(&combine_kernel<64>) : reinterpret_cast<void*>(&combine_kernel<128>);
  return launch_kernel(fn, grid, dim3(kCThreads), smem, stream, args, 0);
}

}  // namespace bd
