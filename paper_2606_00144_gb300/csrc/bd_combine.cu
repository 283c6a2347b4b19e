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
  return std::max(1, std::min(16, kCombineMaxSplit / std::max(1, n_split)));
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

// The error path of a bounded wait, end to end: one warp waits on a shared-memory barrier
// that nothing completes until limit_ns runs out, which records BD_ERR_TIMEOUT in the status
// word exactly as a stalled pipeline wait of the other kernels does, and the kernel returns.
// The second warp watches the shared abort flag the waiting warp raises and stops too.
__global__ void __launch_bounds__(64) wait_probe_kernel(int* status, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    if (threadIdx.x == 0) mbar_wait_for(&bar, 0, status, &abort_flag, limit_ns);
  } else if (threadIdx.x == 32) {
    // a second role that gives up once the first has: the abort flag ends its wait
    mbar_wait_for(&bar, 0, nullptr, &abort_flag, 4 * limit_ns);
  }
  __syncthreads();
}

cudaError_t launch_wait_probe(int* status, long long limit_us, cudaStream_t stream) {
  unsigned long long ns = (unsigned long long)limit_us * 1000ull;
  void* args[] = {&status, &ns};
  return launch_kernel(reinterpret_cast<void*>(&wait_probe_kernel), dim3(1), dim3(64), 0, stream, args, 0);
}

}  // namespace bd
