// The C ABI of libbudgetdraft (include/budgetdraft.h): argument validation on the host
// before any launch, workspace layout, and dispatch to the kernels.
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

int current_sm_count() {
  static int cache[256] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
  if (dev < 256 && cache[dev] > 0) return cache[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
  if (dev < 256) cache[dev] = n;
  return n;
}

cudaError_t launch_kernel(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                          void** args, int cluster_x) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attrs[2];
  unsigned n = 0;
  attrs[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster_x > 0) {
    attrs[n].id = cudaLaunchAttributeClusterDimension;
    attrs[n].val.clusterDim.x = (unsigned)cluster_x;
    attrs[n].val.clusterDim.y = 1;
    attrs[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attrs;
  cfg.numAttrs = n;
  return cudaLaunchKernelExC(&cfg, fn, args);
}

// batch * h_kv with per-sequence lengths: the score, window-LSE and verify kernels keep a
// table of units + 1 ints in shared memory (each plan also checks that its table fits)
constexpr int kMaxRaggedUnits = 4096;

size_t ws_counters_offset() { return kWsHeaderBytes; }
size_t ws_region_offset(int units) { return kWsHeaderBytes + align_up((size_t)units * 4, 256); }

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

cudaError_t make_cache_map(CUtensorMap* map, const void* base, int units, int t_cap, int n_rows, int head_dim,
                           int box_rows) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[3] = {(cuuint64_t)head_dim, (cuuint64_t)n_rows, (cuuint64_t)units};
  const cuuint64_t strides[2] = {(cuuint64_t)head_dim * 2, (cuuint64_t)t_cap * head_dim * 2};
  const cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  const cuuint32_t estride[3] = {1, 1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
                        estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_rows_map(CUtensorMap* map, const void* base, long long n_rows, int head_dim, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {(cuuint64_t)head_dim, (cuuint64_t)n_rows};
  const cuuint64_t strides[1] = {(cuuint64_t)head_dim * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  const cuuint32_t estride[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estride,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace bd

using namespace bd;

namespace {

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

int check_shape(const bd_shape* s) {
  if (!s) return BD_ERR_INVALID_ARG;
  if (s->batch < 1 || s->h_q < 1 || s->h_kv < 1 || s->h_q % s->h_kv != 0 || s->t_ctx < 1 || s->t_cap < s->t_ctx)
    return BD_ERR_INVALID_ARG;
  if (s->head_dim != 64 && s->head_dim != 128) return BD_ERR_UNSUPPORTED;
  // every per-unit row offset must stay addressable by the TMA (rows < 2^31)
  if ((long long)s->batch * s->h_kv * s->t_cap >= (1LL << 31)) return BD_ERR_UNSUPPORTED;
  if (s->seq_lens && !aligned(s->seq_lens, 4)) return BD_ERR_MISALIGNED;
  // per-sequence lengths: the kernels keep a per-unit table in shared memory
  if (s->seq_lens && (long long)s->batch * s->h_kv > kMaxRaggedUnits) return BD_ERR_UNSUPPORTED;
  return BD_OK;
}

int check_tensor(const void* p, uintptr_t align) {
  if (!p) return BD_ERR_INVALID_ARG;
  return aligned(p, align) ? BD_OK : BD_ERR_MISALIGNED;
}

int map_cuda(cudaError_t e) { return e == cudaSuccess ? BD_OK : BD_ERR_CUDA; }

int* status_word(void* ws) { return static_cast<int*>(ws); }
int* counters(void* ws) { return reinterpret_cast<int*>(static_cast<uint8_t*>(ws) + ws_counters_offset()); }
void* region(void* ws, int units) { return static_cast<uint8_t*>(ws) + ws_region_offset(units); }

bool group_supported_by_draft(int g) { return g >= 1 && g <= 16; }

size_t verify_ws(const bd_shape& s, int n_q, bool with_v, bool* ok) {
  VerifyPlan vp;
  *ok = verify_plan(s, n_q, with_v, &vp);
  return *ok ? ws_region_offset(s.batch * s.h_kv) + verify_partials_bytes(s, vp) : 0;
}

}  // namespace

#define BD_TRY(x)                  \
  do {                             \
    const int _st = (x);           \
    if (_st != BD_OK) return _st;  \
  } while (0)

extern "C" {

size_t bd_workspace_size(const bd_shape* shape, int op, int budget, int n_q) {
  if (check_shape(shape) != BD_OK) return 0;
  const bd_shape& s = *shape;
  const int units = s.batch * s.h_kv;
  switch (op) {
    case BD_OP_SELECT: {
      if (n_q < 1 || n_q > s.t_ctx || budget < 1) return 0;
      SelectPlan sp;
      if (!select_plan(s, n_q, budget, 0, 0, 1, &sp)) return 0;
      return ws_region_offset(units) + select_region_bytes(s, sp);
    }
    case BD_OP_DRAFT: {
      if (n_q < 1 || budget < 1) return 0;
      DraftPlan dp;
      if (!draft_plan(s, budget, n_q, &dp)) return 0;
      return ws_region_offset(units) + draft_partials_bytes(s, dp);
    }
    case BD_OP_VERIFY: {
      if (n_q < 1) return 0;
      bool ok_v = false, ok_l = false;
      const size_t a = verify_ws(s, n_q, true, &ok_v);
      const size_t b = verify_ws(s, n_q, false, &ok_l);
      if (!ok_v && !ok_l) return 0;
      return std::max(a, b);
    }
    default:
      return 0;
  }
}

int bd_select_budget(const bd_shape* shape, const void* k_cache, const void* q_window, const float* window_lse,
                     int window, int budget, int n_sink, int n_recent, int chunk, unsigned flags, int32_t* idx_out,
                     int32_t* count_out, void* ws, size_t ws_bytes, void* stream) {
  BD_TRY(check_shape(shape));
  const bd_shape& s = *shape;
  BD_TRY(check_tensor(k_cache, 16));
  BD_TRY(check_tensor(q_window, 16));
  if (window_lse) BD_TRY(check_tensor(window_lse, 4));
  BD_TRY(check_tensor(idx_out, 4));
  BD_TRY(check_tensor(count_out, 4));
  if (window < 1 || window > s.t_ctx || budget < 1 || n_sink < 0 || n_recent < 0 || chunk < 1)
    return BD_ERR_INVALID_ARG;
  if (budget < s.t_ctx && (long long)n_sink + n_recent > budget) return BD_ERR_INVALID_ARG;
  if (flags & ~BD_SELECT_WINDOW_READY) return BD_ERR_INVALID_ARG;
  if ((s.h_q / s.h_kv) * window > 256) return BD_ERR_UNSUPPORTED;
  SelectPlan sp;
  if (!select_plan(s, window, budget, n_sink, n_recent, chunk, &sp)) return BD_ERR_UNSUPPORTED;
  if (!window_lse && sp.need_scores && !sp.self_mode) return BD_ERR_UNSUPPORTED;   // > 128 window rows per KV head
  if (!ws) return BD_ERR_WORKSPACE;
  if (!aligned(ws, 256)) return BD_ERR_MISALIGNED;
  const int units = s.batch * s.h_kv;
  if (ws_bytes < ws_region_offset(units) + select_region_bytes(s, sp)) return BD_ERR_WORKSPACE;
  return map_cuda(launch_select(s, sp, k_cache, q_window, window_lse, window, budget, n_sink, n_recent, chunk,
                                flags, idx_out, count_out, region(ws, units), counters(ws), status_word(ws),
                                static_cast<cudaStream_t>(stream)));
}

int bd_draft_attn(const bd_shape* shape, const void* q, const void* k_cache, const void* v_cache,
                  const int32_t* idx, const int32_t* count, int budget, int step_j, unsigned flags, void* o_out,
                  float* lse_out, void* ws, size_t ws_bytes, void* stream) {
  BD_TRY(check_shape(shape));
  const bd_shape& s = *shape;
  BD_TRY(check_tensor(q, 16));
  BD_TRY(check_tensor(k_cache, 16));
  BD_TRY(check_tensor(v_cache, 16));
  BD_TRY(check_tensor(idx, 4));
  BD_TRY(check_tensor(count, 4));
  BD_TRY(check_tensor(o_out, 16));
  if (lse_out) BD_TRY(check_tensor(lse_out, 4));
  if (budget < 1 || step_j < 0 || (long long)s.t_ctx + step_j >= s.t_cap) return BD_ERR_INVALID_ARG;
  if (flags & ~BD_DRAFT_VIEW_READY) return BD_ERR_INVALID_ARG;
  if (!group_supported_by_draft(s.h_q / s.h_kv)) return BD_ERR_UNSUPPORTED;
  DraftPlan dp;
  if (!draft_plan(s, budget, step_j + 1, &dp)) return BD_ERR_UNSUPPORTED;
  if (!ws) return BD_ERR_WORKSPACE;
  if (!aligned(ws, 256)) return BD_ERR_MISALIGNED;
  const int units = s.batch * s.h_kv;
  if (ws_bytes < ws_region_offset(units) + draft_partials_bytes(s, dp)) return BD_ERR_WORKSPACE;
  return map_cuda(launch_draft(s, dp, q, k_cache, v_cache, idx, count, budget, step_j, flags, o_out, lse_out,
                               region(ws, units), counters(ws), status_word(ws), static_cast<cudaStream_t>(stream)));
}

// Allocation-free bd_draft_attn: the same validation and kernel, with the scratch taken
// from the library's own device array (see bd_draft.cu) instead of a caller workspace.
int bd_draft_attn_static(const bd_shape* shape, const void* q, const void* k_cache, const void* v_cache,
                         const int32_t* idx, const int32_t* count, int budget, int step_j, void* o_out,
                         float* lse_out, void* stream) {
  BD_TRY(check_shape(shape));
  const bd_shape& s = *shape;
  BD_TRY(check_tensor(q, 16));
  BD_TRY(check_tensor(k_cache, 16));
  BD_TRY(check_tensor(v_cache, 16));
  BD_TRY(check_tensor(idx, 4));
  BD_TRY(check_tensor(count, 4));
  BD_TRY(check_tensor(o_out, 16));
  if (lse_out) BD_TRY(check_tensor(lse_out, 4));
  if (budget < 1 || step_j < 0 || (long long)s.t_ctx + step_j >= s.t_cap) return BD_ERR_INVALID_ARG;
  if (!group_supported_by_draft(s.h_q / s.h_kv)) return BD_ERR_UNSUPPORTED;
  DraftPlan dp;
  if (!draft_plan(s, budget, step_j + 1, &dp)) return BD_ERR_UNSUPPORTED;
  const int units = s.batch * s.h_kv;
  if (ws_region_offset(units) + draft_partials_bytes(s, dp) > draft_static_scratch_bytes()) return BD_ERR_WORKSPACE;
  return map_cuda(launch_draft_static(s, dp, q, k_cache, v_cache, idx, count, budget, step_j, o_out, lse_out,
                                      static_cast<cudaStream_t>(stream)));
}

int bd_verify_attn(const bd_shape* shape, const void* q, int n_q, const void* k_cache, const void* v_cache,
                   void* o_out, float* lse_out, void* ws, size_t ws_bytes, void* stream) {
  BD_TRY(check_shape(shape));
  const bd_shape& s = *shape;
  BD_TRY(check_tensor(q, 16));
  BD_TRY(check_tensor(k_cache, 16));
  if (o_out) {
    BD_TRY(check_tensor(v_cache, 16));
    BD_TRY(check_tensor(o_out, 16));
  }
  if (lse_out) BD_TRY(check_tensor(lse_out, 4));
  if (!o_out && !lse_out) return BD_ERR_INVALID_ARG;
  if (n_q < 1 || (long long)s.t_ctx + n_q > s.t_cap) return BD_ERR_INVALID_ARG;
  const bool with_v = o_out != nullptr;
  const long long nq_rows = (long long)(s.h_q / s.h_kv) * n_q;
  if (nq_rows > (with_v ? 768 : 128)) return BD_ERR_UNSUPPORTED;
  VerifyPlan vp;
  if (!verify_plan(s, n_q, with_v, &vp)) return BD_ERR_UNSUPPORTED;
  if (!ws) return BD_ERR_WORKSPACE;
  if (!aligned(ws, 256)) return BD_ERR_MISALIGNED;
  const int units = s.batch * s.h_kv;
  if (ws_bytes < ws_region_offset(units) + verify_partials_bytes(s, vp)) return BD_ERR_WORKSPACE;
  return map_cuda(launch_verify(s, vp, n_q, q, k_cache, v_cache, o_out, lse_out, region(ws, units), counters(ws),
                                status_word(ws), static_cast<cudaStream_t>(stream)));
}

int bd_combine(const float* o_part, const float* lse_part, int n_split, int rows, int head_dim, void* o_out,
               float* lse_out, void* stream) {
  if (n_split < 1 || rows < 0) return BD_ERR_INVALID_ARG;
  if (head_dim != 64 && head_dim != 128) return BD_ERR_UNSUPPORTED;
  if (n_split > kCombineMaxSplit) return BD_ERR_UNSUPPORTED;
  if (rows == 0) return BD_OK;
  BD_TRY(check_tensor(o_part, 16));
  BD_TRY(check_tensor(lse_part, 4));
  BD_TRY(check_tensor(o_out, 16));
  if (lse_out) BD_TRY(check_tensor(lse_out, 4));
  if ((long long)n_split * rows * head_dim >= (1LL << 40)) return BD_ERR_UNSUPPORTED;
  return map_cuda(launch_combine(o_part, lse_part, n_split, rows, head_dim, o_out, lse_out,
                                 static_cast<cudaStream_t>(stream)));
}

int bd_argmax(const void* logits, int dtype, int rows, int vocab, int32_t* ids_out, void* stream) {
  if (dtype != BD_DTYPE_BF16 && dtype != BD_DTYPE_F32) return BD_ERR_INVALID_ARG;
  if (rows < 0 || vocab < 1) return BD_ERR_INVALID_ARG;
  if (rows == 0) return BD_OK;
  // the kernel's element indices (a CTA's range end, a vector batch's first element) stay
  // below 2^31 for rows of up to 2^30 elements
  if (rows > 65535 || vocab > (1 << 30)) return BD_ERR_UNSUPPORTED;
  BD_TRY(check_tensor(logits, dtype == BD_DTYPE_BF16 ? 2 : 4));
  BD_TRY(check_tensor(ids_out, 4));
  return map_cuda(launch_argmax(logits, dtype == BD_DTYPE_BF16, rows, vocab, ids_out,
                                static_cast<cudaStream_t>(stream)));
}

int bd_accept(int batch, int gamma, const int32_t* draft_tokens, const int32_t* verify_tokens,
              int32_t* n_accept_out, int32_t* emit_out, void* stream) {
  if (batch < 0 || gamma < 0) return BD_ERR_INVALID_ARG;
  if (batch == 0) return BD_OK;
  if ((long long)batch * (gamma + 1) >= (1LL << 31)) return BD_ERR_UNSUPPORTED;
  if (gamma > 0) BD_TRY(check_tensor(draft_tokens, 4));
  BD_TRY(check_tensor(verify_tokens, 4));
  if (!n_accept_out && !emit_out) return BD_ERR_INVALID_ARG;
  if (n_accept_out) BD_TRY(check_tensor(n_accept_out, 4));
  if (emit_out) BD_TRY(check_tensor(emit_out, 4));
  return map_cuda(launch_accept(batch, gamma, draft_tokens, verify_tokens, n_accept_out, emit_out,
                                static_cast<cudaStream_t>(stream)));
}

int bd_advance(const bd_shape* shape, int window, int n_q, const int32_t* n_accept, const void* q_verify,
               const float* verify_lse, void* q_window, float* window_lse, int32_t* idx, int32_t* count,
               int idx_capacity, int32_t* advance_out, void* stream) {
  BD_TRY(check_shape(shape));
  const bd_shape& s = *shape;
  if (window < 1 || window > s.t_ctx || n_q < 1 || (long long)s.t_ctx + n_q > s.t_cap) return BD_ERR_INVALID_ARG;
  if ((verify_lse == nullptr) != (window_lse == nullptr)) return BD_ERR_INVALID_ARG;
  if ((idx == nullptr) != (count == nullptr)) return BD_ERR_INVALID_ARG;
  if (idx && idx_capacity < 1) return BD_ERR_INVALID_ARG;
  if (s.batch > 65535 || s.h_q > 65535) return BD_ERR_UNSUPPORTED;
  if (advance_smem(window, s.head_dim) > 200 * 1024) return BD_ERR_UNSUPPORTED;
  BD_TRY(check_tensor(n_accept, 4));
  BD_TRY(check_tensor(q_verify, 16));
  BD_TRY(check_tensor(q_window, 16));
  if (window_lse) {
    BD_TRY(check_tensor(verify_lse, 4));
    BD_TRY(check_tensor(window_lse, 4));
  }
  if (idx) {
    BD_TRY(check_tensor(idx, 4));
    BD_TRY(check_tensor(count, 4));
  }
  if (advance_out) BD_TRY(check_tensor(advance_out, 4));
  return map_cuda(launch_advance(s, window, n_q, n_accept, q_verify, verify_lse, q_window, window_lse, idx, count,
                                 idx_capacity, advance_out, static_cast<cudaStream_t>(stream)));
}

int bd_write_block_rows(const bd_shape* shape, int n_rows, const void* k_rows, const void* v_rows, void* k_cache,
                        void* v_cache, void* stream) {
  BD_TRY(check_shape(shape));
  const bd_shape& s = *shape;
  if (n_rows < 1 || (long long)s.t_ctx + n_rows > s.t_cap) return BD_ERR_INVALID_ARG;
  BD_TRY(check_tensor(k_rows, 16));
  BD_TRY(check_tensor(v_rows, 16));
  BD_TRY(check_tensor(k_cache, 16));
  BD_TRY(check_tensor(v_cache, 16));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (s.seq_lens) return map_cuda(launch_write_rows(s, n_rows, k_rows, v_rows, k_cache, v_cache, st));
  const size_t row = (size_t)s.head_dim * 2;
  const size_t units = (size_t)s.batch * s.h_kv;
  const size_t width = (size_t)n_rows * row;
  const void* src[2] = {k_rows, v_rows};
  void* dst[2] = {k_cache, v_cache};
  for (int i = 0; i < 2; ++i) {
    uint8_t* d = static_cast<uint8_t*>(dst[i]) + (size_t)s.t_ctx * row;
    if (cudaMemcpy2DAsync(d, (size_t)s.t_cap * row, src[i], width, width, units, cudaMemcpyDefault, st) != cudaSuccess)
      return BD_ERR_CUDA;
  }
  return BD_OK;
}

int bd_check_wait_timeout(void* ws, size_t ws_bytes, int limit_us, void* stream) {
  if (!ws) return BD_ERR_INVALID_ARG;
  if (ws_bytes < kWsHeaderBytes) return BD_ERR_WORKSPACE;
  if (limit_us < 1 || limit_us > 2000000) return BD_ERR_INVALID_ARG;
  BD_TRY(check_tensor(ws, 16));
  return map_cuda(launch_wait_probe(status_word(ws), limit_us, static_cast<cudaStream_t>(stream)));
}

int bd_draft_static_status(void* stream) {
  int host = 0;
  if (draft_static_status(&host, static_cast<cudaStream_t>(stream)) != cudaSuccess) return BD_ERR_CUDA;
  return host;
}

int bd_workspace_status(void* ws, void* stream) {
  if (!ws) return BD_ERR_INVALID_ARG;
  int host = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&host, ws, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess) return BD_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, sizeof(int), st) != cudaSuccess) return BD_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return BD_ERR_CUDA;
  return host;
}

const char* bd_strerror(int status) {
  switch (status) {
    case BD_OK: return "ok";
    case BD_ERR_INVALID_ARG: return "invalid argument";
    case BD_ERR_UNSUPPORTED: return "unsupported shape or option";
    case BD_ERR_MISALIGNED: return "misaligned pointer";
    case BD_ERR_WORKSPACE: return "workspace missing or too small";
    case BD_ERR_CUDA: return "CUDA runtime or launch error";
    case BD_ERR_TIMEOUT: return "device-side bounded wait timed out";
    default: return "unknown status";
  }
}

}  // extern "C"
