// Greedy acceptance of a speculative step (Eq. accept; Algorithm 2, accept and bonus
// token): the arg max of every logits row (bd_argmax), then the longest prefix on which the
// drafter's and the verifier's tokens agree plus one verifier token (bd_accept); and the
// cache update that follows (Algorithm 2, Update; bd_advance): the observation window
// slides over the settled block rows and the drafter's sparse view takes their positions.
//
// bd_argmax is a plain streaming reduction: each row is split across a cluster of up to 8
// CTAs; every thread reads batches of 16-byte vectors, takes each batch's maximum with
// NaN-ignoring max instructions and searches a batch for its first maximal element only
// when that maximum beats the thread's best; the CTAs' winners meet in the leading CTA's
// shared memory (distributed shared memory), so no global scratch and no second launch is
// needed.
#include <cooperative_groups.h>

#include <algorithm>
#include <climits>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

namespace cg = cooperative_groups;

constexpr int kAThreads = 512;
constexpr int kAMaxCluster = 8;
constexpr int kAMinPerCta = 4096;   // elements a CTA reads at least before a row is split further

// Maps fp32 bits to an unsigned key with the order of the values: a larger value gives a
// larger key, -0 and +0 share one key (they compare equal), and NaN maps to 0, below every
// number, so it is never chosen.
__device__ __forceinline__ uint32_t order_key(uint32_t f) {
  if ((f & 0x7fffffffu) > 0x7f800000u) return 0u;
  if (f == 0x80000000u) f = 0u;
  return (f & 0x80000000u) ? ~f : (f | 0x80000000u);
}

struct BestOf {
  uint32_t key = 0u;          // 0: nothing comparable seen yet
  uint32_t idx = 0xffffffffu;
  // Elements reach one thread in ascending index order, so a strict comparison keeps the
  // lowest index among equal values.
  __device__ __forceinline__ void take(uint32_t f32_bits, uint32_t i) {
    const uint32_t k = order_key(f32_bits);
    if (k > key) {
      key = k;
      idx = i;
    }
  }
  // (key, lowest index) as one integer whose maximum is the winner.
  __device__ __forceinline__ unsigned long long packed() const {
    return ((unsigned long long)key << 32) | (unsigned long long)(0xffffffffu - idx);
  }
};

template <bool BF16>
__device__ __forceinline__ uint32_t load_bits(const void* row, int i) {
  if (BF16) return (uint32_t)__ldcs(reinterpret_cast<const unsigned short*>(row) + i) << 16;
  return __float_as_uint(__ldcs(reinterpret_cast<const float*>(row) + i));
}

// Elementwise maximum that ignores NaN (max.bf16x2 / fmaxf return the other operand when
// one is NaN, and NaN only when both are).
__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Element e (0..PER_VEC-1) of a 16-byte vector as fp32 bits.
template <bool BF16>
__device__ __forceinline__ uint32_t elem_bits(const uint4& v, int e) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if (BF16) return (e & 1) ? (w[e >> 1] & 0xffff0000u) : (w[e >> 1] << 16);
  return w[e];
}

// A batch of NB vectors at element indices i0[u] (ascending in u): its maximum is found
// with NaN-ignoring max instructions, and only a batch whose maximum beats the thread's
// best so far is searched for the first element equal to it.
template <bool BF16, int NB>
__device__ __forceinline__ void take_batch(BestOf& b, const uint4 (&x)[NB], const uint32_t (&i0)[NB]) {
  constexpr int PER_VEC = BF16 ? 8 : 4;
  uint32_t top_bits;
  if (BF16) {
    uint32_t m[4] = {x[0].x, x[0].y, x[0].z, x[0].w};
#pragma unroll
    for (int u = 1; u < NB; ++u) {
      m[0] = max_bf16x2(m[0], x[u].x);
      m[1] = max_bf16x2(m[1], x[u].y);
      m[2] = max_bf16x2(m[2], x[u].z);
      m[3] = max_bf16x2(m[3], x[u].w);
    }
    const uint32_t p = max_bf16x2(max_bf16x2(m[0], m[1]), max_bf16x2(m[2], m[3]));
    top_bits = __float_as_uint(fmaxf(__uint_as_float(p << 16), __uint_as_float(p & 0xffff0000u)));
  } else {
    float m[4] = {__uint_as_float(x[0].x), __uint_as_float(x[0].y), __uint_as_float(x[0].z),
                  __uint_as_float(x[0].w)};
#pragma unroll
    for (int u = 1; u < NB; ++u) {
      m[0] = fmaxf(m[0], __uint_as_float(x[u].x));
      m[1] = fmaxf(m[1], __uint_as_float(x[u].y));
      m[2] = fmaxf(m[2], __uint_as_float(x[u].z));
      m[3] = fmaxf(m[3], __uint_as_float(x[u].w));
    }
    top_bits = __float_as_uint(fmaxf(fmaxf(m[0], m[1]), fmaxf(m[2], m[3])));
  }
  const uint32_t k = order_key(top_bits);
  if (k > b.key) {
    const float top = __uint_as_float(top_bits);
    uint32_t found = 0xffffffffu;
#pragma unroll
    for (int u = NB - 1; u >= 0; --u)
#pragma unroll
      for (int e = PER_VEC - 1; e >= 0; --e)
        if (__uint_as_float(elem_bits<BF16>(x[u], e)) == top) found = i0[u] + e;   // NaN never equals
    b.key = k;
    b.idx = found;
  }
}

// grid (cluster, rows), clusters of `cluster` CTAs along x: CTA c of row r scans elements
// [c * per_cta, min((c + 1) * per_cta, vocab)).
template <bool BF16>
__global__ void __launch_bounds__(kAThreads) argmax_kernel(const void* logits, int vocab, int per_cta,
                                                           int32_t* ids_out) {
  constexpr int ES = BF16 ? 2 : 4;
  constexpr int PER_VEC = 16 / ES;
  constexpr int NB = 4;
  __shared__ unsigned long long warp_best[kAThreads / 32];
  __shared__ unsigned long long cta_best[kAMaxCluster];
  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x;
  const int row = blockIdx.y;
  const int rank = (int)cluster.block_rank();
  const int n_cta = (int)cluster.num_blocks();

  grid_dependency_wait();
  allow_dependent_launch();

  const char* row_ptr = static_cast<const char*>(logits) + (size_t)row * vocab * ES;
  const int e0 = min(vocab, rank * per_cta), e1 = min(vocab, e0 + per_cta);
  // elements before the first 16-byte boundary, a 16-byte body, then the tail
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(row_ptr + (size_t)e0 * ES);
  const int head = min(e1 - e0, (int)(((16u - (unsigned)(a0 & 15u)) & 15u) / ES));
  const int body0 = e0 + head;
  const int n_vec = (e1 - body0) / PER_VEC;
  const int tail0 = body0 + n_vec * PER_VEC;

  BestOf best;
  if (tid < head) best.take(load_bits<BF16>(row_ptr, e0 + tid), (uint32_t)(e0 + tid));
  const uint4* vec = reinterpret_cast<const uint4*>(row_ptr + (size_t)body0 * ES);
  int v = tid;
  for (; v + (NB - 1) * kAThreads < n_vec; v += NB * kAThreads) {
    uint4 x[NB];
    uint32_t i0[NB];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      x[u] = __ldcs(vec + v + u * kAThreads);
      i0[u] = (uint32_t)(body0 + (v + u * kAThreads) * PER_VEC);
    }
    take_batch<BF16, NB>(best, x, i0);
  }
  for (; v < n_vec; v += kAThreads) {
    uint4 x[1] = {__ldcs(vec + v)};
    const uint32_t i0[1] = {(uint32_t)(body0 + v * PER_VEC)};
    take_batch<BF16, 1>(best, x, i0);
  }
  if (tail0 + tid < e1) best.take(load_bits<BF16>(row_ptr, tail0 + tid), (uint32_t)(tail0 + tid));

  unsigned long long k = best.packed();
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const unsigned long long o = __shfl_xor_sync(0xffffffffu, k, off);
    k = o > k ? o : k;
  }
  if ((tid & 31) == 0) warp_best[tid >> 5] = k;
  __syncthreads();
  if (tid == 0) {
    unsigned long long m = warp_best[0];
#pragma unroll
    for (int w = 1; w < kAThreads / 32; ++w) m = warp_best[w] > m ? warp_best[w] : m;
    unsigned long long* dst = cluster.map_shared_rank(cta_best, 0);
    dst[rank] = m;
  }
  cluster.sync();
  if (rank == 0 && tid == 0) {
    unsigned long long m = cta_best[0];
    for (int c = 1; c < n_cta; ++c) m = cta_best[c] > m ? cta_best[c] : m;
    // a row with no comparable logit (all NaN, or empty) gives id 0
    ids_out[row] = (m >> 32) == 0ull ? 0 : (int32_t)(0xffffffffu - (uint32_t)(m & 0xffffffffull));
  }
}

// One thread per sequence: k = the number of leading positions where drafter and verifier
// agree; emit x_hat[0:k] (equal to x_star[0:k]), then the verifier's token x_star[k] (the
// bonus), then -1 padding.
__global__ void __launch_bounds__(128) accept_kernel(int batch, int gamma, const int32_t* draft_tokens,
                                                     const int32_t* verify_tokens, int32_t* n_accept,
                                                     int32_t* emit) {
  grid_dependency_wait();
  allow_dependent_launch();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  // draft_tokens is pass-major: pass j's token of sequence b sits at [j, b]
  const int32_t* d = draft_tokens + b;
  const int32_t* v = verify_tokens + (size_t)b * (gamma + 1);
  int k = 0;
  while (k < gamma && d[(size_t)k * batch] == v[k]) ++k;
  if (n_accept) n_accept[b] = k;
  if (emit) {
    int32_t* e = emit + (size_t)b * (gamma + 1);
    for (int i = 0; i <= gamma; ++i) e[i] = i < k ? v[i] : (i == k ? v[k] : -1);
  }
}

// ---------------------------------------------------------------------------- bd_advance
constexpr int kVThreads = 128;

struct AdvanceParams {
  const int32_t* n_accept;        // [batch]
  const __nv_bfloat16* q_verify;  // [batch, h_q, n_q, D]
  const float* lse_verify;        // [batch, h_q, n_q] or null
  __nv_bfloat16* q_win;           // [batch, h_q, window, D], slid in place
  float* lse_win;                 // [batch, h_q, window] or null
  int32_t* idx;                   // [batch, h_kv, capacity] or null
  int32_t* count;                 // [batch, h_kv]
  int32_t* advance_out;           // [batch] or null
  int32_t* seq_lens;              // per-sequence context lengths [batch], advanced in place, or null
  int batch, h_q, h_kv, window, n_q, t_ctx, capacity;
};

// grid (h_q, batch).  CTA (h, b) slides the window of query head h of sequence b: new row w
// is old row w + a while that exists, else block row w + a - window.  The new rows are
// staged in shared memory before any is written, so the slide is done in place.  With one
// shared length, a is the batch minimum of the settled counts and CTAs with h < h_kv append
// positions t_ctx .. t_ctx + a - 1 to the view of unit (b, h); with per-sequence lengths,
// a is sequence b's own count and CTA (0, b) appends T_b .. T_b + a - 1 to all of the
// sequence's views, then advances T_b (no other CTA reads it).
template <int D>
__global__ void __launch_bounds__(kVThreads) advance_kernel(const AdvanceParams p) {
  extern __shared__ __align__(16) uint8_t adv_smem[];
  __shared__ int s_min[kVThreads / 32];
  grid_dependency_wait();
  allow_dependent_launch();
  const int tid = threadIdx.x, h = blockIdx.x, b = blockIdx.y;
  int m;
  if (p.seq_lens) {
    m = p.n_accept[b];
  } else {
    m = INT_MAX;
    for (int i = tid; i < p.batch; i += kVThreads) m = min(m, p.n_accept[i]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = min(m, __shfl_xor_sync(0xffffffffu, m, off));
    if ((tid & 31) == 0) s_min[tid >> 5] = m;
    __syncthreads();
    m = s_min[0];
#pragma unroll
    for (int w = 1; w < kVThreads / 32; ++w) m = min(m, s_min[w]);
  }
  const int a = min(max(m, 0), p.n_q - 1) + 1;       // settled rows: the start token + k accepted
  if (h == 0 && tid == 0 && p.advance_out) p.advance_out[b] = a;

  const int W = p.window;
  constexpr int CH = D / 8;                         // 16-byte chunks per row
  uint4* qs = reinterpret_cast<uint4*>(adv_smem);   // [W][CH]
  float* ls = reinterpret_cast<float*>(qs + (size_t)W * CH);
  const size_t bh = (size_t)b * p.h_q + h;
  const uint4* qw = reinterpret_cast<const uint4*>(p.q_win + bh * W * D);
  const uint4* qv = reinterpret_cast<const uint4*>(p.q_verify + bh * p.n_q * D);
  for (int i = tid; i < W * CH; i += kVThreads) {
    const int w = i / CH, c = i % CH, src = w + a;
    qs[i] = src < W ? qw[(size_t)src * CH + c] : qv[(size_t)(src - W) * CH + c];
  }
  if (p.lse_win) {
    for (int w = tid; w < W; w += kVThreads) {
      const int src = w + a;
      ls[w] = src < W ? p.lse_win[bh * W + src] : p.lse_verify[bh * p.n_q + src - W];
    }
  }
  __syncthreads();
  uint4* qo = reinterpret_cast<uint4*>(p.q_win + bh * W * D);
  for (int i = tid; i < W * CH; i += kVThreads) qo[i] = qs[i];
  if (p.lse_win)
    for (int w = tid; w < W; w += kVThreads) p.lse_win[bh * W + w] = ls[w];

  if (p.seq_lens == nullptr) {
    if (p.idx && h < p.h_kv) {
      const size_t u = (size_t)b * p.h_kv + h;
      const int c = p.count[u];
      if (c + a <= p.capacity) {                    // a view without room is left as it is
        for (int i = tid; i < a; i += kVThreads) p.idx[u * p.capacity + c + i] = p.t_ctx + i;
        __syncthreads();
        if (tid == 0) p.count[u] = c + a;
      }
    }
  } else if (h == 0) {
    const int t_b = p.seq_lens[b];
    if (p.idx) {
      for (int g = 0; g < p.h_kv; ++g) {
        const size_t u = (size_t)b * p.h_kv + g;
        const int c = p.count[u];
        if (c + a <= p.capacity) {
          for (int i = tid; i < a; i += kVThreads) p.idx[u * p.capacity + c + i] = t_b + i;
          __syncthreads();
          if (tid == 0) p.count[u] = c + a;
        }
      }
    }
    __syncthreads();
    if (tid == 0) p.seq_lens[b] = t_b + a;
  }
}

// grid (units): rows T_u .. T_u + n_rows - 1 of unit u's K and V rows from dense
// [units][n_rows][D] sources (device or pinned host memory, read through the unified
// address space), for per-sequence lengths.
template <int D>
__global__ void __launch_bounds__(128) write_rows_kernel(const uint4* k_rows, const uint4* v_rows, uint4* k_cache,
                                                         uint4* v_cache, const int32_t* seq_lens, int h_kv,
                                                         int t_cap, int n_rows) {
  grid_dependency_wait();
  allow_dependent_launch();
  constexpr int CH = D / 8;
  const int u = blockIdx.x;
  const int t_u = seq_lens[u / h_kv];
  const size_t src0 = (size_t)u * n_rows * CH;
  const size_t dst0 = ((size_t)u * t_cap + t_u) * CH;
  for (int i = threadIdx.x; i < n_rows * CH; i += blockDim.x) {
    k_cache[dst0 + i] = k_rows[src0 + i];
    v_cache[dst0 + i] = v_rows[src0 + i];
  }
}

cudaError_t launch_write_rows(const bd_shape& s, int n_rows, const void* k_rows, const void* v_rows, void* k_cache,
                              void* v_cache, cudaStream_t stream) {
  const uint4* kr = static_cast<const uint4*>(k_rows);
  const uint4* vr = static_cast<const uint4*>(v_rows);
  uint4* kc = static_cast<uint4*>(k_cache);
  uint4* vc = static_cast<uint4*>(v_cache);
  const int32_t* lens = s.seq_lens;
  int h_kv = s.h_kv, t_cap = s.t_cap;
  void* args[] = {&kr, &vr, &kc, &vc, const_cast<int32_t**>(&lens), &h_kv, &t_cap, &n_rows};
  void* fn = s.head_dim == 64 ? reinterpret_cast<void*>(&write_rows_kernel<64>)
                              : reinterpret_cast<void*>(&write_rows_kernel<128>);
  return launch_kernel(fn, dim3(s.batch * s.h_kv), dim3(128), 0, stream, args, 0);
}

size_t advance_smem(int window, int head_dim) { return (size_t)window * head_dim * 2 + (size_t)window * 4; }

cudaError_t launch_advance(const bd_shape& s, int window, int n_q, const int32_t* n_accept, const void* q_verify,
                           const float* verify_lse, void* q_window, float* window_lse, int32_t* idx, int32_t* count,
                           int capacity, int32_t* advance_out, cudaStream_t stream) {
  AdvanceParams p;
  p.n_accept = n_accept;
  p.q_verify = static_cast<const __nv_bfloat16*>(q_verify);
  p.lse_verify = verify_lse;
  p.q_win = static_cast<__nv_bfloat16*>(q_window);
  p.lse_win = window_lse;
  p.idx = idx;
  p.count = count;
  p.advance_out = advance_out;
  p.seq_lens = const_cast<int32_t*>(s.seq_lens);
  p.batch = s.batch;
  p.h_q = s.h_q;
  p.h_kv = s.h_kv;
  p.window = window;
  p.n_q = n_q;
  p.t_ctx = s.t_ctx;
  p.capacity = capacity;
  const size_t smem = advance_smem(window, s.head_dim);
  void* fn = s.head_dim == 64 ? reinterpret_cast<void*>(&advance_kernel<64>) : reinterpret_cast<void*>(&advance_kernel<128>);
  cudaError_t err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  void* args[] = {&p};
  return launch_kernel(fn, dim3(s.h_q, s.batch), dim3(kVThreads), smem, stream, args, 0);
}

int argmax_cluster(int rows, int vocab) {
  const int want = (2 * current_sm_count() + rows - 1) / std::max(1, rows);
  const int by_size = (vocab + kAMinPerCta - 1) / kAMinPerCta;
  return std::max(1, std::min(kAMaxCluster, std::min(want, by_size)));
}

cudaError_t launch_argmax(const void* logits, bool bf16, int rows, int vocab, int32_t* ids_out,
                          cudaStream_t stream) {
  const int c = argmax_cluster(rows, vocab);
  int per_cta = (vocab + c - 1) / c;
  per_cta = (per_cta + 7) / 8 * 8;   // keeps every CTA's start on the row's 16-byte phase
  void* args[] = {const_cast<void**>(&logits), &vocab, &per_cta, &ids_out};
  void* fn = bf16 ? reinterpret_cast<void*>(&argmax_kernel<true>) : reinterpret_cast<void*>(&argmax_kernel<false>);
  return launch_kernel(fn, dim3(c, rows), dim3(kAThreads), 0, stream, args, c);
}

cudaError_t launch_accept(int batch, int gamma, const int32_t* draft_tokens, const int32_t* verify_tokens,
                          int32_t* n_accept, int32_t* emit, cudaStream_t stream) {
  void* args[] = {&batch, &gamma, const_cast<int32_t**>(&draft_tokens), const_cast<int32_t**>(&verify_tokens),
                  &n_accept, &emit};
  return launch_kernel(reinterpret_cast<void*>(&accept_kernel), dim3((batch + 127) / 128), dim3(128), 0, stream,
                       args, 0);
}

}  // namespace bd
