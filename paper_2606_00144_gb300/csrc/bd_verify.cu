// Verifier block attention (Algorithm 2, Verify) and the window-LSE pass of self-mode
// selection: n_q queries per head at positions t_ctx .. t_ctx+n_q-1 over keys
// [0, t_ctx + i] (causal inside the block), split-K over the key axis.
//
// One CTA = one (sequence, KV head) unit x one contiguous key range:
//   warp 4      TMA producer: 64-key K (and V) tiles, 128-byte swizzled, 3-stage ring;
//   warps 0..3  consumers.  The GQA group's query rows (group * n_q, packed) are the N
//               side of S^T = K Q^T on mma.sync m16n8k16 (keys on M, so 24 rows fill
//               three n8 tiles exactly); P^T is transposed in registers with movmatrix
//               and O^T = V^T P^T accumulates with V^T read by ldmatrix.trans.
// Online softmax runs per query column in the exp2 domain.  Each CTA writes a normalised
// partial (o, lse); the last CTA of a unit to finish merges them (log-sum-exp), so one
// launch produces the final bf16 output.
#include <algorithm>

#include "bd_common.cuh"
#include "bd_internal.h"

namespace bd {

constexpr int kVKeys = 64;            // keys per pipeline stage
constexpr int kVConsumers = 4;        // consumer warps
constexpr int kVThreads = 160;        // + one producer warp
constexpr int kVMaxSplit = 32;

struct VerifyParams {
  const __nv_bfloat16* q;
  __nv_bfloat16* o;
  float* lse;
  float* o_part;       // [n_split][units][nq_rows][D]
  float* lse_part;     // [n_split][units][nq_rows]
  int* counters;       // [units]
  int* status;
  int units, n_q, nq_rows, t_ctx, n_tiles, tiles_per_split, n_split;
  float scale_log2;    // log2(e) / sqrt(D)
};

template <int D, int NT, int WQ, bool WITH_V, int STAGES>
__global__ void __launch_bounds__(kVThreads) verify_kernel(const VerifyParams p,
                                                           const __grid_constant__ CUtensorMap kmap,
                                                           const __grid_constant__ CUtensorMap vmap) {
  constexpr int WK = kVConsumers / WQ;   // consumer warps along keys
  constexpr int SUBS = 4 / WK;           // 16-key sub-tiles per warp per stage
  constexpr int KS = D / 16;
  constexpr uint32_t HALF_BYTES = kVKeys * 128;
  constexpr uint32_t TILE_BYTES = kVKeys * D * 2;
  constexpr uint32_t STAGE_BYTES = (WITH_V ? 2 : 1) * TILE_BYTES;
  constexpr int NQC = 8 * NT * WQ;       // query columns covered by the CTA

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty_bar = full_bar + STAGES;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty_bar + STAGES);
  int* last_flag = const_cast<int*>(abort_flag) + 1;
  uint8_t* stage_base = smem + 1024;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int split = blockIdx.x, unit = blockIdx.y;
  const int tile0 = split * p.tiles_per_split;
  const int ntiles = min(p.tiles_per_split, p.n_tiles - tile0);

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
    if (lane == 0) {
      tma_prefetch_map(&kmap);
      if (WITH_V) tma_prefetch_map(&vmap);
      int issued = 0;
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % STAGES;
        if (t >= STAGES && !mbar_wait(&empty_bar[s], ((t / STAGES) & 1) ^ 1, p.status, abort_flag)) break;
        uint8_t* st = stage_base + s * STAGE_BYTES;
        mbar_arrive_expect_tx(&full_bar[s], STAGE_BYTES);
        const int key0 = (tile0 + t) * kVKeys;
#pragma unroll
        for (int h = 0; h < D / 64; ++h) tma_load_3d(st + h * HALF_BYTES, &kmap, &full_bar[s], 64 * h, key0, unit);
        if (WITH_V) {
#pragma unroll
          for (int h = 0; h < D / 64; ++h)
            tma_load_3d(st + TILE_BYTES + h * HALF_BYTES, &vmap, &full_bar[s], 64 * h, key0, unit);
        }
        issued = t + 1;
      }
      if (*abort_flag) {   // never leave a copy in flight behind an aborted CTA
        for (int t = max(0, issued - STAGES); t < issued; ++t)
          mbar_wait(&full_bar[t % STAGES], (t / STAGES) & 1, p.status, nullptr);
      }
    }
    return;
  }

  // -------------------------------------------------------------------- consumers
  const int wq = warp % WQ, wk = warp / WQ;
  const int gid = lane >> 2, tig = lane & 3;
  const int nq = p.nq_rows;
  const __nv_bfloat16* qbase = p.q + (size_t)unit * nq * D;

  uint32_t bq[NT][KS][2];
  int lim[NT][2];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int row = 8 * (wq * NT + nt) + gid;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
      if (row < nq) {
        bq[nt][ks][0] = __ldg(reinterpret_cast<const uint32_t*>(qbase + row * D + 16 * ks + 2 * tig));
        bq[nt][ks][1] = __ldg(reinterpret_cast<const uint32_t*>(qbase + row * D + 16 * ks + 2 * tig + 8));
      } else {
        bq[nt][ks][0] = 0u;
        bq[nt][ks][1] = 0u;
      }
    }
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int col = 8 * (wq * NT + nt) + 2 * tig + e;
      lim[nt][e] = col < nq ? p.t_ctx + col % p.n_q : -1;
    }
  }

  float m_run[NT][2], l_run[NT][2];
  float oacc[WITH_V ? KS : 1][NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      m_run[nt][e] = -INFINITY;
      l_run[nt][e] = 0.f;
    }
#pragma unroll
    for (int mt = 0; mt < (WITH_V ? KS : 1); ++mt)
#pragma unroll
      for (int c = 0; c < 4; ++c) oacc[mt][nt][c] = 0.f;
  }

  for (int t = 0; t < ntiles; ++t) {
    const int s = t % STAGES;
    if (!mbar_wait(&full_bar[s], (t / STAGES) & 1, p.status, abort_flag)) break;
    const uint32_t kbase = smem_u32(stage_base + s * STAGE_BYTES);
    const uint32_t vbase = kbase + TILE_BYTES;
    const int key_tile0 = (tile0 + t) * kVKeys;
#pragma unroll
    for (int sub = 0; sub < SUBS; ++sub) {
      const int kb = 16 * (wk + WK * sub);
      float sacc[NT][4];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int c = 0; c < 4; ++c) sacc[nt][c] = 0.f;
      // S^T = K Q^T (16 keys x 8*NT query columns)
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        uint32_t a[4];
        ldmatrix_x4(a, kbase + sw128_offset(kb + (lane & 15), 16 * ks + 8 * (lane >> 4), HALF_BYTES));
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_16816(sacc[nt], a, bq[nt][ks][0], bq[nt][ks][1]);
      }
      // online softmax along the keys of every query column
      const int key_a = key_tile0 + kb + gid, key_b = key_a + 8;
      float alpha[NT][2];
      bool rescale = false;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const float x0 = key_a <= lim[nt][e] ? sacc[nt][e] * p.scale_log2 : -INFINITY;
          const float x1 = key_b <= lim[nt][e] ? sacc[nt][2 + e] * p.scale_log2 : -INFINITY;
          float mx = fmaxf(x0, x1);
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
          const float m_new = fmaxf(m_run[nt][e], mx);
          const float m_use = m_new == -INFINITY ? 0.f : m_new;
          const float al = fast_exp2(m_run[nt][e] - m_use);
          const float p0 = fast_exp2(x0 - m_use), p1 = fast_exp2(x1 - m_use);
          alpha[nt][e] = al;
          rescale |= (al != 1.f);
          l_run[nt][e] = l_run[nt][e] * al + (p0 + p1);
          m_run[nt][e] = m_new;
          sacc[nt][e] = p0;
          sacc[nt][2 + e] = p1;
        }
      }
      if (WITH_V) {
        if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
          for (int mt = 0; mt < KS; ++mt)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              oacc[mt][nt][0] *= alpha[nt][0];
              oacc[mt][nt][1] *= alpha[nt][1];
              oacc[mt][nt][2] *= alpha[nt][0];
              oacc[mt][nt][3] *= alpha[nt][1];
            }
        }
        // P^T (keys x queries, bf16) as the B operand: transpose each 8x8 block in registers
        uint32_t bp[NT][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          bp[nt][0] = movmatrix_trans(pack_bf16x2(sacc[nt][0], sacc[nt][1]));
          bp[nt][1] = movmatrix_trans(pack_bf16x2(sacc[nt][2], sacc[nt][3]));
        }
        // O^T += V^T P^T
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) {
          uint32_t a[4];
          ldmatrix_x4_trans(a, vbase + sw128_offset(kb + (lane & 7) + 8 * (lane >> 4),
                                                    16 * mt + 8 * ((lane >> 3) & 1), HALF_BYTES));
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_16816(oacc[mt][nt], a, bp[nt][0], bp[nt][1]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty_bar[s]);
  }

  // column sums of l over the 8 key lanes
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float l = l_run[nt][e];
      l += __shfl_xor_sync(0xffffffffu, l, 4);
      l += __shfl_xor_sync(0xffffffffu, l, 8);
      l += __shfl_xor_sync(0xffffffffu, l, 16);
      l_run[nt][e] = l;
    }

  // ------------------------------------------------------------------ merge the WK warps
  const int ctid = tid;                         // 0..127 (consumer threads)
  named_bar(1, kVConsumers * 32);               // every consumer is done with the stages
  float* scr = reinterpret_cast<float*>(stage_base);
  float* m_s = scr;                             // [WK][NQC]
  float* l_s = m_s + WK * NQC;                  // [WK][NQC]
  float* f_s = l_s + WK * NQC;                  // [WK][NQC]  weight / L
  float* lse_s = f_s + WK * NQC;                // [NQC]
  float* o_s = lse_s + NQC;                     // [WK][NQC][D + 4]
  constexpr int OP = D + 4;
  if (gid == 0) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int col = 8 * (wq * NT + nt) + 2 * tig + e;
        m_s[wk * NQC + col] = m_run[nt][e];
        l_s[wk * NQC + col] = l_run[nt][e];
      }
  }
  if (WITH_V) {
#pragma unroll
    for (int mt = 0; mt < KS; ++mt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int col = 8 * (wq * NT + nt) + 2 * tig;
        const int d0 = 16 * mt + gid;
        float* base = o_s + (size_t)(wk * NQC + col) * OP;
        base[d0] = oacc[mt][nt][0];
        base[OP + d0] = oacc[mt][nt][1];
        base[d0 + 8] = oacc[mt][nt][2];
        base[OP + d0 + 8] = oacc[mt][nt][3];
      }
  }
  named_bar(1, kVConsumers * 32);
  const bool final_direct = (p.n_split == 1);
  for (int col = ctid; col < nq; col += kVConsumers * 32) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < WK; ++w) M = fmaxf(M, m_s[w * NQC + col]);
    const float M_use = M == -INFINITY ? 0.f : M;
    float L = 0.f;
    float f[WK];
#pragma unroll
    for (int w = 0; w < WK; ++w) {
      f[w] = fast_exp2(m_s[w * NQC + col] - M_use);
      L += f[w] * l_s[w * NQC + col];
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int w = 0; w < WK; ++w) f_s[w * NQC + col] = f[w] * inv;
    const float lse = L > 0.f ? (M + log2f(L)) * kLn2 : -INFINITY;
    lse_s[col] = lse;
    const size_t row = (size_t)unit * nq + col;
    if (final_direct) {
      if (p.lse) p.lse[row] = lse;
    } else {
      p.lse_part[(size_t)split * p.units * nq + row] = lse;
    }
  }
  if (WITH_V) {
    named_bar(1, kVConsumers * 32);
    for (int i = ctid; i < nq * (D / 2); i += kVConsumers * 32) {
      const int col = i / (D / 2), d = (i % (D / 2)) * 2;
      float a0 = 0.f, a1 = 0.f;
#pragma unroll
      for (int w = 0; w < WK; ++w) {
        const float fw = f_s[w * NQC + col];
        const float* src = o_s + (size_t)(w * NQC + col) * OP + d;
        a0 += fw * src[0];
        a1 += fw * src[1];
      }
      const size_t row = (size_t)unit * nq + col;
      if (final_direct) {
        *reinterpret_cast<uint32_t*>(p.o + row * D + d) = pack_bf16x2(a0, a1);
      } else {
        *reinterpret_cast<float2*>(p.o_part + ((size_t)split * p.units * nq + row) * D + d) = make_float2(a0, a1);
      }
    }
  }
  if (final_direct) return;

  // ------------------------------------------------------------------ last CTA merges the splits
  __threadfence();
  named_bar(1, kVConsumers * 32);
  if (ctid == 0) {
    const int prev = atomicAdd(&p.counters[unit], 1);
    *last_flag = (prev == p.n_split - 1);
  }
  named_bar(1, kVConsumers * 32);
  if (*last_flag) {
    __threadfence();
    const size_t row0 = (size_t)unit * nq;
    merge_partials<D>(p.o_part + row0 * D, p.lse_part + row0, p.n_split, nq, (size_t)p.units * nq * D,
                      (size_t)p.units * nq, WITH_V ? p.o + row0 * D : nullptr, p.lse ? p.lse + row0 : nullptr,
                      [](int r) { return r; }, scr, ctid, kVConsumers * 32, 1);
    if (ctid == 0) p.counters[unit] = 0;
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

template <int D, int NT, int WQ, bool WITH_V>
void* kernel_ptr() {
  return reinterpret_cast<void*>(&verify_kernel<D, NT, WQ, WITH_V, 3>);
}

void* select_kernel(int d, int nt, int wq, bool with_v) {
#define BD_VK(DD, N, W, V) \
  if (d == DD && nt == N && wq == W && with_v == V) return kernel_ptr<DD, N, W, V>();
  BD_VK(64, 1, 1, true) BD_VK(64, 3, 1, true) BD_VK(64, 3, 2, true) BD_VK(64, 3, 4, true)
  BD_VK(128, 1, 1, true) BD_VK(128, 3, 1, true) BD_VK(128, 3, 2, true) BD_VK(128, 3, 4, true)
  BD_VK(64, 4, 1, false) BD_VK(64, 4, 2, false) BD_VK(64, 4, 4, false)
  BD_VK(128, 4, 1, false) BD_VK(128, 4, 2, false) BD_VK(128, 4, 4, false)
#undef BD_VK
  return nullptr;
}

size_t scratch_bytes(int d, const Variant& v, bool with_v, int n_split, int nq_rows) {
  const int wk = kVConsumers / v.wq;
  const int nqc = 8 * v.nt * v.wq;
  size_t merge = (size_t)(3 * wk * nqc + nqc) * 4 + (with_v ? (size_t)wk * nqc * (d + 4) * 4 : 0);
  size_t weights = (size_t)n_split * nq_rows * 4;
  return std::max(merge, weights);
}

}  // namespace

bool verify_plan(const bd_shape& s, int n_q, bool with_v, VerifyPlan* plan) {
  const int group = s.h_q / s.h_kv;
  const int nq_rows = group * n_q;
  const Variant v = pick_variant(nq_rows, with_v);
  if (v.nt == 0) return false;
  void* k = select_kernel(s.head_dim, v.nt, v.wq, with_v);
  if (!k) return false;
  plan->nq_rows = nq_rows;
  plan->nt = v.nt;
  plan->wq = v.wq;
  plan->with_v = with_v;
  plan->stages = 3;
  const long n_keys = (long)s.t_ctx + n_q;
  plan->n_tiles = (int)((n_keys + kVKeys - 1) / kVKeys);
  const size_t stage_bytes = (size_t)(with_v ? 2 : 1) * kVKeys * s.head_dim * 2;
  // Resident CTAs per SM from the kernel's registers and shared memory.
  size_t smem_core = 1024 + plan->stages * stage_bytes;
  int occ = 1;
  {
    size_t est = 1024 + std::max(plan->stages * stage_bytes,
                                 scratch_bytes(s.head_dim, v, with_v, kVMaxSplit, nq_rows)) + 1024;
    cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)est);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, kVThreads, est) != cudaSuccess || occ < 1) occ = 1;
    (void)cudaGetLastError();
  }
  const int units = s.batch * s.h_kv;
  const int slots = current_sm_count() * occ;
  int n_split = std::max(1, slots / std::max(1, units));
  n_split = std::min(n_split, std::min(plan->n_tiles, kVMaxSplit));
  plan->tiles_per_split = (plan->n_tiles + n_split - 1) / n_split;
  plan->n_split = (plan->n_tiles + plan->tiles_per_split - 1) / plan->tiles_per_split;
  plan->smem_bytes = 1024 + std::max(smem_core - 1024,
                                     scratch_bytes(s.head_dim, v, with_v, plan->n_split, nq_rows)) + 1024;
  return true;
}

size_t verify_partials_bytes(const bd_shape& s, const VerifyPlan& plan) {
  if (plan.n_split <= 1) return 0;
  const size_t rows = (size_t)plan.n_split * s.batch * s.h_kv * plan.nq_rows;
  return align_up(rows * s.head_dim * 4, 256) + align_up(rows * 4, 256);
}

cudaError_t launch_verify(const bd_shape& s, const VerifyPlan& plan, int n_q, const void* q,
                          const void* k_cache, const void* v_cache, void* o_out, float* lse_out,
                          void* ws_region, int* counters, int* status, cudaStream_t stream) {
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
  const size_t rows = (size_t)plan.n_split * units * plan.nq_rows;
  p.o_part = static_cast<float*>(ws_region);
  p.lse_part = reinterpret_cast<float*>(static_cast<uint8_t*>(ws_region) + align_up(rows * s.head_dim * 4, 256));
  p.counters = counters;
  p.status = status;
  p.units = units;
  p.n_q = n_q;
  p.nq_rows = plan.nq_rows;
  p.t_ctx = s.t_ctx;
  p.n_tiles = plan.n_tiles;
  p.tiles_per_split = plan.tiles_per_split;
  p.n_split = plan.n_split;
  p.scale_log2 = kLog2e / sqrtf((float)s.head_dim);
  void* k = select_kernel(s.head_dim, plan.nt, plan.wq, plan.with_v);
  err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem_bytes);
  if (err != cudaSuccess) return err;
  void* args[] = {&p, &kmap, &vmap};
  return cudaLaunchKernel(k, dim3(plan.n_split, units), dim3(kVThreads), args, plan.smem_bytes, stream);
}

}  // namespace bd
