// Warp-level attention over 16-key sub-tiles on mma.sync (shared by the verify and draft
// kernels).  Keys sit on the M side: S^T = K Q^T with the query rows on N (8*NT columns),
// so a GQA group x block of query rows fills n8 tiles without padding to 16.  P^T (fp32)
// is split into two bf16 terms, P = P_hi + P_lo with P_hi = bf16(P) and P_lo = bf16(P - P_hi),
// each 8x8 block transposed in registers with movmatrix to become the B operand, and
// O^T = V^T P_hi^T + V^T P_lo^T accumulates with V^T read by ldmatrix.trans.  The pair
// carries P to about 2^-17 relative, so the weights of O keep nearly fp32 precision: with
// P rounded to one bf16 alone (2^-9), an output element of 1e-3 over a few hundred keys
// could be off by more than 1e-5.  Softmax state (running max m and sum l per query column)
// lives in the exp2 domain.
//
// K/V sub-tiles are read from shared memory in the TMA SWIZZLE_128B layout (sw128_offset).
#pragma once

#include "bd_common.cuh"

namespace bd {

template <int D, int NT, bool WITH_V>
struct WarpAttn {
  static constexpr int KS = D / 16;
  float m[NT][2];
  float l[NT][2];
  float o[WITH_V ? KS : 1][NT][4];

  __device__ __forceinline__ void init() {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        m[nt][e] = -INFINITY;
        l[nt][e] = 0.f;
      }
#pragma unroll
      for (int mt = 0; mt < (WITH_V ? KS : 1); ++mt)
#pragma unroll
        for (int c = 0; c < 4; ++c) o[mt][nt][c] = 0.f;
    }
  }

  // Loads the B fragments of Q^T for query rows 8*(col_tile0 + nt) + gid from a row-major
  // [rows][D] bf16 block; rows >= n_rows read as zero.
  static __device__ __forceinline__ void load_q(uint32_t (&bq)[NT][KS][2], const __nv_bfloat16* q, int n_rows,
                                                int col_tile0, int lane) {
    const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int row = 8 * (col_tile0 + nt) + gid;
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        if (row < n_rows) {
          bq[nt][ks][0] = __ldg(reinterpret_cast<const uint32_t*>(q + row * D + 16 * ks + 2 * tig));
          bq[nt][ks][1] = __ldg(reinterpret_cast<const uint32_t*>(q + row * D + 16 * ks + 2 * tig + 8));
        } else {
          bq[nt][ks][0] = 0u;
          bq[nt][ks][1] = 0u;
        }
      }
    }
  }

  // One 16-key sub-tile at rows kb..kb+15 of the K (and V) tile.  ok(key_offset, nt, e)
  // says whether key kb + key_offset (key_offset = gid or gid + 8) is visible to query
  // column 8*nt + 2*tig + e of this warp.
  template <typename Visible>
  __device__ __forceinline__ void step(uint32_t kbase, uint32_t vbase, uint32_t half_bytes, int kb,
                                       const uint32_t (&bq)[NT][KS][2], float scale_log2, int lane,
                                       Visible ok) {
    const int gid = lane >> 2;
    float s[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int c = 0; c < 4; ++c) s[nt][c] = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
      uint32_t a[4];
      ldmatrix_x4(a, kbase + sw128_offset(kb + (lane & 15), 16 * ks + 8 * (lane >> 4), half_bytes));
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) mma_16816(s[nt], a, bq[nt][ks][0], bq[nt][ks][1]);
    }
    float alpha[NT][2];
    bool rescale = false;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const float x0 = ok(gid, nt, e) ? s[nt][e] * scale_log2 : -INFINITY;
        const float x1 = ok(gid + 8, nt, e) ? s[nt][2 + e] * scale_log2 : -INFINITY;
        float mx = fmaxf(x0, x1);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float m_new = fmaxf(m[nt][e], mx);
        const float m_use = m_new == -INFINITY ? 0.f : m_new;
        const float al = fast_exp2(m[nt][e] - m_use);
        const float p0 = fast_exp2(x0 - m_use), p1 = fast_exp2(x1 - m_use);
        alpha[nt][e] = al;
        rescale |= (al != 1.f);
        l[nt][e] = l[nt][e] * al + (p0 + p1);
        m[nt][e] = m_new;
        s[nt][e] = p0;
        s[nt][2 + e] = p1;
      }
    }
    if (WITH_V) {
      if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
        for (int mt = 0; mt < KS; ++mt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            o[mt][nt][0] *= alpha[nt][0];
            o[mt][nt][1] *= alpha[nt][1];
            o[mt][nt][2] *= alpha[nt][0];
            o[mt][nt][3] *= alpha[nt][1];
          }
      }
      uint32_t bp[NT][2], bl[NT][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        uint32_t h0, l0, h1, l1;
        split_bf16x2(s[nt][0], s[nt][1], h0, l0);
        split_bf16x2(s[nt][2], s[nt][3], h1, l1);
        bp[nt][0] = movmatrix_trans(h0);
        bp[nt][1] = movmatrix_trans(h1);
        bl[nt][0] = movmatrix_trans(l0);
        bl[nt][1] = movmatrix_trans(l1);
      }
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
        uint32_t a[4];
        ldmatrix_x4_trans(a, vbase + sw128_offset(kb + (lane & 7) + 8 * (lane >> 4), 16 * mt + 8 * ((lane >> 3) & 1),
                                                  half_bytes));
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          mma_16816(o[mt][nt], a, bp[nt][0], bp[nt][1]);
          mma_16816(o[mt][nt], a, bl[nt][0], bl[nt][1]);
        }
      }
    }
  }

  // Sums l over the 8 key lanes (after the last step).
  __device__ __forceinline__ void finish_rows() {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        float v = l[nt][e];
        v += __shfl_xor_sync(0xffffffffu, v, 4);
        v += __shfl_xor_sync(0xffffffffu, v, 8);
        v += __shfl_xor_sync(0xffffffffu, v, 16);
        l[nt][e] = v;
      }
  }

  // Writes this warp's state for columns 8*(col_tile0+nt)+2*tig+e into the merge scratch:
  // m_s/l_s [WK][NQC], o_s [WK][NQC][D+4].
  __device__ __forceinline__ void store(float* m_s, float* l_s, float* o_s, int wk, int nqc, int col_tile0,
                                        int lane) const {
    const int gid = lane >> 2, tig = lane & 3;
    if (gid == 0) {
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int col = 8 * (col_tile0 + nt) + 2 * tig + e;
          m_s[wk * nqc + col] = m[nt][e];
          l_s[wk * nqc + col] = l[nt][e];
        }
    }
    if (WITH_V) {
      constexpr int OP = D + 4;
#pragma unroll
      for (int mt = 0; mt < KS; ++mt)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const int col = 8 * (col_tile0 + nt) + 2 * tig;
          const int d0 = 16 * mt + gid;
          float* base = o_s + (size_t)(wk * nqc + col) * OP;
          base[d0] = o[mt][nt][0];
          base[OP + d0] = o[mt][nt][1];
          base[d0 + 8] = o[mt][nt][2];
          base[OP + d0 + 8] = o[mt][nt][3];
        }
    }
  }
};

// Merges the WK warps' states of columns [0, n_cols) from the scratch written by
// WarpAttn::store and emits, per column, a normalised row o (bf16 if o_bf16 else fp32)
// and lse (natural log).  Out-of-CTA addresses: row r of the output block is
// o_dst + r*D, lse_dst[r].  Executed by n_threads threads synchronising on bar_id.
template <int D, int WK, bool WITH_V>
__device__ __forceinline__ void merge_warps_and_store(const float* m_s, const float* l_s, float* f_s,
                                                      const float* o_s, int nqc, int n_cols, float* lse_dst,
                                                      void* o_dst, bool o_bf16, int tid, int n_threads,
                                                      int bar_id) {
  constexpr int OP = D + 4;
  for (int col = tid; col < n_cols; col += n_threads) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < WK; ++w) M = fmaxf(M, m_s[w * nqc + col]);
    const float M_use = M == -INFINITY ? 0.f : M;
    float L = 0.f;
    float f[WK];
#pragma unroll
    for (int w = 0; w < WK; ++w) {
      f[w] = fast_exp2(m_s[w * nqc + col] - M_use);
      L += f[w] * l_s[w * nqc + col];
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int w = 0; w < WK; ++w) f_s[w * nqc + col] = f[w] * inv;
    if (lse_dst) lse_dst[col] = L > 0.f ? (M + log2f(L)) * kLn2 : -INFINITY;
  }
  if (!WITH_V || o_dst == nullptr) return;
  named_bar(bar_id, n_threads);
  for (int i = tid; i < n_cols * (D / 2); i += n_threads) {
    const int col = i / (D / 2), d = (i % (D / 2)) * 2;
    float a0 = 0.f, a1 = 0.f;
#pragma unroll
    for (int w = 0; w < WK; ++w) {
      const float fw = f_s[w * nqc + col];
      const float* src = o_s + (size_t)(w * nqc + col) * OP + d;
      a0 += fw * src[0];
      a1 += fw * src[1];
    }
    if (o_bf16) {
      *reinterpret_cast<uint32_t*>(static_cast<__nv_bfloat16*>(o_dst) + (size_t)col * D + d) = pack_bf16x2(a0, a1);
    } else {
      *reinterpret_cast<float2*>(static_cast<float*>(o_dst) + (size_t)col * D + d) = make_float2(a0, a1);
    }
  }
}

// One-pass form of merge_warps_and_store for the draft pass: each thread owns four
// adjacent output columns of one row and derives that row's merge factors itself from
// the WK warps' (m, l) (broadcast shared-memory loads), so no barrier separates the
// factors from the output.  o_dst rows are D wide (bf16 if OUT_BF16 else fp32, written
// 8 or 16 bytes at a time: o_dst must be 16-byte aligned); lse_dst[r] in natural log.
template <int D, int WK, bool OUT_BF16>
__device__ __forceinline__ void merge_warps_flat(const float* m_s, const float* l_s, const float* o_s, int nqc,
                                                 int n_cols, float* lse_dst, void* o_dst, int tid, int n_threads) {
  constexpr int OP = D + 4;
  constexpr int Q = D / 4;
  for (int i = tid; i < n_cols * Q; i += n_threads) {
    const int col = i / Q, d = (i % Q) * 4;
    float mw[WK];
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < WK; ++w) {
      mw[w] = m_s[w * nqc + col];
      M = fmaxf(M, mw[w]);
    }
    const float M_use = M == -INFINITY ? 0.f : M;
    float L = 0.f;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < WK; ++w) {
      const float f = fast_exp2(mw[w] - M_use);
      L += f * l_s[w * nqc + col];
      const float4 v = *reinterpret_cast<const float4*>(o_s + (size_t)(w * nqc + col) * OP + d);
      a.x += f * v.x;
      a.y += f * v.y;
      a.z += f * v.z;
      a.w += f * v.w;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    a.x *= inv;
    a.y *= inv;
    a.z *= inv;
    a.w *= inv;
    if (d == 0 && lse_dst) lse_dst[col] = L > 0.f ? (M + log2f(L)) * kLn2 : -INFINITY;
    if (OUT_BF16) {
      uint2 packed;
      packed.x = pack_bf16x2(a.x, a.y);
      packed.y = pack_bf16x2(a.z, a.w);
      *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(o_dst) + (size_t)col * D + d) = packed;
    } else {
      *reinterpret_cast<float4*>(static_cast<float*>(o_dst) + (size_t)col * D + d) = a;
    }
  }
}

}  // namespace bd
