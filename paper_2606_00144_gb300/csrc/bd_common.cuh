// Device-side building blocks shared by the speculative-step kernels (sm_103a):
// PTX wrappers for mbarrier, TMA (cp.async.bulk.tensor), cp.async, ldmatrix /
// movmatrix / mma.sync, tcgen05 (TMEM alloc, UMMA, commit, ld), bounded waits and
// the log-sum-exp merge used by every split-K kernel.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "budgetdraft.h"

namespace bd {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// ---------------------------------------------------------------------------------------
// Launch-side parameters shared by kernels and host code
// ---------------------------------------------------------------------------------------
struct WsHeader {          // first 256 bytes of every workspace
  int status;              // first device-side error code (0 = none)
  int pad[63];
};
constexpr size_t kWsHeaderBytes = 256;

__host__ __device__ constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------------------------------
// Small device helpers
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void record_error(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ float fast_exp2(float x) {   // hardware ex2 (MUFU), ex2(-inf) = +0
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Programmatic dependent launch: wait until the preceding grid has completed and its
// memory is visible (a no-op without a programmatic predecessor), then let the next grid
// be scheduled.  Every kernel here calls both before reading any input.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void allow_dependent_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Named barrier over `n` threads (a multiple of 32); id 0 with the whole CTA = __syncthreads.
__device__ __forceinline__ void named_bar(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// Packed fp32 pairs (Blackwell f32x2 FMA and add): two lanes of arithmetic per instruction.
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 r;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mov.b64 rc, {%6, %7};\n\tfma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return r;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  float2 r;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(r.x), "=f"(r.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Two-term bf16 form of a pair of floats: head = bf16x2(x, y) rounded to nearest, tail =
// bf16x2 of what the rounding left over, so that head + tail carries about 16 bits of each
// value's significand (x in the low halves, y in the high halves).
__device__ __forceinline__ void split_bf16x2(float x, float y, uint32_t& head, uint32_t& tail) {
  head = pack_bf16x2(x, y);
  const float hx = __uint_as_float(head << 16), hy = __uint_as_float(head & 0xffff0000u);
  tail = pack_bf16x2(x - hx, y - hy);
}

// Every wait in these kernels gives up after this long (or this many polls) and records
// BD_ERR_TIMEOUT in the workspace status word, so a logic error can never hang the GPU.
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s
constexpr uint32_t kWaitLimitPolls = 1u << 28;

// ---------------------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for the completion of the barrier phase with the given parity.
// `abort_flag` (shared) lets one timed-out role stop the others quickly.  Returns false
// on timeout or abort; the caller then skips its remaining work.
__device__ __forceinline__ bool mbar_wait_for(uint64_t* bar, uint32_t parity, int* status,
                                              volatile int* abort_flag, uint64_t limit_ns) {
  const uint32_t addr = smem_u32(bar);
  if (mbar_test(addr, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 0; i < kWaitLimitPolls; ++i) {
    if (mbar_test(addr, parity)) return true;
    if ((i & 31u) == 31u) {
      if (abort_flag && *abort_flag) return false;
      if (global_timer_ns() - t0 > limit_ns) break;
    }
  }
  record_error(status, BD_ERR_TIMEOUT);
  if (abort_flag) *abort_flag = 1;
  return false;
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int* status,
                                          volatile int* abort_flag) {
  return mbar_wait_for(bar, parity, status, abort_flag, kWaitLimitNs);
}

// ---------------------------------------------------------------------------------------
// TMA (tiled tensor copies global -> shared, completion counted on an mbarrier)
// ---------------------------------------------------------------------------------------
// Starts [p, p + bytes) on its way into L2 (no L1 allocation, nothing to wait for): safe
// before a grid-dependency wait on data the preceding kernel may still write, since L2 is
// where those writes land and the real load after the wait reads through it.  One line per
// thread of [0, n_threads).
__device__ __forceinline__ void prefetch_lines_l2(const void* p, size_t bytes, int tid, int n_threads) {
  const char* c = static_cast<const char*>(p);
  for (size_t off = (size_t)tid * 128; off < bytes; off += (size_t)n_threads * 128)
    asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<uint64_t>(c + off)) : "memory");
}
__device__ __forceinline__ void tma_prefetch_map(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                            int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------------------------------
// cp.async (16-byte global -> shared, L2 only)
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
// 16 bytes copied when `valid`, else 16 zero bytes written (src is not read).
__device__ __forceinline__ void cp_async16_zfill(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// ---------------------------------------------------------------------------------------
// Warp-level tensor core path (mma.sync m16n8k16 bf16 -> fp32)
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}
__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of element (row, col) in a tile stored the way a TMA SWIZZLE_128B box
// writes it: the row's d elements are split into 64-element (128-byte) halves, each half
// a [rows][128 B] block; inside a 1024-byte group of 8 rows the 16-byte chunk c of row r
// sits at chunk c ^ (r % 8).  `half_bytes` = rows * 128.  col must be a multiple of 8.
__device__ __forceinline__ uint32_t sw128_offset(int row, int col, uint32_t half_bytes) {
  const int half = col >> 6;
  const int chunk = (col & 63) >> 3;
  return half * half_bytes + row * 128 + ((chunk ^ (row & 7)) << 4);
}

// ---------------------------------------------------------------------------------------
// tcgen05 (5th-generation tensor core, accumulators in tensor memory)
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulate; one thread issues.
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` once every tcgen05 operation this thread issued so far has completed.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tc_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 32 lanes x 32 consecutive fp32 columns: thread i of the warp gets lane (quadrant*32 + i).
__device__ __forceinline__ void tc_ld_32cols(uint32_t taddr, float (&v)[32]) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

// Shared-memory matrix descriptor for a K-major operand in the 128-byte swizzled layout
// (8-row x 128-byte atoms, atoms stacked every 1024 bytes along M/N).
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t smem_addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((smem_addr & 0x3FFFFu) >> 4);   // start address
  d |= static_cast<uint64_t>(1) << 16;                        // leading byte offset (unused here)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;                // stride byte offset: 8 rows * 128 B
  d |= static_cast<uint64_t>(1) << 46;                        // descriptor version
  d |= static_cast<uint64_t>(2) << 61;                        // swizzle: 128 B
  return d;
}
// Instruction descriptor: kind::f16 with bf16 A/B, fp32 D, both operands K-major.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(m >> 4) << 24);
}

// Context length of the sequence that owns (sequence, KV head) unit `unit` (units are
// sequence-major): seq_lens[unit / h_kv] when per-sequence lengths are given, else t_ctx.
// A length outside [1, t_ctx] is recorded as an argument error and clamped.
__device__ __forceinline__ int unit_context(const int32_t* seq_lens, int unit, int h_kv, int t_ctx, int* status) {
  if (seq_lens == nullptr) return t_ctx;
  int t = seq_lens[unit / h_kv];
  if (t < 1 || t > t_ctx) {
    if (status) record_error(status, BD_ERR_INVALID_ARG);
    t = min(max(t, 1), t_ctx);
  }
  return t;
}

// ---------------------------------------------------------------------------------------
// Log-sum-exp merge of split partials (shared by the fused split-K paths and bd_combine)
// ---------------------------------------------------------------------------------------
// Rows [0, rows) with parts s = 0..n_split-1 at o_part + s*split_stride + r*D (normalised
// fp32 rows) and lse_part + s*lse_split_stride + r.  Output row r goes to o_out + out_row(r)*D
// (bf16) and lse_out[out_row(r)] (natural log).  Executed by `nthreads` threads of one CTA
// that synchronise on named barrier `bar_id`; `w_smem` holds n_split*rows floats.
template <int D, typename RowMap>
__device__ __forceinline__ void merge_partials(const float* o_part, const float* lse_part, int n_split,
                                               int rows, size_t split_stride, size_t lse_split_stride,
                                               __nv_bfloat16* o_out, float* lse_out, RowMap out_row,
                                               float* w_smem, int tid, int nthreads, int bar_id,
                                               float* stage = nullptr, size_t stage_floats = 0) {
  constexpr int D4 = D / 4;
  const int total = rows * D4;
  // The parts were written by other CTAs just before and sit in L2: latency, not bandwidth,
  // decides this merge.  With a staging area big enough, every part row is copied into
  // shared memory by cp.async while the lse loads are in flight too: one round trip.
  const bool staged = o_out != nullptr && stage != nullptr && (size_t)n_split * rows * D <= stage_floats;
  if (staged) {
    for (int i = tid; i < n_split * total; i += nthreads) {
      const int sp = i / total, j = i % total;
      const int r = j / D4, c = (j % D4) * 4;
      cp_async16(stage + (size_t)i * 4, o_part + sp * split_stride + (size_t)r * D + c);
    }
    cp_async_commit();
  }
  // weights exp(lse_s - L) per (split, row); a row's lse values are all requested at once
  for (int r = tid; r < rows; r += nthreads) {
    float mx = -INFINITY;
#pragma unroll 8
    for (int sp = 0; sp < n_split; ++sp) {
      const float l = __ldcg(lse_part + sp * lse_split_stride + r);
      w_smem[sp * rows + r] = l;
      mx = fmaxf(mx, l);
    }
    float tot = 0.f;
    for (int sp = 0; sp < n_split; ++sp) {
      const float w = (mx == -INFINITY) ? 0.f : fast_exp2((w_smem[sp * rows + r] - mx) * kLog2e);
      w_smem[sp * rows + r] = w;
      tot += w;
    }
    const float inv = tot > 0.f ? 1.f / tot : 0.f;
    for (int sp = 0; sp < n_split; ++sp) w_smem[sp * rows + r] *= inv;
    if (lse_out) lse_out[out_row(r)] = (mx == -INFINITY) ? -INFINITY : mx + logf(tot);
  }
  if (staged) cp_async_wait<0>();
  named_bar(bar_id, nthreads);
  if (o_out == nullptr) return;
  for (int i = tid; i < total; i += nthreads) {
    const int r = i / D4, c = (i % D4) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sp = 0; sp < n_split; ++sp) {
      const float w = w_smem[sp * rows + r];
      if (w != 0.f) {
        const float4 v = staged ? *reinterpret_cast<const float4*>(stage + ((size_t)sp * total + i) * 4)
                                : __ldcg(reinterpret_cast<const float4*>(o_part + sp * split_stride + (size_t)r * D + c));
        acc.x += w * v.x;
        acc.y += w * v.y;
        acc.z += w * v.z;
        acc.w += w * v.w;
      }
    }
    uint2 packed;
    packed.x = pack_bf16x2(acc.x, acc.y);
    packed.y = pack_bf16x2(acc.z, acc.w);
    *reinterpret_cast<uint2*>(o_out + (size_t)out_row(r) * D + c) = packed;
  }
}

}  // namespace bd
