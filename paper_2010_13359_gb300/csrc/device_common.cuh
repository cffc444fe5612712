// Device helpers shared by the compress kernels: fp32 element rules of the
// method, Philox4x32-10, sign bit packing, and the TMA / mbarrier primitives
// of the staged (shared-memory pipelined) kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.cuh"

namespace dq {

__host__ __device__ __forceinline__ int64_t min64(int64_t x, int64_t y) { return x < y ? x : y; }
__host__ __device__ __forceinline__ int64_t max64(int64_t x, int64_t y) { return x > y ? x : y; }

__device__ __forceinline__ float4 ld_stream4(const float* p) {
  return __ldcs(reinterpret_cast<const float4*>(p));
}
__device__ __forceinline__ void st_stream4(float* p, float4 v) {
  __stcs(reinterpret_cast<float4*>(p), v);
}

// p = fl(fl(eta * g) + e): error feedback of Algorithm 2, two roundings.
__device__ __forceinline__ float ef_p(float lr, float g, float e) { return __fadd_rn(__fmul_rn(lr, g), e); }

// ((|a0| + |a1|) + |a2|) + |a3|: one chunk's share of the bucket l1 sum.
__device__ __forceinline__ float chunk_abs_sum(float a0, float a1, float a2, float a3) {
  return __fadd_rn(__fadd_rn(__fadd_rn(fabsf(a0), fabsf(a1)), fabsf(a2)), fabsf(a3));
}

// Spread the low 8 bits of x so that bit r lands on bit 4r.
__device__ __forceinline__ uint32_t spread_nibbles(uint32_t x) {
  x &= 0xFFu;
  x = (x | (x << 12)) & 0x000F000Fu;
  x = (x | (x << 6)) & 0x03030303u;
  x = (x | (x << 3)) & 0x11111111u;
  return x;
}

// Packs the signs of one row of 32 chunks (128 elements, 4 words) with four
// ballots.  Bit 4r+k of word u of the row is element k of the chunk in lane
// 8u+r: lane 4u+k spreads byte u of ballot k onto bits 4r+k and lanes
// 4u..4u+3 OR their parts together.  Returns the word in lanes 0, 4, 8, 12.
__device__ __forceinline__ uint32_t pack_sign_row(float p0, float p1, float p2, float p3, int lane) {
  const uint32_t B0 = __ballot_sync(kFullMask, p0 < 0.f);
  const uint32_t B1 = __ballot_sync(kFullMask, p1 < 0.f);
  const uint32_t B2 = __ballot_sync(kFullMask, p2 < 0.f);
  const uint32_t B3 = __ballot_sync(kFullMask, p3 < 0.f);
  const int k = lane & 3, u = (lane >> 2) & 3;
  const uint32_t Bk = (k == 0) ? B0 : (k == 1) ? B1 : (k == 2) ? B2 : B3;
  uint32_t v = spread_nibbles(Bk >> (8 * u)) << k;
  v |= __shfl_xor_sync(kFullMask, v, 1);
  v |= __shfl_xor_sync(kFullMask, v, 2);
  return v;
}

// Philox4x32-10 (Salmon et al., SC'11): 10 rounds, multipliers 0xD2511F53 and
// 0xCD9E8D57, Weyl key increments 0x9E3779B9 and 0xBB67AE85 between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 x, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo_a = 0xD2511F53u * x.x;
    const uint32_t hi_a = __umulhi(0xD2511F53u, x.x);
    const uint32_t lo_b = 0xCD9E8D57u * x.z;
    const uint32_t hi_b = __umulhi(0xCD9E8D57u, x.z);
    x = make_uint4(hi_b ^ x.y ^ k0, lo_b, hi_a ^ x.w ^ k1, lo_a);
  }
  return x;
}

// One element of the b-bit stochastic quantiser: code and the residual p - Q(p).
// t = min(fl(|p| * inv), K); r = floor(t); rounds up iff u < t - r, u the top
// 24 bits of the Philox word; code = K -+ level; Q = sign * fl(s * fl(level/K)),
// +0 at level 0.  With s = 0 the caller passes inv = 0, so every element
// takes level 0 (code K) and keeps e = p.
// No clamp of the level is needed: r <= K, and r = K only when t = K, where
// the fraction is 0 and never rounds up.  The residual is formed as p + mag
// for p < 0 and p - mag otherwise, which equals fl(p - Q) for every level:
// at level 0, mag = fl(s * 0) = +0 and p -+ (+0) = p - (+0).
template <int K>
__device__ __forceinline__ void squant_element(float p, float s, float inv, uint32_t rnd,
                                               const float* level_value, int* code, float* resid) {
  const float t = fminf(__fmul_rn(fabsf(p), inv), (float)K);
  const float r = floorf(t);
  const float f = __fsub_rn(t, r);
  const float u = __fmul_rn(__uint2float_rn(rnd >> 8), 0x1p-24f);
  const int level = (int)r + (u < f ? 1 : 0);
  const bool neg = p < 0.f;
  *code = neg ? K - level : K + level;
  const float mag = __fmul_rn(s, level_value[level]);
  *resid = neg ? __fadd_rn(p, mag) : __fsub_rn(p, mag);
}

// ---------------------------------------------------------------------------
// The server's sum over workers (Algorithm 2, server part).  The order is
// fixed so that the parameters are reproducible bit for bit: the M decoded
// values of an element, padded with +0 to the next power of two P >= M, are
// summed pairwise (x_i <- x_2i + x_2i+1 at every level).  Kernels reach that
// tree from groups of consecutive workers whose size is a power of two: a
// full group is a subtree, a partial last group is padded with +0 inside,
// and the group values are combined by the same rule (padding whole groups
// with +0).  Adding a +0 leaf is done as an addition, so that a -0 partial
// sum becomes +0 exactly where the padded tree says.
// ---------------------------------------------------------------------------
__host__ __device__ constexpr int next_pow2(int n) {
  int p = 1;
  while (p < n) p *= 2;
  return p;
}

// A full group of four consecutive workers: (a + b) + (c + d).
__device__ __forceinline__ float tree4(float a, float b, float c, float d) {
  return __fadd_rn(__fadd_rn(a, b), __fadd_rn(c, d));
}

// The value of a group of four (leaves past M given as +0): a subtree of
// the padded tree when M > 4; for M <= 4 the group is the whole tree, over
// P = next_pow2(M) leaves only.
__device__ __forceinline__ float group4(float a, float b, float c, float d, int M) {
  if (M > 2) return tree4(a, b, c, d);
  return M == 2 ? __fadd_rn(a, b) : a;
}

// Pairwise sum of N values (N fixed at compile time), padded with +0 to
// next_pow2(N).
template <int N>
__device__ __forceinline__ float pairwise_n(const float (&v)[N]) {
  constexpr int P = next_pow2(N);
  float x[P];
#pragma unroll
  for (int i = 0; i < P; ++i) x[i] = i < N ? v[i] : 0.f;
#pragma unroll
  for (int w = 1; w < P; w *= 2)
#pragma unroll
    for (int i = 0; i + w < P; i += 2 * w) x[i] = __fadd_rn(x[i], x[i + w]);
  return x[0];
}

// The same sum for a count known only at run time, fed one value (or one
// group value) at a time in order: a binary counter of complete blocks,
// block L holding the sum of 2^L consecutive values.  LEVELS must exceed
// log2 of the largest count.  result() pads with +0 to the next power of
// two: a block whose right sibling is all padding is added to +0.
template <int LEVELS>
struct PairwiseAcc {
  float lvl[LEVELS];
  uint32_t n = 0;

  __device__ __forceinline__ void push(float x) {
    float c = x;
    bool placed = false;
#pragma unroll
    for (int L = 0; L < LEVELS; ++L) {
      if (!placed) {
        if ((n >> L) & 1u) {
          c = __fadd_rn(lvl[L], c);
        } else {
          lvl[L] = c;
          placed = true;
        }
      }
    }
    ++n;
  }

  __device__ __forceinline__ float result() const {
    float c = 0.f, whole = 0.f;
    bool have = false;
#pragma unroll
    for (int L = 0; L < LEVELS; ++L) {
      if (n == (1u << L)) whole = lvl[L];
      if ((1u << L) < n) {  // the levels below the root of the padded tree
        if ((n >> L) & 1u) {
          c = __fadd_rn(lvl[L], have ? c : 0.f);
          have = true;
        } else if (have) {
          c = __fadd_rn(c, 0.f);
        }
      }
    }
    return (n & (n - 1u)) == 0u ? whole : c;
  }
};

// What a server kernel stores for a parameter w with averaged update q:
// Algorithm 2's step w - q, or (under Optimistic Adam, whose own pass
// follows) q itself.
__device__ __forceinline__ float server_out(const ServerArgs& s, float w, float q) {
  return s.store_q ? q : __fsub_rn(w, q);
}

// ---------------------------------------------------------------------------
// mbarrier + 1-D TMA bulk copy (cp.async.bulk) primitives.  Every wait is
// bounded: after kSpinLimit polls (each may sleep up to kSuspendNs) it sets
// kErrTimeout in the launch's error word and returns false.
// ---------------------------------------------------------------------------

// Programmatic dependent launch: the library launches its kernels with the
// programmatic-stream-serialization attribute, so that a kernel is scheduled
// as the blocks of the kernel before it in the stream exit, instead of after
// the whole grid has drained.  Each kernel first waits for that grid to
// complete (its writes visible); it reads and writes nothing before the
// wait.  No kernel triggers its dependents early: that let the next grid's
// blocks sit waiting on the SMs, and measured up to a third slower per step
// (compress and server alternating on the 25M-parameter workload) against
// 1-9 % faster without it.  Without the attribute the wait is a no-op.
__device__ __forceinline__ void dq_pdl_enter() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Index checks of the checked build (compiled with -DDQGAN_CHECK_BOUNDS):
// dq_in_bounds(cond, err) is cond, and when cond is false it also sets
// kErrBounds in the launch's error word, so that the caller skips the access
// and dqgan_synchronize reports DQGAN_ERR_BOUNDS.  In the normal build it is
// cond alone (where cond holds by construction, the compiler drops it).
__device__ __forceinline__ bool dq_in_bounds(bool cond, uint32_t* err) {
#ifdef DQGAN_CHECK_BOUNDS
  if (!cond) atomicOr(err, kErrBounds);
#else
  (void)err;
#endif
  return cond;
}
constexpr uint32_t kSpinLimit = 1u << 21;
constexpr uint32_t kSuspendNs = 500u;

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity), "r"(kSuspendNs)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, uint32_t* err) {
  for (uint32_t it = 0; it < kSpinLimit; ++it)
    if (mbar_try_wait(bar, parity)) return true;
  atomicOr(err, kErrTimeout);
  return false;
}

// 2-D tiled TMA load of one box of `tmap` at coordinates (x, y) (x counts
// innermost elements; x * element size must be a multiple of 16 bytes).
__device__ __forceinline__ void tma_load_2d(void* dst_smem, const void* tmap, int32_t x, int32_t y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst_smem)),
      "l"(tmap), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

// Orders this thread's earlier generic-proxy shared-memory accesses before
// later async-proxy (TMA) accesses.
__device__ __forceinline__ void fence_proxy_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 2-D tiled TMA store of one box from shared memory to `tmap` at (x, y)
// (x, y >= 0; the part of the box outside the tensor is not written),
// committed as this thread's next bulk group.
__device__ __forceinline__ void tma_store_2d(const void* tmap, int32_t x, int32_t y, const void* src_smem) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(tmap), "r"(x),
               "r"(y), "r"(smem_addr(src_smem))
               : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// Waits until this thread's bulk stores have finished reading shared memory.
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

// Waits until this thread's bulk stores are complete.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Global -> shared bulk copy of `bytes` (multiple of 16, both addresses
// 16-byte aligned); completion counted on `bar`.
__device__ __forceinline__ void tma_load_1d(void* dst_smem, const void* src_gmem, uint32_t bytes,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

}  // namespace dq
