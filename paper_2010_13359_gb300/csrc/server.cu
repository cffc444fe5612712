// Server side of Algorithm 2 (DQGAN), fused into one pass per compressor:
//   decode the M messages, q_hat = fl(sum_m Q_m / M), w = fl(w - q_hat).
// and the worker lookahead w_{t-1/2} = fl(w - h).
//
// Every kernel takes the sum over workers in the one order the library fixes
// (device_common.cuh): the M values padded with +0 to a power of two and
// summed pairwise, reached through groups of consecutive workers (four for
// the sign tables and the generic kernels, two for the b = 2 pair tables).
// The parameters therefore come out the same bit for bit whichever kernel
// runs.
//
// Sign with buckets >= 512: bit-transposed table decode (the column and
// warp-transpose kernels for M <= 32, words staged by TMA; flat buckets or a
// per-bucket slice table with layer segments).  Stochastic quantiser with
// M <= 32: code words staged by TMA, per-worker or pair-table decode (and,
// for 8-bit codes with layer segments and 16 workers, slices from a
// per-bucket table).  The rest -- identity, sign with buckets < 512, more
// than 32 workers -- one thread per 4-element chunk of w walks the M
// messages in groups of four workers.  w is read and written once; every
// kernel waits for the grid before it (programmatic dependent launch).
#include "device_common.cuh"

namespace dq {
namespace {

__device__ __forceinline__ float average(float acc, const ServerArgs& s) {
  return s.M_pow2 ? __fmul_rn(acc, s.inv_M) : __fdiv_rn(acc, (float)s.M);
}

// q_hat = acc / M; with M a power of two the product by the exact 1/M.
template <bool POW2>
__device__ __forceinline__ float average_t(float acc, const ServerArgs& s) {
  if constexpr (POW2) return __fmul_rn(acc, s.inv_M);
  else return __fdiv_rn(acc, (float)s.M);
}

// Applies w_j = fl(w_j - acc_j / M) for the chunk at element j.
__device__ __forceinline__ void apply_chunk(const ServerArgs& s, int64_t j, const float (&acc)[4]) {
  if (j + 3 < s.d) {
    float4 wv = __ldcs(reinterpret_cast<const float4*>(s.w + j));
    wv.x = server_out(s, wv.x, average(acc[0], s));
    wv.y = server_out(s, wv.y, average(acc[1], s));
    wv.z = server_out(s, wv.z, average(acc[2], s));
    wv.w = server_out(s, wv.w, average(acc[3], s));
    __stcs(reinterpret_cast<float4*>(s.w + j), wv);
  } else {
    for (int q = 0; q < 4 && j + q < s.d; ++q) s.w[j + q] = server_out(s, s.w[j + q], average(acc[q], s));
  }
}

// Scaled sign, any bucket: Q_m(p)_j = bit ? -s_m : s_m, message words and
// scales fetched 8 workers at a time, summed as two groups of four.
constexpr int kSumLevels = 11;  // group counts up to 1024 (M <= 4096)

__global__ void __launch_bounds__(256) sign_server_kernel(const ServerArgs s) {
  dq_pdl_enter();
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t j = 4 * c;
  if (j >= s.d) return;
  const int64_t bkt = s.word_bucket ? (int64_t)s.word_bucket[j >> 5] : j / s.bucket;
  const int64_t word = j >> 5;
  const int shift = (int)(j & 31);
  PairwiseAcc<kSumLevels> acc[4];
  for (int m0 = 0; m0 < s.M; m0 += 8) {
    float sc[8];
    uint32_t bits[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      sc[u] = 0.f;
      bits[u] = 0;
      if (m0 + u < s.M) {
        const uint8_t* msg = s.msgs + (int64_t)(m0 + u) * s.msg_stride;
        sc[u] = __ldg(reinterpret_cast<const float*>(msg) + bkt);
        bits[u] = __ldg(reinterpret_cast<const uint32_t*>(msg + s.off_payload) + word) >> shift;
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (m0 + 4 * h < s.M) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float v[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int x = 4 * h + u;
            v[u] = (m0 + x < s.M) ? (((bits[x] >> q) & 1u) ? -sc[x] : sc[x]) : 0.f;  // +0 past M
          }
          acc[q].push(group4(v[0], v[1], v[2], v[3], s.M));
        }
      }
    }
  }
  float sum[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) sum[q] = acc[q].result();
  apply_chunk(s, j, sum);
}

// 32x32 bit transpose across a warp: on entry lane m holds row m; on exit
// lane l holds column l (bit m = bit l of row m).  Five block-swap stages;
// each is a shuffle, a rotate and a bit-select.  The per-lane masks and
// rotate amounts do not depend on the data and are computed once.
struct TransposeLane {
  uint32_t keep[5];
  uint32_t rot[5];
  __device__ __forceinline__ explicit TransposeLane(int lane) {
    const uint32_t masks[5] = {0x0000FFFFu, 0x00FF00FFu, 0x0F0F0F0Fu, 0x33333333u, 0x55555555u};
#pragma unroll
    for (int st = 0; st < 5; ++st) {
      const int jj = 16 >> st;
      const bool lower = (lane & jj) == 0;
      keep[st] = lower ? masks[st] : ~masks[st];
      rot[st] = lower ? jj : 32 - jj;
    }
  }
};

__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x, const TransposeLane& tl) {
#pragma unroll
  for (int st = 0; st < 5; ++st) {
    const uint32_t y = __shfl_xor_sync(kFullMask, x, 16 >> st);
    const uint32_t t = __funnelshift_l(y, y, tl.rot[st]);
    x = (x & tl.keep[st]) | (t & ~tl.keep[st]);
  }
  return x;
}

// Scaled sign, buckets of 512..4096.  One warp per (bucket, slice of up to 32
// message words = 1024 elements), no shared memory and no block barriers.
// Lane m loads worker m's words of the slice (32 contiguous bytes at a time)
// and a warp transpose gives lane l the M sign bits of one element.  The sum
// over workers comes from per-bucket tables of four-worker group values:
// T_g[v] = the group's subtree (a + b) + (c + d) over the leaves
// bit r of v ? -s_{4g+r} : s_{4g+r} (+0 past M), held in registers two
// groups per register -- lane l of register a keeps T_{2a + l/16}[l mod 16]
// -- so that a lookup is one shuffle whose source lane is the group's 4-bit
// field, plus 16 for an odd group (shuffles take the lane index mod 32).
// The NG = ceil(M/4) group values are then summed pairwise, padded with +0
// groups to a power of two: the library's fixed order of the sum.
constexpr int kSliceWords = 32;

// T[a] of groups 2a (lanes 0..15) and 2a + 1 (lanes 16..31) for the
// workers of one 32-worker slab: in_slab of them present, M in all.
template <int NR>
__device__ __forceinline__ void build_group_tables(float my_scale, int in_slab, int M, int lane, float (&T)[NR]) {
  const int pat = lane & 15;
  const int hi = lane >> 4;
#pragma unroll
  for (int a = 0; a < NR; ++a) {
    float leaf[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int wk = 4 * (2 * a + hi) + r;  // <= 31
      const float sc = __shfl_sync(kFullMask, my_scale, wk);
      leaf[r] = wk < in_slab ? (((pat >> r) & 1) ? -sc : sc) : 0.f;
    }
    T[a] = group4(leaf[0], leaf[1], leaf[2], leaf[3], M);
  }
}

// The sum over the NG groups of one element's transposed sign mask x (bit
// m: worker m negative): one lookup per group, then pairwise.
template <int NG, int NR>
__device__ __forceinline__ float group_sum(uint32_t x, const float (&T)[NR]) {
  static_assert(NR == (NG + 1) / 2, "two groups per table register");
  const uint32_t xe = x & 0x0F0F0F0Fu;                          // fields of groups 0, 2, 4, 6
  const uint32_t xo = ((x >> 4) & 0x0F0F0F0Fu) | 0x10101010u;  // groups 1, 3, 5, 7, in lanes 16..31
  float v[NG];
#pragma unroll
  for (int g = 0; g < NG; ++g) v[g] = __shfl_sync(kFullMask, T[g >> 1], (int)(((g & 1) ? xo : xe) >> (8 * (g >> 1))));
  return pairwise_n<NG>(v);
}

// This lane's 8 message words starting at word w0 (zero past the message).
__device__ __forceinline__ void load_words8(const uint32_t* wp, int64_t w0, int64_t nwords, bool active,
                                            uint32_t (&wd)[8]) {
#pragma unroll
  for (int k = 0; k < 8; ++k) wd[k] = 0;
  if (!active) return;
  if (w0 + 7 < nwords) {
    const uint4 lo = __ldcs(reinterpret_cast<const uint4*>(wp));
    const uint4 hi = __ldcs(reinterpret_cast<const uint4*>(wp) + 1);
    wd[0] = lo.x; wd[1] = lo.y; wd[2] = lo.z; wd[3] = lo.w;
    wd[4] = hi.x; wd[5] = hi.y; wd[6] = hi.z; wd[7] = hi.w;
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (w0 + k < nwords) wd[k] = wp[k];
  }
}

// The table sums of 8 transposed words.
template <int NG, int NR>
__device__ __forceinline__ void sums8(const uint32_t (&wd)[8], const float (&T)[NR], const TransposeLane& tl,
                                      float (&out)[8]) {
#pragma unroll
  for (int k = 0; k < 8; ++k) out[k] = group_sum<NG>(warp_transpose32(wd[k], tl), T);
}

// M <= 32 workers in NG = ceil(M / 4) groups; w updated after every 8 words.
// The next 8 words and parameters are fetched before the current ones are
// decoded.
template <int NG, bool POW2>
__global__ void __launch_bounds__(256) sign_server_shfl_kernel(const ServerArgs s) {
  dq_pdl_enter();
  const int lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int words_per_bucket = s.bucket >> 5;
  const int sw = words_per_bucket < kSliceWords ? words_per_bucket : kSliceWords;  // 16 or 32
  const int spb = words_per_bucket / sw;  // slices per bucket
  const int64_t nb = (s.d + s.bucket - 1) / s.bucket;
  const int64_t b = gw / spb;
  if (b >= nb) return;
  const int64_t wbase = b * words_per_bucket + (gw % spb) * sw;
  const int64_t nwords = (s.d + 31) >> 5;
  const TransposeLane tl(lane);
  const uint8_t* my_msg = s.msgs + (int64_t)lane * s.msg_stride;
  const bool active = lane < s.M;
  const float my_scale = active ? __ldg(reinterpret_cast<const float*>(my_msg) + b) : 0.f;
  float T[(NG + 1) / 2];
  build_group_tables(my_scale, s.M, s.M, lane, T);
  const uint32_t* wp = reinterpret_cast<const uint32_t*>(my_msg + s.off_payload) + wbase;
  float* wl = s.w + 32 * wbase + lane;
  const int64_t jmax = s.d - 32 * wbase - lane;  // wl[32 i] is a parameter iff 32 i < jmax
  const int iters = sw / 8;
  uint32_t wd[8];
  float wv[8];
  load_words8(wp, wbase, nwords, active, wd);
#pragma unroll
  for (int k = 0; k < 8; ++k) wv[k] = (32 * k < jmax) ? __ldcs(wl + 32 * k) : 0.f;
#pragma unroll 1
  for (int it = 0; it < iters; ++it) {
    uint32_t wd_next[8];
    float wv_next[8];
    const bool more = it + 1 < iters;
    if (more) {
      load_words8(wp + 8 * (it + 1), wbase + 8 * (it + 1), nwords, active, wd_next);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int64_t off = 32 * (8 * (it + 1) + k);
        wv_next[k] = (off < jmax) ? __ldcs(wl + off) : 0.f;
      }
    }
    float sum[8];
    sums8<NG>(wd, T, tl, sum);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int64_t off = 32 * (8 * it + k);
      if (off < jmax) __stcs(wl + off, server_out(s, wv[k], average_t<POW2>(sum[k], s)));
    }
    if (more) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        wd[k] = wd_next[k];
        wv[k] = wv_next[k];
      }
    }
  }
}

// Buckets of 1024..4096 with M <= 32: the same decode, with the message
// words staged in shared memory by TMA instead of read by the lanes.  A 2-D
// tensor map views the M messages as rows of u32 words; one box is 32 words
// of every worker (M rows of 128 bytes, 128-byte swizzle: the 16-byte chunk c
// of row r sits at chunk c ^ (r mod 8)), so lane m reads its worker's words
// with conflict-free 128-bit shared loads.  Each warp owns two box buffers
// and one mbarrier per buffer: while it decodes slice i it has the copy of
// slice i + 1 in flight.  Waits are bounded (error word on time-out).
// With layer segments (SEG) the slices come from a host-built table in
// which every slice lies inside one bucket (runs of up to 32 words); the
// word box starts at the 16-byte boundary at or before the slice (36 words
// wide, no swizzle) and each lane realigns its worker's 32 words by the
// slice's word offset; the words of a short slice past its rows are read
// but their elements are not stored.
constexpr int kTmaWarps = 8;
constexpr int kTmaBoxBytes = 32 * 32 * 4;
constexpr int kTmaSegBoxBytes = 32 * kSignSegBoxWords * 4;
template <bool SEG>
constexpr int tma_sign_smem_bytes() { return kTmaWarps * 2 * (SEG ? kTmaSegBoxBytes : kTmaBoxBytes) + 1024; }

struct SegSlices {
  const uint32_t* slices;  // per slice {first word, bucket | (rows - 1) << 27}
  int64_t n;
};

template <int NG, bool POW2, bool SEG>
__global__ void __launch_bounds__(32 * kTmaWarps)
sign_server_tma_kernel(const ServerArgs s, const SegSlices seg, const __grid_constant__ CUtensorMap tmap) {
  dq_pdl_enter();
  constexpr int BOX = SEG ? kTmaSegBoxBytes : kTmaBoxBytes;
  constexpr int PITCH = SEG ? 4 * kSignSegBoxWords : 128;  // bytes of a box row
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t bars[kTmaWarps][2];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  // 1024-byte aligned buffers (required by the 128-byte swizzle)
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* base = smem_raw + ((1024u - (raw & 1023u)) & 1023u);
  uint8_t* const buf0 = base + warp * 2 * BOX;  // buffer i at buf0 + i * BOX
  uint64_t* bar = bars[warp];
  if (lane == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    mbar_fence_init();
  }
  __syncwarp();

  const int words_per_bucket = s.bucket >> 5;  // 32..128
  const int spb = words_per_bucket >> 5;       // 32-word slices per bucket
  const int64_t nb = (s.d + s.bucket - 1) / s.bucket;
  const int64_t nslices = SEG ? seg.n : nb * spb;
  const int64_t stride = (int64_t)gridDim.x * kTmaWarps;
  const int32_t x0 = (int32_t)(s.off_payload >> 2);
  const uint32_t box_bytes = (uint32_t)(s.M < 32 ? s.M : 32) * (uint32_t)PITCH;
  const bool active = lane < s.M;
  const TransposeLane tl(lane);

  int64_t sl = (int64_t)blockIdx.x * kTmaWarps + warp;
  struct Slice {
    int64_t word;    // first message word
    int64_t bucket;
    int rows;        // words in the slice, 1..32
  };
  auto slice_of = [&](int64_t slice) -> Slice {
    if constexpr (SEG) {
      const uint2 e = __ldg(reinterpret_cast<const uint2*>(seg.slices) + slice);
      return Slice{(int64_t)e.x, (int64_t)(e.y & 0x7FFFFFFu), (int)(e.y >> 27) + 1};
    } else {
      const int64_t b = slice / spb;
      return Slice{b * words_per_bucket + (slice - b * spb) * 32, b, 32};
    }
  };
  auto box_x = [&](const Slice& c) {
    const int32_t x = x0 + (int32_t)c.word;
    return SEG ? (x & ~3) : x;  // x0 is a multiple of 64 words
  };
  Slice c = sl < nslices ? slice_of(sl) : Slice{0, 0, 0};
  if (sl < nslices && lane == 0) {
    mbar_arrive_expect_tx(&bar[0], box_bytes);
    tma_load_2d(buf0, &tmap, box_x(c), 0, &bar[0]);
  }
  uint32_t it = 0;
  bool ok = true;
  for (; sl < nslices; sl += stride, ++it) {
    const int cur = (int)(it & 1u);
    const int64_t nxt = sl + stride;
    const Slice cn = nxt < nslices ? slice_of(nxt) : Slice{0, 0, 0};
    if (nxt < nslices && lane == 0) {
      fence_proxy_async_shared();  // this warp's reads of that buffer came before
      mbar_arrive_expect_tx(&bar[cur ^ 1], box_bytes);
      tma_load_2d(buf0 + (cur ^ 1) * BOX, &tmap, box_x(cn), 0, &bar[cur ^ 1]);
    }
    const int64_t b = c.bucket;
    const int64_t wbase = c.word;
    const int woff = SEG ? (int)((x0 + wbase) & 3) : 0;  // the slice's first word in the box rows
    float* wl = s.w + 32 * wbase + lane;
    // wl[32 i] is a parameter of this slice iff 32 i < jmax
    const int64_t jmax = min64(s.d - 32 * wbase - lane, 32 * (int64_t)c.rows);
    float wv[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) wv[k] = (32 * k < jmax) ? __ldcs(wl + 32 * k) : 0.f;
    const float my_scale =
        active ? __ldg(reinterpret_cast<const float*>(s.msgs + (int64_t)lane * s.msg_stride) + b) : 0.f;
    float T[(NG + 1) / 2];
    build_group_tables(my_scale, s.M, s.M, lane, T);
    ok = mbar_wait_bounded(&bar[cur], (it >> 1) & 1u, s.err);
    ok = __all_sync(kFullMask, ok);
    if (!ok) break;
    const uint8_t* row = buf0 + cur * BOX + lane * PITCH;
    const int sw = lane & 7;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint32_t wd[8];
      if (active && SEG) {
        // words 8q .. 8q + 11 of the row (16-byte aligned), then the 8 from woff
        const uint4 a = *reinterpret_cast<const uint4*>(row + 32 * q);
        const uint4 bb = *reinterpret_cast<const uint4*>(row + 32 * q + 16);
        const uint4 cc = *reinterpret_cast<const uint4*>(row + 32 * q + 32);
        const uint32_t r[12] = {a.x, a.y, a.z, a.w, bb.x, bb.y, bb.z, bb.w, cc.x, cc.y, cc.z, cc.w};
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t u01 = (woff & 1) ? r[k + 1] : r[k];
          const uint32_t u23 = (woff & 1) ? r[k + 3] : r[k + 2];
          wd[k] = (woff & 2) ? u23 : u01;
        }
      } else if (active) {
        const uint4 lo = *reinterpret_cast<const uint4*>(row + (((2 * q) ^ sw) << 4));
        const uint4 hi = *reinterpret_cast<const uint4*>(row + (((2 * q + 1) ^ sw) << 4));
        wd[0] = lo.x; wd[1] = lo.y; wd[2] = lo.z; wd[3] = lo.w;
        wd[4] = hi.x; wd[5] = hi.y; wd[6] = hi.z; wd[7] = hi.w;
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) wd[k] = 0u;
      }
      float wv_next[8];
      if (q < 3) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int64_t off = 32 * (8 * (q + 1) + k);
          wv_next[k] = (off < jmax) ? __ldcs(wl + off) : 0.f;
        }
      }
      float sum[8];
      sums8<NG>(wd, T, tl, sum);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int64_t off = 32 * (8 * q + k);
        if (off < jmax) __stcs(wl + off, server_out(s, wv[k], average_t<POW2>(sum[k], s)));
      }
      if (q < 3) {
#pragma unroll
        for (int k = 0; k < 8; ++k) wv[k] = wv_next[k];
      }
    }
    __syncwarp();
    c = cn;
  }
  // after a time-out the copy of the next slice may still be in flight
  if (!ok && lane == 0 && sl + stride < nslices)
    mbar_wait_bounded(&bar[(it & 1u) ^ 1u], ((it + 1) >> 1) & 1u, s.err);
}

// Buckets of 1024..4096 with M <= 32 and d >= 32, column form.  Each warp
// owns a contiguous range of 1024-element slices (32 message words).  TMA
// brings the slice's words of every worker (box 32 words x M, 128-byte
// swizzle) and the slice's 1024 parameters (box 32 rows x 32 floats of w
// viewed as rows of 32, 128-byte swizzle) into shared memory.  Lane l reads
// column l, word l of each worker, and transposes the 32 x 32 bit block in
// its own registers, so that it holds the M sign bits of each of the 32
// elements of that word; the worker sum comes from the four-worker group
// tables looked up by shuffle (rebuilt only when the bucket changes).  The
// lane updates its row of 32 parameters in shared memory and one TMA store
// writes the box back.  Per warp two word and two parameter buffers: the
// next slice's boxes load while this one is decoded and updated.
// With layer segments (SEG) every slice lies inside one bucket: a host-built
// table lists each bucket's runs of up to 32 words; the word box starts at
// the 16-byte boundary at or before the slice (36 words wide, no swizzle),
// and a slice shorter than 32 rows, or one that reaches the partial last
// row, updates its parameters with plain loads and stores (a box store would
// overlap the next slice).
// Against sign_server_tma_kernel: no warp transpose, 8 shuffles per element
// at M = 32 instead of 13.
constexpr int kColWarps = 12;
constexpr int kColBox = 4096;        // bytes of a parameter box, and of a word box of the flat form
constexpr int kSegBoxWords = kSignSegBoxWords;

// Per-warp shared memory of the column kernel: two parameter boxes, then two
// word boxes (every swizzled box 1024-byte aligned).
template <bool SEG>
struct ColLayout {
  static constexpr int kWBox = SEG ? 32 * kSegBoxWords * 4 : kColBox;
  static constexpr int kWarpBytes = 2 * kColBox + 2 * kWBox;
  static constexpr int kSmem = kColWarps * kWarpBytes + 1024;  // + alignment slack
  static_assert(kWarpBytes % 1024 == 0, "boxes stay 1024-byte aligned");
};

// In-register transpose of a 32 x 32 bit block: on exit bit m of a[e] is
// bit e of the entry a[m].  Block swaps of 16 and 8 bits by byte permutes,
// then of 4, 2 and 1 bits by shifts and masks.
template <int J>
__device__ __forceinline__ void swap_stage(uint32_t (&a)[32], uint32_t m) {
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    if ((k & J) == 0) {
      const uint32_t x = a[k], y = a[k + J];
      a[k] = (x & m) | ((y << J) & ~m);
      a[k + J] = ((x >> J) & m) | (y & ~m);
    }
  }
}

__device__ __forceinline__ void transpose32_regs(uint32_t (&a)[32]) {
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const uint32_t x = a[k], y = a[k + 16];
    a[k] = __byte_perm(x, y, 0x5410);
    a[k + 16] = __byte_perm(x, y, 0x7632);
  }
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    if ((k & 8) == 0) {
      const uint32_t x = a[k], y = a[k + 8];
      a[k] = __byte_perm(x, y, 0x6240);
      a[k + 8] = __byte_perm(x, y, 0x7351);
    }
  }
  swap_stage<4>(a, 0x0F0F0F0Fu);
  swap_stage<2>(a, 0x33333333u);
  swap_stage<1>(a, 0x55555555u);
}

// The slice table of the layer-segmented form.
template <int NG, bool POW2, bool SEG>
__global__ void __launch_bounds__(32 * kColWarps, 1)
sign_server_col_kernel(const ServerArgs s, const SegSlices seg, const __grid_constant__ CUtensorMap wmap,
                       const __grid_constant__ CUtensorMap pmap) {
  dq_pdl_enter();
  using L = ColLayout<SEG>;
  constexpr int ROWS = 4 * NG < 32 ? 4 * NG : 32;  // message rows that can hold a worker
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t bars[kColWarps][4];  // word boxes 0 and 1, parameter boxes 0 and 1
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* const pbuf = smem_raw + ((1024u - (raw & 1023u)) & 1023u) + warp * L::kWarpBytes;  // + i * kColBox
  uint8_t* const wbuf = pbuf + 2 * kColBox;                                                     // + i * L::kWBox
  uint64_t* wbar = &bars[warp][0];
  uint64_t* pbar = &bars[warp][2];
  if (lane == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(&bars[warp][i], 1);
    mbar_fence_init();
  }
  __syncwarp();

  const int words_per_bucket = s.bucket >> 5;  // 32..128
  const int spb = words_per_bucket >> 5;       // slices per bucket (flat form)
  const int64_t nslices = SEG ? seg.n : ((s.d + s.bucket - 1) / s.bucket) * spb;
  const int64_t nrows = s.d >> 5;              // rows of the parameter map
  const int tail = (int)(s.d & 31);            // elements of the partial row nrows
  const int32_t x0 = (int32_t)(s.off_payload >> 2);
  const uint32_t wbytes = (uint32_t)(s.M < 32 ? s.M : 32) * (SEG ? 4u * kSegBoxWords : 128u);
  // this warp's slices [lo, hi): an even split of nslices over the grid's warps
  const int64_t nwarps = (int64_t)gridDim.x * kColWarps;
  const int64_t gw = (int64_t)blockIdx.x * kColWarps + warp;
  const int64_t lo = nslices * gw / nwarps;
  const int64_t hi = nslices * (gw + 1) / nwarps;
  struct Slice {
    int64_t word;    // first message word = first parameter row
    int64_t bucket;
    int rows;        // words (rows) in the slice, 1..32
  };
  auto slice_of = [&](int64_t sl) -> Slice {
    if constexpr (SEG) {
      const uint2 e = __ldg(reinterpret_cast<const uint2*>(seg.slices) + sl);
      return Slice{(int64_t)e.x, (int64_t)(e.y & 0x7FFFFFFu), (int)(e.y >> 27) + 1};
    } else {
      const int64_t b = sl / spb;
      return Slice{b * words_per_bucket + (sl - b * spb) * 32, b, 32};
    }
  };
  // whether the slice's parameters move as one TMA box: flat, the box starts
  // inside the map (its rows past the map read as zero and are not stored);
  // layer segments, all 32 rows lie inside the map
  auto boxed = [&](const Slice& c) { return SEG ? (c.rows == 32 && c.word + 32 <= nrows) : (c.word < nrows); };
  // lane 0: copies of slice c into buffers i (phases issued and waited for
  // on each barrier are counted; at most one is outstanding)
  uint32_t w_issued0 = 0, w_issued1 = 0, w_done0 = 0, w_done1 = 0;
  uint32_t p_issued0 = 0, p_issued1 = 0, p_done0 = 0, p_done1 = 0;
  auto issue = [&](const Slice& c, int i) {
    if (i) ++w_issued1; else ++w_issued0;
    mbar_arrive_expect_tx(&wbar[i], wbytes);
    const int32_t x = x0 + (int32_t)c.word;
    tma_load_2d(wbuf + i * L::kWBox, &wmap, SEG ? (x & ~3) : x, 0, &wbar[i]);
    if (i) ++p_issued1; else ++p_issued0;
    if (boxed(c)) {
      mbar_arrive_expect_tx(&pbar[i], (uint32_t)kColBox);
      tma_load_2d(pbuf + i * kColBox, &pmap, 0, (int32_t)c.word, &pbar[i]);
    } else {
      mbar_arrive(&pbar[i]);  // nothing to copy: complete the phase
    }
  };
  // byte offset of word `lane` in row m of a swizzled box: chunk (lane / 4) ^ (m mod 8)
  const uint32_t lane_lo = (uint32_t)(lane & 3) << 2;
  const uint32_t lane_chunk = (uint32_t)(lane >> 2);

  Slice c = lo < hi ? slice_of(lo) : Slice{0, 0, 0};
  if (lo < hi && lane == 0) issue(c, 0);
  // worker `lane`'s scale of a bucket; loaded one slice ahead, so that a new
  // bucket's tables do not wait for it
  auto scale_of_bucket = [&](int64_t bkt) -> float {
    return lane < s.M ? __ldg(reinterpret_cast<const float*>(s.msgs + (int64_t)lane * s.msg_stride) + bkt) : 0.f;
  };
  float scale_next = lo < hi ? scale_of_bucket(c.bucket) : 0.f;
  float T[(NG + 1) / 2];
  int64_t table_b = -1;
  uint32_t it = 0;
  bool ok = true;
  for (int64_t sl = lo; sl < hi; ++sl, ++it) {
    const int cur = (int)(it & 1u);
    const bool more = sl + 1 < hi;
    const Slice cn = more ? slice_of(sl + 1) : c;
    if (more && lane == 0) {
      bulk_wait_read_all();        // the store of the previous slice has read its parameter box
      fence_proxy_async_shared();  // this warp's reads of those boxes came before
      issue(cn, cur ^ 1);
    }
    const float scale_cur = scale_next;  // of bucket c.bucket
    if (more && cn.bucket != c.bucket) scale_next = scale_of_bucket(cn.bucket);
    if (c.bucket != table_b) {  // warp-uniform
      table_b = c.bucket;
      const float my_scale = scale_cur;
      build_group_tables(my_scale, s.M, s.M, lane, T);
    }
    ok = mbar_wait_bounded(&wbar[cur], (it >> 1) & 1u, s.err);
    ok = __all_sync(kFullMask, ok);
    if (!ok) break;
    if (cur) ++w_done1; else ++w_done0;
    const uint8_t* const wb = wbuf + cur * L::kWBox;
    const uint32_t seg_off = SEG ? (((uint32_t)(x0 + c.word) & 3u) + (uint32_t)lane) * 4u : 0u;
    uint32_t x[32];
#pragma unroll
    for (int m = 0; m < 32; ++m) {
      x[m] = 0u;
      if (m < ROWS && m < s.M) {
        const uint32_t off = SEG ? (uint32_t)(m * 4 * kSegBoxWords) + seg_off
                                 : (uint32_t)(m * 128) + (((lane_chunk ^ (uint32_t)(m & 7)) << 4) | lane_lo);
        x[m] = *reinterpret_cast<const uint32_t*>(wb + off);
      }
    }
    transpose32_regs(x);  // x[e]: bit m = worker m's sign of element 32 (c.word + lane) + e
    ok = mbar_wait_bounded(&pbar[cur], (it >> 1) & 1u, s.err);
    ok = __all_sync(kFullMask, ok);
    if (!ok) break;
    if (cur) ++p_done1; else ++p_done0;
    const bool in_box = boxed(c);
    const int64_t row = c.word + lane;
    // rows updated with plain loads and stores: flat, the partial last row
    // (rows past it hold no parameters); layer segments, the partial last row
    // of a boxed slice, or every row of a slice without a box
    const bool direct = (SEG && !in_box) ? (lane < c.rows) : (row == nrows && tail != 0);
    const int cnt = row == nrows ? tail : 32;  // parameters in the row
    float* const wg = s.w + 32 * row;
    uint8_t* const prow = pbuf + cur * kColBox + lane * 128;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      float4* slot = reinterpret_cast<float4*>(prow + ((q ^ (lane & 7)) << 4));
      float o[4] = {0.f, 0.f, 0.f, 0.f};
      if (in_box) {
        const float4 wv = *slot;
        o[0] = wv.x; o[1] = wv.y; o[2] = wv.z; o[3] = wv.w;
      }
      if (direct) {
#pragma unroll
        for (int r = 0; r < 4; ++r) o[r] = (4 * q + r < cnt) ? wg[4 * q + r] : 0.f;
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) o[r] = server_out(s, o[r], average_t<POW2>(group_sum<NG>(x[4 * q + r], T), s));
      if (direct) {
#pragma unroll
        for (int r = 0; r < 4; ++r)
          if (4 * q + r < cnt) wg[4 * q + r] = o[r];
      }
      if (in_box) *slot = make_float4(o[0], o[1], o[2], o[3]);
    }
    fence_proxy_async_shared();  // the box writes above, before the store reads them
    __syncwarp();
    if (lane == 0 && in_box) tma_store_2d(&pmap, 0, (int32_t)c.word, pbuf + cur * kColBox);
    __syncwarp();
    c = cn;
  }
  if (lane == 0) {
    bulk_wait_all();  // stores complete before the block's shared memory is released
    // after a time-out, copies already issued may still be in flight
    if (!ok) {
      if (w_issued0 > w_done0) mbar_wait_bounded(&wbar[0], w_done0 & 1u, s.err);
      if (w_issued1 > w_done1) mbar_wait_bounded(&wbar[1], w_done1 & 1u, s.err);
      if (p_issued0 > p_done0) mbar_wait_bounded(&pbar[0], p_done0 & 1u, s.err);
      if (p_issued1 > p_done1) mbar_wait_bounded(&pbar[1], p_done1 & 1u, s.err);
    }
  }
}

// M above 32: workers taken 32 at a time.  With M > 32 the padded tree has
// at least 64 leaves, so each 32-worker slab (the last one padded with +0
// groups) is a subtree: per 8-word chunk of the slice, every slab's sum of
// the chunk's elements goes into a per-element pairwise accumulator over
// slabs, and w is updated once all slabs are in.
constexpr int kSlabLevels = 8;  // up to 128 slabs (M <= 4096)

__global__ void __launch_bounds__(256) sign_server_slabs_kernel(const ServerArgs s) {
  dq_pdl_enter();
  const int lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int words_per_bucket = s.bucket >> 5;
  const int sw = words_per_bucket < kSliceWords ? words_per_bucket : kSliceWords;
  const int spb = words_per_bucket / sw;
  const int64_t nb = (s.d + s.bucket - 1) / s.bucket;
  const int64_t b = gw / spb;
  if (b >= nb) return;
  const int64_t wbase = b * words_per_bucket + (gw % spb) * sw;
  const int64_t nwords = (s.d + 31) >> 5;
  const TransposeLane tl(lane);
  const int nslabs = (s.M + 31) / 32;
  for (int it = 0; it * 8 < sw; ++it) {
    PairwiseAcc<kSlabLevels> acc[8];
    for (int slab = 0; slab < nslabs; ++slab) {
      const int in_slab = min(32, s.M - slab * 32);
      const uint8_t* my_msg = s.msgs + (int64_t)(slab * 32 + lane) * s.msg_stride;
      const float my_scale = (lane < in_slab) ? __ldg(reinterpret_cast<const float*>(my_msg) + b) : 0.f;
      float T[4];
      build_group_tables(my_scale, in_slab, s.M, lane, T);
      const int64_t w0 = wbase + 8 * it;
      uint32_t wd[8];
      load_words8(reinterpret_cast<const uint32_t*>(my_msg + s.off_payload) + w0, w0, nwords, lane < in_slab, wd);
      float v[8];
      sums8<8>(wd, T, tl, v);
#pragma unroll
      for (int k = 0; k < 8; ++k) acc[k].push(v[k]);
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int64_t j = 32 * (wbase + 8 * it + k) + lane;
      if (j < s.d) __stcs(s.w + j, server_out(s, __ldcs(s.w + j), average(acc[k].result(), s)));
    }
  }
}

// b-bit stochastic quantiser: Q_m(p)_j = fl(s_m * V[code]) with
// V[code] = sign(code - K) * fl(|code - K| / K) (so V[K] = +0), summed as
// groups of four workers in the library's pairwise order.  One thread per
// 4-element chunk (a fixed grid strides over the chunks), code words of 8
// workers fetched before they are decoded.  For
// b = 4, 8 V lives in shared memory replicated once per bank (entry c of lane
// l at [c][l]), so the random code lookups of a warp never conflict; for
// b = 2 (V in {-1, 0, +1}) the value is a select.
template <int BITS, bool POW2>
__global__ void __launch_bounds__(256) squant_server_kernel(const ServerArgs s) {
  dq_pdl_enter();
  constexpr int K = (1 << (BITS - 1)) - 1;
  constexpr uint32_t MASK = (1u << BITS) - 1u;
  constexpr int CODES = (BITS == 2) ? 1 : (1 << BITS);
  __shared__ float V[CODES * 32];
  if constexpr (BITS != 2) {
    for (int t = threadIdx.x; t < CODES * 32; t += blockDim.x) {
      const int code = t >> 5;
      const int level = code - K;
      float v = 0.f;
      if (code <= 2 * K && level != 0) {
        const float mag = __fdiv_rn((float)(level < 0 ? -level : level), (float)K);
        v = level < 0 ? -mag : mag;
      }
      V[t] = v;
    }
    __syncthreads();
  }
  const float* Vl = V + (threadIdx.x & 31);
  const int64_t nchunks = (s.d + 3) >> 2;
  for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < nchunks;
       c += (int64_t)gridDim.x * blockDim.x) {
    const int64_t j = 4 * c;
    const int64_t bkt = s.word_bucket ? (int64_t)s.word_bucket[j >> 5] : j / s.bucket;
    const int64_t bitpos = j * BITS;  // a chunk's 4*BITS bits never straddle a word
    const int64_t word = bitpos >> 5;
    const int shift = (int)(bitpos & 31);
    const uint8_t* m_scale = s.msgs + 4 * bkt;
    const uint8_t* m_word = s.msgs + s.off_payload + 4 * word;
    PairwiseAcc<kSumLevels> sum[4];
    for (int m0 = 0; m0 < s.M; m0 += 8) {
      uint32_t bits[8];
      float sc[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const bool ok = m0 + u < s.M;
        const int64_t off = (int64_t)(m0 + u) * s.msg_stride;
        bits[u] = ok ? __ldcs(reinterpret_cast<const uint32_t*>(m_word + off)) >> shift : 0u;
        sc[u] = ok ? __ldg(reinterpret_cast<const float*>(m_scale + off)) : 0.f;
      }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (m0 + 4 * h < s.M) {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float v[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) {
              const int u = 4 * h + x;
              if constexpr (BITS == 2) {
                const uint32_t code = (bits[u] >> (2 * q)) & 3u;
                v[x] = (code == 0) ? -sc[u] : (code == 2 ? sc[u] : 0.f);  // fl(s * 1) = s
              } else if constexpr (BITS == 8) {
                v[x] = __fmul_rn(sc[u], Vl[__byte_perm(bits[u], 0, 0x4440 | q) << 5]);
              } else {
                v[x] = __fmul_rn(sc[u], Vl[((bits[u] >> (q * BITS)) & MASK) << 5]);
              }
              if (m0 + u >= s.M) v[x] = 0.f;  // padding leaves
            }
            sum[q].push(group4(v[0], v[1], v[2], v[3], s.M));
          }
        }
      }
    }
    float acc[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] = sum[q].result();
    if (j + 3 < s.d) {
      float4 wv = __ldcs(reinterpret_cast<const float4*>(s.w + j));
      wv.x = server_out(s, wv.x, average_t<POW2>(acc[0], s));
      wv.y = server_out(s, wv.y, average_t<POW2>(acc[1], s));
      wv.z = server_out(s, wv.z, average_t<POW2>(acc[2], s));
      wv.w = server_out(s, wv.w, average_t<POW2>(acc[3], s));
      __stcs(reinterpret_cast<float4*>(s.w + j), wv);
    } else {
      for (int q = 0; q < 4 && j + q < s.d; ++q)
        s.w[j + q] = server_out(s, s.w[j + q], average_t<POW2>(acc[q], s));
    }
  }
}

// Transpose of a 16 x 16 block of 2-bit entries held one row per register:
// on entry entry e of a[m] is at bits 2e; on exit entry m of a[e] is the old
// entry e of a[m].  Block swaps of 8 and 4 entries by byte permutes, then of
// 2 and 1 entries by shifts and masks (rows k and k + B, S = 2B bits).
template <int B, int S>
__device__ __forceinline__ void swap_stage16(uint32_t (&a)[16], uint32_t m) {
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    if ((k & B) == 0) {
      const uint32_t x = a[k], y = a[k + B];
      a[k] = (x & m) | ((y << S) & ~m);
      a[k + B] = ((x >> S) & m) | (y & ~m);
    }
  }
}

__device__ __forceinline__ void transpose16x2_regs(uint32_t (&a)[16]) {
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const uint32_t x = a[k], y = a[k + 8];
    a[k] = __byte_perm(x, y, 0x5410);
    a[k + 8] = __byte_perm(x, y, 0x7632);
  }
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    if ((k & 4) == 0) {
      const uint32_t x = a[k], y = a[k + 4];
      a[k] = __byte_perm(x, y, 0x6240);
      a[k + 4] = __byte_perm(x, y, 0x7351);
    }
  }
  swap_stage16<2, 4>(a, 0x0F0F0F0Fu);
  swap_stage16<1, 2>(a, 0x33333333u);
}

// b = 2 sums over workers by pair tables.  The decoded value of a 2-bit code
// is v(0, s) = -s, v(1, s) = +0, v(2, s) = +s (code 3 never occurs; 0 here).
// Pair p = workers (2p, 2p + 1), the lowest subtrees of the padded tree once
// M >= 2: lane l holds
//   T_p[l mod 16] = fl(v(l mod 4, s_2p) + v((l / 4) mod 4, s_2p+1)),
// the pair's value for the 4-bit field code_2p | code_2p+1 << 2.  A worker at
// or beyond M has scale 0 and reads as code 1, so it adds a +0 leaf; with
// M = 1 the tree is the single leaf and T_0 holds v(c, s_0) alone.
template <int NP>
__device__ __forceinline__ void build_pair_tables(float my_scale, int lane, int M, float (&T)[NP]) {
  const int ca = lane & 3, cb = (lane >> 2) & 3;
  const float fa = ca == 0 ? -1.f : (ca == 2 ? 1.f : 0.f);  // v(c, s) = f(c) * s exactly
  const float fb = cb == 0 ? -1.f : (cb == 2 ? 1.f : 0.f);
#pragma unroll
  for (int p = 0; p < NP; ++p) {
    const float sa = __shfl_sync(kFullMask, my_scale, 2 * p);
    const float sb = __shfl_sync(kFullMask, my_scale, 2 * p + 1);
    const float va = __fmul_rn(fa, sa);
    T[p] = M == 1 ? va : __fadd_rn(va, __fmul_rn(fb, sb));
  }
}

// The b = 2 server update of this lane's 16 elements in wv (server_out of
// sum_j / M), with the worker sums by pair tables: the lane's code word of
// each worker (16 per set of workers) is transposed so that one register
// holds one element's codes of 16 workers, whose 4-bit pair fields index the
// pair tables by shuffle (the lane index is taken mod 32: the tables repeat
// in lanes 16..31, so the bits above a field do not matter).  The pair
// values are summed pairwise over the padded tree's next_pow2(ceil(M/2))
// pairs (one set: 1, 2, 4 or 8 of them, the level picked by M; two sets:
// the two 8-pair sums added last).
template <int NSET, bool POW2, int FM>
__device__ __forceinline__ void b2_pair_table_update(const uint32_t* words, const ServerArgs& s,
                                                     const float (&T)[8 * NSET], float (&wv)[16]) {
  const int M = FM > 0 ? FM : s.M;
  const int np = next_pow2((M + 1) / 2);  // pairs in the padded tree (NSET = 2: 16)
  float acc[16];
#pragma unroll
  for (int set = 0; set < NSET; ++set) {
    uint32_t z[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      const int m = 16 * set + r;
      z[r] = m < M ? words[32 * m] : 0x55555555u;  // rows past M: level-0 codes (never read past the box)
    }
    transpose16x2_regs(z);
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      float v[8];
#pragma unroll
      for (int p = 0; p < 8; ++p) v[p] = __shfl_sync(kFullMask, T[8 * set + p], (int)(z[e] >> (4 * p)));
      const float a01 = __fadd_rn(v[0], v[1]), a23 = __fadd_rn(v[2], v[3]);
      const float a03 = __fadd_rn(a01, a23);
      const float sum = np >= 8 ? __fadd_rn(a03, __fadd_rn(__fadd_rn(v[4], v[5]), __fadd_rn(v[6], v[7])))
                                : (np == 4 ? a03 : (np == 2 ? a01 : v[0]));
      acc[e] = set == 0 ? sum : __fadd_rn(acc[e], sum);
      if (set + 1 == NSET) wv[e] = server_out(s, wv[e], average_t<POW2>(acc[e], s));
    }
  }
}

// Passes over a lane's 8 elements in the b = 4 per-worker decode (1 or 2).
constexpr int kSquant4Parts = 1;


// b = 4 and 8 load each slice's scale (b = 8: and the lane's parameters)
// one slice ahead; b = 4 writes its parameters back with plain stores
// instead of a TMA store of the box, which frees the box as soon as the
// lanes have read it.  (Both measured faster at d = 25M, M = 16; b = 2
// measured slower with either change and keeps the TMA store and the
// per-slice scale load.)
constexpr bool sq_prefetch(int bits) { return bits != 2; }
constexpr bool sq_direct_store(int bits) { return bits == 4; }

// Whether the squant server stages the parameters by TMA (b = 2 and 4; for
// b = 8 a lane's 16 bytes of w are contiguous across the warp already).
constexpr bool sq_params_boxed(int bits) { return bits != 8; }

// b-bit stochastic quantiser with M <= 32 and buckets of at least 32*32/b
// elements: the code words are staged by TMA like the sign words above (a
// box is 32 words of every worker, M rows of 128 bytes, no swizzle: lane l
// reads word l of row m, one conflict-free 128-byte row per worker).  Lane l
// owns the 32/b consecutive elements of its word; per worker it decodes them
// with the worker's scale (broadcast by shuffle from the lane that loaded it)
// and V[code] (b = 8: the bank-replicated table; b = 4: the worker's 15
// products fl(s * V[c]), one per lane, looked up by shuffle), four workers
// at a time into the group value (a + b) + (c + d), and the groups are
// summed pairwise: the library's fixed order.  b = 2 sums by pair tables
// instead (b2_pair_table_update, NSET sets of 16 workers; tables rebuilt only
// when the bucket changes), which reach the same tree from pairs of workers.
// With layer segments (SEG) a slice may hold words of several buckets: each
// lane then reads the workers' scales of its own word's bucket (b = 2: two
// bit tests per worker and element, then the groups of four).
// For b = 2 and 4 (a lane owns 64 or 32 contiguous bytes of w, which plain
// loads would fetch at a 64- or 32-byte lane stride) the slice's parameters
// come by TMA as well: w viewed as rows of 32 floats (pmap), a box of
// R = 32 (32 / b) / 32 rows with 128-byte swizzle (16-byte chunk c of row r
// at chunk c ^ (r mod 8), so the lanes' 16-byte accesses never conflict),
// loaded with the code words on the same mbarrier and stored back by TMA.
// Rows past the map read as zero and are not stored; the partial last row
// (d mod 32 elements, outside the map) is read and written directly.
// Per warp two buffers of each kind: slice i + 1 loads while slice i is
// decoded.  FM > 0 fixes the worker count at compile time (s.M == FM): the
// per-worker decode then has no tests for workers past M.
template <int BITS, bool POW2, bool SEG, int NSET, int FM>
__global__ void __launch_bounds__(32 * kTmaWarps)
squant_server_tma_kernel(const ServerArgs s, const __grid_constant__ CUtensorMap tmap,
                         const __grid_constant__ CUtensorMap pmap) {
  dq_pdl_enter();
  constexpr int K = (1 << (BITS - 1)) - 1;
  constexpr int EPL = 32 / BITS;  // elements per lane (one code word)
  constexpr int SLICE = 32 * EPL; // elements per slice
  constexpr bool WB = sq_params_boxed(BITS);
  constexpr bool kSqPrefetch = sq_prefetch(BITS);
  constexpr bool kSqDirectStore = sq_direct_store(BITS);
  constexpr int R = SLICE / 32;                 // parameter rows per slice
  constexpr uint32_t PBOX = WB ? R * 128u : 0u;  // bytes of a parameter box (1024-byte multiple)
  constexpr int LPR = 32 / EPL;                 // lanes per parameter row
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t bars[kTmaWarps][2];
  __shared__ float V8[BITS == 8 ? 256 * 32 : 1];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int M = FM > 0 ? FM : s.M;
  const uint32_t box_bytes = (uint32_t)M * 128u;
  const uint32_t raw = smem_addr(smem_raw);
  // parameter boxes of every warp first (1024-byte aligned), then the word boxes
  uint8_t* const pbuf0 = smem_raw + ((1024u - (raw & 1023u)) & 1023u) + warp * 2 * PBOX;  // + i * PBOX
  uint8_t* const buf0 = smem_raw + ((1024u - (raw & 1023u)) & 1023u) + kTmaWarps * 2 * PBOX +
                        warp * 2 * box_bytes;  // + i * box_bytes
  uint64_t* bar = bars[warp];
  if constexpr (BITS == 8) {
    for (int t = threadIdx.x; t < 256 * 32; t += blockDim.x) {
      const int code = t >> 5;
      const int level = code - K;
      float v = 0.f;
      if (code <= 2 * K && level != 0) {
        const float mag = __fdiv_rn((float)(level < 0 ? -level : level), (float)K);
        v = level < 0 ? -mag : mag;
      }
      V8[t] = v;
    }
  }
  float V4 = 0.f;  // b = 4: lane l holds V[l mod 16]
  if constexpr (BITS == 4) {
    const int level = (lane & 15) - K;
    if ((lane & 15) <= 2 * K && level != 0) {
      const float mag = __fdiv_rn((float)(level < 0 ? -level : level), (float)K);
      V4 = level < 0 ? -mag : mag;
    }
  }
  if (lane == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    mbar_fence_init();
  }
  __syncthreads();

  const int spb = s.bucket / SLICE;  // slices per bucket
  const int64_t nb = (s.d + s.bucket - 1) / s.bucket;
  const int64_t nslices = SEG ? (s.d + SLICE - 1) / SLICE : nb * spb;
  const int64_t stride = (int64_t)gridDim.x * kTmaWarps;
  const int32_t x0 = (int32_t)(s.off_payload >> 2);
  const int64_t nrows = s.d >> 5;     // rows of the parameter map
  const int tail = (int)(s.d & 31);   // elements of the partial row nrows
  const bool active = lane < M;
  // slice sl covers code words [32 sl, 32 sl + 32) and parameter rows
  // [R sl, R sl + R): buckets hold whole slices
  auto issue = [&](int64_t sl_, int i) {
    const bool boxed = WB && R * sl_ < nrows;
    mbar_arrive_expect_tx(&bar[i], box_bytes + (boxed ? PBOX : 0u));
    tma_load_2d(buf0 + i * box_bytes, &tmap, x0 + (int32_t)(32 * sl_), 0, &bar[i]);
    if (boxed) tma_load_2d(pbuf0 + i * PBOX, &pmap, 0, (int32_t)(R * sl_), &bar[i]);
  };
  int64_t sl = (int64_t)blockIdx.x * kTmaWarps + warp;
  if (sl < nslices && lane == 0) issue(sl, 0);
  // with layer segments: the bucket of this lane's word, loaded one slice
  // ahead so that the scale load does not wait for it (-1 past d)
  auto word_bucket_of = [&](int64_t sl_) -> int64_t {
    const int64_t j = SLICE * sl_ + EPL * lane;
    return (sl_ < nslices && j < s.d) ? (int64_t)__ldg(s.word_bucket + (j >> 5)) : -1;
  };
  int64_t wb_next = SEG ? word_bucket_of(sl) : 0;
  // (b = 4, 8: two slices ahead, so that the scale can be loaded one ahead)
  int64_t wb_next2 = (SEG && kSqPrefetch) ? word_bucket_of(sl + stride) : 0;
  // b = 4, 8: this lane's worker's scale of the slice's bucket (the bucket
  // of lane 0's word), and (b = 8) the lane's four parameters, loaded one
  // slice ahead
  const float* const lane_scales =
      reinterpret_cast<const float*>(s.msgs + (int64_t)(active ? lane : 0) * s.msg_stride);
  auto load_w4 = [&](int64_t sl_) -> float4 {
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    const int64_t j = SLICE * sl_ + EPL * lane;
    if (sl_ >= nslices) return x;
    if (j + 3 < s.d) return __ldcs(reinterpret_cast<const float4*>(s.w + j));
    if (j < s.d) x.x = s.w[j];
    if (j + 1 < s.d) x.y = s.w[j + 1];
    if (j + 2 < s.d) x.z = s.w[j + 2];
    return x;
  };
  float scale_nx = 0.f;
  if constexpr (kSqPrefetch) {
    const int64_t b0 = SEG ? (int64_t)__shfl_sync(kFullMask, wb_next, 0) : sl / spb;
    scale_nx = (active && sl < nslices && b0 >= 0) ? __ldg(lane_scales + b0) : 0.f;
  }
  float4 w_nx = (kSqPrefetch && !WB) ? load_w4(sl) : make_float4(0.f, 0.f, 0.f, 0.f);
  uint32_t it = 0;
  bool ok = true;
  float T2[8 * NSET];  // b = 2 pair tables of bucket t2_bkt
  int64_t t2_bkt = -1;
  for (; sl < nslices; sl += stride, ++it) {
    const int cur = (int)(it & 1u);
    const int64_t nxt = sl + stride;
    if (nxt < nslices && lane == 0) {
      if constexpr (WB && !kSqDirectStore) bulk_wait_read_all();  // the previous slice's store has read its box
      fence_proxy_async_shared();  // this warp's accesses of those buffers came before
      issue(nxt, cur ^ 1);
    }
    const int64_t wb_cur = wb_next;
    if constexpr (SEG && kSqPrefetch) {
      wb_next = wb_next2;
      wb_next2 = word_bucket_of(nxt + stride);
    } else if constexpr (SEG) {
      wb_next = word_bucket_of(nxt);
    }
    const int64_t b = sl / spb;
    const int64_t j0 = SLICE * sl + EPL * lane;  // this lane's first element
    // the lane's parameters: row pr of the box, 16-byte chunks pc0 ..
    const int pr = lane / LPR;
    const int pc0 = (lane % LPR) * (EPL / 4);
    const bool boxed = WB && R * sl < nrows;
    const bool direct = WB && R * sl + pr == nrows && tail != 0;  // the partial last row
    uint8_t* const prow = pbuf0 + cur * PBOX + pr * 128;
    float wv[EPL];
    if constexpr (!WB && kSqPrefetch) {
      wv[0] = w_nx.x; wv[1] = w_nx.y; wv[2] = w_nx.z; wv[3] = w_nx.w;
      w_nx = load_w4(nxt);
    } else if constexpr (!WB) {
#pragma unroll
      for (int q = 0; q < EPL / 4; ++q) {
        const int64_t j = j0 + 4 * q;
        if (j + 3 < s.d) {
          const float4 x = __ldcs(reinterpret_cast<const float4*>(s.w + j));
          wv[4 * q] = x.x; wv[4 * q + 1] = x.y; wv[4 * q + 2] = x.z; wv[4 * q + 3] = x.w;
        } else {
#pragma unroll
          for (int r = 0; r < 4; ++r) wv[4 * q + r] = (j + r < s.d) ? s.w[j + r] : 0.f;
        }
      }
    }
    // The slice's bucket; with layer segments, each lane's word's bucket, and
    // whether they differ within the slice (warp-uniform).
    int64_t bkt = b, my_bkt = b;
    bool mixed = false;
    if constexpr (SEG) {
      my_bkt = wb_cur;
      bkt = __shfl_sync(kFullMask, my_bkt, 0);  // lane 0's elements always exist
      if (my_bkt < 0) my_bkt = bkt;
      mixed = !__all_sync(kFullMask, my_bkt == bkt);
    }
    float my_scale;
    if constexpr (kSqPrefetch) {
      my_scale = scale_nx;
      const int64_t bn = SEG ? (int64_t)__shfl_sync(kFullMask, wb_next, 0) : nxt / spb;
      scale_nx = (active && nxt < nslices && bn >= 0) ? __ldg(lane_scales + bn) : 0.f;
    } else {
      my_scale = active ? __ldg(reinterpret_cast<const float*>(s.msgs + (int64_t)lane * s.msg_stride) + bkt) : 0.f;
    }
    // A slice that spans buckets holds consecutive ones, bkt .. bkt + nbk - 1
    // (one per 32-element word at most).  Up to four: lane m loads worker m's
    // scales of all of them and each lane picks its own bucket's by shuffle;
    // more (short partial buckets): each lane loads the scales it needs.
    int rel = 0, nbk = 1;
    float sc4[4] = {my_scale, 0.f, 0.f, 0.f};
    if (SEG && mixed) {
      rel = (int)(my_bkt - bkt);
      nbk = __reduce_max_sync(kFullMask, (unsigned)rel) + 1;
      if (nbk <= 4) {
#pragma unroll
        for (int k = 1; k < 4; ++k) sc4[k] = (active && k < nbk) ? __ldg(lane_scales + bkt + k) : 0.f;
      }
    }
    // worker m's scale for this lane's elements (mx: the slice spans buckets;
    // every call passes a constant)
    auto scale_of = [&](bool mx, int m) -> float {
      if (mx) {
        if (nbk > 4) return __ldg(reinterpret_cast<const float*>(s.msgs + (int64_t)m * s.msg_stride) + my_bkt);
        float r = __shfl_sync(kFullMask, sc4[0], m);
#pragma unroll
        for (int k = 1; k < 4; ++k) {
          if (k < nbk) {  // warp-uniform
            const float t = __shfl_sync(kFullMask, sc4[k], m);
            if (rel == k) r = t;
          }
        }
        return r;
      }
      return __shfl_sync(kFullMask, my_scale, m);
    };
    ok = mbar_wait_bounded(&bar[cur], (it >> 1) & 1u, s.err);
    ok = __all_sync(kFullMask, ok);
    if (!ok) break;
    if constexpr (WB) {
#pragma unroll
      for (int q = 0; q < EPL / 4; ++q) {
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (boxed) x = *reinterpret_cast<const float4*>(prow + (((pc0 + q) ^ (pr & 7)) << 4));
        if (direct) {
          const int64_t j = j0 + 4 * q;
          x.x = j < s.d ? s.w[j] : 0.f;
          x.y = j + 1 < s.d ? s.w[j + 1] : 0.f;
          x.z = j + 2 < s.d ? s.w[j + 2] : 0.f;
          x.w = j + 3 < s.d ? s.w[j + 3] : 0.f;
        }
        wv[4 * q] = x.x; wv[4 * q + 1] = x.y; wv[4 * q + 2] = x.z; wv[4 * q + 3] = x.w;
      }
    }
    const uint32_t* words = reinterpret_cast<const uint32_t*>(buf0 + cur * box_bytes) + lane;
    const float* V8l = V8 + lane;
    // The per-worker decode (b = 4, 8, and b = 2 on slices that span layer
    // segments) takes the lane's elements in kParts passes of NE (b = 4: two
    // passes of 4, which halves the live sums at the cost of reading each
    // code word and scale twice).
    constexpr int kParts = BITS == 4 ? kSquant4Parts : 1;
    constexpr int NE = EPL / kParts;
    // one worker's decoded values of this lane's elements e0 .. e0 + NE - 1
    auto decode_part = [&](bool MX, uint32_t word, float sc, int e0, float (&v)[NE]) {
      if constexpr (BITS == 2) {
        // code 0: -s, 1: +0, 2: +s (fl(s * 1) = s): one bit test picks +0,
        // one the sign
        const float nsc = -sc;
#pragma unroll
        for (int e = 0; e < NE; ++e) {
          const bool zero = (word >> (2 * (e0 + e))) & 1u;
          v[e] = zero ? 0.f : (((word >> (2 * (e0 + e) + 1)) & 1u) ? sc : nsc);
        }
        return;
      }
      // b = 4: lane c first forms this worker's decoded value of code c mod 16,
      // fl(s * V[c mod 16]); each element then fetches its value with one
      // shuffle (the lane index is taken mod 32 and the values repeat in lanes
      // 16..31, so the bits above the element's code need no mask).  (With
      // layer segments the lanes' scales may differ: look up V[c] and multiply
      // by the lane's own scale instead.)
      const float T4 = (BITS == 4) ? __fmul_rn(MX ? 1.0f : sc, V4) : 0.f;
#pragma unroll
      for (int e = 0; e < NE; ++e) {
        if constexpr (BITS == 4) {
          v[e] = __shfl_sync(kFullMask, T4, (int)(word >> (4 * (e0 + e))));
          if (MX) v[e] = __fmul_rn(sc, v[e]);
        } else {
          v[e] = __fmul_rn(sc, V8l[__byte_perm(word, 0u, 0x4440u | (uint32_t)(e0 + e)) * 32u]);
        }
      }
    };
    float acc[EPL] = {};
    if constexpr (BITS == 2) {
      if (!(SEG && mixed)) {
        if (bkt != t2_bkt) {
          build_pair_tables<8 * NSET>(my_scale, lane, M, T2);
          t2_bkt = bkt;
        }
        b2_pair_table_update<NSET, POW2, FM>(words, s, T2, wv);
      }
    }
    // groups of four workers, G = (a + b) + (c + d) with +0 past M, combined
    // as the padded tree over the next_pow2(ceil(M / 4)) <= 8 groups: G0;
    // G0 + G1; (G0 + G1) + (G2 + G3); then + ((G4 + G5) + (G6 + G7)), groups
    // past M being +0 (M is warp-uniform, so are the branches)
    const bool per_worker = BITS != 2 || (SEG && mixed);
    // (slices that span buckets take their own instance of the decode, so
    // that the common one carries none of their scale handling)
    auto per_worker_sums = [&](bool mx) {
#pragma unroll
      for (int part = 0; part < kParts; ++part) {
        const int e0 = part * NE;
        // group value of workers m .. m + 3 into g
        auto group = [&](int m, float (&g)[NE]) {
          // the group's code words and scales first (a worker past M is not read)
          uint32_t wd[4];
          float sc[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const bool here = m + u < M;  // warp-uniform
            wd[u] = here ? words[32 * (m + u)] : 0u;
            sc[u] = here ? scale_of(mx, m + u) : 0.f;
          }
          float va[NE], vb[NE];
          decode_part(mx, wd[0], sc[0], e0, va);
          decode_part(mx, wd[1], sc[1], e0, vb);
          const bool h1 = m + 1 < M;
#pragma unroll
          for (int e = 0; e < NE; ++e) g[e] = M == 1 ? va[e] : __fadd_rn(va[e], h1 ? vb[e] : 0.f);
          if (M <= 2) return;
          decode_part(mx, wd[2], sc[2], e0, va);
          decode_part(mx, wd[3], sc[3], e0, vb);
          const bool h2 = m + 2 < M, h3 = m + 3 < M;
#pragma unroll
          for (int e = 0; e < NE; ++e) g[e] = __fadd_rn(g[e], __fadd_rn(h2 ? va[e] : 0.f, h3 ? vb[e] : 0.f));
        };
        // x <- x + (value of groups i, i + 1), the second +0 past M
        auto add_pair = [&](int i, float (&x)[NE]) {
          float t[NE], g[NE];
          group(4 * i, t);
          if (4 * (i + 1) < M) {
            group(4 * (i + 1), g);
          } else {
#pragma unroll
            for (int e = 0; e < NE; ++e) g[e] = 0.f;
          }
#pragma unroll
          for (int e = 0; e < NE; ++e) x[e] = __fadd_rn(x[e], __fadd_rn(t[e], g[e]));
        };
        float r[NE];
        group(0, r);
        if (M > 4) {
          float g[NE];
          group(4, g);
#pragma unroll
          for (int e = 0; e < NE; ++e) r[e] = __fadd_rn(r[e], g[e]);
          if (M > 8) {
            add_pair(2, r);
            if (M > 16) {
              float h[NE];
              group(16, h);
              if (M > 20) {
                group(20, g);
              } else {
#pragma unroll
                for (int e = 0; e < NE; ++e) g[e] = 0.f;
              }
#pragma unroll
              for (int e = 0; e < NE; ++e) h[e] = __fadd_rn(h[e], g[e]);
              if (M > 24) {
                add_pair(6, h);
              } else {
#pragma unroll
                for (int e = 0; e < NE; ++e) h[e] = __fadd_rn(h[e], 0.f);
              }
#pragma unroll
              for (int e = 0; e < NE; ++e) r[e] = __fadd_rn(r[e], h[e]);
            }
          }
        }
#pragma unroll
        for (int e = 0; e < NE; ++e) acc[e0 + e] = r[e];
      }
    };
    if (per_worker) {
      if constexpr (SEG) {
        if (mixed) per_worker_sums(true);
        else per_worker_sums(false);
      } else {
        per_worker_sums(false);
      }
    }
#pragma unroll
    for (int q = 0; q < EPL / 4; ++q) {
      const int64_t j = j0 + 4 * q;
      float o[4];
#pragma unroll
      for (int r = 0; r < 4; ++r)
        o[r] = per_worker ? server_out(s, wv[4 * q + r], average_t<POW2>(acc[4 * q + r], s)) : wv[4 * q + r];
      if constexpr (WB && kSqDirectStore) {
        if (R * sl + pr < nrows) __stcs(reinterpret_cast<float4*>(s.w + j), make_float4(o[0], o[1], o[2], o[3]));
        if (direct) {
#pragma unroll
          for (int r = 0; r < 4; ++r)
            if (j + r < s.d) s.w[j + r] = o[r];
        }
      } else if constexpr (WB) {
        if (boxed)
          *reinterpret_cast<float4*>(prow + (((pc0 + q) ^ (pr & 7)) << 4)) = make_float4(o[0], o[1], o[2], o[3]);
        if (direct) {
#pragma unroll
          for (int r = 0; r < 4; ++r)
            if (j + r < s.d) s.w[j + r] = o[r];
        }
      } else if (j + 3 < s.d) {
        __stcs(reinterpret_cast<float4*>(s.w + j), make_float4(o[0], o[1], o[2], o[3]));
      } else {
#pragma unroll
        for (int r = 0; r < 4; ++r)
          if (j + r < s.d) s.w[j + r] = o[r];
      }
    }
    if constexpr (WB && !kSqDirectStore) fence_proxy_async_shared();  // the box writes above, before the store reads them
    __syncwarp();
    if (WB && !kSqDirectStore && lane == 0 && boxed) tma_store_2d(&pmap, 0, (int32_t)(R * sl), pbuf0 + cur * PBOX);
    __syncwarp();
  }
  if (lane == 0) {
    if constexpr (WB && !kSqDirectStore) bulk_wait_all();  // stores complete before the block's shared memory is released
    // after a time-out, the copy of the next slice may still be in flight
    if (!ok && sl + stride < nslices) mbar_wait_bounded(&bar[(it & 1u) ^ 1u], ((it + 1) >> 1) & 1u, s.err);
  }
}

// 8-bit codes with layer segments and 16 workers: the slices come from a
// host-built table of each bucket's code words in runs of up to 32, so no
// slice spans two buckets (the per-lane bucket lookups and the mixed-slice
// decode of the kernel above are not needed).  The word box starts at the
// 16-byte boundary at or before the slice (36 words wide, no swizzle); lane l
// takes word first + l of every worker when l < rows.  The decode and the
// sum over workers are the b = 8 ones above: level table replicated per
// shared-memory bank, groups of four workers (a + b) + (c + d), the four
// group values added pairwise.  The slice's scale, the next slice's table
// entry and the lane's four parameters are loaded one slice ahead.
template <bool POW2>
__global__ void __launch_bounds__(32 * kTmaWarps)
squant8_server_table_kernel(const ServerArgs s, const SegSlices seg, const __grid_constant__ CUtensorMap tmap) {
  dq_pdl_enter();
  constexpr int K = 127;
  constexpr int M = 16;
  constexpr int RW = kSignSegBoxWords;                       // words per box row
  constexpr uint32_t kBoxBytes = (uint32_t)M * RW * 4u;      // 2304: a multiple of 128
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t bars[kTmaWarps][2];
  __shared__ float V8[256 * 32];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* const buf0 = smem_raw + ((128u - (raw & 127u)) & 127u) + warp * 2 * kBoxBytes;  // + i * kBoxBytes
  uint64_t* bar = bars[warp];
  for (int t = threadIdx.x; t < 256 * 32; t += blockDim.x) {
    const int code = t >> 5;
    const int level = code - K;
    float v = 0.f;
    if (code <= 2 * K && level != 0) {
      const float mag = __fdiv_rn((float)(level < 0 ? -level : level), (float)K);
      v = level < 0 ? -mag : mag;
    }
    V8[t] = v;
  }
  if (lane == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    mbar_fence_init();
  }
  __syncthreads();

  const int64_t nslices = seg.n;
  const int64_t stride = (int64_t)gridDim.x * kTmaWarps;
  const int32_t x0 = (int32_t)(s.off_payload >> 2);  // a multiple of 64 words
  const bool active = lane < M;
  struct Slice {
    int64_t word;    // first code word
    int64_t bucket;
    int rows;        // code words in the slice, 1..32 (0: none)
  };
  auto slice_of = [&](int64_t sl_) -> Slice {
    if (sl_ >= nslices) return Slice{0, 0, 0};
    const uint2 e = __ldg(reinterpret_cast<const uint2*>(seg.slices) + sl_);
    return Slice{(int64_t)e.x, (int64_t)(e.y & 0x7FFFFFFu), (int)(e.y >> 27) + 1};
  };
  auto issue = [&](const Slice& c, int i) {
    mbar_arrive_expect_tx(&bar[i], kBoxBytes);
    tma_load_2d(buf0 + i * kBoxBytes, &tmap, (x0 + (int32_t)c.word) & ~3, 0, &bar[i]);
  };
  const float* const lane_scales =
      reinterpret_cast<const float*>(s.msgs + (int64_t)(active ? lane : 0) * s.msg_stride);
  // the lane's four parameters of slice c (none past its rows or past d)
  auto load_w4 = [&](const Slice& c) -> float4 {
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (lane >= c.rows) return x;
    const int64_t j = 4 * (c.word + lane);
    if (j + 3 < s.d) return __ldcs(reinterpret_cast<const float4*>(s.w + j));
    if (j < s.d) x.x = s.w[j];
    if (j + 1 < s.d) x.y = s.w[j + 1];
    if (j + 2 < s.d) x.z = s.w[j + 2];
    return x;
  };
  int64_t sl = (int64_t)blockIdx.x * kTmaWarps + warp;
  Slice c = slice_of(sl);
  Slice cn = slice_of(sl + stride);
  if (sl < nslices && lane == 0) issue(c, 0);
  float scale_nx = (active && sl < nslices) ? __ldg(lane_scales + c.bucket) : 0.f;
  float4 w_nx = load_w4(c);
  uint32_t it = 0;
  bool ok = true;
  for (; sl < nslices; sl += stride, ++it) {
    const int cur = (int)(it & 1u);
    const int64_t nxt = sl + stride;
    const Slice cnn = slice_of(nxt + stride);  // the table entry one slice further
    if (nxt < nslices && lane == 0) {
      fence_proxy_async_shared();  // this warp's reads of that buffer came before
      issue(cn, cur ^ 1);
    }
    const float my_scale = scale_nx;
    scale_nx = (active && nxt < nslices) ? __ldg(lane_scales + cn.bucket) : 0.f;
    const float wv[4] = {w_nx.x, w_nx.y, w_nx.z, w_nx.w};
    w_nx = load_w4(cn);
    ok = mbar_wait_bounded(&bar[cur], (it >> 1) & 1u, s.err);
    ok = __all_sync(kFullMask, ok);
    if (!ok) break;
    const uint32_t* words = reinterpret_cast<const uint32_t*>(buf0 + cur * kBoxBytes) + (int)((x0 + c.word) & 3) + lane;
    const float* V8l = V8 + lane;
    // group value of workers m .. m + 3: (a + b) + (c + d)
    auto group = [&](int m, float (&g)[4]) {
      uint32_t wd[4];
      float sc[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        wd[u] = words[RW * (m + u)];
        sc[u] = __shfl_sync(kFullMask, my_scale, m + u);
      }
      float v[4][4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          v[u][e] = __fmul_rn(sc[u], V8l[__byte_perm(wd[u], 0u, 0x4440u | (uint32_t)e) * 32u]);
#pragma unroll
      for (int e = 0; e < 4; ++e) g[e] = __fadd_rn(__fadd_rn(v[0][e], v[1][e]), __fadd_rn(v[2][e], v[3][e]));
    };
    float g0[4], g1[4], r[4];
    group(0, g0);
    group(4, g1);
#pragma unroll
    for (int e = 0; e < 4; ++e) r[e] = __fadd_rn(g0[e], g1[e]);
    group(8, g0);
    group(12, g1);
#pragma unroll
    for (int e = 0; e < 4; ++e) r[e] = __fadd_rn(r[e], __fadd_rn(g0[e], g1[e]));
    if (lane < c.rows) {
      const int64_t j = 4 * (c.word + lane);
      float o[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) o[e] = server_out(s, wv[e], average_t<POW2>(r[e], s));
      if (j + 3 < s.d) {
        __stcs(reinterpret_cast<float4*>(s.w + j), make_float4(o[0], o[1], o[2], o[3]));
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (j + e < s.d) s.w[j + e] = o[e];
      }
    }
    __syncwarp();
    c = cn;
    cn = cnn;
  }
  // after a time-out, the copy of the next slice may still be in flight
  if (!ok && lane == 0 && sl + stride < nslices)
    mbar_wait_bounded(&bar[(it & 1u) ^ 1u], ((it + 1) >> 1) & 1u, s.err);
}

// Identity: the messages are the p vectors themselves, summed in groups of
// four workers in the library's pairwise order.
__global__ void __launch_bounds__(256) identity_server_kernel(const ServerArgs s) {
  dq_pdl_enter();
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t j = 4 * c;
  if (j >= s.d) return;
  PairwiseAcc<kSumLevels> sum[4];
  const bool vec = j + 3 < s.d;
  for (int m0 = 0; m0 < s.M; m0 += 4) {
    float4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);  // +0 leaves past M and past d
      if (m0 + u < s.M) {
        const float* vals = reinterpret_cast<const float*>(s.msgs + (int64_t)(m0 + u) * s.msg_stride);
        if (vec) {
          v[u] = __ldcs(reinterpret_cast<const float4*>(vals + j));
        } else {
          v[u].x = vals[j];
          if (j + 1 < s.d) v[u].y = vals[j + 1];
          if (j + 2 < s.d) v[u].z = vals[j + 2];
        }
      }
    }
    sum[0].push(group4(v[0].x, v[1].x, v[2].x, v[3].x, s.M));
    sum[1].push(group4(v[0].y, v[1].y, v[2].y, v[3].y, s.M));
    sum[2].push(group4(v[0].z, v[1].z, v[2].z, v[3].z, s.M));
    sum[3].push(group4(v[0].w, v[1].w, v[2].w, v[3].w, s.M));
  }
  float acc[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) acc[q] = sum[q].result();
  apply_chunk(s, j, acc);
}

__global__ void __launch_bounds__(256)
lookahead_kernel(const float* __restrict__ w, const float* __restrict__ h, float* __restrict__ out,
                 int64_t d) {
  dq_pdl_enter();
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t j = 4 * c;
  if (j + 3 < d) {
    const float4 wv = __ldg(reinterpret_cast<const float4*>(w + j));
    const float4 hv = __ldcs(reinterpret_cast<const float4*>(h + j));
    __stcs(reinterpret_cast<float4*>(out + j),
           make_float4(__fsub_rn(wv.x, hv.x), __fsub_rn(wv.y, hv.y), __fsub_rn(wv.z, hv.z),
                       __fsub_rn(wv.w, hv.w)));
  } else {
    for (int64_t jj = j; jj < d; ++jj) out[jj] = __fsub_rn(w[jj], h[jj]);
  }
}

// Optimistic Adam over all parameters from q_hat (written by the server
// kernel), every operation rounded once in this order:
//   m = b1 m + (1 - b1) q;  v = b2 v + ((1 - b2) q) q;
//   m_hat = m / c1, v_hat = v / c2 (with bias correction);
//   u = m_hat / (sqrt(v_hat) + eps), 0 where m_hat = 0 (adaptive), else m_hat;
//   w = w - alpha (2 u - u_prev);  u_prev = u.
// One thread per 4 parameters, 16-byte streaming loads and stores.
__device__ __forceinline__ float oadam_element(const OAdamArgs& a, float q, float& m, float& v, float& u, float w) {
  m = __fadd_rn(__fmul_rn(a.beta1, m), __fmul_rn(a.one_m_beta1, q));
  v = __fadd_rn(__fmul_rn(a.beta2, v), __fmul_rn(__fmul_rn(a.one_m_beta2, q), q));
  const float mh = a.bias_correction ? __fdiv_rn(m, a.c1) : m;
  const float vh = a.bias_correction ? __fdiv_rn(v, a.c2) : v;
  float un = mh;
  if (a.adaptive) un = (mh == 0.f) ? 0.f : __fdiv_rn(mh, __fadd_rn(__fsqrt_rn(vh), a.eps));
  const float step = __fsub_rn(__fmul_rn(2.f, un), u);
  u = un;
  return __fsub_rn(w, __fmul_rn(a.alpha, step));
}

__global__ void __launch_bounds__(256) oadam_update_kernel(const OAdamArgs a) {
  dq_pdl_enter();
  const int64_t j = 4 * ((int64_t)blockIdx.x * blockDim.x + threadIdx.x);
  if (j + 3 < a.d) {
    const float4 q = __ldcs(reinterpret_cast<const float4*>(a.q + j));
    float4 m = __ldcs(reinterpret_cast<const float4*>(a.m + j));
    float4 v = __ldcs(reinterpret_cast<const float4*>(a.v + j));
    float4 u = __ldcs(reinterpret_cast<const float4*>(a.u + j));
    float4 w = __ldcs(reinterpret_cast<const float4*>(a.w + j));
    w.x = oadam_element(a, q.x, m.x, v.x, u.x, w.x);
    w.y = oadam_element(a, q.y, m.y, v.y, u.y, w.y);
    w.z = oadam_element(a, q.z, m.z, v.z, u.z, w.z);
    w.w = oadam_element(a, q.w, m.w, v.w, u.w, w.w);
    __stcs(reinterpret_cast<float4*>(a.m + j), m);
    __stcs(reinterpret_cast<float4*>(a.v + j), v);
    __stcs(reinterpret_cast<float4*>(a.u + j), u);
    __stcs(reinterpret_cast<float4*>(a.w + j), w);
  } else {
    for (int64_t jj = j; jj < a.d; ++jj) a.w[jj] = oadam_element(a, a.q[jj], a.m[jj], a.v[jj], a.u[jj], a.w[jj]);
  }
}

template <int NG, bool POW2, bool SEG>
cudaError_t launch_sign_tma(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream) {
  auto kern = sign_server_tma_kernel<NG, POW2, SEG>;
  constexpr int smem = tma_sign_smem_bytes<SEG>();
  int dev = 0;
  cudaError_t st = cudaGetDevice(&dev);
  if (st != cudaSuccess) return st;
  static int blocks_for[64] = {0};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (blocks_for[dev] == 0) {
    if ((st = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
      return st;
    int sms = 0, per_sm = 0;
    if ((st = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return st;
    if ((st = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 32 * kTmaWarps, smem)) != cudaSuccess)
      return st;
    blocks_for[dev] = sms * (per_sm > 0 ? per_sm : 1);
  }
  const int64_t warps = SEG ? x.seg_nslices : ((s.d + s.bucket - 1) / s.bucket) * (s.bucket / 1024);
  const int64_t need = (warps + kTmaWarps - 1) / kTmaWarps;
  const unsigned blocks = (unsigned)(need < blocks_for[dev] ? need : blocks_for[dev]);
  if (blocks == 0) return cudaSuccess;
  launch_pdl(kern, dim3(blocks), dim3(32 * kTmaWarps), smem, stream, s, SegSlices{x.seg_slices, x.seg_nslices},
             *s.sign_words_map);
  return cudaGetLastError();
}

template <int NG, bool POW2, bool SEG>
cudaError_t launch_sign_col(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream) {
  auto kern = sign_server_col_kernel<NG, POW2, SEG>;
  constexpr int smem = ColLayout<SEG>::kSmem;
  int dev = 0;
  cudaError_t st = cudaGetDevice(&dev);
  if (st != cudaSuccess) return st;
  static int blocks_for[64] = {0};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (blocks_for[dev] == 0) {
    if ((st = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
      return st;
    int sms = 0, per_sm = 0;
    if ((st = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return st;
    if ((st = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 32 * kColWarps, smem)) != cudaSuccess)
      return st;
    blocks_for[dev] = sms * (per_sm > 0 ? per_sm : 1);
  }
  const int64_t nslices = SEG ? x.seg_nslices : ((s.d + s.bucket - 1) / s.bucket) * (s.bucket / 1024);
  const int64_t need = (nslices + kColWarps - 1) / kColWarps;
  const unsigned blocks = (unsigned)(need < blocks_for[dev] ? need : blocks_for[dev]);
  if (blocks == 0) return cudaSuccess;
  launch_pdl(kern, dim3(blocks), dim3(32 * kColWarps), smem, stream, s, SegSlices{x.seg_slices, x.seg_nslices}, *s.sign_words_map,
                                                  *x.params_map);
  return cudaGetLastError();
}

// The column kernel pays once every resident warp has several slices: with
// one or two the latency of a slice's chain (copies in, transpose, store)
// shows and the bit-transpose kernel is as fast or faster.
bool sign_col_pays(int64_t nslices) {
  static int sms[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (sms[dev] == 0 && cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return false;
  return nslices >= 4ll * sms[dev] * kColWarps;
}

template <int BITS, bool POW2, bool SEG, int NSET, int FM = 0>
cudaError_t launch_squant_tma(const ServerArgs& s, const CUtensorMap* params_map, cudaStream_t stream) {
  auto kern = squant_server_tma_kernel<BITS, POW2, SEG, NSET, FM>;
  constexpr int pbox = sq_params_boxed(BITS) ? 32 * (32 / BITS) * 4 : 0;  // bytes of a parameter box
  const int smem = kTmaWarps * 2 * (pbox + s.M * 128) + 1024;  // + alignment slack
  int dev = 0;
  cudaError_t st = cudaGetDevice(&dev);
  if (st != cudaSuccess) return st;
  if ((st = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess) return st;
  int sms = 0, per_sm = 0;
  if ((st = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return st;
  if ((st = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 32 * kTmaWarps, smem)) != cudaSuccess)
    return st;
  const int64_t nslices = SEG ? (s.d + 32 * (32 / BITS) - 1) / (32 * (32 / BITS))
                              : ((s.d + s.bucket - 1) / s.bucket) * (s.bucket / (32 * (32 / BITS)));
  const int64_t need = (nslices + kTmaWarps - 1) / kTmaWarps;
  const int64_t cap = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
  // (b = 8 takes no parameter map: the word map stands in for the unused argument)
  launch_pdl(kern, dim3((unsigned)(need < cap ? need : cap)), dim3(32 * kTmaWarps), smem, stream,
      s, *s.squant_words_map, sq_params_boxed(BITS) ? *params_map : *s.squant_words_map);
  return cudaGetLastError();
}

cudaError_t launch_squant8_table(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream) {
  auto kern = squant8_server_table_kernel<true>;
  constexpr int smem = kTmaWarps * 2 * 16 * kSignSegBoxWords * 4 + 128;  // + alignment slack
  int dev = 0;
  cudaError_t st = cudaGetDevice(&dev);
  if (st != cudaSuccess) return st;
  static int blocks_for[64] = {0};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (blocks_for[dev] == 0) {
    if ((st = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
      return st;
    int sms = 0, per_sm = 0;
    if ((st = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return st;
    if ((st = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 32 * kTmaWarps, smem)) != cudaSuccess)
      return st;
    blocks_for[dev] = sms * (per_sm > 0 ? per_sm : 1);
  }
  const int64_t need = (x.seg_nslices + kTmaWarps - 1) / kTmaWarps;
  const unsigned blocks = (unsigned)(need < blocks_for[dev] ? need : blocks_for[dev]);
  if (blocks == 0) return cudaSuccess;
  launch_pdl(kern, dim3(blocks), dim3(32 * kTmaWarps), smem, stream, s, SegSlices{x.seg_slices, x.seg_nslices},
             *s.squant_words_map);
  return cudaGetLastError();
}

unsigned chunk_blocks(int64_t d, int threads) {
  const int64_t chunks = (d + 3) / 4;
  return (unsigned)((chunks + threads - 1) / threads);
}

}  // namespace

cudaError_t launch_sign_server(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream,
                               uint64_t* launches) {
  if (s.word_bucket) {  // buckets restart at layer segments
    if (x.seg_slices && s.sign_words_map && s.bucket >= 1024 && s.M <= 32) {
      const bool p2 = s.M_pow2 != 0;
      // the column kernel where it pays (as for flat buckets), else the
      // warp-transpose kernel; DQGAN_SIGN_SERVER fixes the choice
      const bool col = x.params_map != nullptr && (x.path == 1 || (x.path == 0 && sign_col_pays(x.seg_nslices)));
      cudaError_t st;
#define DQ_SIGN_SEG(NG)                                                                                     \
  st = col ? (p2 ? launch_sign_col<NG, true, true>(s, x, stream) : launch_sign_col<NG, false, true>(s, x, stream)) \
           : (p2 ? launch_sign_tma<NG, true, true>(s, x, stream) : launch_sign_tma<NG, false, true>(s, x, stream))
      switch ((s.M + 3) / 4) {
        case 1: DQ_SIGN_SEG(1); break;
        case 2: DQ_SIGN_SEG(2); break;
        case 3: DQ_SIGN_SEG(3); break;
        case 4: DQ_SIGN_SEG(4); break;
        case 5: DQ_SIGN_SEG(5); break;
        case 6: DQ_SIGN_SEG(6); break;
        case 7: DQ_SIGN_SEG(7); break;
        default: DQ_SIGN_SEG(8); break;
      }
#undef DQ_SIGN_SEG
      *launches += 1;
      return st;
    }
    launch_pdl(sign_server_kernel, dim3(chunk_blocks(s.d, 256)), dim3(256), 0, stream, s);  // per-element scale lookup
    *launches += 1;
    return cudaGetLastError();
  }
  if (s.bucket >= 1024 && s.M <= 32 && s.sign_words_map != nullptr) {
    const bool p2 = s.M_pow2 != 0;
    const bool col = x.params_map != nullptr &&
                     (x.path == 1 || (x.path == 0 && sign_col_pays(((s.d + s.bucket - 1) / s.bucket) * (s.bucket / 1024))));
    cudaError_t st;
#define DQ_SIGN_TMA(NG)                                                                           \
  st = col ? (p2 ? launch_sign_col<NG, true, false>(s, x, stream) : launch_sign_col<NG, false, false>(s, x, stream)) \
           : (p2 ? launch_sign_tma<NG, true, false>(s, x, stream) : launch_sign_tma<NG, false, false>(s, x, stream))
    switch ((s.M + 3) / 4) {
      case 1: DQ_SIGN_TMA(1); break;
      case 2: DQ_SIGN_TMA(2); break;
      case 3: DQ_SIGN_TMA(3); break;
      case 4: DQ_SIGN_TMA(4); break;
      case 5: DQ_SIGN_TMA(5); break;
      case 6: DQ_SIGN_TMA(6); break;
      case 7: DQ_SIGN_TMA(7); break;
      default: DQ_SIGN_TMA(8); break;
    }
#undef DQ_SIGN_TMA
    *launches += 1;
    return st;
  }
  if (s.bucket >= 512) {
    const int64_t nb = (s.d + s.bucket - 1) / s.bucket;
    const int64_t wpb = s.bucket >= 1024 ? s.bucket / 1024 : 1;  // warps per bucket
    const int64_t warps = nb * wpb;
    const unsigned blocks = (unsigned)((warps + 7) / 8);
    if (s.M > 32) {
      launch_pdl(sign_server_slabs_kernel, dim3(blocks), dim3(256), 0, stream, s);
    } else {
      const int ng = (s.M + 3) / 4;
      const bool p2 = s.M_pow2 != 0;
#define DQ_SIGN_SERVER(NG) \
      (p2 ? launch_pdl(sign_server_shfl_kernel<NG, true>, dim3(blocks), dim3(256), 0, stream, s) \
          : launch_pdl(sign_server_shfl_kernel<NG, false>, dim3(blocks), dim3(256), 0, stream, s))
      switch (ng) {
        case 1: DQ_SIGN_SERVER(1); break;
        case 2: DQ_SIGN_SERVER(2); break;
        case 3: DQ_SIGN_SERVER(3); break;
        case 4: DQ_SIGN_SERVER(4); break;
        case 5: DQ_SIGN_SERVER(5); break;
        case 6: DQ_SIGN_SERVER(6); break;
        case 7: DQ_SIGN_SERVER(7); break;
        default: DQ_SIGN_SERVER(8); break;
      }
#undef DQ_SIGN_SERVER
    }
  } else {
    launch_pdl(sign_server_kernel, dim3(chunk_blocks(s.d, 256)), dim3(256), 0, stream, s);
  }
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_squant_server(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream,
                                 uint64_t* launches) {
  const CUtensorMap* params_map = x.params_map;
  if (s.word_bucket && x.seg_slices && s.squant_words_map != nullptr && s.bits == 8 && s.M == 16) {
    // 8-bit codes, layer segments, 16 workers: slices from the per-bucket table
    const cudaError_t st = launch_squant8_table(s, x, stream);
    *launches += 1;
    return st;
  }
  if (s.squant_words_map != nullptr && s.M <= 32 && s.bucket >= 32 * (32 / s.bits) &&
      (params_map != nullptr || !sq_params_boxed(s.bits))) {
    const bool p2 = s.M_pow2 != 0;
    cudaError_t st = cudaErrorInvalidValue;
#define DQ_SQ_TMA(B, NSET)                                                                              \
  st = s.word_bucket ? (p2 ? launch_squant_tma<B, true, true, NSET>(s, params_map, stream)              \
                           : launch_squant_tma<B, false, true, NSET>(s, params_map, stream))            \
                     : (p2 ? launch_squant_tma<B, true, false, NSET>(s, params_map, stream)             \
                           : launch_squant_tma<B, false, false, NSET>(s, params_map, stream))
    switch (s.bits) {
      case 2:
        if (s.M == 16 && !s.word_bucket) st = launch_squant_tma<2, true, false, 1, 16>(s, params_map, stream);
        else if (s.M <= 16) DQ_SQ_TMA(2, 1);
        else DQ_SQ_TMA(2, 2);
        break;
      case 4:
        if (s.M == 16 && !s.word_bucket) st = launch_squant_tma<4, true, false, 1, 16>(s, params_map, stream);
        else DQ_SQ_TMA(4, 1);
        break;
      case 8:
        if (s.M == 16)
          st = s.word_bucket ? launch_squant_tma<8, true, true, 1, 16>(s, params_map, stream)
                             : launch_squant_tma<8, true, false, 1, 16>(s, params_map, stream);
        else DQ_SQ_TMA(8, 1);
        break;
    }
#undef DQ_SQ_TMA
    *launches += 1;
    return st;
  }
  const unsigned chunk_grid = chunk_blocks(s.d, 256);
  const unsigned blocks = chunk_grid < 152u * 6u ? chunk_grid : 152u * 6u;  // V is built once per block
  const bool p2 = s.M_pow2 != 0;
  switch (s.bits) {
    case 2: p2 ? launch_pdl(squant_server_kernel<2, true>, dim3(blocks), dim3(256), 0, stream, s)
               : launch_pdl(squant_server_kernel<2, false>, dim3(blocks), dim3(256), 0, stream, s); break;
    case 4: p2 ? launch_pdl(squant_server_kernel<4, true>, dim3(blocks), dim3(256), 0, stream, s)
               : launch_pdl(squant_server_kernel<4, false>, dim3(blocks), dim3(256), 0, stream, s); break;
    case 8: p2 ? launch_pdl(squant_server_kernel<8, true>, dim3(blocks), dim3(256), 0, stream, s)
               : launch_pdl(squant_server_kernel<8, false>, dim3(blocks), dim3(256), 0, stream, s); break;
    default: return cudaErrorInvalidValue;
  }
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_identity_server(const ServerArgs& s, cudaStream_t stream, uint64_t* launches) {
  launch_pdl(identity_server_kernel, dim3(chunk_blocks(s.d, 256)), dim3(256), 0, stream, s);
  *launches += 1;
  return cudaGetLastError();
}


cudaError_t launch_oadam_update(const OAdamArgs& a, cudaStream_t stream, uint64_t* launches) {
  launch_pdl(oadam_update_kernel, dim3(chunk_blocks(a.d, 256)), dim3(256), 0, stream, a);
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_lookahead(const float* w, const float* h, float* out, int64_t d,
                             cudaStream_t stream, uint64_t* launches) {
  launch_pdl(lookahead_kernel, dim3(chunk_blocks(d, 256)), dim3(256), 0, stream, w, h, out, d);
  *launches += 1;
  return cudaGetLastError();
}

}  // namespace dq

namespace dq {

namespace {

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link
// against libcuda); nullptr if it is unavailable.
EncodeFn tensor_map_encoder() {
  static EncodeFn encode = nullptr;
  static bool looked_up = false;
  if (!looked_up) {
    looked_up = true;
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      encode = reinterpret_cast<EncodeFn>(fn);
  }
  return encode;
}

}  // namespace

bool encode_words_map(const uint8_t* msgs, int64_t msg_stride, int64_t off_payload, int64_t payload_words,
                      int32_t M, bool swizzle128, int32_t box_words, CUtensorMap* out) {
  const EncodeFn encode = tensor_map_encoder();
  if (!encode || M < 1 || (swizzle128 && box_words != 32)) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)(off_payload / 4 + payload_words), (cuuint64_t)M};
  const cuuint64_t strides[1] = {(cuuint64_t)msg_stride};
  const cuuint32_t box[2] = {(cuuint32_t)box_words, (cuuint32_t)(M < 32 ? M : 32)};
  const cuuint32_t elem[2] = {1u, 1u};
  return encode(out, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint8_t*>(msgs), dims, strides, box, elem,
                CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_params_map(float* w, int64_t d, int32_t box_rows, CUtensorMap* out) {
  const EncodeFn encode = tensor_map_encoder();
  if (!encode || d < 32 || ((uintptr_t)w & 15u) != 0 || box_rows < 1 || box_rows > 256) return false;
  const cuuint64_t dims[2] = {32u, (cuuint64_t)(d / 32)};
  const cuuint64_t strides[1] = {128u};
  const cuuint32_t box[2] = {32u, (cuuint32_t)box_rows};
  const cuuint32_t elem[2] = {1u, 1u};
  return encode(out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, w, dims, strides, box, elem, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace dq
