// Top-k compressor of Algorithm 2 (Section 2.4, Theorem 1), worker and server.
//
// Worker: keep the k entries of p = fl(fl(eta*g) + e) with the largest |p_j|
// (ties to the lower index), send them as (u32 index, f32 value) records in
// ascending index order, and keep e_j = p_j - p_j (+0) at the kept entries
// and e_j = p_j elsewhere.  |p_j| is ordered by its bit pattern with the sign
// cleared (a 31-bit key), so the k-th largest key T is found by a three-digit
// radix select (11 + 10 + 10 bits) without sorting.
//
// Two kernels per call, one pass over the dense vectors:
//   1. form (tiles of 4096 elements): p -> e in place, h (optional), and the
//      tile's candidates -- the elements whose key is at least a threshold
//      tau carried over from the worker's previous call (15/16 of its T) --
//      written in index order to the tile's slot, with the tile's count.
//   2. select-and-compact, one cluster of 8 CTAs per worker.  The candidates
//      are split evenly over the 8 CTAs (by their index order, through a
//      prefix of the tile counts); each CTA histograms the top, then the
//      middle, then the low digit of its share, the cluster sums each
//      histogram through distributed shared memory, and every CTA selects
//      the same T and the number `need` of keys equal to T that are kept
//      (the lowest indices).  If T >= tau, every key >= T was a candidate
//      and T is exact; otherwise (first call, or T fell below the carried
//      threshold) each CTA histograms the top digit over its tiles of p,
//      re-extracts the elements whose top digit reaches the selected one,
//      and the selection is repeated.  Kept records are then written at
//      position (number of keys > T before it) + min(number of keys == T
//      before it, need), the per-CTA counts taken from the CTA's own
//      histograms.
// The carried threshold only decides how much work the first pass saves the
// second; the result is the same bit for bit either way.
//
// Server: w_j -= (sum over workers of the value recorded for j, absent
// workers as +0, in the library's pairwise order) / M at the indices some
// worker sent; elsewhere the sum is +0 and w is unchanged.  Up to 64
// workers, one thread per record in two launches: the records scatter their
// values into per-worker rows and set their worker's bit in a per-index
// mask, then the lowest worker of each index sums the index's values and
// updates w_j.  Above 64 workers, a first kernel finds where each worker's
// records of each 256-index tile start, and one thread per record searches
// the other workers' records of its tile.
#include <atomic>

#include <cooperative_groups.h>

#include "device_common.cuh"
#include "internal.cuh"

namespace dq {
namespace {

namespace cg = cooperative_groups;

constexpr int kTile = 4096;                                   // elements per tile
constexpr int kFormThreads = 256;                             // threads of a form block
constexpr int kFormRows = kTile / (4 * kFormThreads);         // float4 rows per form thread
constexpr int kCluster = 8;                                   // CTAs per worker in the select kernel
constexpr int kSelThreads = 512;                              // threads of a select CTA
constexpr int kSelRows = kTile / (4 * kSelThreads);           // float4 rows per select thread
constexpr int kBins0 = 2048, kBins1 = 1024;                   // 11-bit, then 10-bit digits
constexpr int kStateWords = 32;
constexpr int kChunkTiles = 2048;                             // tile prefixes a select CTA holds at once
constexpr int kCacheCap = 20480;                              // candidates a select CTA keeps on chip
constexpr int kBatch = 8;                                     // candidate loads in flight per thread
constexpr int kSrvTile = 256;                                 // indices per server tile
constexpr int kSrvThreads = 256;
constexpr uint32_t kTauValid = 0x80000000u;                   // flag bit of the carried threshold word

// State words.  ST_TAU (the carried threshold: kTauValid | key, or 0 for
// none) is the last word, so that a caller may clear the others and keep it.
enum : int { ST_TAU = kStateWords - 1 };

__host__ __device__ constexpr int64_t tiles_of(int64_t d) { return (d + kTile - 1) / kTile; }
__host__ __device__ constexpr int64_t round64(int64_t x) { return (x + 63) / 64 * 64; }

// Per-worker scratch, in u32 words: state | tile counts | the 8 CTAs'
// private tile-prefix arrays (nt + 1 each) | candidate slots (kTile uint2
// per tile).
__host__ __device__ constexpr int64_t head_words(int64_t d) {
  return round64(kStateWords + tiles_of(d) + kCluster * (tiles_of(d) + 1));
}
__host__ __device__ constexpr int64_t row_words(int64_t d) { return head_words(d) + 2 * tiles_of(d) * kTile; }
__host__ __device__ constexpr int64_t srv_tiles(int64_t d) { return (d + kSrvTile - 1) / kSrvTile; }

struct RowScratch {
  uint32_t* state;
  uint32_t* cnt;
  uint32_t* gpre;  // kCluster arrays of nt + 1 words
  uint2* cand;
};

__device__ __forceinline__ RowScratch row_scratch(void* base, int64_t d, int row) {
  uint32_t* p = reinterpret_cast<uint32_t*>(base) + (int64_t)row * row_words(d);
  RowScratch r;
  r.state = p;
  r.cnt = r.state + kStateWords;
  r.gpre = r.cnt + tiles_of(d);
  r.cand = reinterpret_cast<uint2*>(p + head_words(d));
  return r;
}

__device__ __forceinline__ uint32_t key_of(float v) { return __float_as_uint(v) & 0x7FFFFFFFu; }
__device__ __forceinline__ uint32_t key_bits(uint32_t bits) { return bits & 0x7FFFFFFFu; }

// hist[bin] += 1 for each lane of `mask` (the lanes that call it together)
// with `valid`: lanes with the same bin are counted by one atomic.  (The
// candidates of a call lie within a few binades above the carried threshold,
// so their top digits fall into a few bins, and plain per-lane atomics on
// them serialise.)
__device__ __forceinline__ void warp_hist_add(uint32_t* hist, uint32_t bin, bool valid, unsigned mask) {
  const unsigned peers = __match_any_sync(mask, valid ? bin : 0xFFFFFFFFu);
  if (valid && (int)(threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(hist + bin, (uint32_t)__popc(peers));
}

// Block-wide exclusive scan of one value per thread; *total gets the sum.
// `warp_sums` is shared memory of NT/32 words.  Two barriers.
template <int NT>
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* total, uint32_t* warp_sums) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(kFullMask, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  uint32_t before = 0, sum = 0;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) {
    const uint32_t s = warp_sums[w];
    if (w < warp) before += s;
    sum += s;
  }
  __syncthreads();
  *total = sum;
  return before + x - v;
}

// Block-wide sum of one value per thread (two barriers).
template <int NT>
__device__ __forceinline__ uint32_t block_sum(uint32_t v, uint32_t* warp_sums) {
  uint32_t total;
  block_exclusive_scan<NT>(v, &total, warp_sums);
  return total;
}

// Digit selection in a shared-memory histogram of BINS counts: the digit b
// with count(> b) < k_rem <= count(>= b); *digit = b, *krem = k_rem -
// count(> b) (shared-memory outputs, valid after the call for all threads;
// left as they were when no digit qualifies).
template <int NT, int BINS>
__device__ void block_select(const uint32_t* hist, uint32_t k_rem, uint32_t* digit, uint32_t* krem,
                             uint32_t* warp_sums) {
  constexpr int kPer = BINS / NT;  // bins per thread, taken in descending digit order
  static_assert(kPer >= 1 && kPer * NT == BINS, "bins must be a multiple of the block size");
  uint32_t cnt[kPer];
  uint32_t local = 0;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    cnt[q] = hist[BINS - 1 - ((int)threadIdx.x * kPer + q)];
    local += cnt[q];
  }
  uint32_t total;
  uint32_t cum = block_exclusive_scan<NT>(local, &total, warp_sums);
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    if (cum < k_rem && k_rem <= cum + cnt[q]) {
      *digit = (uint32_t)(BINS - 1 - ((int)threadIdx.x * kPer + q));
      *krem = k_rem - cum;
    }
    cum += cnt[q];
  }
  __syncthreads();
}

// Writes one tile's flagged elements to its candidate slot in index order.
// Element order in the tile: row i, thread t, component q is tile offset
// 4 * (i * NT + t) + q.  Per lane and row at most 4 flags, per warp and row
// at most 128, so the R <= 4 row counts share one 32-bit warp scan (8 bits
// each).  `totals` is shared memory of NT/32 words.  Returns the tile's
// count (in every thread); one barrier, two when `reuse` (the caller writes
// `totals` again afterwards).
template <int NT, int R, bool REUSE>
__device__ __forceinline__ uint32_t write_tile_candidates(const float (&v)[R][4], const uint32_t (&cmask)[R],
                                                          int64_t tile0, uint2* slot, uint32_t* totals,
                                                          uint32_t* err) {
  static_assert(R <= 4, "four 8-bit row counts per word");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t packed = 0;
#pragma unroll
  for (int i = 0; i < R; ++i) packed |= (uint32_t)__popc(cmask[i]) << (8 * i);
  uint32_t incl = packed;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(kFullMask, incl, off);
    if (lane >= off) incl += y;
  }
  const uint32_t excl = incl - packed;
  if (lane == 31) totals[warp] = incl;
  __syncthreads();
  uint32_t done = 0;
#pragma unroll
  for (int i = 0; i < R; ++i) {
    uint32_t row_before = 0, row_total = 0;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) {
      const uint32_t f = (totals[w] >> (8 * i)) & 0xFFu;
      if (w < warp) row_before += f;
      row_total += f;
    }
    uint32_t pos = done + row_before + ((excl >> (8 * i)) & 0xFFu);
    done += row_total;
    if (cmask[i]) {
      const int64_t j = tile0 + 4 * ((int64_t)i * NT + threadIdx.x);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if ((cmask[i] >> q) & 1u) {
          if (dq_in_bounds(pos < (uint32_t)kTile, err)) slot[pos] = make_uint2((uint32_t)(j + q), __float_as_uint(v[i][q]));
          ++pos;
        }
    }
  }
  if constexpr (REUSE) __syncthreads();
  return done;
}

// ---------------------------------------------------------------------------
// 1. p = fl(fl(eta g) + e) into e; h = fl(fl(eta g) + p) (corrected at the kept
// entries by the second kernel); candidates with key >= the carried
// threshold (none without one).  Element order in a tile: row i,
// thread t, component q is tile offset 4 * (i * 256 + t) + q, so warp w of
// row i covers the 128 consecutive offsets of group g = 8 i + w.  Candidate
// values wait in shared memory (flagged in a bitmask) until the block's one
// barrier; then each warp writes its groups' candidates to the tile's slot
// in index order.
// ---------------------------------------------------------------------------
template <bool KEEP_H>
__global__ void __launch_bounds__(kFormThreads, 6) topk_form_kernel(const CompressArgs a, void* scratch) {
  dq_pdl_enter();
  constexpr int kGroups = kTile / 128;
  __shared__ float vstage[kTile];
  __shared__ uint32_t flags[kTile / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  const float* g = a.g + (int64_t)row * a.g_stride;
  float* e = a.e + (int64_t)(worker - a.row0) * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)(worker - a.row0) * a.ld : nullptr;
  RowScratch rs = row_scratch(scratch, a.d, worker - a.row0);
  const uint32_t tau_word = rs.state[ST_TAU];
  const bool has_tau = (tau_word & kTauValid) != 0;
  const uint32_t tau = tau_word & 0x7FFFFFFFu;
  const int64_t tile = blockIdx.x;
  const int64_t tile0 = tile * kTile;
#pragma unroll
  for (int i = 0; i < kFormRows; ++i) {
    const int off = 4 * (i * kFormThreads + (int)threadIdx.x);
    const int64_t j = tile0 + off;
    float v[4];
    int nvalid = 0;
    if (j + 3 < a.d) {
      const float4 gv = __ldcs(reinterpret_cast<const float4*>(g + j));
      const float4 ev = __ldcs(reinterpret_cast<const float4*>(e + j));
      const float gq[4] = {gv.x, gv.y, gv.z, gv.w};
      const float eq[4] = {ev.x, ev.y, ev.z, ev.w};
      float hv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float s = __fmul_rn(a.lr, gq[q]);
        v[q] = __fadd_rn(s, eq[q]);
        hv[q] = __fadd_rn(s, v[q]);
      }
      __stcs(reinterpret_cast<float4*>(e + j), make_float4(v[0], v[1], v[2], v[3]));
      if constexpr (KEEP_H) __stcs(reinterpret_cast<float4*>(h + j), make_float4(hv[0], hv[1], hv[2], hv[3]));
      nvalid = 4;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        v[q] = 0.f;
        if (j + q < a.d) {
          const float s = __fmul_rn(a.lr, g[j + q]);
          v[q] = __fadd_rn(s, e[j + q]);
          e[j + q] = v[q];
          if constexpr (KEEP_H) h[j + q] = __fadd_rn(s, v[q]);
          nvalid = q + 1;
        }
      }
    }
    uint32_t bits = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q < nvalid) {
        const uint32_t key = key_of(v[q]);
        if (has_tau && key >= tau) {
          bits |= 1u << q;
          vstage[off + q] = v[q];
        }
      }
    }
    // 8 lanes' 4 flag bits form one 32-bit word of the tile's bitmask
    uint32_t word = bits << (4 * (lane & 7));
    word |= __shfl_xor_sync(kFullMask, word, 1);
    word |= __shfl_xor_sync(kFullMask, word, 2);
    word |= __shfl_xor_sync(kFullMask, word, 4);
    if ((lane & 7) == 0) flags[off >> 5] = word;
  }
  __syncthreads();
  // group offsets: every warp scans the 32 groups' counts (group = lane)
  uint32_t gc = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) gc += __popc(flags[lane * 4 + q]);
  uint32_t incl = gc;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFullMask, incl, o);
    if (lane >= o) incl += y;
  }
  const uint32_t total = __shfl_sync(kFullMask, incl, 31);
  uint2* slot = rs.cand + tile * kTile;
  static_assert(kGroups == kFormRows * (kFormThreads / 32), "one group per warp and row");
#pragma unroll
  for (int i = 0; i < kFormRows; ++i) {
    const int grp = i * (kFormThreads / 32) + warp;
    const uint32_t gbase = __shfl_sync(kFullMask, incl - gc, grp);
    const uint32_t lane_bits = (flags[grp * 4 + (lane >> 3)] >> (4 * (lane & 7))) & 0xFu;
    const uint32_t n = __popc(lane_bits);
    uint32_t x = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFullMask, x, o);
      if (lane >= o) x += y;
    }
    uint32_t pos = gbase + x - n;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if ((lane_bits >> q) & 1u) {
        const int off = grp * 128 + lane * 4 + q;
        if (dq_in_bounds(pos < (uint32_t)kTile, a.err))  // a tile holds at most kTile candidates
          slot[pos] = make_uint2((uint32_t)(tile0 + off), __float_as_uint(vstage[off]));
        ++pos;
      }
    }
  }
  if (threadIdx.x == 0) rs.cnt[tile] = total;
}

// ---------------------------------------------------------------------------
// 2. Select T over the candidates and write the kept records (a cluster of
// kCluster CTAs per worker).
// ---------------------------------------------------------------------------
struct SelectSmem {
  uint32_t hist_t[kBins0];          // this CTA's top-digit histogram (read by the cluster)
  uint32_t hist_a[kBins1];          // this CTA's middle-digit histogram (read by the cluster)
  uint32_t hist_b[kBins1];          // this CTA's low-digit histogram (read by the cluster)
  uint32_t full[kBins0];            // a whole histogram (top digit; then the cluster's sums)
  uint32_t tpre[kChunkTiles + 1];   // candidate prefix at the chunk's tiles
  uint32_t warp_sums[kSelThreads / 32];
  uint32_t sel[6];
  uint32_t pre_t[kBins0];           // the same three histograms summed over the CTAs of lower rank
  uint32_t pre_a[kBins1];
  uint32_t pre_b[kBins1];
  uint32_t span[2];                 // first and last tile overlapping this CTA's share
  uint2 cache[kCacheCap];           // this CTA's share of the candidates, when it fits
};

// Tile counts a select thread holds in registers (all tiles, when nt fits).
constexpr int kRegTiles = 4;

// The tile of candidate f: the largest i < n with tpre[i] <= f (tpre
// non-decreasing, tpre[0] <= f < tpre[n]; an empty tile repeats its
// successor's prefix, so the tile found holds f), in a fixed number of
// halving steps (n <= kChunkTiles).  Used where the share is not kept on
// chip; filling the on-chip copy uses the tile map instead (a search per
// candidate, with the lanes reading scattered prefixes, conflicts in the
// shared-memory banks).
__device__ __forceinline__ int tile_of(const uint32_t* tpre, int n, uint32_t f) {
  int lo = 0;
#pragma unroll
  for (int step = kChunkTiles / 2; step >= 1; step >>= 1) {
    const int mid = lo + step;
    if (mid < n && tpre[mid] <= f) lo = mid;
  }
  return lo;
}

// Candidate f (prefix coordinates of tpre) of the chunk starting at tile tc0.
__device__ __forceinline__ uint2 chunk_candidate(const uint2* cand, const uint32_t* tpre, int n, int64_t tc0,
                                                 uint32_t f) {
  const int i = tile_of(tpre, n, f);
  return cand[(tc0 + i) * kTile + (f - tpre[i])];
}

// Sums the cluster's copies of one histogram into sm.full[0, BINS), and
// those of the CTAs of lower rank than this one into pre[0, BINS) (from which
// the CTA's first record position follows).  The cluster barrier publishes
// every CTA's counts; each histogram buffer is written once per selection
// round, so no barrier is needed after the reads.
template <int BINS>
__device__ __forceinline__ void cluster_sum(cg::cluster_group& cluster, uint32_t* local, uint32_t* pre,
                                            int rank, SelectSmem& sm) {
  cluster.sync();
  for (int i = threadIdx.x; i < BINS; i += kSelThreads) {
    uint32_t s = 0, below = 0;
#pragma unroll
    for (int r = 0; r < kCluster; ++r) {
      const uint32_t x = cluster.map_shared_rank(local, r)[i];
      if (r < rank) below += x;
      s += x;
    }
    sm.full[i] = s;
    pre[i] = below;
  }
  __syncthreads();
}

template <bool KEEP_H>
__global__ void __cluster_dims__(kCluster, 1, 1) __launch_bounds__(kSelThreads, 1)
topk_select_kernel(const CompressArgs a, int64_t k, void* scratch) {
  // launched as a programmatic dependent of the form kernel: its tile counts,
  // candidates and p are complete and visible after this wait
  dq_pdl_enter();
  extern __shared__ __align__(16) unsigned char smem_raw[];
  SelectSmem& sm = *reinterpret_cast<SelectSmem*>(smem_raw);
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  float* e = a.e + (int64_t)(worker - a.row0) * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)(worker - a.row0) * a.ld : nullptr;
  const float* g = a.g + (int64_t)row * a.g_stride;
  uint2* rec = reinterpret_cast<uint2*>(a.msg + (int64_t)row * a.msg_stride);
  RowScratch rs = row_scratch(scratch, a.d, worker - a.row0);
  const int64_t nt = tiles_of(a.d);
  uint32_t* gpre = rs.gpre + (int64_t)rank * (nt + 1);  // this CTA's private prefix array
  const uint32_t tau_word = rs.state[ST_TAU];
  const uint32_t tau = tau_word & 0x7FFFFFFFu;
  bool fast = (tau_word & kTauValid) != 0;
  const bool reg_tiles = nt <= (int64_t)kSelThreads * kRegTiles;

  // the first pass's tile counts
  uint32_t cnt_r[kRegTiles];
#pragma unroll
  for (int q = 0; q < kRegTiles; ++q) {
    const int64_t t = (int64_t)threadIdx.x * kRegTiles + q;
    cnt_r[q] = (fast && reg_tiles && t < nt) ? rs.cnt[t] : 0u;
  }
  uint32_t b0 = 0;  // top digit of T

  // This CTA's share: candidates [F0, F1) in prefix coordinates, lying in
  // tiles [ta, tb).  With one chunk, sm.tpre[i] is the prefix at tile ta + i.
  int64_t ta = 0, tb = 0;
  uint32_t F0 = 0, F1 = 0;
  bool one_chunk = true, cached = false;
  uint32_t lo1 = 0, hi1 = 0;  // the share's bounds when it is one chunk

  // Loads the prefix of tiles [tc0, tc0 + n] from gpre into sm.tpre.
  auto load_chunk = [&](int64_t tc0, int n) {
    for (int i = threadIdx.x; i <= n; i += kSelThreads) sm.tpre[i] = gpre[tc0 + i];
    __syncthreads();
  };

  const int64_t t0 = nt * rank / kCluster, t1 = nt * (rank + 1) / kCluster;  // this CTA's tiles

  auto set_up = [&]() {
    if (fast && reg_tiles) {
      // the tile counts are in registers: one scan gives every prefix
      uint32_t local = 0;
#pragma unroll
      for (int q = 0; q < kRegTiles; ++q) local += cnt_r[q];
      uint32_t N;
      const uint32_t ex = block_exclusive_scan<kSelThreads>(local, &N, sm.warp_sums);
      F0 = (uint32_t)((uint64_t)N * rank / kCluster);
      F1 = (uint32_t)((uint64_t)N * (rank + 1) / kCluster);
      if (threadIdx.x == 0) {
        sm.span[0] = 0xFFFFFFFFu;
        sm.span[1] = 0;
      }
      __syncthreads();
      uint32_t p = ex;
#pragma unroll
      for (int q = 0; q < kRegTiles; ++q) {
        const uint32_t t = threadIdx.x * kRegTiles + q;
        if (cnt_r[q] > 0 && p < F1 && p + cnt_r[q] > F0) {
          atomicMin(&sm.span[0], t);
          atomicMax(&sm.span[1], t);
        }
        p += cnt_r[q];
      }
      __syncthreads();
      if (F0 < F1) {
        ta = sm.span[0];
        tb = (int64_t)sm.span[1] + 1;
      } else {
        ta = tb = 0;
      }
      p = ex;
#pragma unroll
      for (int q = 0; q < kRegTiles; ++q) {
        const int64_t t = (int64_t)threadIdx.x * kRegTiles + q;
        if (t >= ta && t < tb) sm.tpre[t - ta] = p;
        p += cnt_r[q];
        if (t + 1 == tb) sm.tpre[tb - ta] = p;
      }
      __syncthreads();
      one_chunk = true;
    } else if (fast) {
      // all tiles' prefix through this CTA's private array in global memory
      uint32_t N = 0;
      for (int64_t base = 0; base < nt; base += kSelThreads) {
        const int64_t t = base + threadIdx.x;
        N += block_sum<kSelThreads>(t < nt ? rs.cnt[t] : 0u, sm.warp_sums);
      }
      F0 = (uint32_t)((uint64_t)N * rank / kCluster);
      F1 = (uint32_t)((uint64_t)N * (rank + 1) / kCluster);
      if (threadIdx.x == 0) {
        sm.span[0] = 0xFFFFFFFFu;
        sm.span[1] = 0;
      }
      __syncthreads();
      uint32_t run = 0;
      for (int64_t base = 0; base < nt; base += kSelThreads) {
        const int64_t t = base + threadIdx.x;
        const uint32_t c = t < nt ? rs.cnt[t] : 0u;
        uint32_t total;
        const uint32_t p = run + block_exclusive_scan<kSelThreads>(c, &total, sm.warp_sums);
        if (t < nt) {
          gpre[t] = p;
          if (c > 0 && p < F1 && p + c > F0) {
            atomicMin(&sm.span[0], (uint32_t)t);
            atomicMax(&sm.span[1], (uint32_t)t);
          }
        }
        run += total;
      }
      if (threadIdx.x == 0) gpre[nt] = run;
      __syncthreads();
      if (F0 < F1) {
        ta = sm.span[0];
        tb = (int64_t)sm.span[1] + 1;
      } else {
        ta = tb = 0;
      }
      one_chunk = (tb - ta) <= kChunkTiles;
      if (one_chunk && tb > ta) load_chunk(ta, (int)(tb - ta));
    } else {
      // re-extract this CTA's tiles from p: every element with top digit >= b0
      for (int64_t t = t0; t < t1; ++t) {
        const int64_t tile0 = t * kTile;
        float v[kSelRows][4];
        uint32_t cmask[kSelRows];
#pragma unroll
        for (int i = 0; i < kSelRows; ++i) {
          const int64_t j = tile0 + 4 * ((int64_t)i * kSelThreads + threadIdx.x);
          cmask[i] = 0;
          if (j + 3 < a.d) {
            const float4 x = *reinterpret_cast<const float4*>(e + j);
            v[i][0] = x.x; v[i][1] = x.y; v[i][2] = x.z; v[i][3] = x.w;
#pragma unroll
            for (int q = 0; q < 4; ++q)
              if ((key_of(v[i][q]) >> 20) >= b0) cmask[i] |= 1u << q;
          } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              v[i][q] = (j + q < a.d) ? e[j + q] : 0.f;
              if (j + q < a.d && (key_of(v[i][q]) >> 20) >= b0) cmask[i] |= 1u << q;
            }
          }
        }
        const uint32_t n = write_tile_candidates<kSelThreads, kSelRows, true>(v, cmask, tile0,
                                                                              rs.cand + t * kTile, sm.warp_sums, a.err);
        if (threadIdx.x == 0) rs.cnt[t] = n;
      }
      __syncthreads();
      // prefix of this CTA's own tiles, from 0
      uint32_t run = 0;
      for (int64_t base = t0; base < t1; base += kSelThreads) {
        const int64_t t = base + threadIdx.x;
        const uint32_t c = t < t1 ? rs.cnt[t] : 0u;
        uint32_t total;
        const uint32_t p = run + block_exclusive_scan<kSelThreads>(c, &total, sm.warp_sums);
        if (t < t1) gpre[t] = p;
        run += total;
      }
      if (threadIdx.x == 0) gpre[t1] = run;
      __syncthreads();
      ta = t0;
      tb = t1;
      F0 = 0;
      F1 = run;
      one_chunk = (tb - ta) <= kChunkTiles;
      if (one_chunk && tb > ta) load_chunk(ta, (int)(tb - ta));
    }
    cached = false;
    lo1 = hi1 = 0;
    if (one_chunk && tb > ta) {
      lo1 = max(F0, sm.tpre[0]);
      hi1 = min(F1, sm.tpre[tb - ta]);
      cached = hi1 - lo1 <= (uint32_t)kCacheCap;
    }
  };

  // Runs body(candidate) over this CTA's share, kBatch loads in flight per
  // thread; with `fill`, also keeps the share on chip.
  // (body(candidate, valid) is called by every thread of the block the same
  // number of times, so it may use warp collectives.)
  auto for_each = [&](auto&& body, bool fill) {
    if (fill) {
      // The share becomes the on-chip copy (cached: one chunk of tiles
      // [ta, tb), candidates [lo1, hi1)).  First every candidate slot gets
      // its tile: each tile with candidates in the share marks its first
      // slot with its number, and a block-wide running maximum over the
      // slots carries each mark forward (the marks grow with the slot).  The
      // cost does not depend on how the candidates spread over the tiles,
      // and the loads below need no search.
      const int n = (int)(tb - ta);
      const uint32_t S = hi1 - lo1;
      for (uint32_t f = threadIdx.x; f < S; f += kSelThreads) sm.cache[f].x = 0u;
      __syncthreads();
      for (int i = threadIdx.x; i < n; i += kSelThreads) {
        const uint32_t a0 = sm.tpre[i], a1 = sm.tpre[i + 1];
        if (a0 < a1 && a1 > lo1 && a0 < hi1) sm.cache[max(a0, lo1) - lo1].x = (uint32_t)i;
      }
      __syncthreads();
      const uint32_t per = (S + kSelThreads - 1) / kSelThreads;
      const uint32_t g0 = min(threadIdx.x * per, S), g1 = min(g0 + per, S);
      uint32_t run = 0;
      for (uint32_t f = g0; f < g1; ++f) run = max(run, sm.cache[f].x);
      // exclusive running maximum over the threads' runs
      {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        uint32_t x = run;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const uint32_t y = __shfl_up_sync(kFullMask, x, off);
          if (lane >= off) x = max(x, y);
        }
        if (lane == 31) sm.warp_sums[warp] = x;
        __syncthreads();
        uint32_t before = 0;
#pragma unroll
        for (int w = 0; w < kSelThreads / 32; ++w)
          if (w < warp) before = max(before, sm.warp_sums[w]);
        const uint32_t up = __shfl_up_sync(kFullMask, x, 1);
        run = max(before, lane > 0 ? up : 0u);
        __syncthreads();
      }
      for (uint32_t f = g0; f < g1; ++f) {
        run = max(run, sm.cache[f].x);
        sm.cache[f].x = run;
      }
      __syncthreads();
      for (uint32_t base = lo1; base < hi1; base += kSelThreads * kBatch) {
        uint2 c[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const uint32_t f = base + u * kSelThreads + threadIdx.x;
          c[u] = make_uint2(0u, 0u);
          if (f < hi1) {
            const uint32_t i = sm.cache[f - lo1].x;
            c[u] = rs.cand[(ta + i) * kTile + (f - sm.tpre[i])];
          }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const uint32_t f = base + u * kSelThreads + threadIdx.x;
          if (f < hi1) sm.cache[f - lo1] = c[u];
          body(c[u], f < hi1);
        }
      }
      __syncthreads();
      return;
    }
    if (cached) {
      for (uint32_t base = lo1; base < hi1; base += kSelThreads) {
        const uint32_t f = base + threadIdx.x;
        body(f < hi1 ? sm.cache[f - lo1] : make_uint2(0u, 0u), f < hi1);
      }
      return;
    }
    for (int64_t tc0 = ta; tc0 < tb; tc0 += kChunkTiles) {
      const int n = (int)min64(kChunkTiles, tb - tc0);
      if (!one_chunk) load_chunk(tc0, n);
      const uint32_t lo = max(F0, sm.tpre[0]), hi = min(F1, sm.tpre[n]);
      for (uint32_t base = lo; base < hi; base += kSelThreads * kBatch) {
        uint2 c[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const uint32_t f = base + u * kSelThreads + threadIdx.x;
          c[u] = (f < hi) ? chunk_candidate(rs.cand, sm.tpre, n, tc0, f) : make_uint2(0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const uint32_t f = base + u * kSelThreads + threadIdx.x;
          if (fill && f < hi) sm.cache[f - lo] = c[u];
          body(c[u], f < hi);
        }
      }
      if (!one_chunk) __syncthreads();  // sm.tpre is reloaded for the next chunk
    }
  };

  // Histogram of the top digit over all of p in this CTA's tiles.
  auto histogram_p = [&]() {
    for (int64_t t = t0; t < t1; ++t) {
#pragma unroll
      for (int i = 0; i < kSelRows; ++i) {
        const int64_t j = t * kTile + 4 * ((int64_t)i * kSelThreads + threadIdx.x);
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (j + 3 < a.d) {
          x = *reinterpret_cast<const float4*>(e + j);
        } else {
          if (j < a.d) x.x = e[j];
          if (j + 1 < a.d) x.y = e[j + 1];
          if (j + 2 < a.d) x.z = e[j + 2];
        }
        // (all of p: its top digits spread over many bins, so plain atomics)
        if (j < a.d) atomicAdd(&sm.hist_t[key_of(x.x) >> 20], 1u);
        if (j + 1 < a.d) atomicAdd(&sm.hist_t[key_of(x.y) >> 20], 1u);
        if (j + 2 < a.d) atomicAdd(&sm.hist_t[key_of(x.z) >> 20], 1u);
        if (j + 3 < a.d) atomicAdd(&sm.hist_t[key_of(x.w) >> 20], 1u);
      }
    }
    __syncthreads();
  };

  uint32_t T = 0, need = 0;
  for (int attempt = 0; attempt < 2; ++attempt) {
    if (attempt > 0) cluster.sync();  // every CTA is done reading the first round's histograms
    for (int i = threadIdx.x; i < kBins0; i += kSelThreads) sm.hist_t[i] = 0;
    for (int i = threadIdx.x; i < kBins1; i += kSelThreads) {
      sm.hist_a[i] = 0;
      sm.hist_b[i] = 0;
    }
    __syncthreads();
    // top digit: over the candidates, or over all of p
    bool filled = false;
    if (fast) {
      set_up();
      for_each(
          [&](uint2 c, bool valid) {
            warp_hist_add(sm.hist_t, key_bits(c.y) >> 20, valid, kFullMask);
          },
          cached);
      filled = cached;
    } else {
      histogram_p();
    }
    cluster_sum<kBins0>(cluster, sm.hist_t, sm.pre_t, rank, sm);
    if (threadIdx.x == 0) {
      sm.sel[0] = 0;
      sm.sel[1] = (uint32_t)k;
    }
    __syncthreads();
    block_select<kSelThreads, kBins0>(sm.full, (uint32_t)k, &sm.sel[0], &sm.sel[1], sm.warp_sums);
    b0 = sm.sel[0];
    const uint32_t krem0 = sm.sel[1];
    if (!fast) set_up();  // candidates: every element with top digit >= b0
    // middle digit
    for_each(
        [&](uint2 c, bool valid) {
          const uint32_t key = key_bits(c.y);
          if (valid && (key >> 20) == b0) atomicAdd(&sm.hist_a[(key >> 10) & 1023u], 1u);
        },
        cached && !filled);
    cluster_sum<kBins1>(cluster, sm.hist_a, sm.pre_a, rank, sm);
    if (threadIdx.x == 0) {
      sm.sel[2] = 0;
      sm.sel[3] = krem0;
    }
    __syncthreads();
    block_select<kSelThreads, kBins1>(sm.full, krem0, &sm.sel[2], &sm.sel[3], sm.warp_sums);
    const uint32_t hi21 = (b0 << 10) | sm.sel[2];
    const uint32_t krem1 = sm.sel[3];
    // low digit
    for_each(
        [&](uint2 c, bool valid) {
          const uint32_t key = key_bits(c.y);
          if (valid && (key >> 10) == hi21) atomicAdd(&sm.hist_b[key & 1023u], 1u);
        },
        false);
    cluster_sum<kBins1>(cluster, sm.hist_b, sm.pre_b, rank, sm);
    if (threadIdx.x == 0) {
      sm.sel[4] = 0;
      sm.sel[5] = krem1;
    }
    __syncthreads();
    block_select<kSelThreads, kBins1>(sm.full, krem1, &sm.sel[4], &sm.sel[5], sm.warp_sums);
    T = (hi21 << 10) | sm.sel[4];
    need = sm.sel[5];
    // T is exact when every key >= T was a candidate, i.e. T >= tau (the
    // same decision in every CTA of the cluster).
    if (!fast || T >= tau) break;
    fast = false;
  }

  // Every read of another CTA's shared memory is done: arrive at the
  // cluster barrier now, wait for the others only before leaving (no CTA
  // leaves while another may still read its shared memory).
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");

  // Keys above and equal to T in the shares of the CTAs before this one, from
  // the histogram sums over them: top digit above b0, or middle digit above
  // T's, or low digit above T's; and keys equal to T.
  uint32_t gt_before = 0, tie_before = 0;
  {
    const uint32_t b1 = (T >> 10) & 1023u, b2 = T & 1023u;
    uint32_t part = 0;
    for (int i = threadIdx.x; i < kBins0; i += kSelThreads)
      if ((uint32_t)i > b0) part += sm.pre_t[i];
    for (int i = threadIdx.x; i < kBins1; i += kSelThreads) {
      if ((uint32_t)i > b1) part += sm.pre_a[i];
      if ((uint32_t)i > b2) part += sm.pre_b[i];
    }
    gt_before = block_sum<kSelThreads>(part, sm.warp_sums);
    tie_before = sm.pre_b[b2];
  }

  // Kept records: position = (keys > T before) + min(keys == T before, need).
  auto keep = [&](uint2 c) {
    const uint32_t j = c.x;
    const float p = __uint_as_float(c.y);
    const float ej = __fsub_rn(p, p);
    e[j] = ej;
    if constexpr (KEEP_H) h[j] = __fadd_rn(__fmul_rn(a.lr, g[j]), ej);
  };
  if (cached) {
    // Each warp takes kEmitRows rows of 32 consecutive candidates; ballots
    // rank the lanes, one exchange of the warps' counts ranks the warps.
    constexpr int kEmitRows = 8;
    constexpr int kWarps = kSelThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t lt = (1u << lane) - 1u;
    for (uint32_t base = lo1; base < hi1; base += kWarps * kEmitRows * 32) {
      const uint32_t seg = base + (uint32_t)warp * kEmitRows * 32;
      uint2 c[kEmitRows];
      uint32_t gtb[kEmitRows], tieb[kEmitRows];
      uint32_t wg = 0, wt = 0;
#pragma unroll
      for (int u = 0; u < kEmitRows; ++u) {
        const uint32_t f = seg + 32u * u + lane;
        const bool valid = f < hi1;
        c[u] = valid ? sm.cache[f - lo1] : make_uint2(0u, 0u);
        const uint32_t key = key_bits(c[u].y);
        gtb[u] = __ballot_sync(kFullMask, valid && key > T);
        tieb[u] = __ballot_sync(kFullMask, valid && key == T);
        wg += __popc(gtb[u]);
        wt += __popc(tieb[u]);
      }
      if (lane == 0) sm.warp_sums[warp] = wg | (wt << 16);
      __syncthreads();
      uint32_t before = 0, total = 0;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const uint32_t v = sm.warp_sums[w];
        if (w < warp) before += v;
        total += v;
      }
      __syncthreads();
      uint32_t rg = gt_before + (before & 0xFFFFu), rt = tie_before + (before >> 16);
#pragma unroll
      for (int u = 0; u < kEmitRows; ++u) {
        const uint32_t my_g = rg + __popc(gtb[u] & lt), my_t = rt + __popc(tieb[u] & lt);
        const bool is_gt = (gtb[u] >> lane) & 1u, is_tie = (tieb[u] >> lane) & 1u;
        if (is_gt || (is_tie && my_t < need)) {
          const uint32_t pos = my_g + min(my_t, need);
          if (dq_in_bounds(pos < (uint64_t)k, a.err)) {  // always true; keeps the write inside the message
            rec[pos] = c[u];
            keep(c[u]);
          }
        }
        rg += __popc(gtb[u]);
        rt += __popc(tieb[u]);
      }
      gt_before += total & 0xFFFFu;
      tie_before += total >> 16;
    }
  } else {
    auto emit = [&](uint2 c, bool valid) {
      const uint32_t key = key_bits(c.y);
      const bool is_gt = valid && key > T;
      const bool is_tie = valid && key == T;
      uint32_t total;
      const uint32_t ex = block_exclusive_scan<kSelThreads>((uint32_t)is_gt | ((uint32_t)is_tie << 16), &total,
                                                            sm.warp_sums);
      const uint32_t ties = tie_before + (ex >> 16);
      if (is_gt || (is_tie && ties < need)) {
        const uint32_t pos = gt_before + (ex & 0xFFFFu) + min(ties, need);
        if (dq_in_bounds(pos < (uint64_t)k, a.err)) {  // always true; keeps the write inside the message
          rec[pos] = c;
          keep(c);
        }
      }
      gt_before += total & 0xFFFFu;
      tie_before += total >> 16;
    };
    for (int64_t tc0 = ta; tc0 < tb; tc0 += kChunkTiles) {
      const int n = (int)min64(kChunkTiles, tb - tc0);
      if (!one_chunk) load_chunk(tc0, n);
      const uint32_t lo = max(F0, sm.tpre[0]), hi = min(F1, sm.tpre[n]);
      for (uint32_t base = lo; base < hi; base += kSelThreads * kBatch) {
        uint2 c[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const uint32_t f = base + u * kSelThreads + threadIdx.x;
          c[u] = (f < hi) ? chunk_candidate(rs.cand, sm.tpre, n, tc0, f) : make_uint2(0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) emit(c[u], base + u * kSelThreads + threadIdx.x < hi);
      }
      __syncthreads();
    }
  }

  // For the next call: the candidate threshold, 15/16 of T.
  if (rank == 0 && threadIdx.x == 0) {
    const float t_next = __fmul_rn(__uint_as_float(T), 0.9375f);
    rs.state[ST_TAU] = kTauValid | key_of(t_next);
  }
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Server.  starts[m][t] = first record of worker m whose index is in tile t
// or later (t in [0, nts]); record r writes the tiles (tile(r-1), tile(r)],
// and the last record also (tile(k-1), nts].
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) topk_server_starts_kernel(const ServerArgs s, uint32_t* starts) {
  dq_pdl_enter();
  const int m = blockIdx.y;
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31;
  const int64_t nts = srv_tiles(s.d);
  const uint2* msg = reinterpret_cast<const uint2*>(s.msgs + (int64_t)m * s.msg_stride);
  uint32_t* st = starts + (int64_t)m * (nts + 1);
  // this record fills the tiles [t_a, t_b] with r (empty range: t_a > t_b)
  int64_t t_a = 1, t_b = 0;
  if (r < s.k) {
    const int64_t tile = min64(msg[r].x / kSrvTile, nts - 1);
    const int64_t prev = (r == 0) ? -1 : min64(msg[r - 1].x / kSrvTile, nts - 1);
    t_a = prev + 1;
    t_b = tile;
  }
  for (int64_t t = t_a; t <= t_b && t < t_a + 32; ++t) st[t] = (uint32_t)r;
  // long runs (sparse stretches of the index range) are written by the whole warp
  uint32_t longs = __ballot_sync(kFullMask, t_b - t_a >= 32);
  while (longs) {
    const int src = __ffs(longs) - 1;
    longs &= longs - 1;
    const int64_t a = __shfl_sync(kFullMask, t_a, src), bnd = __shfl_sync(kFullMask, t_b, src);
    const uint32_t val = (uint32_t)__shfl_sync(kFullMask, r, src);
    for (int64_t t = a + 32 + lane; t <= bnd; t += 32) st[t] = val;
  }
  // after the last record: the tiles up to nts point past the end
  const uint32_t last = __ballot_sync(kFullMask, r == s.k - 1);
  if (last) {
    const int src = __ffs(last) - 1;
    const int64_t a = __shfl_sync(kFullMask, t_b, src) + 1;
    for (int64_t t = a + lane; t <= nts; t += 32) st[t] = (uint32_t)s.k;
  }
}

template <bool POW2>
__device__ __forceinline__ float srv_average(float acc, const ServerArgs& s) {
  if constexpr (POW2) return __fmul_rn(acc, s.inv_M);
  else return __fdiv_rn(acc, (float)s.M);
}

// Server for M <= kSrvMaskMaxM: two launches over the M * k records, with
// two tables in the scratch -- a worker mask per index (u64; all zero
// between calls) and a value row per worker (d floats, never cleared).
//   1. scatter: record (m, r) with index j writes its value to row m at j
//      and sets bit m of j's mask.
//   2. reduce: the record of the lowest worker in j's mask owns j.  It sums
//      the values of the workers in the mask, in worker order with the
//      absent workers as +0 leaves (the library's pairwise order), updates
//      w_j and clears j's mask.  The other records of j read its mask
//      before or after the owner clears it; either way their own bit is not
//      its lowest, so they do nothing.
// Indices nobody sent have the sum +0 and keep w_j; with store_q the q_hat
// buffer is cleared before the scatter.
constexpr int kSrvMaskMaxM = 64;


struct SrvTables {
  unsigned long long* mask;  // d masks
  float* vals;               // row m at vals + m * ldv
  int64_t ldv;
};

__host__ __device__ constexpr int64_t srv_mask_table_words(int64_t d, int32_t nworkers) {
  return 2 * round64(d) + (int64_t)nworkers * round64(d);
}

inline SrvTables srv_tables(void* scratch, int64_t d, int32_t rows) {
  uint32_t* base = reinterpret_cast<uint32_t*>(scratch) + row_words(d) * rows;
  SrvTables t;
  t.mask = reinterpret_cast<unsigned long long*>(base);
  t.vals = reinterpret_cast<float*>(base + 2 * round64(d));
  t.ldv = round64(d);
  return t;
}

__global__ void __launch_bounds__(kSrvThreads) topk_server_scatter_kernel(const ServerArgs s, SrvTables t) {
  dq_pdl_enter();
  const int m = blockIdx.y;
  const int64_t r = (int64_t)blockIdx.x * kSrvThreads + threadIdx.x;
  if (r >= s.k) return;
  const uint2 rec = reinterpret_cast<const uint2*>(s.msgs + (int64_t)m * s.msg_stride)[r];
  // records come from the compressor and are below d
  if (!dq_in_bounds((int64_t)rec.x < s.d, s.err)) return;
  t.vals[(int64_t)m * t.ldv + rec.x] = __uint_as_float(rec.y);
  atomicOr(t.mask + rec.x, 1ull << m);
}

template <bool POW2, int P>
__global__ void __launch_bounds__(kSrvThreads) topk_server_reduce_kernel(const ServerArgs s, SrvTables t) {
  const int m = blockIdx.y;
  const int64_t r = (int64_t)blockIdx.x * kSrvThreads + threadIdx.x;
  if (r >= s.k) return;
  const uint2 rec = reinterpret_cast<const uint2*>(s.msgs + (int64_t)m * s.msg_stride)[r];
  const int64_t j = rec.x;
  if (j >= s.d) return;  // skipped by the scatter (and reported there by the checked build)
  // the scatter grid has completed and its writes are visible (the record
  // was complete before the scatter ran)
  dq_pdl_enter();
  const unsigned long long mask = t.mask[j];
  // the owner: bit m set and no bit below it
  if (!((mask >> m) & 1ull) || (mask & ((1ull << m) - 1ull))) return;
  const float v = __uint_as_float(rec.y);
  float sum;
  if ((mask & (mask - 1ull)) == 0ull) {
    sum = P == 1 ? v : __fadd_rn(v, 0.f);  // one value among +0 leaves
  } else {
    // the padded tree itself: chunks of C leaves (workers), each summed
    // pairwise from its values (+0 where a worker is absent), then the
    // P / C chunk sums pairwise -- the chunks are the tree's subtrees
    constexpr int C = P < 16 ? P : 16;
    float part[P / C];
#pragma unroll
    for (int c = 0; c < P / C; ++c) {
      const uint32_t bits = (uint32_t)(mask >> (C * c)) & (uint32_t)((1ull << C) - 1ull);
      float x[C];
#pragma unroll
      for (int u = 0; u < C; ++u) {
        const int who = C * c + u;
        x[u] = 0.f;
        if ((bits >> u) & 1u) x[u] = who == m ? v : t.vals[(int64_t)who * t.ldv + j];
      }
#pragma unroll
      for (int width = C / 2; width >= 1; width /= 2)
#pragma unroll
        for (int i = 0; i < width; ++i) x[i] = __fadd_rn(x[2 * i], x[2 * i + 1]);
      part[c] = x[0];
    }
#pragma unroll
    for (int width = P / C / 2; width >= 1; width /= 2)
#pragma unroll
      for (int i = 0; i < width; ++i) part[i] = __fadd_rn(part[2 * i], part[2 * i + 1]);
    sum = part[0];
  }
  s.w[j] = server_out(s, s.w[j], srv_average<POW2>(sum, s));
  t.mask[j] = 0ull;
}

// One thread per record of every worker.  The record of the lowest worker
// holding index j owns j: it sums the values recorded for j over all M
// workers (absent ones as +0 leaves) in the library's pairwise order and
// applies w_j -= sum / M; the others find an earlier worker holding j and
// stop.  Each search looks only at the other worker's
// records in j's tile of kSrvTile indices (the starts table), and the
// searches in kSrvGroup workers' lists advance in lockstep so that their
// loads are in flight together.
constexpr int kSrvGroup = 8;

template <bool POW2>
__global__ void __launch_bounds__(kSrvThreads) topk_server_owner_kernel(const ServerArgs s, const uint32_t* starts) {
  dq_pdl_enter();
  const int64_t id = (int64_t)blockIdx.x * kSrvThreads + threadIdx.x;
  if (id >= (int64_t)s.M * s.k) return;
  const int m = (int)(id / s.k);
  const int64_t r = id - (int64_t)m * s.k;
  const uint2 mine = reinterpret_cast<const uint2*>(s.msgs + (int64_t)m * s.msg_stride)[r];
  const uint32_t j = mine.x;
  if (!dq_in_bounds((int64_t)j < s.d, s.err)) return;  // records come from the compressor and are < d
  const int64_t nts = srv_tiles(s.d);
  const int64_t t = j / kSrvTile;
  PairwiseAcc<13> sum;  // M <= 4096
  for (int m2 = 0; m2 < m; ++m2) sum.push(0.f);  // no earlier worker holds j (else it owns j)
  sum.push(__uint_as_float(mine.y));
  for (int m0 = 0; m0 < s.M; m0 += kSrvGroup) {
    uint32_t lo[kSrvGroup], hi[kSrvGroup], end[kSrvGroup];
#pragma unroll
    for (int u = 0; u < kSrvGroup; ++u) {
      const int m2 = m0 + u;
      lo[u] = hi[u] = 0;
      if (m2 < s.M && m2 != m) {
        const uint32_t* st = starts + (int64_t)m2 * (nts + 1);
        lo[u] = (uint32_t)min64(st[t], s.k);
        hi[u] = (uint32_t)min64(st[t + 1], s.k);
      }
      end[u] = hi[u];
    }
    // lower bound of j in every range, one halving step for all at a time
    bool active = true;
    while (active) {
      uint32_t x[kSrvGroup];
#pragma unroll
      for (int u = 0; u < kSrvGroup; ++u) {
        x[u] = 0;
        if (lo[u] < hi[u]) {
          const uint2* rec = reinterpret_cast<const uint2*>(s.msgs + (int64_t)(m0 + u) * s.msg_stride);
          x[u] = rec[lo[u] + ((hi[u] - lo[u]) >> 1)].x;
        }
      }
      active = false;
#pragma unroll
      for (int u = 0; u < kSrvGroup; ++u) {
        if (lo[u] < hi[u]) {
          const uint32_t mid = lo[u] + ((hi[u] - lo[u]) >> 1);
          if (x[u] < j) lo[u] = mid + 1;
          else hi[u] = mid;
          active |= lo[u] < hi[u];
        }
      }
    }
    float val[kSrvGroup];
    bool has[kSrvGroup];
#pragma unroll
    for (int u = 0; u < kSrvGroup; ++u) {
      has[u] = false;
      val[u] = 0.f;
      if (lo[u] < end[u]) {
        const uint2* rec = reinterpret_cast<const uint2*>(s.msgs + (int64_t)(m0 + u) * s.msg_stride);
        const uint2 x = rec[lo[u]];
        has[u] = x.x == j;
        val[u] = __uint_as_float(x.y);
      }
    }
#pragma unroll
    for (int u = 0; u < kSrvGroup; ++u) {
      if (has[u] && m0 + u < m) return;  // an earlier worker owns j
      if (m0 + u > m && m0 + u < s.M) sum.push(has[u] ? val[u] : 0.f);
    }
  }
  s.w[j] = __fsub_rn(s.w[j], srv_average<POW2>(sum.result(), s));
}

}  // namespace

size_t topk_scratch_bytes(int64_t d, int32_t rows, int32_t nworkers) {
  // the server's tables: masks and value rows (M <= kSrvMaskMaxM), or the
  // record-range table of the owner kernel (more workers); none for 0
  const int64_t server_words = nworkers <= 0 ? 0
                               : nworkers <= kSrvMaskMaxM ? srv_mask_table_words(d, nworkers)
                                                          : round64((int64_t)nworkers * (srv_tiles(d) + 1));
  return (size_t)(row_words(d) * rows + server_words) * 4u;
}

// Raises a kernel's dynamic shared memory limit when its static plus dynamic
// shared memory exceeds the default 48 KB.  The attribute belongs to the
// function on the current device, so what has been set is remembered per
// device ordinal (`done` has kSmemDevices slots; the value only grows).
// Several host threads may race to set it; setting it twice is harmless.
constexpr int kSmemDevices = 64;

template <typename K>
cudaError_t ensure_smem(K kernel, size_t bytes, size_t static_bytes, std::atomic<size_t> (&done)[kSmemDevices]) {
  if (bytes + static_bytes <= 48u * 1024u) return cudaSuccess;
  int dev = 0;
  cudaError_t st = cudaGetDevice(&dev);
  if (st != cudaSuccess) return st;
  const bool cached = dev >= 0 && dev < kSmemDevices;
  if (cached && done[dev].load(std::memory_order_acquire) >= bytes) return cudaSuccess;
  st = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (st == cudaSuccess && cached) {
    size_t cur = done[dev].load(std::memory_order_relaxed);
    while (cur < bytes && !done[dev].compare_exchange_weak(cur, bytes, std::memory_order_release)) {
    }
  }
  return st;
}

cudaError_t launch_topk_compress(const CompressArgs& a, int64_t k, bool keep_h, void* scratch,
                                 cudaStream_t stream, uint64_t* launches) {
  static std::atomic<size_t> smem_done[2][kSmemDevices];
  const unsigned rows = (unsigned)a.nworkers;
  const dim3 tiles((unsigned)tiles_of(a.d), rows);
  const dim3 clusters(kCluster, rows);
  const size_t smem = sizeof(SelectSmem);
  cudaError_t st;
  if (keep_h) {
    if ((st = ensure_smem(topk_select_kernel<true>, smem, 0, smem_done[1])) != cudaSuccess) return st;
    launch_pdl(topk_form_kernel<true>, tiles, dim3(kFormThreads), 0, stream, a, scratch);
    if ((st = cudaGetLastError()) != cudaSuccess) return st;
    st = launch_pdl(topk_select_kernel<true>, clusters, dim3(kSelThreads), smem, stream, a, k, scratch);
  } else {
    if ((st = ensure_smem(topk_select_kernel<false>, smem, 0, smem_done[0])) != cudaSuccess) return st;
    launch_pdl(topk_form_kernel<false>, tiles, dim3(kFormThreads), 0, stream, a, scratch);
    if ((st = cudaGetLastError()) != cudaSuccess) return st;
    st = launch_pdl(topk_select_kernel<false>, clusters, dim3(kSelThreads), smem, stream, a, k, scratch);
  }
  *launches += st == cudaSuccess ? 2 : 1;
  return st;
}

cudaError_t launch_topk_server(const ServerArgs& s, void* scratch, int32_t rows, cudaStream_t stream,
                                uint64_t* launches) {
  if (s.M <= kSrvMaskMaxM) {
    const SrvTables t = srv_tables(scratch, s.d, rows);
    const dim3 grid((unsigned)((s.k + kSrvThreads - 1) / kSrvThreads), (unsigned)s.M);
    if (s.store_q) {  // the dense q_hat buffer: +0 wherever nobody sent an index
      const cudaError_t st = cudaMemsetAsync(s.w, 0, (size_t)s.d * sizeof(float), stream);
      if (st != cudaSuccess) return st;
    }
    launch_pdl(topk_server_scatter_kernel, grid, dim3(kSrvThreads), 0, stream, s, t);
    cudaError_t st = cudaGetLastError();
    if (st != cudaSuccess) return st;
    // the reduce kernel's blocks read their records while the scatter's last
    // blocks finish, then wait for the scatter grid
    st = cudaErrorInvalidValue;
    switch (next_pow2(s.M)) {
#define DQ_TOPK_REDUCE(P)                                                                             \
  case P:                                                                                             \
    st = s.M_pow2 ? launch_pdl(topk_server_reduce_kernel<true, P>, grid, dim3(kSrvThreads), 0, stream, s, t) \
                  : launch_pdl(topk_server_reduce_kernel<false, P>, grid, dim3(kSrvThreads), 0, stream, s, t); \
    break;
      DQ_TOPK_REDUCE(1) DQ_TOPK_REDUCE(2) DQ_TOPK_REDUCE(4) DQ_TOPK_REDUCE(8) DQ_TOPK_REDUCE(16)
      DQ_TOPK_REDUCE(32) DQ_TOPK_REDUCE(64)
#undef DQ_TOPK_REDUCE
    }
    // (a failure here would leave the scatter's mask bits set; the launch has
    // the scatter's grid and block, which were just accepted)
    *launches += st == cudaSuccess ? 2 : 1;
    return st;
  }
  if (s.store_q) return cudaErrorNotSupported;  // the owner kernel is sparse
  uint32_t* starts = reinterpret_cast<uint32_t*>(scratch) + row_words(s.d) * rows;
  const int64_t n = (int64_t)s.M * s.k;
  launch_pdl(topk_server_starts_kernel, dim3((unsigned)((s.k + 255) / 256), (unsigned)s.M), dim3(256), 0, stream, s, starts);
  const unsigned blocks = (unsigned)((n + kSrvThreads - 1) / kSrvThreads);
  if (s.M_pow2) launch_pdl(topk_server_owner_kernel<true>, dim3(blocks), dim3(kSrvThreads), 0, stream, s, starts);
  else launch_pdl(topk_server_owner_kernel<false>, dim3(blocks), dim3(kSrvThreads), 0, stream, s, starts);
  *launches += 2;
  return cudaGetLastError();
}

}  // namespace dq
