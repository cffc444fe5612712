// Worker side of Algorithm 2 with the top-k compressor (Section 2.4, Theorem 1):
// keep the k entries of p = fl(fl(eta*g) + e) with the largest |p_j| (ties to
// the lower index), send them as (u32 index, f32 value) records in ascending
// index order, and keep e_j = +0 at the kept entries and e_j = p_j elsewhere.
//
// |p_j| is ordered by its bit pattern with the sign cleared (a 31-bit key),
// so the k-th largest key is found by a three-digit radix select (11 + 10 +
// 10 bits) without sorting:
//   1. pass over g, e (tiles of 4096): p -> e in place, h (optional), and a
//      block-shared histogram of the top 11 key bits, merged into global;
//   2. one block finds the digit b0 holding the k-th largest key;
//   3. pass over p: per tile, count keys with digit > b0 (all kept) and append
//      the indices with digit == b0 to a candidate list, histogramming their
//      middle digit;
//   4-6. the middle and low digits are selected on the (short) candidate list,
//      giving the threshold key T and the number `need` of keys equal to T
//      that are kept (the lowest indices among them);
//   7. per-tile counts of candidates above T and equal to T;
//   8. one block scans the tiles: output offset of every tile;
//   9. pass over p: each tile writes its kept records in index order (block
//      scan) and zeroes e at the kept entries.
// Every histogram and counter is returned to zero by the stage that consumes
// it, so the scratch needs no clearing between calls.
#include "internal.cuh"

namespace dq {
namespace {

constexpr int kTile = 4096;          // elements per tile
constexpr int kThreads = 256;        // threads per tile block
constexpr int kRows = kTile / (4 * kThreads);  // 4 rows of 256 chunks
constexpr int kBins0 = 2048, kBins1 = 1024, kBins2 = 1024;
constexpr int kStateWords = 32;

// state words
enum : int { ST_B0 = 0, ST_KREM0, ST_CAND, ST_B1, ST_KREM1, ST_T, ST_NEED };

__host__ __device__ __forceinline__ int64_t tiles_of(int64_t d) { return (d + kTile - 1) / kTile; }

// Per-worker scratch, in u32 words.
struct RowScratch {
  uint32_t* hist0;
  uint32_t* hist1;
  uint32_t* hist2;
  uint32_t* state;
  uint32_t* tile_above;
  uint32_t* gt_count;
  uint32_t* tie_count;
  uint32_t* ties_before;
  uint32_t* out_off;
  uint32_t* cand;
};

__host__ __device__ __forceinline__ int64_t row_words(int64_t d) {
  const int64_t nt = tiles_of(d);
  const int64_t w = kBins0 + kBins1 + kBins2 + kStateWords + 5 * nt + d;
  return (w + 63) / 64 * 64;
}

__device__ __forceinline__ RowScratch row_scratch(void* base, int64_t d, int row) {
  uint32_t* p = reinterpret_cast<uint32_t*>(base) + (int64_t)row * row_words(d);
  const int64_t nt = tiles_of(d);
  RowScratch r;
  r.hist0 = p;
  r.hist1 = r.hist0 + kBins0;
  r.hist2 = r.hist1 + kBins1;
  r.state = r.hist2 + kBins2;
  r.tile_above = r.state + kStateWords;
  r.gt_count = r.tile_above + nt;
  r.tie_count = r.gt_count + nt;
  r.ties_before = r.tie_count + nt;
  r.out_off = r.ties_before + nt;
  r.cand = r.out_off + nt;
  return r;
}

__device__ __forceinline__ uint32_t key_of(float v) { return __float_as_uint(v) & 0x7FFFFFFFu; }

// Block-wide exclusive scan of one value per thread (kThreads threads).
// Returns the exclusive prefix; *total receives the block sum.
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* total) {
  __shared__ uint32_t warp_sums[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(kFullMask, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  uint32_t warp_prefix = 0, sum = 0;
#pragma unroll
  for (int w = 0; w < kThreads / 32; ++w) {
    const uint32_t s = warp_sums[w];
    if (w < warp) warp_prefix += s;
    sum += s;
  }
  __syncthreads();
  *total = sum;
  return warp_prefix + x - v;
}

// ---------------------------------------------------------------------------
// 1. p = fl(fl(eta g) + e) into e; h = fl(fl(eta g) + p) (fixed up at the kept
// entries in stage 9); histogram of the top key digit.
// ---------------------------------------------------------------------------
template <bool KEEP_H>
__global__ void __launch_bounds__(kThreads) topk_form_kernel(const CompressArgs a, void* scratch) {
  __shared__ uint32_t hist[kBins0];
  for (int i = threadIdx.x; i < kBins0; i += kThreads) hist[i] = 0;
  __syncthreads();
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  const float* g = a.g + (int64_t)row * a.g_stride;
  float* e = a.e + (int64_t)worker * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)worker * a.ld : nullptr;
  const int64_t tile0 = (int64_t)blockIdx.x * kTile;
#pragma unroll
  for (int i = 0; i < kRows; ++i) {
    const int64_t j = tile0 + 4 * ((int64_t)i * kThreads + threadIdx.x);
    if (j + 3 < a.d) {
      const float4 gv = __ldcs(reinterpret_cast<const float4*>(g + j));
      const float4 ev = __ldcs(reinterpret_cast<const float4*>(e + j));
      const float gq[4] = {gv.x, gv.y, gv.z, gv.w};
      const float eq[4] = {ev.x, ev.y, ev.z, ev.w};
      float pv[4], hv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float s = __fmul_rn(a.lr, gq[q]);
        pv[q] = __fadd_rn(s, eq[q]);
        hv[q] = __fadd_rn(s, pv[q]);
        atomicAdd(&hist[key_of(pv[q]) >> 20], 1u);
      }
      __stcs(reinterpret_cast<float4*>(e + j), make_float4(pv[0], pv[1], pv[2], pv[3]));
      if constexpr (KEEP_H) __stcs(reinterpret_cast<float4*>(h + j), make_float4(hv[0], hv[1], hv[2], hv[3]));
    } else {
      for (int64_t jj = j; jj < a.d && jj < j + 4; ++jj) {
        const float s = __fmul_rn(a.lr, g[jj]);
        const float pv = __fadd_rn(s, e[jj]);
        e[jj] = pv;
        if constexpr (KEEP_H) h[jj] = __fadd_rn(s, pv);
        atomicAdd(&hist[key_of(pv) >> 20], 1u);
      }
    }
  }
  __syncthreads();
  RowScratch rs = row_scratch(scratch, a.d, row);
  for (int i = threadIdx.x; i < kBins0; i += kThreads)
    if (hist[i]) atomicAdd(&rs.hist0[i], hist[i]);
}

// ---------------------------------------------------------------------------
// Digit selection: in a histogram of `bins` counts, find the digit b with
// count(> b) < k_rem <= count(>= b); store b and k_rem - count(> b); zero the
// histogram.  One block of 1024 threads per worker row.
// ---------------------------------------------------------------------------
__device__ void select_digit(uint32_t* hist, int bins, uint32_t k_rem, uint32_t* out_digit,
                             uint32_t* out_krem) {
  __shared__ uint32_t warp_sums[32];
  const int per = bins / 1024;  // 1 or 2 bins per thread, taken in descending digit order
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t cnt[2] = {0, 0};
  uint32_t local = 0;
  for (int q = 0; q < per; ++q) {
    const int pos = threadIdx.x * per + q;  // position in descending order
    cnt[q] = hist[bins - 1 - pos];
    local += cnt[q];
  }
  uint32_t x = local;
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(kFullMask, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  uint32_t before = 0;
  for (int w = 0; w < warp; ++w) before += warp_sums[w];
  uint32_t cum = before + x - local;  // count of digits above this thread's first
  for (int q = 0; q < per; ++q) {
    const int pos = threadIdx.x * per + q;
    if (cum < k_rem && k_rem <= cum + cnt[q]) {
      *out_digit = (uint32_t)(bins - 1 - pos);
      *out_krem = k_rem - cum;
    }
    cum += cnt[q];
  }
  __syncthreads();
  for (int q = 0; q < per; ++q) hist[bins - 1 - (threadIdx.x * per + q)] = 0;
}

__global__ void __launch_bounds__(1024) topk_select0_kernel(int64_t d, int64_t k, void* scratch) {
  RowScratch rs = row_scratch(scratch, d, blockIdx.y);
  select_digit(rs.hist0, kBins0, (uint32_t)k, &rs.state[ST_B0], &rs.state[ST_KREM0]);
}

// ---------------------------------------------------------------------------
// 3. Per tile: count digit0 > b0, append digit0 == b0 to the candidates and
// histogram their middle digit.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) topk_filter_kernel(const CompressArgs a, void* scratch) {
  __shared__ uint32_t hist[kBins1];
  __shared__ uint32_t tile_above;
  for (int i = threadIdx.x; i < kBins1; i += kThreads) hist[i] = 0;
  if (threadIdx.x == 0) tile_above = 0;
  __syncthreads();
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  const float* p = a.e + (int64_t)worker * a.ld;
  RowScratch rs = row_scratch(scratch, a.d, row);
  const uint32_t b0 = rs.state[ST_B0];
  const int lane = threadIdx.x & 31;
  const int64_t tile0 = (int64_t)blockIdx.x * kTile;
  uint32_t above = 0;
#pragma unroll
  for (int i = 0; i < kRows; ++i) {
    const int64_t j = tile0 + 4 * ((int64_t)i * kThreads + threadIdx.x);
    uint32_t keys[4] = {0, 0, 0, 0};
    int nvalid = 0;
    if (j + 3 < a.d) {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(p + j));
      keys[0] = key_of(v.x); keys[1] = key_of(v.y); keys[2] = key_of(v.z); keys[3] = key_of(v.w);
      nvalid = 4;
    } else {
      for (int q = 0; q < 4 && j + q < a.d; ++q) { keys[q] = key_of(p[j + q]); nvalid = q + 1; }
    }
    uint32_t cmask = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q < nvalid) {
        const uint32_t dg = keys[q] >> 20;
        above += (dg > b0);
        if (dg == b0) {
          cmask |= 1u << q;
          atomicAdd(&hist[(keys[q] >> 10) & 1023u], 1u);
        }
      }
    }
    // warp-aggregated append of the candidates
    const uint32_t n = __popc(cmask);
    uint32_t incl = n;
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(kFullMask, incl, off);
      if (lane >= off) incl += y;
    }
    const uint32_t wtotal = __shfl_sync(kFullMask, incl, 31);
    uint32_t wbase = 0;
    if (lane == 31 && wtotal) wbase = atomicAdd(&rs.state[ST_CAND], wtotal);
    wbase = __shfl_sync(kFullMask, wbase, 31);
    uint32_t pos = wbase + incl - n;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (cmask & (1u << q)) rs.cand[pos++] = (uint32_t)(j + q);
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) above += __shfl_xor_sync(kFullMask, above, off);
  if (lane == 0 && above) atomicAdd(&tile_above, above);
  __syncthreads();
  for (int i = threadIdx.x; i < kBins1; i += kThreads)
    if (hist[i]) atomicAdd(&rs.hist1[i], hist[i]);
  if (threadIdx.x == 0) rs.tile_above[blockIdx.x] = tile_above;
}

__global__ void __launch_bounds__(1024) topk_select1_kernel(int64_t d, void* scratch) {
  RowScratch rs = row_scratch(scratch, d, blockIdx.y);
  select_digit(rs.hist1, kBins1, rs.state[ST_KREM0], &rs.state[ST_B1], &rs.state[ST_KREM1]);
}

// 5. histogram of the low digit over candidates whose middle digit is b1.
__global__ void __launch_bounds__(kThreads) topk_cand_hist_kernel(const CompressArgs a, void* scratch) {
  __shared__ uint32_t hist[kBins2];
  for (int i = threadIdx.x; i < kBins2; i += kThreads) hist[i] = 0;
  __syncthreads();
  const int row = blockIdx.y;
  const float* p = a.e + (int64_t)(a.worker0 + row) * a.ld;
  RowScratch rs = row_scratch(scratch, a.d, row);
  const uint32_t ncand = rs.state[ST_CAND], b1 = rs.state[ST_B1];
  for (uint32_t c = blockIdx.x * kThreads + threadIdx.x; c < ncand; c += gridDim.x * kThreads) {
    const uint32_t key = key_of(p[rs.cand[c]]);
    if (((key >> 10) & 1023u) == b1) atomicAdd(&hist[key & 1023u], 1u);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kBins2; i += kThreads)
    if (hist[i]) atomicAdd(&rs.hist2[i], hist[i]);
}

__global__ void __launch_bounds__(1024) topk_select2_kernel(int64_t d, void* scratch) {
  RowScratch rs = row_scratch(scratch, d, blockIdx.y);
  __shared__ uint32_t b2;
  select_digit(rs.hist2, kBins2, rs.state[ST_KREM1], &b2, &rs.state[ST_NEED]);
  __syncthreads();
  if (threadIdx.x == 0) rs.state[ST_T] = (rs.state[ST_B0] << 20) | (rs.state[ST_B1] << 10) | b2;
}

// 7. per-tile counts of candidates above the threshold and equal to it.
__global__ void __launch_bounds__(kThreads) topk_cand_count_kernel(const CompressArgs a, void* scratch) {
  const int row = blockIdx.y;
  const float* p = a.e + (int64_t)(a.worker0 + row) * a.ld;
  RowScratch rs = row_scratch(scratch, a.d, row);
  const uint32_t ncand = rs.state[ST_CAND], T = rs.state[ST_T];
  for (uint32_t c = blockIdx.x * kThreads + threadIdx.x; c < ncand; c += gridDim.x * kThreads) {
    const uint32_t j = rs.cand[c];
    const uint32_t key = key_of(p[j]);
    if (key > T) atomicAdd(&rs.gt_count[j / kTile], 1u);
    else if (key == T) atomicAdd(&rs.tie_count[j / kTile], 1u);
  }
}

// 8. tile offsets: ties before each tile, kept records before each tile.
__global__ void __launch_bounds__(kThreads) topk_offsets_kernel(int64_t d, void* scratch) {
  RowScratch rs = row_scratch(scratch, d, blockIdx.y);
  const int64_t nt = tiles_of(d);
  const uint32_t need = rs.state[ST_NEED];
  uint32_t ties_run = 0, out_run = 0;
  for (int64_t t0 = 0; t0 < nt; t0 += kThreads) {
    const int64_t t = t0 + threadIdx.x;
    const uint32_t tie = (t < nt) ? rs.tie_count[t] : 0u;
    uint32_t tie_total;
    const uint32_t tie_before = ties_run + block_exclusive_scan(tie, &tie_total);
    uint32_t taken = 0;
    if (tie_before < need) taken = min(tie, need - tie_before);
    const uint32_t sel = (t < nt) ? rs.tile_above[t] + rs.gt_count[t] + taken : 0u;
    uint32_t sel_total;
    const uint32_t off = out_run + block_exclusive_scan(sel, &sel_total);
    if (t < nt) {
      rs.ties_before[t] = tie_before;
      rs.out_off[t] = off;
      rs.gt_count[t] = 0;
      rs.tie_count[t] = 0;
    }
    ties_run += tie_total;
    out_run += sel_total;
  }
  if (threadIdx.x == 0) rs.state[ST_CAND] = 0;
}

// 9. write the kept records of each tile in index order; e = +0 there.
// Element order in a tile is row-major: row i (1024 elements) is split over
// the 8 warps, 128 elements each, 4 per lane.  Each lane counts its keys
// above T and equal to T, packed as (above | ties << 16) (a tile holds at
// most 4096 of either), a warp shuffle scan ranks the lanes and one block
// exchange of the 32 warp-row totals ranks the warps: one barrier per tile.
template <bool KEEP_H>
__global__ void __launch_bounds__(kThreads)
topk_compact_kernel(const CompressArgs a, int64_t k, void* scratch) {
  __shared__ uint32_t totals[kRows][kThreads / 32];
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  float* e = a.e + (int64_t)worker * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)worker * a.ld : nullptr;
  const float* g = a.g + (int64_t)row * a.g_stride;
  uint2* rec = reinterpret_cast<uint2*>(a.msg + (int64_t)row * a.msg_stride);
  RowScratch rs = row_scratch(scratch, a.d, row);
  const uint32_t T = rs.state[ST_T], need = rs.state[ST_NEED];
  const uint32_t tie_rank0 = rs.ties_before[blockIdx.x];
  const uint32_t out0 = rs.out_off[blockIdx.x];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t tile0 = (int64_t)blockIdx.x * kTile;
  float v[kRows][4];
  uint32_t gmask[kRows], tmask[kRows], excl[kRows];
#pragma unroll
  for (int i = 0; i < kRows; ++i) {
    const int64_t j = tile0 + 4 * ((int64_t)i * kThreads + threadIdx.x);
    int nvalid = 0;
    if (j + 3 < a.d) {
      const float4 x = __ldcs(reinterpret_cast<const float4*>(e + j));
      v[i][0] = x.x; v[i][1] = x.y; v[i][2] = x.z; v[i][3] = x.w;
      nvalid = 4;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        v[i][q] = (j + q < a.d) ? e[j + q] : 0.f;
        if (j + q < a.d) nvalid = q + 1;
      }
    }
    gmask[i] = 0;
    tmask[i] = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q < nvalid) {
        const uint32_t key = key_of(v[i][q]);
        if (key > T) gmask[i] |= 1u << q;
        else if (key == T) tmask[i] |= 1u << q;
      }
    }
    const uint32_t packed = (uint32_t)__popc(gmask[i]) | ((uint32_t)__popc(tmask[i]) << 16);
    uint32_t incl = packed;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(kFullMask, incl, off);
      if (lane >= off) incl += y;
    }
    excl[i] = incl - packed;
    if (lane == 31) totals[i][warp] = incl;
  }
  __syncthreads();
  uint32_t before = 0;  // packed counts of the tile's earlier warp-rows
#pragma unroll
  for (int i = 0; i < kRows; ++i) {
    uint32_t row_before = 0, row_total = 0;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) {
      const uint32_t t = totals[i][w];
      if (w < warp) row_before += t;
      row_total += t;
    }
    const uint32_t pre = before + row_before + excl[i];
    before += row_total;
    if ((gmask[i] | tmask[i]) == 0) continue;
    uint32_t R = tie_rank0 + (pre >> 16);  // global rank of this lane's first tie
    const uint32_t sel_ties_before = min(R, need) - min(tie_rank0, need);
    uint32_t pos = out0 + (pre & 0xFFFFu) + sel_ties_before;
    const int64_t j = tile0 + 4 * ((int64_t)i * kThreads + threadIdx.x);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      bool take = (gmask[i] >> q) & 1u;
      if ((tmask[i] >> q) & 1u) {
        take = R < need;
        ++R;
      }
      if (take && pos < k) {  // pos < k always holds; the guard keeps writes in the message
        rec[pos++] = make_uint2((uint32_t)(j + q), __float_as_uint(v[i][q]));
        e[j + q] = __fsub_rn(v[i][q], v[i][q]);
        if constexpr (KEEP_H) h[j + q] = __fadd_rn(__fmul_rn(a.lr, g[j + q]), e[j + q]);
      }
    }
  }
}

}  // namespace

size_t topk_scratch_bytes(int64_t d, int32_t nworkers) {
  return (size_t)row_words(d) * 4u * (size_t)nworkers;
}

cudaError_t launch_topk_compress(const CompressArgs& a, int64_t k, bool keep_h, void* scratch,
                                 cudaStream_t stream, uint64_t* launches) {
  const unsigned rows = (unsigned)a.nworkers;
  const dim3 tiles((unsigned)tiles_of(a.d), rows);
  const dim3 one(1, rows);
  // candidate-list kernels: a fixed grid that strides over the device-side count
  const dim3 cgrid((unsigned)((tiles_of(a.d) + 3) / 4 < 1184 ? (tiles_of(a.d) + 3) / 4 : 1184), rows);
  if (keep_h) topk_form_kernel<true><<<tiles, kThreads, 0, stream>>>(a, scratch);
  else topk_form_kernel<false><<<tiles, kThreads, 0, stream>>>(a, scratch);
  topk_select0_kernel<<<one, 1024, 0, stream>>>(a.d, k, scratch);
  topk_filter_kernel<<<tiles, kThreads, 0, stream>>>(a, scratch);
  topk_select1_kernel<<<one, 1024, 0, stream>>>(a.d, scratch);
  topk_cand_hist_kernel<<<cgrid, kThreads, 0, stream>>>(a, scratch);
  topk_select2_kernel<<<one, 1024, 0, stream>>>(a.d, scratch);
  topk_cand_count_kernel<<<cgrid, kThreads, 0, stream>>>(a, scratch);
  topk_offsets_kernel<<<one, kThreads, 0, stream>>>(a.d, scratch);
  if (keep_h) topk_compact_kernel<true><<<tiles, kThreads, 0, stream>>>(a, k, scratch);
  else topk_compact_kernel<false><<<tiles, kThreads, 0, stream>>>(a, k, scratch);
  *launches += 9;
  return cudaGetLastError();
}

}  // namespace dq
