// Worker side of Algorithm 2 (DQGAN) for the dense compressors: fused
//   p = fl(fl(eta * g) + e)            error feedback
//   Q(p) and its packed message         scaled sign / b-bit stochastic / identity
//   e = fl(p - Q(p))                    residual, written in place
//   h = fl(fl(eta * g) + e)             lookahead offset (optional)
// in one pass over g and e.
//
// Mapping: a bucket is cut into 4-element chunks; a warp reads rows of 32
// consecutive chunks (512 contiguous bytes) with 128-bit loads and keeps them
// in registers until the bucket's scale is known, so g and e are read once
// and e is written once.  The bucket's l1 sum is taken in the library's fixed
// order: lane l adds the chunk sums ((|a0|+|a1|)+|a2|)+|a3| of chunks
// l, l+32, l+64, ... in increasing order, then five xor-shuffle rounds with
// partners 16, 8, 4, 2, 1 combine the 32 lane totals.  The max-abs scale of
// the stochastic quantiser is exact in any order.
#include "device_common.cuh"

namespace dq {
namespace {

// Loads this thread's CPL chunks c = c0 + CSTRIDE i of the bucket [base, end)
// and forms p.  Elements outside the bucket read as 0 and give p = 0.  sg (if
// HOLD) receives fl(eta * g) for the lookahead.
template <int CPL, bool HOLD, int CSTRIDE = 32>
__device__ __forceinline__ void load_and_form(const CompressArgs& a, const float* g, const float* e,
                                              int64_t base, int64_t end, int c0, bool full,
                                              float (&p)[CPL][4], float (&sg)[HOLD ? CPL : 1][4]) {
  const int nchunk = a.bucket >> 2;
  if (full) {
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
      const int c = c0 + CSTRIDE * i;
      float4 gv = make_float4(0.f, 0.f, 0.f, 0.f), ev = gv;
      if (c < nchunk) {
        gv = ld_stream4(g + base + 4 * c);
        ev = ld_stream4(e + base + 4 * c);
      }
      const float gq[4] = {gv.x, gv.y, gv.z, gv.w};
      const float eq[4] = {ev.x, ev.y, ev.z, ev.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float s = __fmul_rn(a.lr, gq[q]);
        p[i][q] = (c < nchunk) ? __fadd_rn(s, eq[q]) : 0.f;
        if constexpr (HOLD) sg[i][q] = s;
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
      const int c = c0 + CSTRIDE * i;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int64_t j = base + 4 * c + q;
        const bool ok = (c < nchunk) && (j < end);
        const float gq = ok ? g[j] : 0.f;
        const float eq = ok ? e[j] : 0.f;
        const float s = __fmul_rn(a.lr, gq);
        p[i][q] = ok ? __fadd_rn(s, eq) : 0.f;
        if constexpr (HOLD) sg[i][q] = s;
      }
    }
  }
}

// Stores the new residual (and lookahead offset) of one chunk.
template <bool KEEP_H, bool HOLD, int CPL>
__device__ __forceinline__ void store_chunk(const CompressArgs& a, const float* g, float* e, float* h,
                                            int64_t j, bool full, int nvalid, const float (&en)[4],
                                            const float (&sg)[HOLD ? CPL : 1][4], int i) {
  if (full) {
    st_stream4(e + j, make_float4(en[0], en[1], en[2], en[3]));
    if constexpr (KEEP_H) {
      float s4[4];
      if constexpr (HOLD) {
#pragma unroll
        for (int q = 0; q < 4; ++q) s4[q] = sg[i][q];
      } else {
        const float4 gv = __ldg(reinterpret_cast<const float4*>(g + j));
        s4[0] = __fmul_rn(a.lr, gv.x);
        s4[1] = __fmul_rn(a.lr, gv.y);
        s4[2] = __fmul_rn(a.lr, gv.z);
        s4[3] = __fmul_rn(a.lr, gv.w);
      }
      st_stream4(h + j, make_float4(__fadd_rn(s4[0], en[0]), __fadd_rn(s4[1], en[1]),
                                    __fadd_rn(s4[2], en[2]), __fadd_rn(s4[3], en[3])));
    }
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q < nvalid) {
        e[j + q] = en[q];
        if constexpr (KEEP_H) {
          float s;
          if constexpr (HOLD) s = sg[i][q];
          else s = __fmul_rn(a.lr, g[j + q]);
          h[j + q] = __fadd_rn(s, en[q]);
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Scaled sign, s_b = ||p_b||_1 / n_b (Section 2.4; error-feedback sign
// compressor of Section 3.1).  Bit = (p < 0); Q(p) = bit ? -s_b : s_b.
//
// WPB warps share a bucket (4 for 4096, 2 for 2048, 1 up to 1024); each
// thread holds CPT chunks in registers.  Warp w of a bucket owns the chunk
// rows w*CPT .. w*CPT+CPT-1 (row r = chunks 32r .. 32r+31, contiguous in
// memory), so lane l holds the chunk sums of positions r of the l1 chain
// "lane l adds chunks l, l+32, l+64, ... in order".  With one warp the chain
// runs in registers; with several, the chunk sums go through shared memory
// and warp 0 runs the chains, so the sum is the same whatever WPB is.
// ---------------------------------------------------------------------------

template <int CPT, int WPB, bool KEEP_H, bool SEG>
__global__ void __launch_bounds__(32 * WPB * (WPB < 4 ? 4 / WPB : 1))
sign_compress_kernel(const CompressArgs a) {
  dq_pdl_enter();
  constexpr bool HOLD = KEEP_H && CPT <= 8;
  constexpr int BPC = WPB < 4 ? 4 / WPB : 1;  // buckets per CTA (CTA = max(4, WPB) warps)
  constexpr int CHAIN = 32 * CPT * WPB;
  __shared__ float chain[WPB > 1 ? BPC * CHAIN : 1];
  __shared__ float scale_sh[BPC];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int slot = warp / WPB;  // bucket within the CTA
  const int wib = warp % WPB;   // warp within the bucket
  const int64_t b = (int64_t)blockIdx.x * BPC + slot;
  const bool valid = b < a.nb;
  if (WPB == 1 && !valid) return;  // no barriers below for a single warp per bucket
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  const float* g = a.g + (int64_t)row * a.g_stride;
  float* e = a.e + (int64_t)(worker - a.row0) * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)(worker - a.row0) * a.ld : nullptr;
  uint8_t* msg = a.msg + (int64_t)row * a.msg_stride;

  // flat buckets: [b n, b n + n) clipped to d; layer buckets (SEG): the table
  const int64_t base = SEG ? (valid ? a.bstart[b] : 0) : b * a.bucket;
  const int64_t end = SEG ? (valid ? a.bstart[b + 1] : 0) : a.d;  // elements at or past `end` are not this bucket's
  const int64_t count = SEG ? end - base : (valid ? min64((int64_t)a.bucket, a.d - base) : 0);
  const bool full = (count == a.bucket);
  const int nchunk = a.bucket >> 2;
  const int row0 = wib * CPT;  // first chunk row of this warp

  float p[CPT][4];
  float sg[HOLD ? CPT : 1][4];
  if (valid) {
    load_and_form<CPT, HOLD>(a, g, e, base, end, 32 * row0 + lane, full, p, sg);
  } else {
#pragma unroll
    for (int i = 0; i < CPT; ++i)
#pragma unroll
      for (int q = 0; q < 4; ++q) p[i][q] = 0.f;
  }

  float s;
  if constexpr (WPB == 1) {
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < CPT; ++i)
      acc = __fadd_rn(acc, __fadd_rn(__fadd_rn(__fadd_rn(fabsf(p[i][0]), fabsf(p[i][1])), fabsf(p[i][2])),
                                     fabsf(p[i][3])));
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) acc = __fadd_rn(acc, __shfl_xor_sync(kFullMask, acc, off));
    s = __fdiv_rn(acc, (float)count);
  } else {
    float* ch = chain + slot * CHAIN;
#pragma unroll
    for (int i = 0; i < CPT; ++i)
      ch[(row0 + i) * 32 + lane] =
          __fadd_rn(__fadd_rn(__fadd_rn(fabsf(p[i][0]), fabsf(p[i][1])), fabsf(p[i][2])), fabsf(p[i][3]));
    __syncthreads();
    if (wib == 0) {
      float acc = 0.f;
#pragma unroll 8
      for (int r = 0; r < CPT * WPB; ++r) acc = __fadd_rn(acc, ch[r * 32 + lane]);
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) acc = __fadd_rn(acc, __shfl_xor_sync(kFullMask, acc, off));
      if (lane == 0) scale_sh[slot] = valid ? __fdiv_rn(acc, (float)count) : 0.f;
    }
    __syncthreads();
    s = scale_sh[slot];
    if (!valid) return;
  }
  if (wib == 0 && lane == 0) reinterpret_cast<float*>(msg)[b] = s;

  uint32_t* words = reinterpret_cast<uint32_t*>(msg + a.off_payload);
  const int64_t word0 = base >> 5;
  const int64_t word_end = SEG ? (end + 31) >> 5 : (a.d + 31) >> 5;  // buckets start on word boundaries
  const int words_in_bucket = a.bucket >> 5;
#pragma unroll
  for (int i = 0; i < CPT; ++i) {
    const uint32_t wv = pack_sign_row(p[i][0], p[i][1], p[i][2], p[i][3], lane);
    if ((lane & 3) == 0 && lane < 16) {
      const int wib_word = 4 * (row0 + i) + (lane >> 2);
      if (wib_word < words_in_bucket && word0 + wib_word < word_end) words[word0 + wib_word] = wv;
    }
    const int c = 32 * (row0 + i) + lane;
    if (c < nchunk) {
      const int64_t j = base + 4 * c;
      const int nvalid = (int)min64(4, end - j);
      if (nvalid > 0) {
        float en[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) en[q] = __fsub_rn(p[i][q], p[i][q] < 0.f ? -s : s);
        store_chunk<KEEP_H, HOLD, CPT>(a, g, e, h, j, full, nvalid, en, sg, i);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// b-bit stochastic quantiser of Hou et al. (Section 2.4, proof of Theorem 2),
// and QSGD's variant with the l2 scale (Eq. (qsgd)):
// s_b = max |p_j| (or ||p_b||_2), levels B_r = r / K, K = 2^(b-1) - 1; |p_j| K / s_b rounds
// up from r = floor(.) iff u < frac(.), u the 24-bit Philox4x32-10 draw of
// counter (j div 4, worker, step, 0x51) word j mod 4; code = K +- level.
// ---------------------------------------------------------------------------
// L2 = false: s_b = max |p_j| (Hou et al.); L2 = true: s_b = fl(sqrt(sum p_j^2))
// (QSGD), the sum of squares in the fixed chain order of the scaled sign.
template <int CPT, int WPB, int BITS, bool KEEP_H, bool L2, bool SEG>
__global__ void __launch_bounds__(32 * WPB * (WPB < 4 ? 4 / WPB : 1))
squant_compress_kernel(const CompressArgs a) {
  dq_pdl_enter();
  constexpr int K = (1 << (BITS - 1)) - 1;
  constexpr bool HOLD = KEEP_H && CPT <= 8;
  constexpr int BPC = WPB < 4 ? 4 / WPB : 1;  // buckets per CTA (CTA = max(4, WPB) warps)
  constexpr int CHAIN = 32 * CPT * WPB;
  // b = 2, 4 with the max-abs scale and one warp per bucket: lane l takes the
  // CPT consecutive chunks CPT l .. CPT l + CPT - 1, which hold whole code
  // words, so its codes are packed without shuffles (the max is the same in
  // any order; the l2 chain order of QSGD needs the interleaved mapping).
  constexpr bool LC = WPB == 1 && !L2 && BITS < 8 && (CPT * 4 * BITS) % 32 == 0;
  constexpr int CPW = 8 / BITS;  // chunks per code word
  __shared__ float level_value[K + 1];        // fl(r / K)
  __shared__ float warp_max[BPC * WPB];
  __shared__ float chain[(L2 && WPB > 1) ? BPC * CHAIN : 1];
  for (int r = threadIdx.x; r <= K; r += blockDim.x) level_value[r] = __fdiv_rn((float)r, (float)K);
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int slot = warp / WPB;  // bucket within the CTA
  const int wib = warp % WPB;   // warp within the bucket
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  const float* g = a.g + (int64_t)row * a.g_stride;
  float* e = a.e + (int64_t)(worker - a.row0) * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)(worker - a.row0) * a.ld : nullptr;
  uint8_t* msg = a.msg + (int64_t)row * a.msg_stride;

  // With one warp per bucket the grid is persistent: a warp takes buckets b,
  // b + stride, ... (the level table above is built once per CTA, not once
  // per four buckets) and, with layer segments, loads the next bucket's
  // bounds from the table while it quantises this one, so the data loads of
  // a bucket never wait for the table.  Otherwise one bucket per warp.
  constexpr bool PERSIST = WPB == 1;
  const int64_t bstride = (int64_t)gridDim.x * BPC;
  int64_t b = (int64_t)blockIdx.x * BPC + slot;
  int64_t next_base = 0, next_end = 0;
  if (PERSIST && SEG && b < a.nb) {
    next_base = a.bstart[b];
    next_end = a.bstart[b + 1];
  }
  for (;; b += bstride) {
  const bool valid = b < a.nb;
  if (WPB == 1 && !valid) return;

  // flat buckets: [b n, b n + n) clipped to d; layer buckets (SEG): the table
  int64_t base, end;  // elements at or past `end` are not this bucket's
  if constexpr (PERSIST && SEG) {
    base = next_base;
    end = next_end;
    if (b + bstride < a.nb) {
      next_base = a.bstart[b + bstride];
      next_end = a.bstart[b + bstride + 1];
    }
  } else {
    base = SEG ? (valid ? a.bstart[b] : 0) : b * a.bucket;
    end = SEG ? (valid ? a.bstart[b + 1] : 0) : a.d;
  }
  const int64_t count = SEG ? end - base : (valid ? min64((int64_t)a.bucket, a.d - base) : 0);
  const bool full = (count == a.bucket);
  const int nchunk = a.bucket >> 2;
  const int row0 = wib * CPT;  // first chunk row of this warp

  float p[CPT][4];
  float sg[HOLD ? CPT : 1][4];
  if (valid) {
    load_and_form<CPT, HOLD, LC ? 1 : 32>(a, g, e, base, end, LC ? CPT * lane : 32 * row0 + lane, full, p, sg);
  } else {
#pragma unroll
    for (int i = 0; i < CPT; ++i)
#pragma unroll
      for (int q = 0; q < 4; ++q) p[i][q] = 0.f;
  }

  float mx = 0.f;
  if constexpr (!L2) {
    // s = max |p| over the bucket (exact in any order)
#pragma unroll
    for (int i = 0; i < CPT; ++i)
#pragma unroll
      for (int q = 0; q < 4; ++q) mx = fmaxf(mx, fabsf(p[i][q]));
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(kFullMask, mx, off));
    if constexpr (WPB > 1) {
      if (lane == 0) warp_max[warp] = mx;
      __syncthreads();
#pragma unroll
      for (int w = 0; w < WPB; ++w) mx = fmaxf(mx, warp_max[slot * WPB + w]);
      if (!valid) return;
    }
  } else {
    // s = sqrt of the sum of squares in the chain order
    float cs[CPT];
#pragma unroll
    for (int i = 0; i < CPT; ++i)
      cs[i] = __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(p[i][0], p[i][0]), __fmul_rn(p[i][1], p[i][1])),
                                  __fmul_rn(p[i][2], p[i][2])),
                        __fmul_rn(p[i][3], p[i][3]));
    float acc = 0.f;
    if constexpr (WPB == 1) {
#pragma unroll
      for (int i = 0; i < CPT; ++i) acc = __fadd_rn(acc, cs[i]);
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) acc = __fadd_rn(acc, __shfl_xor_sync(kFullMask, acc, off));
      mx = __fsqrt_rn(acc);
    } else {
      float* ch = chain + slot * CHAIN;
#pragma unroll
      for (int i = 0; i < CPT; ++i) ch[(row0 + i) * 32 + lane] = cs[i];
      __syncthreads();
      if (wib == 0) {
#pragma unroll 8
        for (int r = 0; r < CPT * WPB; ++r) acc = __fadd_rn(acc, ch[r * 32 + lane]);
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) acc = __fadd_rn(acc, __shfl_xor_sync(kFullMask, acc, off));
        if (lane == 0) warp_max[slot * WPB] = __fsqrt_rn(acc);
      }
      __syncthreads();
      mx = warp_max[slot * WPB];
      if (!valid) return;
    }
  }
  const float s = mx;
  if (wib == 0 && lane == 0) reinterpret_cast<float*>(msg)[b] = s;
  const float inv = (s > 0.f) ? __fdiv_rn((float)K, s) : 0.f;

  uint32_t* words = reinterpret_cast<uint32_t*>(msg + a.off_payload);
  const int64_t nwords = (a.d * BITS + 31) >> 5;
  uint32_t lc_word = 0;  // LC: the code word being filled
#pragma unroll
  for (int i = 0; i < CPT; ++i) {
    const int c = LC ? CPT * lane + i : 32 * (row0 + i) + lane;
    const int64_t j = base + 4 * c;
    const int64_t cg = j >> 2;  // global chunk index = Philox counter word 0
    const int nvalid = (c < nchunk) ? (int)max64(0, min64(4, end - j)) : 0;
    const uint4 r4 = philox4x32_10(make_uint4((uint32_t)cg, (uint32_t)worker, a.step, kSquantTag),
                                   a.seed_lo, a.seed_hi);
    const uint32_t rq[4] = {r4.x, r4.y, r4.z, r4.w};
    uint32_t chunk_bits = 0;
    float en[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      int code;
      squant_element<K>(p[i][q], s, inv, rq[q], level_value, &code, &en[q]);
      if (q < nvalid) chunk_bits |= (uint32_t)code << (q * BITS);
    }
    // pack: a chunk is 4*BITS bits; 32 / (4*BITS) neighbouring chunks share a word
    uint32_t wv = chunk_bits;
    int64_t widx;
    bool writer;
    if constexpr (LC) {
      // this lane's chunks c - CPW + 1 .. c complete a word
      lc_word |= chunk_bits << (4 * BITS * (i % CPW));
      wv = lc_word;
      widx = (cg - (CPW - 1)) / CPW;
      writer = (i + 1) % CPW == 0;
      if (writer) lc_word = 0;
    } else if constexpr (BITS == 8) {
      widx = cg;
      writer = true;
    } else if constexpr (BITS == 4) {
      wv <<= 16 * (lane & 1);
      wv |= __shfl_xor_sync(kFullMask, wv, 1);
      widx = cg >> 1;
      writer = (lane & 1) == 0;
    } else {
      wv <<= 8 * (lane & 3);
      wv |= __shfl_xor_sync(kFullMask, wv, 1);
      wv |= __shfl_xor_sync(kFullMask, wv, 2);
      widx = cg >> 2;
      writer = (lane & 3) == 0;
    }
    // a code word holds 32 / BITS elements of one bucket (buckets start on
    // multiples of 32): write the words that start inside this bucket
    const int c_first = LC ? c - (CPW - 1) : c;  // the word's first chunk
    if (writer && c_first < nchunk && widx < nwords && (!SEG || widx * (32 / BITS) < end)) words[widx] = wv;
    if (nvalid > 0) store_chunk<KEEP_H, HOLD, CPT>(a, g, e, h, j, full, nvalid, en, sg, i);
  }
  if constexpr (!PERSIST) break;
  }
}

// ---------------------------------------------------------------------------
// Identity: the message is p itself and e = fl(p - p) = 0.
// ---------------------------------------------------------------------------
template <bool KEEP_H>
__global__ void __launch_bounds__(256)
identity_compress_kernel(const CompressArgs a) {
  dq_pdl_enter();
  const int row = blockIdx.y;
  const int worker = a.worker0 + row;
  const float* g = a.g + (int64_t)row * a.g_stride;
  float* e = a.e + (int64_t)(worker - a.row0) * a.ld;
  float* h = KEEP_H ? a.h + (int64_t)(worker - a.row0) * a.ld : nullptr;
  float* vals = reinterpret_cast<float*>(a.msg + (int64_t)row * a.msg_stride);
  const int64_t nchunks = (a.d + 3) >> 2;
  for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < nchunks;
       c += (int64_t)gridDim.x * blockDim.x) {
    const int64_t j = 4 * c;
    if (j + 3 < a.d) {
      const float4 gv = ld_stream4(g + j);
      const float4 ev = ld_stream4(e + j);
      const float gq[4] = {gv.x, gv.y, gv.z, gv.w};
      const float eq[4] = {ev.x, ev.y, ev.z, ev.w};
      float pv[4], en[4], hv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float s = __fmul_rn(a.lr, gq[q]);
        pv[q] = __fadd_rn(s, eq[q]);
        en[q] = __fsub_rn(pv[q], pv[q]);
        hv[q] = __fadd_rn(s, en[q]);
      }
      st_stream4(vals + j, make_float4(pv[0], pv[1], pv[2], pv[3]));
      st_stream4(e + j, make_float4(en[0], en[1], en[2], en[3]));
      if constexpr (KEEP_H) st_stream4(h + j, make_float4(hv[0], hv[1], hv[2], hv[3]));
    } else {
      for (int64_t jj = j; jj < a.d; ++jj) {
        const float s = __fmul_rn(a.lr, g[jj]);
        const float pv = __fadd_rn(s, e[jj]);
        const float en = __fsub_rn(pv, pv);
        vals[jj] = pv;
        e[jj] = en;
        if constexpr (KEEP_H) h[jj] = __fadd_rn(s, en);
      }
    }
  }
}

template <int CPT, int WPB>
cudaError_t sign_dispatch_keep(const CompressArgs& a, bool keep_h, cudaStream_t stream) {
  constexpr int BPC = WPB < 4 ? 4 / WPB : 1;
  constexpr int THREADS = 32 * WPB * BPC;
  const dim3 grid((unsigned)((a.nb + BPC - 1) / BPC), (unsigned)a.nworkers);
  const bool seg = a.bstart != nullptr;
  if (keep_h) {
    if (seg) launch_pdl(sign_compress_kernel<CPT, WPB, true, true>, grid, dim3(THREADS), 0, stream, a);
    else launch_pdl(sign_compress_kernel<CPT, WPB, true, false>, grid, dim3(THREADS), 0, stream, a);
  } else {
    if (seg) launch_pdl(sign_compress_kernel<CPT, WPB, false, true>, grid, dim3(THREADS), 0, stream, a);
    else launch_pdl(sign_compress_kernel<CPT, WPB, false, false>, grid, dim3(THREADS), 0, stream, a);
  }
  return cudaGetLastError();
}

template <int CPT, int WPB, int BITS, bool L2>
cudaError_t squant_dispatch_keep(const CompressArgs& a, bool keep_h, cudaStream_t stream) {
  constexpr int BPC = WPB < 4 ? 4 / WPB : 1;
  constexpr int THREADS = 32 * WPB * BPC;
  const bool seg = a.bstart != nullptr;
  int64_t gx = (a.nb + BPC - 1) / BPC;
  if (WPB == 1) {
    // persistent over buckets: about four waves of resident CTAs in all rows
    static int sms[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64) {
      if (sms[dev] == 0 && cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        sms[dev] = 0;
      if (sms[dev] > 0) {
        const int64_t cap = ((int64_t)sms[dev] * 4 * (2048 / THREADS) + a.nworkers - 1) / a.nworkers;
        gx = gx < cap ? gx : (cap > 0 ? cap : 1);
      }
    }
  }
  const dim3 grid((unsigned)gx, (unsigned)a.nworkers);
  if (keep_h) {
    if (seg) launch_pdl(squant_compress_kernel<CPT, WPB, BITS, true, L2, true>, grid, dim3(THREADS), 0, stream, a);
    else launch_pdl(squant_compress_kernel<CPT, WPB, BITS, true, L2, false>, grid, dim3(THREADS), 0, stream, a);
  } else {
    if (seg) launch_pdl(squant_compress_kernel<CPT, WPB, BITS, false, L2, true>, grid, dim3(THREADS), 0, stream, a);
    else launch_pdl(squant_compress_kernel<CPT, WPB, BITS, false, L2, false>, grid, dim3(THREADS), 0, stream, a);
  }
  return cudaGetLastError();
}

template <int CPT, int WPB>
cudaError_t squant_dispatch_bits(const CompressArgs& a, bool keep_h, bool l2, cudaStream_t stream) {
  switch (a.bits) {
    case 2: return l2 ? squant_dispatch_keep<CPT, WPB, 2, true>(a, keep_h, stream)
                      : squant_dispatch_keep<CPT, WPB, 2, false>(a, keep_h, stream);
    case 4: return l2 ? squant_dispatch_keep<CPT, WPB, 4, true>(a, keep_h, stream)
                      : squant_dispatch_keep<CPT, WPB, 4, false>(a, keep_h, stream);
    case 8: return l2 ? squant_dispatch_keep<CPT, WPB, 8, true>(a, keep_h, stream)
                      : squant_dispatch_keep<CPT, WPB, 8, false>(a, keep_h, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_sign_compress(const CompressArgs& a, bool keep_h, cudaStream_t stream,
                                 uint64_t* launches) {
  cudaError_t st;
  switch (a.bucket) {
    case 32: case 64: case 128: st = sign_dispatch_keep<1, 1>(a, keep_h, stream); break;
    case 256: st = sign_dispatch_keep<2, 1>(a, keep_h, stream); break;
    case 512: st = sign_dispatch_keep<4, 1>(a, keep_h, stream); break;
    case 1024: st = sign_dispatch_keep<2, 4>(a, keep_h, stream); break;
    case 2048: st = sign_dispatch_keep<2, 8>(a, keep_h, stream); break;
    case 4096: st = sign_dispatch_keep<2, 16>(a, keep_h, stream); break;
    default: return cudaErrorInvalidValue;
  }
  *launches += 1;
  return st;
}

cudaError_t launch_squant_compress(const CompressArgs& a, bool keep_h, bool l2, cudaStream_t stream,
                                   uint64_t* launches) {
  cudaError_t st;
  switch (a.bucket) {
    case 32: case 64: case 128: st = squant_dispatch_bits<1, 1>(a, keep_h, l2, stream); break;
    case 256: st = squant_dispatch_bits<2, 1>(a, keep_h, l2, stream); break;
    case 512: st = squant_dispatch_bits<4, 1>(a, keep_h, l2, stream); break;
    case 1024: st = squant_dispatch_bits<8, 1>(a, keep_h, l2, stream); break;
    case 2048: st = squant_dispatch_bits<2, 8>(a, keep_h, l2, stream); break;
    case 4096: st = squant_dispatch_bits<2, 16>(a, keep_h, l2, stream); break;
    default: return cudaErrorInvalidValue;
  }
  *launches += 1;
  return st;
}

cudaError_t launch_identity_compress(const CompressArgs& a, bool keep_h, cudaStream_t stream,
                                     uint64_t* launches) {
  const int64_t nchunks = (a.d + 3) / 4;
  const int64_t blocks = min64((nchunks + 255) / 256, 152 * 8);
  const dim3 grid((unsigned)max64(blocks, 1), (unsigned)a.nworkers);
  if (keep_h) launch_pdl(identity_compress_kernel<true>, grid, dim3(256), 0, stream, a);
  else launch_pdl(identity_compress_kernel<false>, grid, dim3(256), 0, stream, a);
  *launches += 1;
  return cudaGetLastError();
}

}  // namespace dq
