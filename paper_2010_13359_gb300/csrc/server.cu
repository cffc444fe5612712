// Server side of Algorithm 2 (DQGAN), fused into one pass per compressor:
//   decode the M messages, q_hat = fl(sum_m Q_m / M), w = fl(w - q_hat).
// and the worker lookahead w_{t-1/2} = fl(w - h).
//
// Dense compressors: one thread per 4-element chunk of w; the thread walks
// the M messages in worker order and keeps 4 fp32 accumulators.  Message
// bytes per chunk are a word (or part of one) and one scale per worker, read
// with plain coalesced loads; w is read and written once with 128-bit loads.
#include "internal.cuh"

namespace dq {
namespace {

__device__ __forceinline__ float average(float acc, const ServerArgs& s) {
  return s.M_pow2 ? __fmul_rn(acc, s.inv_M) : __fdiv_rn(acc, (float)s.M);
}

// Applies w_j = fl(w_j - acc_j / M) for the chunk at element j.
__device__ __forceinline__ void apply_chunk(const ServerArgs& s, int64_t j, const float (&acc)[4]) {
  if (j + 3 < s.d) {
    float4 wv = __ldcs(reinterpret_cast<const float4*>(s.w + j));
    wv.x = __fsub_rn(wv.x, average(acc[0], s));
    wv.y = __fsub_rn(wv.y, average(acc[1], s));
    wv.z = __fsub_rn(wv.z, average(acc[2], s));
    wv.w = __fsub_rn(wv.w, average(acc[3], s));
    __stcs(reinterpret_cast<float4*>(s.w + j), wv);
  } else {
    for (int q = 0; q < 4 && j + q < s.d; ++q) s.w[j + q] = __fsub_rn(s.w[j + q], average(acc[q], s));
  }
}

// Scaled sign: Q_m(p)_j = bit ? -s_m : s_m.
__global__ void __launch_bounds__(256) sign_server_kernel(const ServerArgs s) {
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t j = 4 * c;
  if (j >= s.d) return;
  const int64_t bkt = j / s.bucket;
  const int64_t word = j >> 5;
  const int shift = (int)(j & 31);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int m = 0; m < s.M; ++m) {
    const uint8_t* msg = s.msgs + (int64_t)m * s.msg_stride;
    const float sc = __ldg(reinterpret_cast<const float*>(msg) + bkt);
    const uint32_t bits = __ldg(reinterpret_cast<const uint32_t*>(msg + s.off_payload) + word) >> shift;
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] = __fadd_rn(acc[q], ((bits >> q) & 1u) ? -sc : sc);
  }
  apply_chunk(s, j, acc);
}

// b-bit stochastic quantiser: Q_m(p)_j = sign * fl(s_m * fl(level / K)), +0 at level 0.
template <int BITS>
__global__ void __launch_bounds__(256) squant_server_kernel(const ServerArgs s) {
  constexpr int K = (1 << (BITS - 1)) - 1;
  constexpr uint32_t MASK = (1u << BITS) - 1u;
  __shared__ float level_value[K + 1];
  for (int r = threadIdx.x; r <= K; r += blockDim.x) level_value[r] = __fdiv_rn((float)r, (float)K);
  __syncthreads();
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t j = 4 * c;
  if (j >= s.d) return;
  const int64_t bkt = j / s.bucket;
  const int64_t bitpos = j * BITS;  // a chunk's 4*BITS bits never straddle a word
  const int64_t word = bitpos >> 5;
  const int shift = (int)(bitpos & 31);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int m = 0; m < s.M; ++m) {
    const uint8_t* msg = s.msgs + (int64_t)m * s.msg_stride;
    const float sc = __ldg(reinterpret_cast<const float*>(msg) + bkt);
    const uint32_t bits = __ldg(reinterpret_cast<const uint32_t*>(msg + s.off_payload) + word) >> shift;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int level = (int)((bits >> (q * BITS)) & MASK) - K;
      float v = 0.f;
      if (level != 0) {
        const float mag = __fmul_rn(sc, level_value[level < 0 ? -level : level]);
        v = level < 0 ? -mag : mag;
      }
      acc[q] = __fadd_rn(acc[q], v);
    }
  }
  apply_chunk(s, j, acc);
}

// Identity: the messages are the p vectors themselves.
__global__ void __launch_bounds__(256) identity_server_kernel(const ServerArgs s) {
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t j = 4 * c;
  if (j >= s.d) return;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int m = 0; m < s.M; ++m) {
    const float* vals = reinterpret_cast<const float*>(s.msgs + (int64_t)m * s.msg_stride);
    if (j + 3 < s.d) {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(vals + j));
      acc[0] = __fadd_rn(acc[0], v.x);
      acc[1] = __fadd_rn(acc[1], v.y);
      acc[2] = __fadd_rn(acc[2], v.z);
      acc[3] = __fadd_rn(acc[3], v.w);
    } else {
      for (int q = 0; q < 4 && j + q < s.d; ++q) acc[q] = __fadd_rn(acc[q], vals[j + q]);
    }
  }
  apply_chunk(s, j, acc);
}

// Top-k: every worker's records are sorted by index, so whether an index
// appears in worker m's list is a binary search.  The thread holding the
// first occurrence (lowest worker) of an index sums that index's values over
// all workers in worker order and applies the update; the others do nothing.
__device__ __forceinline__ bool find_index(const uint2* rec, int64_t k, uint32_t idx, float* val) {
  int64_t lo = 0, hi = k;  // search [lo, hi)
  while (lo < hi) {
    const int64_t mid = (lo + hi) >> 1;
    const uint32_t v = __ldg(&rec[mid].x);
    if (v < idx) lo = mid + 1;
    else hi = mid;
  }
  if (lo < k) {
    const uint2 r = __ldg(&rec[lo]);
    if (r.x == idx) {
      *val = __uint_as_float(r.y);
      return true;
    }
  }
  return false;
}

__global__ void __launch_bounds__(256) topk_server_kernel(const ServerArgs s) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (tid >= (int64_t)s.M * s.k) return;
  const int m = (int)(tid / s.k);
  const int64_t r = tid - (int64_t)m * s.k;
  const uint2 mine = __ldg(reinterpret_cast<const uint2*>(s.msgs + (int64_t)m * s.msg_stride) + r);
  const uint32_t idx = mine.x;
  if (idx >= s.d) return;  // records come from the compressor and are < d; never write past w
  float v;
  for (int m2 = 0; m2 < m; ++m2) {
    const uint2* rec = reinterpret_cast<const uint2*>(s.msgs + (int64_t)m2 * s.msg_stride);
    if (find_index(rec, s.k, idx, &v)) return;  // an earlier worker owns this index
  }
  float acc = __fadd_rn(0.f, __uint_as_float(mine.y));
  for (int m2 = m + 1; m2 < s.M; ++m2) {
    const uint2* rec = reinterpret_cast<const uint2*>(s.msgs + (int64_t)m2 * s.msg_stride);
    if (find_index(rec, s.k, idx, &v)) acc = __fadd_rn(acc, v);
  }
  s.w[idx] = __fsub_rn(s.w[idx], average(acc, s));
}

__global__ void __launch_bounds__(256)
lookahead_kernel(const float* __restrict__ w, const float* __restrict__ h, float* __restrict__ out,
                 int64_t d) {
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

unsigned chunk_blocks(int64_t d, int threads) {
  const int64_t chunks = (d + 3) / 4;
  return (unsigned)((chunks + threads - 1) / threads);
}

}  // namespace

cudaError_t launch_sign_server(const ServerArgs& s, cudaStream_t stream, uint64_t* launches) {
  sign_server_kernel<<<chunk_blocks(s.d, 256), 256, 0, stream>>>(s);
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_squant_server(const ServerArgs& s, cudaStream_t stream, uint64_t* launches) {
  const unsigned blocks = chunk_blocks(s.d, 256);
  switch (s.bits) {
    case 2: squant_server_kernel<2><<<blocks, 256, 0, stream>>>(s); break;
    case 4: squant_server_kernel<4><<<blocks, 256, 0, stream>>>(s); break;
    case 8: squant_server_kernel<8><<<blocks, 256, 0, stream>>>(s); break;
    default: return cudaErrorInvalidValue;
  }
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_identity_server(const ServerArgs& s, cudaStream_t stream, uint64_t* launches) {
  identity_server_kernel<<<chunk_blocks(s.d, 256), 256, 0, stream>>>(s);
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_topk_server(const ServerArgs& s, cudaStream_t stream, uint64_t* launches) {
  const int64_t n = (int64_t)s.M * s.k;
  topk_server_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(s);
  *launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_lookahead(const float* w, const float* h, float* out, int64_t d,
                             cudaStream_t stream, uint64_t* launches) {
  lookahead_kernel<<<chunk_blocks(d, 256), 256, 0, stream>>>(w, h, out, d);
  *launches += 1;
  return cudaGetLastError();
}

}  // namespace dq
