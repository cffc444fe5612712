// Internal declarations of the sm_103a DQGAN library (not part of the C-ABI).
//
// Every kernel computes in IEEE binary32 with explicit round-to-nearest
// intrinsics (__fmul_rn, __fadd_rn, __fsub_rn, __fdiv_rn), which the compiler
// never contracts into fused multiply-adds; the library is also built with
// -fmad=false.  That makes messages and residuals reproducible bit for bit.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <cuda.h>

#include <utility>

#include "dqgan.h"

namespace dq {

constexpr unsigned kFullMask = 0xffffffffu;
// Bits of the device error word a handle's kernels share.
constexpr uint32_t kErrTimeout = 1u;  // a bounded wait gave up
constexpr uint32_t kErrBounds = 2u;   // checked build: an index check skipped an access
// Counter word 3 of the Philox4x32-10 draws of the stochastic quantiser.
constexpr uint32_t kSquantTag = 0x51u;

struct Layout {
  int64_t off_scales;
  int64_t off_payload;
  int64_t total;
};

// Host-side layout of one message (see dqgan.h); returns false on a bad config.
bool message_layout(const dqgan_config& cfg, Layout* out);

// Records `msg` as this thread's last error (dqgan_last_error(NULL)); returns code.
int set_thread_error(int code, const char* msg);

// Arguments shared by every worker-side (compress) kernel.  One launch covers
// `nworkers` consecutive workers starting at `worker0`; launch row y (blockIdx.y)
// is worker worker0 + y.
struct CompressArgs {
  const float* g;      // gradient of row y at g + y * g_stride
  int64_t g_stride;    // floats, multiple of 4
  float* e;            // residual of worker w at e + (w - row0) * ld (library-owned)
  float* h;            // lookahead offset of worker w at h + (w - row0) * ld, or nullptr
  int64_t ld;          // floats, multiple of 64
  uint8_t* msg;        // message of row y at msg + y * msg_stride
  int64_t msg_stride;  // bytes
  int64_t d;
  int64_t nb;          // buckets: ceil(d / bucket), or the sum over layer segments
  const int64_t* bstart;  // nb + 1 bucket starts (layer segments), or nullptr: b * bucket
  int64_t off_payload; // byte offset of the payload section in a message
  float lr;
  int32_t bucket;
  int32_t bits;
  int32_t worker0;
  int32_t nworkers;
  int32_t row0;        // the worker whose residual is row 0 (the handle's first local worker)
  uint32_t seed_lo, seed_hi;
  uint32_t step;
  uint32_t* err;       // device error word (bit 0: a bounded wait timed out)
};

// Optimistic Adam on the server's averaged update (Daskalakis et al., the
// CPOAdam family): one dense pass after the server kernel has written q_hat.
struct OAdamArgs {
  const float* q;       // q_hat, d floats
  float* w;             // parameters, updated in place
  float* m;             // first moments
  float* v;             // second moments
  float* u;             // the previous step's normalised update u_prev
  int64_t d;
  float alpha;
  float beta1, one_m_beta1;  // b1 and fl(1 - b1)
  float beta2, one_m_beta2;  // b2 and fl(1 - b2)
  float eps;
  float c1, c2;         // fl(1 - b1^t), fl(1 - b2^t) at this step (bias correction)
  int32_t adaptive;     // 1: u = m_hat / (sqrt(v_hat) + eps); 0: u = m_hat
  int32_t bias_correction;
};

// Arguments of the server (decode + average + update) kernels.
struct ServerArgs {
  const uint8_t* msgs;  // message m at msgs + m * msg_stride
  int64_t msg_stride;
  float* w;             // d parameters, updated in place
  int64_t d;
  int64_t k;            // top-k records per message
  int64_t off_payload;
  int32_t M;
  int32_t bucket;
  int32_t bits;
  float inv_M;          // exact 1/M when M is a power of two
  int32_t M_pow2;       // 1 if M is a power of two (then x/M == x * inv_M exactly)
  uint32_t* err;        // device error word (bit 0: a bounded wait timed out)
  const uint32_t* word_bucket;  // bucket of each 32-element word (layer segments), or nullptr: j / bucket
  const CUtensorMap* sign_words_map;    // TMA map of the M messages' sign words, or nullptr
  const CUtensorMap* squant_words_map;  // TMA map of the M messages' code words, or nullptr
  int32_t store_q;      // 1: write q_hat itself where w - q_hat would go (w is then a q_hat buffer,
                        // dense: top-k writes +0 at the indices nobody sent)
};

// The sign server's further inputs, also the quantiser server's slice table
// (kept out of ServerArgs, which every server kernel takes as its parameter
// block).
struct SignServerExtras {
  const CUtensorMap* params_map;  // TMA map of w as rows of 32 floats, or nullptr
  int32_t path;                   // buckets >= 1024, M <= 32: 0 by size, 1 column kernel, 2 bit-transpose kernel
  const uint32_t* seg_slices;     // layer segments: per slice {first word, bucket | (rows - 1) << 27}, or nullptr
  int64_t seg_nslices;
};

// TMA tensor map over the payload words of M messages: a 2-D array of u32,
// rows = workers (M), columns = message words up to the end of the payload;
// boxes of box_words words (a multiple of 4; 32 with the 128-byte swizzle)
// x min(M, 32) workers, zero fill outside.  Returns false if the driver entry
// point or the encoding fails.
bool encode_words_map(const uint8_t* msgs, int64_t msg_stride, int64_t off_payload, int64_t payload_words,
                      int32_t M, bool swizzle128, int32_t box_words, CUtensorMap* out);
// Width in words of the sign server's word boxes with layer segments: a box
// starts at the 16-byte boundary at or before its 32-word slice.
constexpr int kSignSegBoxWords = 36;

// TMA tensor map over the parameters: floor(d / 32) rows of 32 fp32 (the
// partial last row, if any, is outside it), boxes of 32 floats x box_rows
// rows (32 for the sign server's column kernel; 32 * (32 / b) / 32 for the
// b-bit quantiser's server at b = 2, 4), 128-byte swizzle, zero fill.  Needs
// d >= 32 and w 16-byte aligned.
bool encode_params_map(float* w, int64_t d, int32_t box_rows, CUtensorMap* out);

// Launches `kern` as a programmatic dependent launch (see dq_pdl_enter in
// device_common.cuh: every kernel launched this way waits for its
// predecessor's grid before touching memory).  Returns the launch status.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              Args&&... args) {
  cudaLaunchConfig_t lc = {};
  lc.gridDim = grid;
  lc.blockDim = block;
  lc.dynamicSmemBytes = smem;
  lc.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = attr;
  lc.numAttrs = 1;
  return cudaLaunchKernelEx(&lc, kern, std::forward<Args>(args)...);
}

// Kernel launchers: each enqueues its kernels on `stream`, adds the number of
// kernels it launched to *launches and returns the launch status.
cudaError_t launch_sign_compress(const CompressArgs& a, bool keep_h, cudaStream_t stream,
                                 uint64_t* launches);
// l2_scale = false: Hou et al.'s max-abs scale; true: QSGD's l2 scale.
cudaError_t launch_squant_compress(const CompressArgs& a, bool keep_h, bool l2_scale, cudaStream_t stream,
                                   uint64_t* launches);
cudaError_t launch_identity_compress(const CompressArgs& a, bool keep_h, cudaStream_t stream,
                                     uint64_t* launches);

// Scratch of the top-k path: `rows` rows (one per local worker) and the
// server's tables for `nworkers` messages (none for 0).  A row needs no
// clearing between calls: every call rewrites its tile counts, tile prefixes
// and candidates in full.  Only the row's last state word carries over -- the
// candidate threshold of the worker's previous call (0 before the first),
// which decides how much work the first pass saves and never a result.  The
// server's per-index worker masks (up to 64 workers) must be zero when the
// scratch is created; each server call clears the masks it set.
size_t topk_scratch_bytes(int64_t d, int32_t rows, int32_t nworkers);
cudaError_t launch_topk_compress(const CompressArgs& a, int64_t k, bool keep_h, void* scratch,
                                 cudaStream_t stream, uint64_t* launches);

cudaError_t launch_sign_server(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream,
                               uint64_t* launches);
// x.params_map: encode_params_map(w, d, 32 * (32 / bits) / 32) for bits 2 and
// 4, or nullptr (then those widths take the kernel without TMA); with layer
// segments and 8-bit codes, x.seg_slices lists each bucket's code words in
// runs of up to 32 (and the words map has 36-word boxes).
cudaError_t launch_squant_server(const ServerArgs& s, const SignServerExtras& x, cudaStream_t stream,
                                 uint64_t* launches);
cudaError_t launch_identity_server(const ServerArgs& s, cudaStream_t stream, uint64_t* launches);
// scratch: topk_scratch_bytes(d, rows, M); the server's table follows the rows.
cudaError_t launch_topk_server(const ServerArgs& s, void* scratch, int32_t rows, cudaStream_t stream,
                               uint64_t* launches);

// Enqueues one kernel that polls an mbarrier nobody arrives on `polls` times
// and then sets kErrTimeout in *err (the bounded-wait path, on demand).
cudaError_t launch_wait_selftest(uint32_t polls, uint32_t* err, cudaStream_t stream, uint64_t* launches);
uint32_t wait_selftest_max_polls();

// Optimistic Adam over all d parameters from q_hat (one dense pass).
cudaError_t launch_oadam_update(const OAdamArgs& a, cudaStream_t stream, uint64_t* launches);

cudaError_t launch_lookahead(const float* w, const float* h, float* out, int64_t d,
                             cudaStream_t stream, uint64_t* launches);

}  // namespace dq
