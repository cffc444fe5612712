/*
 * dqgan.h -- C-ABI of the GB300 (sm_103a) DQGAN hot path.
 *
 * One iteration of Algorithm 2 (DQGAN) of "A Distributed Training Algorithm
 * of Generative Adversarial Networks with Quantized Gradients" (Chen, Yang,
 * Shen, Pang; arXiv 2010.13359) for M workers that live as separate buffers
 * on ONE GPU:
 *
 *   worker m (Algorithm 2, worker part):
 *     w_{t-1/2} = w_{t-1} - [eta F(w_{t-3/2}) + e_{t-1}]       lookahead
 *     p_t       = eta F(w_{t-1/2}; xi_t) + e_{t-1}               error feedback
 *     p_hat_t   = Q(p_t), packed into a message                  compression
 *     e_t       = p_t - p_hat_t                                  residual
 *   server (Algorithm 2, server part):
 *     q_hat_t = (1/M) sum_m p_hat_t^(m);   w_t = w_{t-1} - q_hat_t
 *
 * Q is a delta-approximate compressor (Definition 1, Section 3.1): the scaled
 * sign of Section 2.4 (one l1 scale per bucket), top-k (Theorem 1), the b-bit
 * stochastic quantiser of Hou et al. with an l_inf scale per bucket (Section
 * 2.4, proof of Theorem 2), the same quantiser with QSGD's l2 scale (Eq.
 * (qsgd)), or the identity.  The caller supplies
 * the stochastic gradients F(.; xi) -- the GAN forward/backward pass is not
 * part of this library.
 *
 * Conventions for every call:
 *   - Every call returns a status (DQGAN_OK or a negative DQGAN_ERR_*) and
 *     never aborts or exits.  On error, dqgan_last_error() describes it.
 *   - Device pointers are CUDA device (or managed) addresses on the device
 *     that was current when the handle was created; they must be non-NULL
 *     and 16-byte aligned unless stated otherwise.
 *   - Work is enqueued asynchronously on the handle's stream (the
 *     cuda_stream of the config).  Asynchronous CUDA errors surface at
 *     dqgan_synchronize() (or at any later call that checks).
 *   - The library owns the residuals e, the lookahead offsets h, its scratch
 *     space and the step counter t.  The caller owns gradients, messages and
 *     parameters.
 *   - Arithmetic is IEEE binary32 with one rounding per operation (no fused
 *     multiply-add), so compressed messages and residuals are reproducible
 *     bit for bit from identical state.
 *   - A handle may be used from one host thread at a time.
 */
#ifndef DQGAN_H_
#define DQGAN_H_

#include <stdint.h>

#if defined(__GNUC__)
#define DQGAN_API __attribute__((visibility("default")))
#else
#define DQGAN_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define DQGAN_OK 0
#define DQGAN_ERR_INVALID_ARG (-1) /* bad config, index, size, NULL or misaligned pointer */
#define DQGAN_ERR_OOM (-2)         /* device allocation failed */
#define DQGAN_ERR_CUDA (-3)        /* a CUDA runtime call or kernel launch failed */
#define DQGAN_ERR_UNSUPPORTED (-4) /* valid request this build does not provide */
#define DQGAN_ERR_TIMEOUT (-5)     /* a bounded device-side wait gave up */
#define DQGAN_ERR_BOUNDS (-6)      /* checked build only: an index check skipped an out-of-range access */

/* Compressors Q (Section 2.4, Section 3.2). */
#define DQGAN_SIGN 0     /* scaled sign, s_b = ||p_b||_1 / n_b per bucket */
#define DQGAN_TOPK 1     /* k entries of largest |p_j|, ties to the lower index */
#define DQGAN_SQUANT 2   /* b-bit stochastic quantiser, s_b = ||p_b||_inf */
#define DQGAN_IDENTITY 3 /* no compression (uncompressed distributed OMD) */
#define DQGAN_QSGD 4     /* b-bit stochastic quantiser, s_b = ||p_b||_2 (Eq. (qsgd)) */

/* Config flags. */
#define DQGAN_KEEP_LOOKAHEAD 1u /* keep h = eta F + e per worker for the lookahead */

/*
 * Problem description.  56 bytes, no implicit padding.
 *   d           parameters in the flat vector w = [theta, phi] (Section 2.1);
 *               1 <= d <= 2^32 - 1.
 *   k           top-k only: entries kept per worker, 1 <= k <= d.
 *   lr          step size eta of Algorithm 2, finite.
 *   M           workers, 1 <= M <= 4096.
 *   compressor  DQGAN_SIGN / TOPK / SQUANT / IDENTITY / QSGD.
 *   bucket      sign, squant, qsgd: elements per scale, a power of two in
 *               [32, 4096]; the last bucket may be partial.  Ignored otherwise.
 *   bits        squant, qsgd: bits per code b in {2, 4, 8}.
 *   flags       0 or DQGAN_KEEP_LOOKAHEAD.
 *   seed        64-bit key of the Philox4x32-10 draws of the squant rounding.
 *   cuda_stream the cudaStream_t all work is enqueued on (NULL: legacy stream).
 */
typedef struct dqgan_config {
  int64_t d;
  int64_t k;
  float lr;
  int32_t M;
  int32_t compressor;
  int32_t bucket;
  int32_t bits;
  uint32_t flags;
  uint64_t seed;
  void* cuda_stream;
} dqgan_config;

typedef struct dqgan_handle dqgan_handle;

/*
 * Message layout (one per worker, `dqgan_message_bytes` bytes, a multiple of
 * 256; every section starts at a multiple of 256 bytes; nb = ceil(d/bucket)):
 *   SIGN:     [nb fp32 scales s_b][ceil(d/32) u32 words]; bit (j mod 32) of
 *             word (j div 32) is 1 iff p_j < 0 (so -0 and +0 send +s_b);
 *             Q(p)_j = bit ? -s_b : +s_b.  Bits past d are 0.
 *   SQUANT:   [nb fp32 scales s_b = max |p_j|][ceil(d*b/32) u32 words]; the
 *             b-bit code of element j sits at bit (j*b) mod 32 of word
 *             (j*b) div 32; code = K + sign(p_j) * level, K = 2^(b-1) - 1,
 *             level in [0, K]; Q(p)_j = sign * fl(s_b * fl(level / K)) and +0
 *             for level 0.  Bits past d*b are 0.
 *   QSGD:     as SQUANT with s_b = fl(sqrt(sum_j p_j^2)), the sum of squares
 *             taken in the same fixed order as the SIGN l1 sum (chunks of 4,
 *             ((x0^2+x1^2)+x2^2)+x3^2; lane l of 32 adds chunks l, l+32, ...;
 *             xor rounds 16, 8, 4, 2, 1).
 *   TOPK:     k records {u32 index j, f32 p_j}, ascending index.
 *   IDENTITY: d fp32 values p_j.
 * Bytes between sections are not written by the library.
 */

/* Host-only (no CUDA call): message size and section offsets for a config.
 * Returns DQGAN_OK or DQGAN_ERR_INVALID_ARG; any output pointer may be NULL. */
DQGAN_API int dqgan_message_layout(const dqgan_config* cfg, int64_t* scales_offset,
                         int64_t* payload_offset, int64_t* total_bytes);

/* Host-only: validate a config without touching the GPU.  DQGAN_OK or
 * DQGAN_ERR_INVALID_ARG (text in dqgan_last_error(NULL)). */
DQGAN_API int dqgan_validate_config(const dqgan_config* cfg);

/*
 * Create a handle for Algorithm 2 with the given config (the problem
 * statement dqgan_create(d, M, compressor, lr, buckets) plus the fields the
 * compressors need).  Allocates on the current device: e (M x d fp32, zero:
 * e_0 = 0), h (M x d fp32, zero, only with DQGAN_KEEP_LOOKAHEAD: F(w_{-1/2})
 * is taken as 0 so that w_{1/2} = w_0), and top-k scratch (per worker row
 * about 8 bytes per parameter for the candidates; for M <= 64 the server's
 * per-index worker masks and per-worker value rows, 8 + 4M bytes per
 * parameter, else a table of record ranges).  Sets t = 1.
 * *out receives the handle; on error *out is NULL and
 * dqgan_last_error(NULL) holds the reason, and nothing stays allocated.
 * Test hook: with the environment variable DQGAN_TEST_FAIL_ALLOC=N set, the
 * N-th device allocation this thread makes from this call on (through later
 * calls as well) fails as out of memory, once.
 */
DQGAN_API int dqgan_create(const dqgan_config* cfg, dqgan_handle** out);

/* Release everything the handle owns (synchronises its stream first).
 * NULL is accepted and is a no-op. */
DQGAN_API int dqgan_destroy(dqgan_handle* h);

/* Bytes of one worker's message (see the layout above); -1 for a NULL handle. */
DQGAN_API int64_t dqgan_message_bytes(const dqgan_handle* h);

/*
 * Worker step of Algorithm 2 for worker i at the current step t:
 *   p = fl(fl(eta * g_j) + e_j); message = pack(Q(p)); e = fl(p - Q(p));
 *   with DQGAN_KEEP_LOOKAHEAD also h = fl(fl(eta * g_j) + e_j) (new e).
 * g:       d fp32, caller-owned, read only (F(w_{t-1/2}^(i); xi_t^(i))): device
 *          memory, or pinned host memory (cudaHostAlloc / cudaMallocHost), which
 *          the kernels then read in place over the host link.
 * out_msg: device, dqgan_message_bytes() bytes, caller-owned, written.
 * Updates e^(i) (and h^(i)).  0 <= i < M.  Does not advance t.
 */
DQGAN_API int dqgan_worker_compress(dqgan_handle* h, int32_t i, const float* g, void* out_msg);

/*
 * The worker step for all M workers in one launch per kernel stage.
 * g_all:    worker m's gradient at g_all + m * g_stride (floats), device or
 *           pinned host memory as for dqgan_worker_compress; g_stride >= d and a
 *           multiple of 4.
 * msgs_all: device, worker m's message at msgs_all + m * dqgan_message_bytes().
 */
DQGAN_API int dqgan_workers_compress_all(dqgan_handle* h, const float* g_all, int64_t g_stride,
                               void* msgs_all);

/*
 * The worker step for workers first .. first + count - 1 in one launch per
 * kernel stage (the part of Algorithm 2 one rank runs when the M workers are
 * sharded over several GPUs: each rank compresses its workers into its rows
 * of the message buffer, the ranks all-gather the messages -- the push and
 * pull of Section 2.3 -- and every rank runs the same server step).
 * g:    worker first + r's gradient at g + r * g_stride (floats), device or
 *       pinned host memory; g_stride >= d and a multiple of 4.
 * msgs: device, worker first + r's message at msgs + r * dqgan_message_bytes().
 * The workers must lie in the handle's local range (all M unless
 * dqgan_set_local_workers chose fewer).
 */
DQGAN_API int dqgan_workers_compress_range(dqgan_handle* h, int32_t first, int32_t count, const float* g,
                                           int64_t g_stride, void* msgs);

/*
 * Keep the worker state (residuals e, lookahead offsets h, top-k scratch) of
 * workers first .. first + count - 1 only, instead of all M: the handle of
 * one rank when the M workers are sharded over several GPUs.  The server
 * step still averages all M messages.  Only before the first step (step
 * counter 1, else DQGAN_ERR_INVALID_ARG); replaces the state with zeroed
 * rows for the range (DQGAN_ERR_OOM if that fails; the handle then keeps its
 * old state).  Afterwards the per-worker calls accept only workers in the
 * range, dqgan_workers_compress_all is refused unless the range is all M,
 * and the checkpoint state holds the range's rows.  Synchronous.
 */
DQGAN_API int dqgan_set_local_workers(dqgan_handle* h, int32_t first, int32_t count);

/*
 * Server step of Algorithm 2, fused: decode the M messages, average them
 * (q_hat = fl(S / M), S the sum over workers in one fixed order: the M
 * decoded values, padded with +0 to the next power of two, summed pairwise
 * -- at every level x_i = fl(x_2i + x_2i+1) -- so the result does not depend
 * on the kernel that runs), and update the parameters in place,
 * w = fl(w - q_hat), or apply the server rule dqgan_set_server_optimizer
 * chose.  Then t <- t + 1.
 * msgs_all: device, M messages back to back (stride dqgan_message_bytes()).
 * params:   device, d fp32, caller-owned, read and written.
 * SIGN with bucket >= 1024 and M <= 32 has two server kernels with the same
 * results; the library picks by size.  The environment
 * variable DQGAN_SIGN_SERVER, read by dqgan_create, fixes the choice for the
 * handle: "col" (per-lane bit transpose, parameters staged by TMA; needs
 * d >= 32) or "tma" (warp bit transpose).  Any other value: by size.
 */
DQGAN_API int dqgan_server_aggregate_update(dqgan_handle* h, const void* msgs_all, float* params);

/*
 * Lookahead of Algorithm 2 for worker i: out = fl(params - h^(i)), i.e.
 * w_{t-1/2}^(i) = w_{t-1} - [eta F(w_{t-3/2}^(i)) + e_{t-1}^(i)].  Needs
 * DQGAN_KEEP_LOOKAHEAD (else DQGAN_ERR_UNSUPPORTED).  At t = 1, h = 0 and
 * the result is params.  params, out_w_half: device, d fp32.
 */
DQGAN_API int dqgan_worker_lookahead(dqgan_handle* h, int32_t i, const float* params, float* out_w_half);

/* Wait for the handle's stream.  DQGAN_ERR_CUDA if any enqueued work failed;
 * DQGAN_ERR_TIMEOUT if a bounded device-side wait of an enqueued kernel gave
 * up since the last call (the error word is then cleared, the handle and the
 * CUDA context stay usable, and the results of the steps since the last
 * successful synchronize are undefined).  In the checked build (compiled
 * with -DDQGAN_CHECK_BOUNDS, libdqgan_checked.so) also DQGAN_ERR_BOUNDS when
 * an index check in a kernel skipped an out-of-range access, or when the
 * guard zones around the top-k scratch were written; the word is cleared
 * and the guards restored the same way. */
DQGAN_API int dqgan_synchronize(dqgan_handle* h);

/*
 * Failure-detection self-test.  The paper has no counterpart: it checks the
 * library's own fault handling.  Enqueues on the handle's stream one kernel
 * that initialises an mbarrier expecting one arrival, polls it `polls` times
 * (each poll may sleep up to 0.5 us; 0 means the limit every library wait
 * uses, 2^21 polls, about a second) while nothing arrives, then sets the
 * time-out bit of the handle's error word and returns -- the same path every
 * bounded wait in the library takes when a transfer never completes.  The
 * next dqgan_synchronize returns DQGAN_ERR_TIMEOUT and clears the word; the
 * residuals, lookahead offsets and step counter are untouched.
 * Returns DQGAN_OK, DQGAN_ERR_INVALID_ARG (polls above 2^21) or DQGAN_ERR_CUDA.
 */
DQGAN_API int dqgan_selftest_wait_timeout(dqgan_handle* h, uint32_t polls);

/* Copy worker i's residual e^(i) (d fp32) to / from dst / src, which may be a
 * host or a device pointer (any alignment).  Synchronous. */
DQGAN_API int dqgan_get_residual(dqgan_handle* h, int32_t i, float* dst);
DQGAN_API int dqgan_set_residual(dqgan_handle* h, int32_t i, const float* src);

/* Same for the lookahead offset h^(i); DQGAN_ERR_UNSUPPORTED without
 * DQGAN_KEEP_LOOKAHEAD. */
DQGAN_API int dqgan_get_lookahead(dqgan_handle* h, int32_t i, float* dst);
DQGAN_API int dqgan_set_lookahead(dqgan_handle* h, int32_t i, const float* src);

/* Current step t (1-based) and its setter (t >= 1); -1 for a NULL handle. */
DQGAN_API int64_t dqgan_get_step(const dqgan_handle* h);
DQGAN_API int dqgan_set_step(dqgan_handle* h, int64_t t);

/*
 * Checkpoint / resume.  The state is a 64-byte header (magic, d, M,
 * compressor, flags, t, server rule, local worker range) followed by e
 * (one d fp32 row per local worker), with DQGAN_KEEP_LOOKAHEAD h (the same
 * rows), and under DQGAN_SERVER_OADAM m, v and
 * u_prev (d fp32 each; the rule's parameters are not stored: set the same
 * rule on the handle before loading).  host buffers of at least
 * dqgan_state_bytes() bytes.  Synchronous.  Loading checks that the header
 * matches the handle's config (else DQGAN_ERR_INVALID_ARG).
 */
DQGAN_API int64_t dqgan_state_bytes(const dqgan_handle* h);
DQGAN_API int dqgan_save_state(dqgan_handle* h, void* host_dst, int64_t bytes);
DQGAN_API int dqgan_load_state(dqgan_handle* h, const void* host_src, int64_t bytes);

/*
 * Per-layer bucketing (the layer-wise variant of Section 2.4's bucketed
 * compressors): buckets restart at every layer boundary instead of tiling
 * the flat vector w = [theta, phi].  offsets: host array of nseg + 1
 * int64, 0 = offsets[0] < offsets[1] < ... < offsets[nseg] = d, the inner
 * ones multiples of 32; segment i is [offsets[i], offsets[i+1]) and is cut
 * into buckets of `bucket` elements from its own start, its last bucket
 * partial.  Buckets are numbered in element order, so a message holds one
 * scale per bucket of every segment, then the same payload as without
 * segments; dqgan_message_bytes() reflects the new size (the config-only
 * dqgan_message_layout() describes the flat layout).  nseg = 0 with
 * offsets = NULL returns to flat buckets.  Only for DQGAN_SIGN, SQUANT and
 * QSGD (else DQGAN_ERR_UNSUPPORTED), and only before the first step
 * (step counter 1; else DQGAN_ERR_INVALID_ARG).  Synchronous; allocates
 * small device tables: nb + 1 int64 bucket starts, one u32 per 32 elements,
 * and for DQGAN_SIGN (and 8-bit codes with 16 workers) a table of each
 * bucket's message words in runs of up to 32 (8 bytes per run), from which
 * the servers take slices that never span two buckets; DQGAN_ERR_OOM if an
 * allocation fails (the handle is then left with flat buckets).  Other widths and
 * worker counts look up each 32-element word's bucket.
 */
DQGAN_API int dqgan_set_segments(dqgan_handle* h, const int64_t* offsets, int32_t nseg);

/*
 * Server update rule.  Algorithm 2's server steps w = fl(w - q_hat)
 * (DQGAN_SERVER_OMD, the default).  DQGAN_SERVER_OADAM replaces that step by
 * Optimistic Adam on the averaged update q_hat -- the optimizer family of the
 * CPOAdam systems Section 4 compares against, for which the paper prints no
 * rule; this is the rule of Daskalakis, Ilyas, Syrgkanis and Zeng, "Training
 * GANs with Optimism" (ICLR 2018).  Per parameter j, in fp32 with one
 * rounding per operation in this order (one dense pass after the server
 * kernel, which then writes q_hat to a library-owned buffer):
 *   m = b1 m + (1 - b1) q_hat;   v = b2 v + ((1 - b2) q_hat) q_hat;
 *   m_hat = m / (1 - b1^t), v_hat = v / (1 - b2^t)   (DQGAN_OADAM_BIAS_CORRECTION,
 *                                    b^t the fp32 product of t factors, t the step);
 *   u = m_hat / (sqrt(v_hat) + eps), u = 0 where m_hat = 0   (DQGAN_OADAM_ADAPTIVE),
 *   else u = m_hat;
 *   w = w - alpha (2 u - u_prev);   u_prev = u.
 * m, v and u_prev start at 0 and are library-owned (with the q_hat buffer,
 * 4 x d fp32).  With
 * b1 = 0, no DQGAN_OADAM_ADAPTIVE and alpha = 1 the update is
 * w_t = w_{t-1} - 2 q_hat_t + q_hat_{t-1}, the one-line OMD recurrence of
 * Section 2.2.  With top-k messages every parameter moves, not only the
 * indices sent.  28 bytes, no implicit padding.
 */
#define DQGAN_SERVER_OMD 0
#define DQGAN_SERVER_OADAM 1
#define DQGAN_OADAM_ADAPTIVE 1u
#define DQGAN_OADAM_BIAS_CORRECTION 2u

typedef struct dqgan_server_optimizer {
  int32_t kind;    /* DQGAN_SERVER_OMD or DQGAN_SERVER_OADAM */
  uint32_t flags;  /* DQGAN_OADAM_ADAPTIVE | DQGAN_OADAM_BIAS_CORRECTION */
  float alpha;     /* step size, finite */
  float beta1;     /* in [0, 1) */
  float beta2;     /* in [0, 1) */
  float eps;       /* >= 0, finite */
  uint32_t reserved; /* 0 */
} dqgan_server_optimizer;

/* Choose the server update rule; only before the first step (step counter
 * 1, else DQGAN_ERR_INVALID_ARG).  DQGAN_SERVER_OADAM allocates m, v, u_prev
 * and the q_hat buffer (4 x d fp32, zero; DQGAN_ERR_OOM if that fails) and
 * adds m, v, u_prev to the
 * checkpoint state; DQGAN_SERVER_OMD frees them.  DQGAN_ERR_UNSUPPORTED for
 * DQGAN_TOPK with more than 64 workers.  Synchronous. */
DQGAN_API int dqgan_set_server_optimizer(dqgan_handle* h, const dqgan_server_optimizer* opt);

/* Copy the Optimistic Adam state to dst (host or device, d fp32):
 * which = 0: m, 1: v, 2: u_prev.  DQGAN_ERR_UNSUPPORTED under DQGAN_SERVER_OMD.
 * Synchronous. */
DQGAN_API int dqgan_get_server_state(dqgan_handle* h, int32_t which, float* dst);

/* Kernels this handle has launched so far. */
DQGAN_API uint64_t dqgan_launch_count(const dqgan_handle* h);

/*
 * Top-k worker step without any device allocation.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory (code inside a host framework that owns all device memory
 * under a fixed plan, or a hot path that must not risk an allocation), which
 * rules out dqgan_create.  It computes exactly what dqgan_worker_compress
 * does for DQGAN_TOPK (same kernels, same bits):
 *   p = fl(fl(lr * g_j) + e_j); out_msg = the k records {u32 j, f32 p_j} of
 *   the k largest |p_j| (ties to the lower index), ascending index;
 *   e_j = +0 at the kept entries and p_j elsewhere.
 * g:       device, d fp32, read only.
 * e:       device, d fp32, caller-owned residual, read and written.
 * out_msg: device, at least 8*k bytes, written.
 * All three 16-byte aligned.  1 <= d <= DQGAN_NOALLOC_MAX_D (2^20); 1 <= k <= d.
 * cuda_stream: the cudaStream_t to enqueue on (NULL: legacy stream).
 * Scratch: a fixed array of DQGAN_NOALLOC_SCRATCH_BYTES (8.75 MiB) in this
 * library's device memory, reserved on every GPU that loads the library
 * until the process exits.  Nothing is allocated or freed.  The first call
 * on a device looks up the array's device address (cudaGetSymbolAddress) and
 * keeps it for the life of the process: make that first call before any
 * stream capture, and do not reset the device while the library is loaded.
 * The kernels rewrite the array's counts, prefixes and candidates in full on
 * every call, so nothing needs clearing; the one word that carries over from
 * call to call is the previous call's candidate threshold, which only
 * decides how much work the first pass saves and never changes a result.
 * All calls share the array: calls whose work overlaps on the GPU (other
 * streams, other host threads) race and give wrong results.
 * Returns DQGAN_OK, DQGAN_ERR_INVALID_ARG (sizes beyond the limit, NULL or
 * misaligned pointers) or DQGAN_ERR_CUDA; the reason is in
 * dqgan_last_error(NULL).
 */
#define DQGAN_NOALLOC_MAX_D (1 << 20)
#define DQGAN_NOALLOC_SCRATCH_BYTES (35 << 18)
DQGAN_API int dqgan_topk_compress_noalloc(const float* g, float* e, void* out_msg, int64_t d, int64_t k,
                                          float lr, void* cuda_stream);

/* Text of the last error on this handle, or of the last failed
 * create / validate / layout call in this thread when h is NULL.
 * Never NULL; valid until the next call on the same handle / thread. */
DQGAN_API const char* dqgan_last_error(const dqgan_handle* h);

#ifdef __cplusplus
}
#endif

#endif /* DQGAN_H_ */
