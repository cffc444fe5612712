// C-ABI of the DQGAN hot path (declared in include/dqgan.h): argument
// checking, ownership of the per-worker state (residuals e, lookahead offsets
// h, top-k scratch, step t) and dispatch to the kernels.  Every entry point
// returns a status and never aborts.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "internal.cuh"

struct dqgan_handle {
  dqgan_config cfg;
  cudaStream_t stream = nullptr;
  int device = 0;
  int64_t ld = 0;  // row stride of e and h, floats
  int64_t nb = 0;
  dq::Layout lay{};
  float* e = nullptr;
  float* h = nullptr;
  void* scratch = nullptr;
  size_t scratch_bytes = 0;
  uint32_t* err_word = nullptr;  // device error word written by bounded waits
  int64_t* seg_bstart = nullptr;     // layer segments: nb + 1 bucket starts (device)
  uint32_t* seg_wbucket = nullptr;   // layer segments: bucket of every 32-element word (device)
  uint32_t* seg_slices = nullptr;    // layer segments, sign and 8-bit codes: {first word, bucket | (rows - 1) << 27} per slice
  int64_t seg_nslices = 0;
  CUtensorMap words_map;         // TMA map of the last message buffer the server saw
  const void* words_map_msgs = nullptr;
  bool words_map_ok = false;
  CUtensorMap params_map;        // TMA map of the last parameter vector the sign / squant server saw
  const float* params_map_w = nullptr;
  bool params_map_ok = false;
  int32_t sign_path = 0;         // DQGAN_SIGN_SERVER at creation: 0 auto, 1 col, 2 tma
  dqgan_server_optimizer opt{};  // server update rule (kind DQGAN_SERVER_OMD: w = w - q_hat)
  float* opt_m = nullptr;        // Optimistic Adam: m, v, u_prev and the server's q_hat
  float* opt_v = nullptr;        // (d fp32 each, rows of one allocation)
  float* opt_u = nullptr;
  float* opt_q = nullptr;
  float pow1 = 1.f, pow2 = 1.f;  // b1^pow_t, b2^pow_t as fp32 running products
  int64_t pow_t = 0;
  int32_t row0 = 0;              // the handle holds the state of workers [row0, row0 + nlocal)
  int32_t nlocal = 0;            // (all M unless dqgan_set_local_workers chose a range)
  int64_t t = 1;
  uint64_t launches = 0;
  std::string err;
};

namespace {

// A named NVTX range over one host call (worker compress, server update,
// lookahead), so that profilers show the hot-path stages by name; without
// a profiler attached the push and pop do nothing.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

thread_local std::string tl_err;

int set_error(dqgan_handle* h, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (h) h->err = buf;
  else tl_err = buf;
  return code;
}

// Every device allocation of the library goes through dq_malloc.  For the
// tests of the out-of-memory paths, the environment variable
// DQGAN_TEST_FAIL_ALLOC=N, read by dqgan_create, makes the N-th allocation
// made by this thread from then on fail with cudaErrorMemoryAllocation
// (nothing is allocated); N counts on through later calls such as
// dqgan_set_segments, and the hook is spent once it fires.
thread_local int64_t tl_fail_countdown = 0;

void arm_allocation_failure() {
  tl_fail_countdown = 0;
  if (const char* v = std::getenv("DQGAN_TEST_FAIL_ALLOC")) {
    const long long n = std::atoll(v);
    if (n > 0) tl_fail_countdown = n;
  }
}

cudaError_t dq_malloc(void** p, size_t bytes) {
  if (tl_fail_countdown > 0 && --tl_fail_countdown == 0) {
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMalloc(p, bytes);
}

template <typename T>
cudaError_t dq_malloc(T** p, size_t bytes) {
  void* q = nullptr;
  const cudaError_t st = dq_malloc(&q, bytes);
  *p = static_cast<T*>(q);
  return st;
}

// The top-k scratch.  In the checked build (-DDQGAN_CHECK_BOUNDS) it sits
// between two guard zones of kScratchGuard bytes of kGuardByte, which
// dqgan_synchronize checks; otherwise it is a plain allocation.
#ifdef DQGAN_CHECK_BOUNDS
constexpr size_t kScratchGuard = 64u << 10;
#else
constexpr size_t kScratchGuard = 0;
#endif
constexpr unsigned char kGuardByte = 0xA5;

cudaError_t scratch_alloc(void** scratch, size_t bytes) {
  *scratch = nullptr;
  void* base = nullptr;
  cudaError_t st = dq_malloc(&base, bytes + 2 * kScratchGuard);
  if (st != cudaSuccess) return st;
  if (kScratchGuard && (st = cudaMemset(base, kGuardByte, bytes + 2 * kScratchGuard)) != cudaSuccess) {
    cudaFree(base);
    return st;
  }
  *scratch = static_cast<char*>(base) + kScratchGuard;
  return cudaSuccess;
}

void scratch_free(void* scratch) {
  if (scratch) cudaFree(static_cast<char*>(scratch) - kScratchGuard);
}

// Checked build: whether both guard zones of the scratch still hold
// kGuardByte (restoring them if not).
bool scratch_guards_intact(void* scratch, size_t bytes) {
  if (!kScratchGuard || !scratch) return true;
  std::vector<unsigned char> host(2 * kScratchGuard);
  char* lo = static_cast<char*>(scratch) - kScratchGuard;
  char* hi = static_cast<char*>(scratch) + bytes;
  if (cudaMemcpy(host.data(), lo, kScratchGuard, cudaMemcpyDeviceToHost) != cudaSuccess ||
      cudaMemcpy(host.data() + kScratchGuard, hi, kScratchGuard, cudaMemcpyDeviceToHost) != cudaSuccess)
    return false;
  for (unsigned char c : host)
    if (c != kGuardByte) {
      cudaMemset(lo, kGuardByte, kScratchGuard);
      cudaMemset(hi, kGuardByte, kScratchGuard);
      return false;
    }
  return true;
}

bool is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }
bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Returns an empty string for a valid config, else the reason.
std::string check_config(const dqgan_config* c) {
  char buf[256];
  if (!c) return "config is NULL";
  if (c->d < 1 || c->d > 0xFFFFFFFFll) {
    snprintf(buf, sizeof buf, "d = %lld outside [1, 2^32 - 1]", (long long)c->d);
    return buf;
  }
  if (c->M < 1 || c->M > 4096) {
    snprintf(buf, sizeof buf, "M = %d outside [1, 4096]", c->M);
    return buf;
  }
  if (!std::isfinite(c->lr)) return "lr is not finite";
  if (c->flags & ~DQGAN_KEEP_LOOKAHEAD) return "unknown flag bits";
  switch (c->compressor) {
    case DQGAN_SIGN:
    case DQGAN_SQUANT:
    case DQGAN_QSGD:
      if (!is_pow2(c->bucket) || c->bucket < 32 || c->bucket > 4096) {
        snprintf(buf, sizeof buf, "bucket = %d is not a power of two in [32, 4096]", c->bucket);
        return buf;
      }
      if (c->compressor != DQGAN_SIGN && c->bits != 2 && c->bits != 4 && c->bits != 8) {
        snprintf(buf, sizeof buf, "bits = %d not in {2, 4, 8}", c->bits);
        return buf;
      }
      break;
    case DQGAN_TOPK:
      if (c->k < 1 || c->k > c->d) {
        snprintf(buf, sizeof buf, "k = %lld outside [1, d]", (long long)c->k);
        return buf;
      }
      break;
    case DQGAN_IDENTITY:
      break;
    default:
      snprintf(buf, sizeof buf, "unknown compressor %d", c->compressor);
      return buf;
  }
  return "";
}

int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

int cuda_fail(dqgan_handle* h, cudaError_t e, const char* what) {
  return set_error(h, DQGAN_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

dq::CompressArgs compress_args(dqgan_handle* h, const float* g, int64_t g_stride, void* msg,
                               int64_t msg_stride, int32_t worker0, int32_t nworkers) {
  dq::CompressArgs a{};
  a.g = g;
  a.g_stride = g_stride;
  a.e = h->e;
  a.h = h->h;
  a.ld = h->ld;
  a.msg = reinterpret_cast<uint8_t*>(msg);
  a.msg_stride = msg_stride;
  a.d = h->cfg.d;
  a.nb = h->nb;
  a.bstart = h->seg_bstart;
  a.off_payload = h->lay.off_payload;
  a.lr = h->cfg.lr;
  a.bucket = h->cfg.bucket;
  a.bits = h->cfg.bits;
  a.worker0 = worker0;
  a.nworkers = nworkers;
  a.row0 = h->row0;
  a.seed_lo = (uint32_t)(h->cfg.seed & 0xFFFFFFFFu);
  a.seed_hi = (uint32_t)(h->cfg.seed >> 32);
  a.step = (uint32_t)h->t;
  a.err = h->err_word;
  return a;
}

int run_compress(dqgan_handle* h, const dq::CompressArgs& a) {
  NvtxRange range("dqgan worker compress");
  const bool keep = (h->cfg.flags & DQGAN_KEEP_LOOKAHEAD) != 0;
  cudaError_t st = cudaSuccess;
  switch (h->cfg.compressor) {
    case DQGAN_SIGN: st = dq::launch_sign_compress(a, keep, h->stream, &h->launches); break;
    case DQGAN_SQUANT: st = dq::launch_squant_compress(a, keep, false, h->stream, &h->launches); break;
    case DQGAN_QSGD: st = dq::launch_squant_compress(a, keep, true, h->stream, &h->launches); break;
    case DQGAN_IDENTITY: st = dq::launch_identity_compress(a, keep, h->stream, &h->launches); break;
    case DQGAN_TOPK: {
      // scratch rows: one per worker
      st = dq::launch_topk_compress(a, h->cfg.k, keep, h->scratch, h->stream, &h->launches);
      break;
    }
  }
  if (st != cudaSuccess) return cuda_fail(h, st, "compress launch");
  return DQGAN_OK;
}

int check_worker(dqgan_handle* h, int32_t i) {
  if (i < h->row0 || i >= h->row0 + h->nlocal)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "worker %d outside the handle's workers [%d, %d)", i, h->row0,
                     h->row0 + h->nlocal);
  return DQGAN_OK;
}

int copy_rows(dqgan_handle* h, float* base, int32_t i, void* dst, const void* src) {
  float* row = base + (int64_t)(i - h->row0) * h->ld;
  cudaError_t st;
  if (dst) st = cudaMemcpyAsync(dst, row, (size_t)h->cfg.d * 4, cudaMemcpyDefault, h->stream);
  else st = cudaMemcpyAsync(row, src, (size_t)h->cfg.d * 4, cudaMemcpyDefault, h->stream);
  if (st != cudaSuccess) return cuda_fail(h, st, "copy");
  st = cudaStreamSynchronize(h->stream);
  if (st != cudaSuccess) return cuda_fail(h, st, "copy sync");
  return DQGAN_OK;
}

// b^t as the fp32 product of t factors, t the handle's step (the bias
// corrections of Optimistic Adam); advanced one factor per step, recomputed
// after the step counter is set.
void advance_powers(dqgan_handle* h) {
  if (h->pow_t > h->t) {
    h->pow1 = h->pow2 = 1.f;
    h->pow_t = 0;
  }
  while (h->pow_t < h->t) {
    const float n1 = h->pow1 * h->opt.beta1, n2 = h->pow2 * h->opt.beta2;
    if (n1 == h->pow1 && n2 == h->pow2) {  // a fixed point (0, or a subnormal that rounds to itself)
      h->pow_t = h->t;
      break;
    }
    h->pow1 = n1;
    h->pow2 = n2;
    ++h->pow_t;
  }
}

dq::OAdamArgs oadam_args(dqgan_handle* h, float* params) {
  advance_powers(h);
  dq::OAdamArgs a{};
  a.q = h->opt_q;
  a.w = params;
  a.m = h->opt_m;
  a.v = h->opt_v;
  a.u = h->opt_u;
  a.d = h->cfg.d;
  a.alpha = h->opt.alpha;
  a.beta1 = h->opt.beta1;
  a.one_m_beta1 = 1.f - h->opt.beta1;
  a.beta2 = h->opt.beta2;
  a.one_m_beta2 = 1.f - h->opt.beta2;
  a.eps = h->opt.eps;
  a.bias_correction = (h->opt.flags & DQGAN_OADAM_BIAS_CORRECTION) ? 1 : 0;
  a.adaptive = (h->opt.flags & DQGAN_OADAM_ADAPTIVE) ? 1 : 0;
  a.c1 = a.bias_correction ? 1.f - h->pow1 : 1.f;
  a.c2 = a.bias_correction ? 1.f - h->pow2 : 1.f;
  return a;
}

int64_t opt_state_floats(const dqgan_handle* h) {
  return h->opt_m ? 3 * h->cfg.d : 0;
}

struct StateHeader {
  char magic[8];
  int64_t d;
  int64_t k;
  int64_t t;
  int32_t M;
  int32_t compressor;
  int32_t bucket;
  int32_t bits;
  uint32_t flags;
  uint32_t server_kind;  // DQGAN_SERVER_OMD, or DQGAN_SERVER_OADAM (then m, v, u_prev follow e and h)
  int32_t row0;          // the local workers [row0, row0 + nlocal) whose rows follow
  int32_t nlocal;
};
static_assert(sizeof(StateHeader) == 64, "state header layout");
constexpr int64_t kHeaderBytes = 64;

}  // namespace

namespace dq {

int set_thread_error(int code, const char* msg) { return set_error(nullptr, code, "%s", msg); }

bool message_layout(const dqgan_config& c, Layout* out) {
  if (!check_config(&c).empty()) return false;
  const int64_t nb = (c.compressor == DQGAN_SIGN || c.compressor == DQGAN_SQUANT || c.compressor == DQGAN_QSGD)
                         ? (c.d + c.bucket - 1) / c.bucket
                         : 0;
  Layout L{0, 0, 0};
  switch (c.compressor) {
    case DQGAN_SIGN:
      L.off_payload = round_up(4 * nb, 256);
      L.total = round_up(L.off_payload + 4 * ((c.d + 31) / 32), 256);
      break;
    case DQGAN_SQUANT:
    case DQGAN_QSGD:
      L.off_payload = round_up(4 * nb, 256);
      L.total = round_up(L.off_payload + 4 * ((c.d * c.bits + 31) / 32), 256);
      break;
    case DQGAN_TOPK:
      L.total = round_up(8 * c.k, 256);
      break;
    case DQGAN_IDENTITY:
      L.total = round_up(4 * c.d, 256);
      break;
  }
  *out = L;
  return true;
}

}  // namespace dq

extern "C" {

int dqgan_validate_config(const dqgan_config* cfg) {
  const std::string why = check_config(cfg);
  if (!why.empty()) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "%s", why.c_str());
  return DQGAN_OK;
}

int dqgan_message_layout(const dqgan_config* cfg, int64_t* scales_offset, int64_t* payload_offset,
                         int64_t* total_bytes) {
  const std::string why = check_config(cfg);
  if (!why.empty()) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "%s", why.c_str());
  dq::Layout L;
  dq::message_layout(*cfg, &L);
  if (scales_offset) *scales_offset = L.off_scales;
  if (payload_offset) *payload_offset = L.off_payload;
  if (total_bytes) *total_bytes = L.total;
  return DQGAN_OK;
}

int dqgan_create(const dqgan_config* cfg, dqgan_handle** out) {
  if (!out) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  const std::string why = check_config(cfg);
  if (!why.empty()) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "%s", why.c_str());
  arm_allocation_failure();
  dqgan_handle* h = new (std::nothrow) dqgan_handle();
  if (!h) return set_error(nullptr, DQGAN_ERR_OOM, "host allocation failed");
  h->cfg = *cfg;
  h->stream = reinterpret_cast<cudaStream_t>(cfg->cuda_stream);
  if (const char* path = std::getenv("DQGAN_SIGN_SERVER")) {
    if (std::strcmp(path, "col") == 0) h->sign_path = 1;
    else if (std::strcmp(path, "tma") == 0) h->sign_path = 2;
  }
  dq::message_layout(*cfg, &h->lay);
  h->nb = (cfg->d + cfg->bucket - 1) / (cfg->bucket > 0 ? cfg->bucket : 1);
  h->ld = round_up(cfg->d, 64);
  cudaError_t st = cudaGetDevice(&h->device);
  if (st != cudaSuccess) {
    delete h;
    return set_error(nullptr, DQGAN_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(st));
  }
  const size_t rows_bytes = (size_t)cfg->M * (size_t)h->ld * sizeof(float);
  auto fail_oom = [&](const char* what, cudaError_t e) {
    cudaGetLastError();
    if (h->e) cudaFree(h->e);
    if (h->h) cudaFree(h->h);
    scratch_free(h->scratch);
    if (h->err_word) cudaFree(h->err_word);
    delete h;
    return set_error(nullptr, e == cudaErrorMemoryAllocation ? DQGAN_ERR_OOM : DQGAN_ERR_CUDA,
                     "%s: %s", what, cudaGetErrorString(e));
  };
  if ((st = dq_malloc(&h->err_word, 256)) != cudaSuccess) return fail_oom("allocating the error word", st);
  if ((st = cudaMemsetAsync(h->err_word, 0, 256, h->stream)) != cudaSuccess) return fail_oom("zeroing the error word", st);
  if ((st = dq_malloc(&h->e, rows_bytes)) != cudaSuccess) return fail_oom("allocating e", st);
  if (cfg->flags & DQGAN_KEEP_LOOKAHEAD)
    if ((st = dq_malloc(&h->h, rows_bytes)) != cudaSuccess) return fail_oom("allocating h", st);
  if (cfg->compressor == DQGAN_TOPK) {
    h->scratch_bytes = dq::topk_scratch_bytes(cfg->d, cfg->M, cfg->M);
    if ((st = scratch_alloc(&h->scratch, h->scratch_bytes)) != cudaSuccess)
      return fail_oom("allocating top-k scratch", st);
  }
  if ((st = cudaMemsetAsync(h->e, 0, rows_bytes, h->stream)) != cudaSuccess) return fail_oom("zeroing e", st);
  if (h->h && (st = cudaMemsetAsync(h->h, 0, rows_bytes, h->stream)) != cudaSuccess)
    return fail_oom("zeroing h", st);
  if (h->scratch && (st = cudaMemsetAsync(h->scratch, 0, h->scratch_bytes, h->stream)) != cudaSuccess)
    return fail_oom("zeroing scratch", st);
  if ((st = cudaStreamSynchronize(h->stream)) != cudaSuccess) return fail_oom("create sync", st);
  h->t = 1;
  h->row0 = 0;
  h->nlocal = cfg->M;
  *out = h;
  return DQGAN_OK;
}

int dqgan_destroy(dqgan_handle* h) {
  if (!h) return DQGAN_OK;
  cudaStreamSynchronize(h->stream);
  if (h->e) cudaFree(h->e);
  if (h->h) cudaFree(h->h);
  scratch_free(h->scratch);
  if (h->err_word) cudaFree(h->err_word);
  if (h->seg_bstart) cudaFree(h->seg_bstart);
  if (h->seg_wbucket) cudaFree(h->seg_wbucket);
  if (h->seg_slices) cudaFree(h->seg_slices);
  if (h->opt_m) cudaFree(h->opt_m);
  const cudaError_t st = cudaGetLastError();
  delete h;
  if (st != cudaSuccess) return set_error(nullptr, DQGAN_ERR_CUDA, "destroy: %s", cudaGetErrorString(st));
  return DQGAN_OK;
}

int64_t dqgan_message_bytes(const dqgan_handle* h) { return h ? h->lay.total : -1; }

int dqgan_set_segments(dqgan_handle* h, const int64_t* offsets, int32_t nseg) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  const dqgan_config& c = h->cfg;
  if (c.compressor != DQGAN_SIGN && c.compressor != DQGAN_SQUANT && c.compressor != DQGAN_QSGD)
    return set_error(h, DQGAN_ERR_UNSUPPORTED, "layer segments apply to the bucketed compressors only");
  if (h->t != 1) return set_error(h, DQGAN_ERR_INVALID_ARG, "layer segments must be set before the first step");
  if (nseg < 0 || (nseg > 0 && !offsets) || (nseg == 0 && offsets))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "nseg = %d with offsets %s", nseg, offsets ? "set" : "NULL");
  std::vector<int64_t> starts;
  if (nseg > 0) {
    if (offsets[0] != 0 || offsets[nseg] != c.d)
      return set_error(h, DQGAN_ERR_INVALID_ARG, "offsets must run from 0 to d = %lld", (long long)c.d);
    for (int32_t i = 0; i < nseg; ++i) {
      if (offsets[i + 1] <= offsets[i])
        return set_error(h, DQGAN_ERR_INVALID_ARG, "offsets must increase (offset %d)", i + 1);
      if (i > 0 && (offsets[i] & 31))
        return set_error(h, DQGAN_ERR_INVALID_ARG, "offset %d = %lld is not a multiple of 32", i,
                         (long long)offsets[i]);
    }
    for (int32_t i = 0; i < nseg; ++i)
      for (int64_t j = offsets[i]; j < offsets[i + 1]; j += c.bucket) starts.push_back(j);
    starts.push_back(c.d);
  }
  cudaError_t st = cudaStreamSynchronize(h->stream);  // no step is in flight; tables are replaced
  if (st != cudaSuccess) return cuda_fail(h, st, "synchronize");
  if (h->seg_bstart) cudaFree(h->seg_bstart);
  if (h->seg_wbucket) cudaFree(h->seg_wbucket);
  if (h->seg_slices) cudaFree(h->seg_slices);
  h->seg_bstart = nullptr;
  h->seg_wbucket = nullptr;
  h->seg_slices = nullptr;
  h->seg_nslices = 0;
  h->words_map_msgs = nullptr;  // the payload moves with the scale section
  dq::message_layout(c, &h->lay);
  h->nb = (c.d + c.bucket - 1) / c.bucket;
  if (nseg == 0) return DQGAN_OK;
  const int64_t nb = (int64_t)starts.size() - 1;
  const int64_t nwords = (c.d + 31) / 32;
  std::vector<uint32_t> wb((size_t)nwords);
  for (int64_t b = 0; b < nb; ++b)
    for (int64_t w = starts[b] / 32; w < (starts[b + 1] + 31) / 32; ++w) wb[(size_t)w] = (uint32_t)b;
  // sign server slices: each bucket's words in runs of up to 32 (every bucket
  // starts on a word: inner segment offsets are multiples of 32)
  std::vector<uint32_t> slices;
  if (c.compressor == DQGAN_SIGN)
    for (int64_t b = 0; b < nb; ++b) {
      const int64_t we = (starts[b + 1] + 31) / 32;
      for (int64_t w = starts[b] / 32; w < we; w += 32) {
        const int64_t rows = we - w < 32 ? we - w : 32;
        slices.push_back((uint32_t)w);
        slices.push_back((uint32_t)b | (uint32_t)(rows - 1) << 27);
      }
    }
  // 8-bit codes with 16 workers (four codes per word; buckets start on
  // multiples of 32 elements): the quantiser server's slices, each bucket's
  // code words in runs of up to 32, so that no slice spans two buckets
  if ((c.compressor == DQGAN_SQUANT || c.compressor == DQGAN_QSGD) && c.bits == 8 && c.M == 16)
    for (int64_t b = 0; b < nb; ++b) {
      const int64_t we = (starts[b + 1] + 3) / 4;
      for (int64_t w = starts[b] / 4; w < we; w += 32) {
        const int64_t rows = we - w < 32 ? we - w : 32;
        slices.push_back((uint32_t)w);
        slices.push_back((uint32_t)b | (uint32_t)(rows - 1) << 27);
      }
    }
  if ((st = dq_malloc(&h->seg_bstart, starts.size() * sizeof(int64_t))) != cudaSuccess ||
      (st = dq_malloc(&h->seg_wbucket, wb.size() * sizeof(uint32_t))) != cudaSuccess ||
      (!slices.empty() && (st = dq_malloc(&h->seg_slices, slices.size() * sizeof(uint32_t))) != cudaSuccess)) {
    if (h->seg_bstart) cudaFree(h->seg_bstart);
    if (h->seg_wbucket) cudaFree(h->seg_wbucket);
    h->seg_bstart = nullptr;
    h->seg_wbucket = nullptr;
    h->seg_slices = nullptr;
    cudaGetLastError();
    return set_error(h, st == cudaErrorMemoryAllocation ? DQGAN_ERR_OOM : DQGAN_ERR_CUDA, "segment tables: %s",
                     cudaGetErrorString(st));
  }
  if ((st = cudaMemcpy(h->seg_bstart, starts.data(), starts.size() * sizeof(int64_t), cudaMemcpyHostToDevice)) !=
          cudaSuccess ||
      (st = cudaMemcpy(h->seg_wbucket, wb.data(), wb.size() * sizeof(uint32_t), cudaMemcpyHostToDevice)) !=
          cudaSuccess ||
      (h->seg_slices && (st = cudaMemcpy(h->seg_slices, slices.data(), slices.size() * sizeof(uint32_t),
                                         cudaMemcpyHostToDevice)) != cudaSuccess)) {
    cudaFree(h->seg_bstart);
    cudaFree(h->seg_wbucket);
    if (h->seg_slices) cudaFree(h->seg_slices);
    h->seg_bstart = nullptr;
    h->seg_wbucket = nullptr;
    h->seg_slices = nullptr;
    return cuda_fail(h, st, "copying the segment tables");
  }
  h->seg_nslices = (int64_t)slices.size() / 2;
  h->nb = nb;
  h->lay.off_payload = round_up(4 * nb, 256);
  const int64_t payload_words = c.compressor == DQGAN_SIGN ? nwords : (c.d * c.bits + 31) / 32;
  h->lay.total = round_up(h->lay.off_payload + 4 * payload_words, 256);
  return DQGAN_OK;
}

int dqgan_worker_compress(dqgan_handle* h, int32_t i, const float* g, void* out_msg) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (int r = check_worker(h, i)) return r;
  if (!g || !out_msg) return set_error(h, DQGAN_ERR_INVALID_ARG, "NULL gradient or message pointer");
  if (!aligned16(g) || !aligned16(out_msg))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "gradient and message must be 16-byte aligned");
  return run_compress(h, compress_args(h, g, 0, out_msg, 0, i, 1));
}

int dqgan_workers_compress_all(dqgan_handle* h, const float* g_all, int64_t g_stride, void* msgs_all) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!g_all || !msgs_all) return set_error(h, DQGAN_ERR_INVALID_ARG, "NULL gradient or message pointer");
  if (!aligned16(g_all) || !aligned16(msgs_all))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "gradients and messages must be 16-byte aligned");
  if (g_stride < h->cfg.d || (g_stride & 3))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "g_stride = %lld must be >= d and a multiple of 4",
                     (long long)g_stride);
  if (h->nlocal != h->cfg.M)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "the handle holds workers [%d, %d) only: use dqgan_workers_compress_range",
                     h->row0, h->row0 + h->nlocal);
  return run_compress(h, compress_args(h, g_all, g_stride, msgs_all, h->lay.total, 0, h->cfg.M));
}

int dqgan_workers_compress_range(dqgan_handle* h, int32_t first, int32_t count, const float* g, int64_t g_stride,
                                 void* msgs) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (count < 1 || first < h->row0 || (int64_t)first + count > (int64_t)h->row0 + h->nlocal)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "workers [%d, %d) outside the handle's workers [%d, %d)", first,
                     first + count, h->row0, h->row0 + h->nlocal);
  if (!g || !msgs) return set_error(h, DQGAN_ERR_INVALID_ARG, "NULL gradient or message pointer");
  if (!aligned16(g) || !aligned16(msgs))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "gradients and messages must be 16-byte aligned");
  if (g_stride < h->cfg.d || (g_stride & 3))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "g_stride = %lld must be >= d and a multiple of 4",
                     (long long)g_stride);
  return run_compress(h, compress_args(h, g, g_stride, msgs, h->lay.total, first, count));
}

int dqgan_set_local_workers(dqgan_handle* h, int32_t first, int32_t count) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (h->t != 1) return set_error(h, DQGAN_ERR_INVALID_ARG, "local workers must be set before the first step");
  if (count < 1 || first < 0 || (int64_t)first + count > h->cfg.M)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "workers [%d, %d) outside [0, %d)", first, first + count, h->cfg.M);
  cudaError_t st = cudaStreamSynchronize(h->stream);  // no step in flight
  if (st != cudaSuccess) return cuda_fail(h, st, "synchronize");
  const size_t rows_bytes = (size_t)count * (size_t)h->ld * sizeof(float);
  const size_t scratch_bytes =
      h->cfg.compressor == DQGAN_TOPK ? dq::topk_scratch_bytes(h->cfg.d, count, h->cfg.M) : 0;
  float *e = nullptr, *hh = nullptr;
  void* scratch = nullptr;
  auto fail = [&](const char* what, cudaError_t err) {
    cudaGetLastError();
    if (e) cudaFree(e);
    if (hh) cudaFree(hh);
    scratch_free(scratch);
    return set_error(h, err == cudaErrorMemoryAllocation ? DQGAN_ERR_OOM : DQGAN_ERR_CUDA, "%s: %s", what,
                     cudaGetErrorString(err));
  };
  if ((st = dq_malloc(&e, rows_bytes)) != cudaSuccess) return fail("allocating e", st);
  if (h->h && (st = dq_malloc(&hh, rows_bytes)) != cudaSuccess) return fail("allocating h", st);
  if (scratch_bytes && (st = scratch_alloc(&scratch, scratch_bytes)) != cudaSuccess)
    return fail("allocating top-k scratch", st);
  if ((st = cudaMemset(e, 0, rows_bytes)) != cudaSuccess || (hh && (st = cudaMemset(hh, 0, rows_bytes)) != cudaSuccess) ||
      (scratch && (st = cudaMemset(scratch, 0, scratch_bytes)) != cudaSuccess))
    return fail("zeroing the worker state", st);
  cudaFree(h->e);
  if (h->h) cudaFree(h->h);
  scratch_free(h->scratch);
  h->e = e;
  h->h = hh;
  h->scratch = scratch;
  h->scratch_bytes = scratch_bytes;
  h->row0 = first;
  h->nlocal = count;
  return DQGAN_OK;
}

int dqgan_server_aggregate_update(dqgan_handle* h, const void* msgs_all, float* params) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!msgs_all || !params) return set_error(h, DQGAN_ERR_INVALID_ARG, "NULL message or parameter pointer");
  if (!aligned16(msgs_all) || !aligned16(params))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "messages and parameters must be 16-byte aligned");
  NvtxRange range("dqgan server aggregate update");
  dq::ServerArgs s{};
  s.msgs = reinterpret_cast<const uint8_t*>(msgs_all);
  s.msg_stride = h->lay.total;
  s.w = params;
  s.d = h->cfg.d;
  s.k = h->cfg.k;
  s.off_payload = h->lay.off_payload;
  s.M = h->cfg.M;
  s.bucket = h->cfg.bucket;
  s.bits = h->cfg.bits;
  s.M_pow2 = is_pow2(h->cfg.M) ? 1 : 0;
  s.inv_M = 1.0f / (float)h->cfg.M;
  s.err = h->err_word;
  s.word_bucket = h->seg_wbucket;
  s.sign_words_map = nullptr;
  s.squant_words_map = nullptr;
  // Optimistic Adam: the server kernel writes q_hat to the handle's buffer,
  // then one dense pass updates m, v, u_prev and the parameters
  const bool oadam = h->opt_m != nullptr;
  if (oadam) {
    s.w = h->opt_q;
    s.store_q = 1;
  }
  float* const target = s.w;
  const bool flat = h->seg_wbucket == nullptr;
  // sign, buckets >= 1024, M <= 32: the TMA kernels (flat: 32-word boxes,
  // 128-byte swizzle; layer segments: 36-word boxes without swizzle)
  const bool tma_sign = h->cfg.compressor == DQGAN_SIGN && h->cfg.bucket >= 1024 && h->cfg.M <= 32 &&
                        (flat || h->seg_slices != nullptr);
  const bool tma_squant = (h->cfg.compressor == DQGAN_SQUANT || h->cfg.compressor == DQGAN_QSGD) &&
                          h->cfg.M <= 32 && h->cfg.bucket >= 32 * (32 / h->cfg.bits);
  if (tma_sign || tma_squant) {
    if (h->words_map_msgs != msgs_all) {
      const int64_t payload_words = tma_sign ? (s.d + 31) / 32 : (s.d * s.bits + 31) / 32;
      // 36-word boxes wherever slices come from a table (layer segments:
      // the sign server, and the quantiser server with 8-bit codes)
      const bool table = !flat && h->seg_slices != nullptr;
      h->words_map_ok = dq::encode_words_map(s.msgs, s.msg_stride, s.off_payload, payload_words, s.M,
                                             tma_sign && flat, table ? dq::kSignSegBoxWords : 32, &h->words_map);
      h->words_map_msgs = msgs_all;
    }
    if (h->words_map_ok) (tma_sign ? s.sign_words_map : s.squant_words_map) = &h->words_map;
  }
  dq::SignServerExtras x{};
  x.path = h->sign_path;
  x.seg_slices = h->seg_slices;
  x.seg_nslices = h->seg_nslices;
  // parameter boxes: 32 rows for the sign column kernel, one slice of
  // 32 * (32 / b) elements for the b = 2, 4 quantiser server
  const bool boxed_squant = tma_squant && s.squant_words_map && h->cfg.bits != 8;
  if (((tma_sign && s.sign_words_map) || boxed_squant) && s.d >= 32) {
    if (h->params_map_w != target) {
      const int32_t rows = boxed_squant ? 32 / h->cfg.bits : 32;
      h->params_map_ok = dq::encode_params_map(target, s.d, rows, &h->params_map);
      h->params_map_w = target;
    }
    if (h->params_map_ok) x.params_map = &h->params_map;
  }
  cudaError_t st = cudaSuccess;
  switch (h->cfg.compressor) {
    case DQGAN_SIGN: st = dq::launch_sign_server(s, x, h->stream, &h->launches); break;
    case DQGAN_SQUANT:
    case DQGAN_QSGD: st = dq::launch_squant_server(s, x, h->stream, &h->launches); break;
    case DQGAN_IDENTITY: st = dq::launch_identity_server(s, h->stream, &h->launches); break;
    case DQGAN_TOPK: st = dq::launch_topk_server(s, h->scratch, h->nlocal, h->stream, &h->launches); break;
  }
  if (st != cudaSuccess) return cuda_fail(h, st, "server launch");
  if (oadam) {
    st = dq::launch_oadam_update(oadam_args(h, params), h->stream, &h->launches);
    if (st != cudaSuccess) return cuda_fail(h, st, "optimizer launch");
  }
  h->t += 1;
  return DQGAN_OK;
}

int dqgan_worker_lookahead(dqgan_handle* h, int32_t i, const float* params, float* out_w_half) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!(h->cfg.flags & DQGAN_KEEP_LOOKAHEAD))
    return set_error(h, DQGAN_ERR_UNSUPPORTED, "lookahead needs DQGAN_KEEP_LOOKAHEAD");
  if (int r = check_worker(h, i)) return r;
  if (!params || !out_w_half) return set_error(h, DQGAN_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(params) || !aligned16(out_w_half))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
  NvtxRange range("dqgan worker lookahead");
  const cudaError_t st = dq::launch_lookahead(params, h->h + (int64_t)i * h->ld, out_w_half, h->cfg.d,
                                              h->stream, &h->launches);
  if (st != cudaSuccess) return cuda_fail(h, st, "lookahead launch");
  return DQGAN_OK;
}

int dqgan_synchronize(dqgan_handle* h) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  cudaError_t st = cudaStreamSynchronize(h->stream);
  if (st == cudaSuccess) st = cudaGetLastError();
  if (st != cudaSuccess) return cuda_fail(h, st, "synchronize");
  uint32_t word = 0;
  st = cudaMemcpy(&word, h->err_word, sizeof word, cudaMemcpyDeviceToHost);
  if (st != cudaSuccess) return cuda_fail(h, st, "reading the error word");
  if (word != 0) cudaMemset(h->err_word, 0, sizeof word);
  if (!scratch_guards_intact(h->scratch, h->scratch_bytes))
    return set_error(h, DQGAN_ERR_BOUNDS, "the guard zones around the top-k scratch were written");
  if (word & dq::kErrBounds)
    return set_error(h, DQGAN_ERR_BOUNDS, "an index check skipped an out-of-range access (error word 0x%x)", word);
  if (word != 0)
    return set_error(h, DQGAN_ERR_TIMEOUT, "a bounded device-side wait gave up (error word 0x%x)", word);
  return DQGAN_OK;
}

int dqgan_selftest_wait_timeout(dqgan_handle* h, uint32_t polls) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  const uint32_t max_polls = dq::wait_selftest_max_polls();
  if (polls > max_polls)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "polls must be at most %u", max_polls);
  if (polls == 0) polls = max_polls;
  const cudaError_t st = dq::launch_wait_selftest(polls, h->err_word, h->stream, &h->launches);
  if (st != cudaSuccess) return cuda_fail(h, st, "self-test launch");
  return DQGAN_OK;
}

int dqgan_get_residual(dqgan_handle* h, int32_t i, float* dst) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (int r = check_worker(h, i)) return r;
  if (!dst) return set_error(h, DQGAN_ERR_INVALID_ARG, "dst is NULL");
  return copy_rows(h, h->e, i, dst, nullptr);
}

int dqgan_set_residual(dqgan_handle* h, int32_t i, const float* src) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (int r = check_worker(h, i)) return r;
  if (!src) return set_error(h, DQGAN_ERR_INVALID_ARG, "src is NULL");
  return copy_rows(h, h->e, i, nullptr, src);
}

int dqgan_get_lookahead(dqgan_handle* h, int32_t i, float* dst) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!h->h) return set_error(h, DQGAN_ERR_UNSUPPORTED, "lookahead needs DQGAN_KEEP_LOOKAHEAD");
  if (int r = check_worker(h, i)) return r;
  if (!dst) return set_error(h, DQGAN_ERR_INVALID_ARG, "dst is NULL");
  return copy_rows(h, h->h, i, dst, nullptr);
}

int dqgan_set_lookahead(dqgan_handle* h, int32_t i, const float* src) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!h->h) return set_error(h, DQGAN_ERR_UNSUPPORTED, "lookahead needs DQGAN_KEEP_LOOKAHEAD");
  if (int r = check_worker(h, i)) return r;
  if (!src) return set_error(h, DQGAN_ERR_INVALID_ARG, "src is NULL");
  return copy_rows(h, h->h, i, nullptr, src);
}

int64_t dqgan_get_step(const dqgan_handle* h) { return h ? h->t : -1; }

int dqgan_set_step(dqgan_handle* h, int64_t t) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (t < 1 || t > 0xFFFFFFFFll) return set_error(h, DQGAN_ERR_INVALID_ARG, "step %lld outside [1, 2^32)", (long long)t);
  h->t = t;
  return DQGAN_OK;
}

int64_t dqgan_state_bytes(const dqgan_handle* h) {
  if (!h) return -1;
  const int64_t rows = (int64_t)h->nlocal * h->cfg.d * 4;
  return kHeaderBytes + rows * (h->h ? 2 : 1) + 4 * opt_state_floats(h);
}

int dqgan_save_state(dqgan_handle* h, void* host_dst, int64_t bytes) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!host_dst || bytes < dqgan_state_bytes(h))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "state buffer NULL or smaller than %lld bytes",
                     (long long)dqgan_state_bytes(h));
  uint8_t* dst = reinterpret_cast<uint8_t*>(host_dst);
  StateHeader hd{};
  memcpy(hd.magic, "DQGANST1", 8);
  hd.d = h->cfg.d;
  hd.k = h->cfg.k;
  hd.t = h->t;
  hd.M = h->cfg.M;
  hd.compressor = h->cfg.compressor;
  hd.bucket = h->cfg.bucket;
  hd.bits = h->cfg.bits;
  hd.flags = h->cfg.flags;
  hd.server_kind = h->opt_m ? (uint32_t)DQGAN_SERVER_OADAM : (uint32_t)DQGAN_SERVER_OMD;
  hd.row0 = h->row0;
  hd.nlocal = h->nlocal;
  memset(dst, 0, kHeaderBytes);
  memcpy(dst, &hd, sizeof hd);
  const size_t row = (size_t)h->cfg.d * 4;
  uint8_t* out = dst + kHeaderBytes;
  for (int which = 0; which < (h->h ? 2 : 1); ++which) {
    float* base = which == 0 ? h->e : h->h;
    cudaError_t st = cudaMemcpy2DAsync(out, row, base, (size_t)h->ld * 4, row, (size_t)h->nlocal,
                                       cudaMemcpyDefault, h->stream);
    if (st != cudaSuccess) return cuda_fail(h, st, "save state copy");
    out += row * (size_t)h->nlocal;
  }
  if (h->opt_m) {
    cudaError_t st = cudaMemcpy2DAsync(out, row, h->opt_m, (size_t)round_up(h->cfg.d, 64) * 4, row, 3,
                                       cudaMemcpyDefault, h->stream);  // m, v, u_prev rows
    if (st != cudaSuccess) return cuda_fail(h, st, "save state copy");
  }
  const cudaError_t st = cudaStreamSynchronize(h->stream);
  if (st != cudaSuccess) return cuda_fail(h, st, "save state sync");
  return DQGAN_OK;
}

int dqgan_load_state(dqgan_handle* h, const void* host_src, int64_t bytes) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!host_src || bytes < dqgan_state_bytes(h))
    return set_error(h, DQGAN_ERR_INVALID_ARG, "state buffer NULL or smaller than %lld bytes",
                     (long long)dqgan_state_bytes(h));
  const uint8_t* src = reinterpret_cast<const uint8_t*>(host_src);
  StateHeader hd;
  memcpy(&hd, src, sizeof hd);
  if (memcmp(hd.magic, "DQGANST1", 8) != 0 || hd.d != h->cfg.d || hd.M != h->cfg.M ||
      hd.compressor != h->cfg.compressor || hd.flags != h->cfg.flags || hd.k != h->cfg.k ||
      hd.bucket != h->cfg.bucket || hd.bits != h->cfg.bits || hd.t < 1 ||
      hd.server_kind != (h->opt_m ? (uint32_t)DQGAN_SERVER_OADAM : (uint32_t)DQGAN_SERVER_OMD) ||
      hd.row0 != h->row0 || hd.nlocal != h->nlocal)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "state header does not match this handle's config");
  const size_t row = (size_t)h->cfg.d * 4;
  const uint8_t* in = src + kHeaderBytes;
  for (int which = 0; which < (h->h ? 2 : 1); ++which) {
    float* base = which == 0 ? h->e : h->h;
    cudaError_t st = cudaMemcpy2DAsync(base, (size_t)h->ld * 4, in, row, row, (size_t)h->nlocal,
                                       cudaMemcpyDefault, h->stream);
    if (st != cudaSuccess) return cuda_fail(h, st, "load state copy");
    in += row * (size_t)h->nlocal;
  }
  if (h->opt_m) {
    cudaError_t st = cudaMemcpy2DAsync(h->opt_m, (size_t)round_up(h->cfg.d, 64) * 4, in, row, row, 3,
                                       cudaMemcpyDefault, h->stream);  // m, v, u_prev rows
    if (st != cudaSuccess) return cuda_fail(h, st, "load state copy");
  }
  const cudaError_t st = cudaStreamSynchronize(h->stream);
  if (st != cudaSuccess) return cuda_fail(h, st, "load state sync");
  h->t = hd.t;
  h->pow_t = h->t + 1;  // recompute b^t at the next server step
  return DQGAN_OK;
}

int dqgan_set_server_optimizer(dqgan_handle* h, const dqgan_server_optimizer* opt) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!opt) return set_error(h, DQGAN_ERR_INVALID_ARG, "optimizer is NULL");
  if (h->t != 1) return set_error(h, DQGAN_ERR_INVALID_ARG, "the server rule must be set before the first step");
  if (opt->kind != DQGAN_SERVER_OMD && opt->kind != DQGAN_SERVER_OADAM)
    return set_error(h, DQGAN_ERR_INVALID_ARG, "unknown server rule %d", opt->kind);
  if (opt->kind == DQGAN_SERVER_OADAM) {
    if (opt->flags & ~(DQGAN_OADAM_ADAPTIVE | DQGAN_OADAM_BIAS_CORRECTION) || opt->reserved != 0)
      return set_error(h, DQGAN_ERR_INVALID_ARG, "unknown optimizer flag bits");
    if (!std::isfinite(opt->alpha) || !std::isfinite(opt->eps) || opt->eps < 0.f)
      return set_error(h, DQGAN_ERR_INVALID_ARG, "alpha must be finite and eps finite and >= 0");
    if (!(opt->beta1 >= 0.f && opt->beta1 < 1.f) || !(opt->beta2 >= 0.f && opt->beta2 < 1.f))
      return set_error(h, DQGAN_ERR_INVALID_ARG, "beta1 and beta2 must lie in [0, 1)");
    if (h->cfg.compressor == DQGAN_TOPK && h->cfg.M > 64)
      return set_error(h, DQGAN_ERR_UNSUPPORTED, "Optimistic Adam with top-k messages takes at most 64 workers");
  }
  cudaError_t st = cudaStreamSynchronize(h->stream);  // no step in flight
  if (st != cudaSuccess) return cuda_fail(h, st, "synchronize");
  if (h->opt_m) cudaFree(h->opt_m);
  h->opt_m = h->opt_v = h->opt_u = h->opt_q = nullptr;
  h->opt = *opt;
  h->pow1 = h->pow2 = 1.f;
  h->pow_t = 0;
  if (opt->kind == DQGAN_SERVER_OMD) return DQGAN_OK;
  const int64_t ld = round_up(h->cfg.d, 64);
  if ((st = dq_malloc(&h->opt_m, (size_t)(4 * ld) * 4)) != cudaSuccess) {
    cudaGetLastError();
    h->opt_m = nullptr;
    h->opt.kind = DQGAN_SERVER_OMD;
    return set_error(h, st == cudaErrorMemoryAllocation ? DQGAN_ERR_OOM : DQGAN_ERR_CUDA,
                     "allocating the optimizer state: %s", cudaGetErrorString(st));
  }
  h->opt_v = h->opt_m + ld;
  h->opt_u = h->opt_v + ld;
  h->opt_q = h->opt_u + ld;
  if ((st = cudaMemset(h->opt_m, 0, (size_t)(4 * ld) * 4)) != cudaSuccess)
    return cuda_fail(h, st, "zeroing the optimizer state");
  return DQGAN_OK;
}

int dqgan_get_server_state(dqgan_handle* h, int32_t which, float* dst) {
  if (!h) return set_error(nullptr, DQGAN_ERR_INVALID_ARG, "handle is NULL");
  if (!h->opt_m) return set_error(h, DQGAN_ERR_UNSUPPORTED, "the server rule keeps no state");
  if (which < 0 || which > 2 || !dst) return set_error(h, DQGAN_ERR_INVALID_ARG, "which must be 0, 1 or 2 and dst set");
  const float* src = which == 0 ? h->opt_m : (which == 1 ? h->opt_v : h->opt_u);
  cudaError_t st = cudaMemcpyAsync(dst, src, (size_t)h->cfg.d * 4, cudaMemcpyDefault, h->stream);
  if (st == cudaSuccess) st = cudaStreamSynchronize(h->stream);
  if (st != cudaSuccess) return cuda_fail(h, st, "copying the optimizer state");
  return DQGAN_OK;
}

uint64_t dqgan_launch_count(const dqgan_handle* h) { return h ? h->launches : 0; }

const char* dqgan_last_error(const dqgan_handle* h) { return h ? h->err.c_str() : tl_err.c_str(); }

}  // extern "C"
