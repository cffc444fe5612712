/*
 * DQGAN oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded CPU statement of one iteration of
 * Algorithm 2 (DQGAN) of Chen, Yang, Shen, Pang, "A Distributed Training
 * Algorithm of Generative Adversarial Networks with Quantized Gradients"
 * (arXiv 2010.13359).  Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark may load this file.  It shares no code,
 * header, table or constant with the CUDA library: every format and every
 * rule below is restated here from the paper and from the readings that the
 * design notes list where the paper is silent.
 *
 * Arithmetic: IEEE-754 binary32, round to nearest even, one rounding per
 * operation.  The file must be compiled with -ffp-contract=off (no fused
 * multiply-add) and without -ffast-math.  fp32 is the precision of the
 * paper's own implementation (Section 4, "full-precision (float32)"), and the
 * integer decisions of the method (sign bits, top-k membership, quantisation
 * codes) are taken in that precision on both sides.
 *
 * Parity pins: every function here is checked by the CPU tests against the
 * closed forms, identities and brute-force enumerations that the paper fixes
 * (Definition 1, Theorem 1, Theorem 2's moment identities, the error-feedback
 * recurrence of Appendix B, and the one-line OMD recurrence of Section 2.2).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#if defined(__FAST_MATH__)
#error "the oracle must not be compiled with -ffast-math"
#endif

enum { ORC_SIGN = 0, ORC_TOPK = 1, ORC_SQUANT = 2, ORC_IDENTITY = 3, ORC_QSGD = 4 };

/* Counter word 3 of every Philox draw made by the stochastic quantiser. */
#define ORC_TAG_SQUANT 0x51u

typedef struct orc_cfg {
  int64_t d;        /* parameters in the flat vector w = [theta, phi] */
  int64_t k;        /* top-k: entries kept per worker */
  float lr;         /* step size eta of Algorithm 2 */
  int32_t M;        /* workers */
  int32_t compressor;
  int32_t bucket;   /* sign / stochastic quantiser: elements per scale */
  int32_t bits;     /* stochastic quantiser: bits per code */
  int32_t keep_lookahead; /* 1: also produce h = eta*F + e (Algorithm 2) */
  uint64_t seed;
  int32_t nseg;     /* 0: buckets tile the flat vector; else the number of  */
                    /* layer segments, each bucketed on its own             */
  const int64_t* seg; /* nseg + 1 offsets: 0 = seg[0] < seg[1] < ... = d    */
} orc_cfg;

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As   */
/* Easy as 1, 2, 3", SC 2011): ten rounds of the 4x32 Philox S-box with the  */
/* Weyl key schedule.  Round multipliers 0xD2511F53 and 0xCD9E8D57; key      */
/* increments 0x9E3779B9 and 0xBB67AE85, applied between rounds.             */
/* ------------------------------------------------------------------------ */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t prod_a = (uint64_t)0xD2511F53u * (uint64_t)x0;
    uint64_t prod_b = (uint64_t)0xCD9E8D57u * (uint64_t)x2;
    uint32_t y0 = (uint32_t)(prod_b >> 32) ^ x1 ^ k0;
    uint32_t y1 = (uint32_t)prod_b;
    uint32_t y2 = (uint32_t)(prod_a >> 32) ^ x3 ^ k1;
    uint32_t y3 = (uint32_t)prod_a;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The uniform draw u in [0, 1) of the stochastic quantiser for element j of
 * worker i at step t: the top 24 bits of Philox output word (j mod 4) of the
 * counter (j div 4, i, t, TAG), keyed by the 64-bit seed split low/high. */
float orc_squant_uniform(uint64_t seed, int32_t worker, int64_t step, int64_t j) {
  uint32_t ctr[4] = {(uint32_t)(j >> 2), (uint32_t)worker, (uint32_t)step, ORC_TAG_SQUANT};
  uint32_t key[2] = {(uint32_t)(seed & 0xFFFFFFFFu), (uint32_t)(seed >> 32)};
  uint32_t out[4];
  orc_philox4x32_10(ctr, key, out);
  uint32_t x = out[j & 3];
  return (float)(x >> 8) * 0x1p-24f;
}

/* ------------------------------------------------------------------------ */
/* Message layout.  Every section starts at a multiple of 256 bytes and the  */
/* whole message is padded to a multiple of 256 bytes; padding is zero.      */
/*   sign:     [nb fp32 scales][ceil(d/32) u32 words]                        */
/*             bit (j mod 32) of word (j div 32) is 1 iff p_j < 0            */
/*   squant, qsgd: [nb fp32 scales][ceil(d*b/32) u32 words]                  */
/*             code j sits in bits [(j*b) mod 32, +b) of word (j*b) div 32   */
/*   top-k:    k records {u32 index, f32 value}, ascending index             */
/*   identity: d fp32 values                                                 */
/* ------------------------------------------------------------------------ */
static int64_t round256(int64_t x) { return (x + 255) / 256 * 256; }

/* ------------------------------------------------------------------------ */
/* Buckets.  Without segments, bucket b covers [b*n, min((b+1)*n, d)).  With */
/* layer segments (the per-layer variant of Section 2.4's bucketing), each   */
/* segment [seg[i], seg[i+1]) is cut into buckets of n from its own start,   */
/* the last one partial; buckets are numbered in element order.             */
/* ------------------------------------------------------------------------ */
int64_t orc_bucket_count(const orc_cfg* c) {
  if (c->nseg <= 0) return (c->d + c->bucket - 1) / c->bucket;
  int64_t nb = 0;
  for (int32_t i = 0; i < c->nseg; ++i) nb += (c->seg[i + 1] - c->seg[i] + c->bucket - 1) / c->bucket;
  return nb;
}

/* starts[0..nb]: bucket b covers [starts[b], starts[b+1]). */
void orc_bucket_starts(const orc_cfg* c, int64_t* starts) {
  int64_t b = 0;
  if (c->nseg <= 0) {
    int64_t nb = orc_bucket_count(c);
    for (b = 0; b < nb; ++b) starts[b] = b * c->bucket;
    starts[nb] = c->d;
    return;
  }
  for (int32_t i = 0; i < c->nseg; ++i)
    for (int64_t j = c->seg[i]; j < c->seg[i + 1]; j += c->bucket) starts[b++] = j;
  starts[b] = c->d;
}

int64_t orc_layout(const orc_cfg* c, int64_t* off_scales, int64_t* off_payload) {
  int64_t nb = (c->compressor == ORC_TOPK || c->compressor == ORC_IDENTITY) ? 0 : orc_bucket_count(c);
  *off_scales = 0;
  switch (c->compressor) {
    case ORC_SIGN: {
      int64_t words = (c->d + 31) / 32;
      *off_payload = round256(4 * nb);
      return round256(*off_payload + 4 * words);
    }
    case ORC_SQUANT:
    case ORC_QSGD: {
      int64_t words = (c->d * c->bits + 31) / 32;
      *off_payload = round256(4 * nb);
      return round256(*off_payload + 4 * words);
    }
    case ORC_TOPK:
      *off_payload = 0;
      return round256(8 * c->k);
    case ORC_IDENTITY:
      *off_payload = 0;
      return round256(4 * c->d);
  }
  return -1;
}

/* ------------------------------------------------------------------------ */
/* Scaled sign (Section 2.4: the sign function with a scaling factor; the    */
/* error-feedback sign compressor cited in Section 3.1).  The paper does not */
/* print the scale; the reading taken is the mean absolute value of the     */
/* bucket, s = ||x_b||_1 / n_b, the least-squares scale for the pattern      */
/* sign(x_b).  The l1 sum is taken in one fixed order so that the scale,    */
/* and through the residual every later step, is reproducible:             */
/*   - the bucket (zero-padded to `bucket` elements) is cut into 4-element  */
/*     chunks c = 0, 1, ...; a chunk's sum is ((|a0|+|a1|)+|a2|)+|a3|;       */
/*   - lane l in 0..31 adds, in increasing c, the sums of the chunks with   */
/*     c mod 32 == l to a running total that starts at 0;                   */
/*   - the 32 lane totals are combined by five exchange rounds with         */
/*     partners l xor 16, 8, 4, 2, 1, each lane taking own + partner.       */
/* The scale is then fl(l1 / n_b), n_b the real (unpadded) bucket length.   */
/* ------------------------------------------------------------------------ */
float orc_sign_l1(const float* x, int64_t count, int32_t bucket) {
  float lane[32];
  for (int l = 0; l < 32; ++l) lane[l] = 0.0f;
  int64_t chunks = bucket / 4;
  for (int64_t c = 0; c < chunks; ++c) {
    float a[4];
    for (int q = 0; q < 4; ++q) {
      int64_t j = 4 * c + q;
      a[q] = (j < count) ? fabsf(x[j]) : 0.0f;
    }
    float chunk_sum = ((a[0] + a[1]) + a[2]) + a[3];
    lane[c % 32] = lane[c % 32] + chunk_sum;
  }
  for (int off = 16; off >= 1; off /= 2) {
    float next[32];
    for (int l = 0; l < 32; ++l) next[l] = lane[l] + lane[l ^ off];
    for (int l = 0; l < 32; ++l) lane[l] = next[l];
  }
  return lane[0];
}

float orc_sign_scale(const float* x, int64_t count, int32_t bucket) {
  return orc_sign_l1(x, count, bucket) / (float)count;
}

/* ------------------------------------------------------------------------ */
/* QSGD scale (Section 2.4, Eq. (qsgd) of Alistarh et al.): the l2 norm of  */
/* the bucket, s = fl(sqrt(sum_j x_j^2)).  The sum of squares is taken in    */
/* the same fixed order as the scaled sign's l1 sum: a chunk's share is      */
/* ((x0*x0 + x1*x1) + x2*x2) + x3*x3, lane l adds chunks l, l+32, ... in     */
/* increasing order, then the five exchange rounds 16, 8, 4, 2, 1.          */
/* ------------------------------------------------------------------------ */
float orc_qsgd_sumsq(const float* x, int64_t count, int32_t bucket) {
  float lane[32];
  for (int l = 0; l < 32; ++l) lane[l] = 0.0f;
  int64_t chunks = bucket / 4;
  for (int64_t c = 0; c < chunks; ++c) {
    float sq[4];
    for (int q = 0; q < 4; ++q) {
      int64_t j = 4 * c + q;
      float v = (j < count) ? x[j] : 0.0f;
      sq[q] = v * v;
    }
    float chunk_sum = ((sq[0] + sq[1]) + sq[2]) + sq[3];
    lane[c % 32] = lane[c % 32] + chunk_sum;
  }
  for (int off = 16; off >= 1; off /= 2) {
    float next[32];
    for (int l = 0; l < 32; ++l) next[l] = lane[l] + lane[l ^ off];
    for (int l = 0; l < 32; ++l) lane[l] = next[l];
  }
  return lane[0];
}

float orc_qsgd_scale(const float* x, int64_t count, int32_t bucket) {
  return sqrtf(orc_qsgd_sumsq(x, count, bucket));
}

/* ------------------------------------------------------------------------ */
/* m-bit stochastic quantiser of Hou et al. (Section 2.4, Appendix A proof   */
/* of Theorem 2) with s = ||v_b||_inf per bucket and uniform levels          */
/* B_r = r / K, K = 2^(b-1) - 1.  A code is the signed level shifted by K,   */
/* so codes lie in [0, 2K] and fit in b bits.                               */
/* ------------------------------------------------------------------------ */
float orc_squant_decode(int32_t code, float s, int32_t K) {
  int32_t level = code - K;
  if (level == 0) return 0.0f;
  float mag = s * ((float)abs(level) / (float)K);
  return level < 0 ? -mag : mag;
}

/* The b-bit stochastic rounding of one bucket with scale s: the l_inf norm
 * for Hou et al.'s quantiser, the l2 norm for QSGD (Section 2.4). */
static void squant_bucket(const orc_cfg* c, int32_t worker, int64_t step, int64_t start,
                          int64_t count, const float* p, float* s_out, int32_t* codes) {
  int32_t K = (1 << (c->bits - 1)) - 1;
  float s = 0.0f;
  if (c->compressor == ORC_QSGD) {
    s = orc_qsgd_scale(p, count, c->bucket);
  } else {
    for (int64_t j = 0; j < count; ++j) {
      float a = fabsf(p[j]);
      if (a > s) s = a;
    }
  }
  *s_out = s;
  if (s == 0.0f) {
    for (int64_t j = 0; j < count; ++j) codes[j] = K;
    return;
  }
  float inv = (float)K / s;
  for (int64_t j = 0; j < count; ++j) {
    float t = fabsf(p[j]) * inv;
    if (t > (float)K) t = (float)K;
    float r = floorf(t);
    float f = t - r;
    float u = orc_squant_uniform(c->seed, worker, step, start + j);
    int32_t level = (int32_t)r + (u < f ? 1 : 0);
    if (level > K) level = K;
    codes[j] = (p[j] < 0.0f) ? K - level : K + level;
  }
}

/* ------------------------------------------------------------------------ */
/* Top-k (Section 2.4; Theorem 1 and its proof in Appendix A): keep the k   */
/* entries of largest magnitude.  Magnitude order is the order of the bit   */
/* pattern with the sign bit cleared; ties go to the lower index.           */
/* ------------------------------------------------------------------------ */
typedef struct { uint32_t key; int64_t index; } topk_item;

static int topk_order(const void* a, const void* b) {
  const topk_item* x = (const topk_item*)a;
  const topk_item* y = (const topk_item*)b;
  if (x->key != y->key) return x->key > y->key ? -1 : 1;
  if (x->index != y->index) return x->index < y->index ? -1 : 1;
  return 0;
}

static uint32_t magnitude_key(float v) {
  uint32_t bits;
  memcpy(&bits, &v, 4);
  return bits & 0x7FFFFFFFu;
}

/* Marks selected[j] = 1 for the k chosen entries of p (d entries). */
void orc_topk_select(const float* p, int64_t d, int64_t k, uint8_t* selected) {
  topk_item* items = (topk_item*)malloc((size_t)d * sizeof(topk_item));
  for (int64_t j = 0; j < d; ++j) {
    items[j].key = magnitude_key(p[j]);
    items[j].index = j;
  }
  qsort(items, (size_t)d, sizeof(topk_item), topk_order);
  memset(selected, 0, (size_t)d);
  for (int64_t r = 0; r < k; ++r) selected[items[r].index] = 1;
  free(items);
}

/* ------------------------------------------------------------------------ */
/* Decode of elements [j0, j1) of one message: q[j - j0] = Q(p)_j as the    */
/* server sees it.  starts: the nb + 1 bucket starts (sign, quantisers).    */
/* ------------------------------------------------------------------------ */
static void decode_range(const orc_cfg* c, const uint8_t* msg, const int64_t* starts, int64_t nb,
                         int64_t j0, int64_t j1, float* q) {
  int64_t off_s, off_p;
  orc_layout(c, &off_s, &off_p);
  switch (c->compressor) {
    case ORC_SIGN:
    case ORC_SQUANT:
    case ORC_QSGD: {
      const float* scales = (const float*)(msg + off_s);
      const uint32_t* words = (const uint32_t*)(msg + off_p);
      int32_t K = (1 << (c->bits - 1)) - 1;
      uint32_t mask = (1u << c->bits) - 1u;
      /* the bucket holding j0: the last b with starts[b] <= j0 */
      int64_t lo = 0, hi = nb;
      while (hi - lo > 1) {
        int64_t mid = (lo + hi) / 2;
        if (starts[mid] <= j0) lo = mid;
        else hi = mid;
      }
      int64_t b = lo;
      for (int64_t j = j0; j < j1; ++j) {
        while (starts[b + 1] <= j) ++b;
        if (c->compressor == ORC_SIGN) {
          int neg = (words[j >> 5] >> (j & 31)) & 1u;
          q[j - j0] = neg ? -scales[b] : scales[b];
        } else {
          int64_t bitpos = j * c->bits;
          int32_t code = (int32_t)((words[bitpos >> 5] >> (bitpos & 31)) & mask);
          q[j - j0] = orc_squant_decode(code, scales[b], K);
        }
      }
      break;
    }
    case ORC_TOPK: {
      for (int64_t j = j0; j < j1; ++j) q[j - j0] = 0.0f;
      /* records ascend by index: the first one at or after j0 */
      int64_t lo = 0, hi = c->k;
      while (lo < hi) {
        int64_t mid = (lo + hi) / 2;
        uint32_t idx;
        memcpy(&idx, msg + 8 * mid, 4);
        if ((int64_t)idx < j0) lo = mid + 1;
        else hi = mid;
      }
      for (int64_t r = lo; r < c->k; ++r) {
        uint32_t idx;
        float val;
        memcpy(&idx, msg + 8 * r, 4);
        if ((int64_t)idx >= j1) break;
        memcpy(&val, msg + 8 * r + 4, 4);
        q[idx - j0] = val;
      }
      break;
    }
    case ORC_IDENTITY:
      memcpy(q, msg + 4 * j0, (size_t)(j1 - j0) * 4);
      break;
  }
}

static int64_t* bucket_starts_alloc(const orc_cfg* c, int64_t* nb_out) {
  int64_t nb = (c->compressor == ORC_TOPK || c->compressor == ORC_IDENTITY) ? 0 : orc_bucket_count(c);
  int64_t* starts = (int64_t*)malloc((size_t)(nb + 1) * 8);
  if (nb > 0) orc_bucket_starts(c, starts);
  else starts[0] = c->d;
  *nb_out = nb;
  return starts;
}

/* Dense decode of one message: q = Q(p) as the server sees it. */
void orc_decode(const orc_cfg* c, const uint8_t* msg, float* q) {
  int64_t nb;
  int64_t* starts = bucket_starts_alloc(c, &nb);
  decode_range(c, msg, starts, nb, 0, c->d, q);
  free(starts);
}

/* ------------------------------------------------------------------------ */
/* The sum over the M workers of Algorithm 2's server, in one fixed order   */
/* (the paper leaves the order open; fixing it makes the parameters        */
/* reproducible bit for bit): the M values, padded with +0 to the next     */
/* power of two P >= M, are summed pairwise -- at every level x_i becomes  */
/* x_2i + x_2i+1 -- until one value is left.  x: P floats, overwritten.    */
/* ------------------------------------------------------------------------ */
float orc_pairwise_sum(float* x, int32_t M) {
  int32_t P = 1;
  while (P < M) P *= 2;
  for (int32_t i = M; i < P; ++i) x[i] = 0.0f;
  for (int32_t width = 1; width < P; width *= 2)
    for (int32_t i = 0; i < P; i += 2 * width) x[i] = x[i] + x[i + width];
  return x[0];
}

/* ------------------------------------------------------------------------ */
/* Worker step of Algorithm 2 for worker `worker` at iteration `step`:      */
/*   p = eta * F + e          (F = g, the worker's stochastic gradient)     */
/*   p_hat = Q(p), packed into msg                                          */
/*   e = p - p_hat                                                          */
/*   h = eta * F + e          (kept for the next lookahead, only if asked)  */
/* g: d floats (read); e, h: d floats (read/write); msg: the layout above.  */
/* ------------------------------------------------------------------------ */
void orc_worker_step(const orc_cfg* c, int32_t worker, int64_t step, const float* g, float* e,
                     float* h, uint8_t* msg) {
  int64_t d = c->d;
  int64_t off_s, off_p;
  int64_t total = orc_layout(c, &off_s, &off_p);
  memset(msg, 0, (size_t)total);

  float* p = (float*)malloc((size_t)(d > 0 ? d : 1) * 4);
  float* q = (float*)malloc((size_t)(d > 0 ? d : 1) * 4);
  for (int64_t j = 0; j < d; ++j) {
    float step_g = c->lr * g[j];
    p[j] = step_g + e[j];
  }

  switch (c->compressor) {
    case ORC_SIGN: {
      float* scales = (float*)(msg + off_s);
      uint32_t* words = (uint32_t*)(msg + off_p);
      int64_t nb = orc_bucket_count(c);
      int64_t* starts = (int64_t*)malloc((size_t)(nb + 1) * 8);
      orc_bucket_starts(c, starts);
      for (int64_t b = 0; b < nb; ++b) {
        int64_t start = starts[b];
        int64_t count = starts[b + 1] - start;
        float s = orc_sign_scale(p + start, count, c->bucket);
        scales[b] = s;
        for (int64_t j = start; j < start + count; ++j) {
          int neg = p[j] < 0.0f;
          if (neg) words[j >> 5] |= 1u << (j & 31);
          q[j] = neg ? -s : s;
        }
      }
      free(starts);
      break;
    }
    case ORC_SQUANT:
    case ORC_QSGD: {
      float* scales = (float*)(msg + off_s);
      uint32_t* words = (uint32_t*)(msg + off_p);
      int32_t K = (1 << (c->bits - 1)) - 1;
      int64_t nb = orc_bucket_count(c);
      int64_t* starts = (int64_t*)malloc((size_t)(nb + 1) * 8);
      orc_bucket_starts(c, starts);
      int32_t* codes = (int32_t*)malloc((size_t)c->bucket * 4);
      for (int64_t b = 0; b < nb; ++b) {
        int64_t start = starts[b];
        int64_t count = starts[b + 1] - start;
        squant_bucket(c, worker, step, start, count, p + start, &scales[b], codes);
        for (int64_t j = 0; j < count; ++j) {
          int64_t bitpos = (start + j) * c->bits;
          words[bitpos >> 5] |= (uint32_t)codes[j] << (bitpos & 31);
          q[start + j] = orc_squant_decode(codes[j], scales[b], K);
        }
      }
      free(codes);
      free(starts);
      break;
    }
    case ORC_TOPK: {
      uint8_t* selected = (uint8_t*)malloc((size_t)(d > 0 ? d : 1));
      orc_topk_select(p, d, c->k, selected);
      int64_t r = 0;
      for (int64_t j = 0; j < d; ++j) {
        if (selected[j]) {
          uint32_t idx = (uint32_t)j;
          memcpy(msg + 8 * r, &idx, 4);
          memcpy(msg + 8 * r + 4, &p[j], 4);
          ++r;
          q[j] = p[j];
        } else {
          q[j] = 0.0f;
        }
      }
      free(selected);
      break;
    }
    case ORC_IDENTITY:
      memcpy(msg, p, (size_t)d * 4);
      for (int64_t j = 0; j < d; ++j) q[j] = p[j];
      break;
  }

  for (int64_t j = 0; j < d; ++j) e[j] = p[j] - q[j];
  if (c->keep_lookahead && h != NULL) {
    for (int64_t j = 0; j < d; ++j) {
      float step_g = c->lr * g[j];
      h[j] = step_g + e[j];
    }
  }
  free(p);
  free(q);
}

/* ------------------------------------------------------------------------ */
/* Server step of Algorithm 2: q_hat = (1/M) sum_m p_hat^(m), the sum taken */
/* by orc_pairwise_sum, then w = w - q_hat.  Elements are handled a chunk   */
/* at a time (every message's values of the chunk decoded first) only to   */
/* bound the memory; each element's arithmetic is the one stated.          */
/* msgs: M messages, message m at msgs + m * msg_stride.  w: d floats.      */
/* ------------------------------------------------------------------------ */
#define ORC_SERVER_CHUNK 4096

/* The averaged update q_hat of Algorithm 2's server for elements [j0, j1),
 * element j written to q_hat[j - j0]: the sum over workers taken by
 * orc_pairwise_sum, then divided by M.  Each element depends on that element alone, so disjoint
 * ranges may run concurrently. */
void orc_server_average_range(const orc_cfg* c, const uint8_t* msgs, int64_t msg_stride, float* q_hat,
                              int64_t j0, int64_t j1) {
  int32_t M = c->M;
  int32_t P = 1;
  while (P < M) P *= 2;
  int64_t nb;
  int64_t* starts = bucket_starts_alloc(c, &nb);
  float* q = (float*)malloc((size_t)M * ORC_SERVER_CHUNK * 4);
  float* x = (float*)malloc((size_t)P * 4);
  for (int64_t c0 = j0; c0 < j1; c0 += ORC_SERVER_CHUNK) {
    int64_t c1 = c0 + ORC_SERVER_CHUNK < j1 ? c0 + ORC_SERVER_CHUNK : j1;
    for (int32_t m = 0; m < M; ++m)
      decode_range(c, msgs + (int64_t)m * msg_stride, starts, nb, c0, c1, q + (int64_t)m * ORC_SERVER_CHUNK);
    for (int64_t j = c0; j < c1; ++j) {
      for (int32_t m = 0; m < M; ++m) x[m] = q[(int64_t)m * ORC_SERVER_CHUNK + (j - c0)];
      float sum = orc_pairwise_sum(x, M);
      q_hat[j - j0] = sum / (float)M;
    }
  }
  free(x);
  free(q);
  free(starts);
}

/* The server step (w = w - q_hat) restricted to elements [j0, j1). */
void orc_server_step_range(const orc_cfg* c, const uint8_t* msgs, int64_t msg_stride, float* w, int64_t j0,
                           int64_t j1) {
  float* q_hat = (float*)malloc((size_t)(j1 > j0 ? j1 - j0 : 1) * 4);
  orc_server_average_range(c, msgs, msg_stride, q_hat, j0, j1);
  for (int64_t j = j0; j < j1; ++j) w[j] = w[j] - q_hat[j - j0];
  free(q_hat);
}

void orc_server_step(const orc_cfg* c, const uint8_t* msgs, int64_t msg_stride, float* w) {
  orc_server_step_range(c, msgs, msg_stride, w, 0, c->d);
}

/* ------------------------------------------------------------------------ */
/* Optimistic Adam on the server (the CPOAdam family that Section 4 compares */
/* against).  The paper prints no rule for it; the reading taken is the     */
/* Optimistic Adam of Daskalakis, Ilyas, Syrgkanis and Zeng ("Training GANs  */
/* with Optimism", ICLR 2018), fed the averaged update q_hat of Algorithm 2  */
/* in place of the plain step w = w - q_hat:                                 */
/*   m = b1 m + (1 - b1) q_hat,   v = b2 v + ((1 - b2) q_hat) q_hat          */
/*   with bias correction m_hat = m / (1 - b1^t), v_hat = v / (1 - b2^t),   */
/*   else m_hat = m, v_hat = v                                               */
/*   adaptive: u = m_hat / (sqrt(v_hat) + eps), and u = 0 where m_hat = 0;  */
/*   else u = m_hat (the identity preconditioner)                           */
/*   w = w - alpha (2 u - u_prev),   u_prev = u                              */
/* in fp32, one rounding per operation in the order written; b^t is the     */
/* product of t factors b taken left to right.  m, v, u_prev start at 0.    */
/* With b1 = 0, the identity preconditioner and alpha = 1 the update is     */
/* w_t = w_{t-1} - 2 q_hat_t + q_hat_{t-1}, the one-line OMD recurrence of  */
/* Section 2.2.                                                              */
/* ------------------------------------------------------------------------ */
typedef struct orc_oadam {
  float alpha;
  float beta1;
  float beta2;
  float eps;
  int32_t adaptive;         /* 1: divide by sqrt(v_hat) + eps */
  int32_t bias_correction;  /* 1: divide m, v by 1 - b^t */
} orc_oadam;

float orc_pow_steps(float b, int64_t t) {
  float r = 1.0f;
  for (int64_t i = 0; i < t; ++i) r = r * b;
  return r;
}

/* One Optimistic Adam step at iteration t (1-based) on n elements. */
void orc_oadam_update(const orc_oadam* p, int64_t t, int64_t n, const float* q_hat, float* m, float* v, float* u,
                      float* w) {
  float one_m_b1 = 1.0f - p->beta1;
  float one_m_b2 = 1.0f - p->beta2;
  float c1 = p->bias_correction ? 1.0f - orc_pow_steps(p->beta1, t) : 1.0f;
  float c2 = p->bias_correction ? 1.0f - orc_pow_steps(p->beta2, t) : 1.0f;
  for (int64_t j = 0; j < n; ++j) {
    float g = q_hat[j];
    float mj = p->beta1 * m[j] + one_m_b1 * g;
    float vj = p->beta2 * v[j] + (one_m_b2 * g) * g;
    float mh = p->bias_correction ? mj / c1 : mj;
    float vh = p->bias_correction ? vj / c2 : vj;
    float uj = mh;
    if (p->adaptive) uj = (mh == 0.0f) ? 0.0f : mh / (sqrtf(vh) + p->eps);
    float step = 2.0f * uj - u[j];
    w[j] = w[j] - p->alpha * step;
    m[j] = mj;
    v[j] = vj;
    u[j] = uj;
  }
}

/* The server step with Optimistic Adam on elements [j0, j1): q_hat as in   */
/* orc_server_average_range, then orc_oadam_update (m, v, u: d floats).      */
void orc_server_step_oadam_range(const orc_cfg* c, const uint8_t* msgs, int64_t msg_stride, const orc_oadam* p,
                                 int64_t t, float* m, float* v, float* u, float* w, int64_t j0, int64_t j1) {
  float* q_hat = (float*)malloc((size_t)(j1 > j0 ? j1 - j0 : 1) * 4);
  orc_server_average_range(c, msgs, msg_stride, q_hat, j0, j1);
  orc_oadam_update(p, t, j1 - j0, q_hat, m + j0, v + j0, u + j0, w + j0);
  free(q_hat);
}

/* Lookahead of Algorithm 2: w_{t-1/2} = w_{t-1} - h, h = eta*F_prev + e_prev. */
void orc_lookahead(int64_t d, const float* w, const float* h, float* out) {
  for (int64_t j = 0; j < d; ++j) out[j] = w[j] - h[j];
}
