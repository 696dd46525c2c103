// GB300 (sm_103a) verification step of speculative cascades with the
// vocabulary split across W GPUs (include/sc_shard.h).
//
// Each rank holds the logits of a contiguous range of tokens of every row.
// The step is Algorithm 4 with Algorithm 5's target, for the deferral rules of
// Table 1 (and delta = 1, delta = 0), written as five phases with an
// all-gather of a small message between consecutive phases:
//
//   pass 1   grid (unit, slice): every CTA reads one slice of kL logits of a
//            row pair (or of the bonus target row) with coalesced 16-byte
//            loads, all of them in flight before any arithmetic, and reduces
//            it to (max, sum of 2^{fma(y, k, -fl(max k))}) per row; a second
//            kernel merges the rank's slices per unit           -> message 1
//   decide   one thread per unit merges the W ranks' partials in double
//            precision, in rank order (identical on every rank): M, S, max q,
//            max p, delta by the rule, and the acceptance test; OPT pairs in
//            the band need D_TV: a grid (pair, slice) sums the residual
//            weights max(0, 2^{b + c} - 2^a) = S_q max(0, p - q) over the
//            rank's part of those rows                           -> message 2
//   accept   one thread per sequence finishes the band pairs (Eq. 10),
//            settles j*, and a grid (sequence, slice) sums the weights of the
//            row to draw from -- the residual of row j*, or p of the bonus
//            row -- per 256-token segment (warp scans in double) -> message 3
//   draw     one warp per sequence finds the rank, slice, segment and token
//            holding u R in ascending token order; only the rank holding it
//            rescans that one segment                            -> message 4
//   finish   one thread per sequence takes the drawing rank's token.
//
// Every sum that a later phase splits again (rank totals into slices, slices
// into segments, segments into lanes) is formed in the same order by the
// same code in both places, so a search never falls between two levels; a
// rounding gap at the bottom level falls back to the last positive weight of
// the segment.

#include "sc_shard.h"

#include <cuda_runtime.h>

#include <cfloat>
#include <cmath>
#include <cstdint>

namespace {

constexpr int kT = 256;                 // threads per CTA
constexpr int kWarps = kT / 32;         // warps per CTA
constexpr int kSeg = 256;               // tokens per segment: one warp, 8 per lane
constexpr int kSegs = 32;               // segments per slice
constexpr int kL = kSeg * kSegs;        // 8192 tokens per slice
constexpr int kRounds = kSegs / kWarps; // segments per warp per slice

enum UnitKind : int { kAccepted = 0, kRejected = 1, kNeedTV = 2, kBonus = 3, kBad = 4 };

// Decision state of one unit (row pair (b, j < gamma) or bonus row (b, gamma)).
struct UnitState {
  double Sq, Sp;      // sums of 2^{fma(y, k, -R)} over the whole row
  double maxq, maxp;  // max_v q(v), max_v p(v)
  double L;           // log2 p(x) - log2 q(x) (both finite)
  float Rq, Rp;       // exponent references fl(M k)
  float c;            // log2(S_q / S_p) rounded to f32: the residual weights' shift
  int kind;           // UnitKind
  int xq0, xp0;       // q(x) = 0, p(x) = 0 (masked logits at the draft token)
};

struct SeqState {
  int jstar;  // first rejection, or gamma
  int bad;    // a data error in the sequence
};

struct Geom {
  int B, gamma, W, rank;
  int begin[SC_SHARD_MAX + 1];
  int width;  // tokens of this rank
  int slots;  // slices of kL tokens of this rank
  long long ld;
  float k;    // log2(e) / T in f32
  double kd;  // log2(e) / T in double
  int rule;
  double alpha;
};

size_t align16(size_t n) { return (n + 15) & ~static_cast<size_t>(15); }

struct Msg1 {
  float4 *rec;  // [units] (m_q, s_q, m_p, s_p) of this rank
  float2 *x;    // [pairs] the draft token's logits (q, p), from the rank holding it
};
__host__ __device__ inline Msg1 msg1_at(void *base, int B, int gamma) {
  const size_t units = static_cast<size_t>(B) * (gamma + 1);
  char *p = static_cast<char *>(base);
  return Msg1{reinterpret_cast<float4 *>(p), reinterpret_cast<float2 *>(p + units * sizeof(float4))};
}
size_t msg_bytes(int B, int gamma, int k) {
  const size_t units = static_cast<size_t>(B) * (gamma + 1), pairs = static_cast<size_t>(B) * gamma;
  switch (k) {
    case 1: return align16(units * sizeof(float4)) + align16(pairs * sizeof(float2));
    case 2: return align16(pairs * sizeof(double));
    case 3: return align16(static_cast<size_t>(B) * sizeof(double));
    case 4: return align16(static_cast<size_t>(B) * sizeof(int32_t));
    default: return 0;
  }
}

// Workspace of one rank.  The per-sequence and per-unit states come first, at
// offsets that do not depend on the shard's width (sc_shard_finish does not know it).
struct Work {
  SeqState *seq;       // [B]
  UnitState *unit;     // [units]
  float4 *slot_rec;    // [units][slots]
  float *tv_slot;      // [pairs][slots]
  double *seg_tot;     // [B][slots][kSegs]
  double *slot_mass;   // [B][slots]
};
__host__ __device__ inline size_t work_layout(int B, int gamma, int slots, void *base, Work *w) {
  const size_t units = static_cast<size_t>(B) * (gamma + 1), pairs = static_cast<size_t>(B) * gamma;
  const size_t sizes[6] = {static_cast<size_t>(B) * sizeof(SeqState), units * sizeof(UnitState),
                           units * slots * sizeof(float4), pairs * slots * sizeof(float),
                           static_cast<size_t>(B) * slots * kSegs * sizeof(double),
                           static_cast<size_t>(B) * slots * sizeof(double)};
  size_t off[6], total = 0;
  for (int i = 0; i < 6; ++i) {
    off[i] = total;
    total += (sizes[i] + 255) & ~static_cast<size_t>(255);
  }
  if (w != nullptr) {
    char *p = static_cast<char *>(base);
    w->seq = reinterpret_cast<SeqState *>(p + off[0]);
    w->unit = reinterpret_cast<UnitState *>(p + off[1]);
    w->slot_rec = reinterpret_cast<float4 *>(p + off[2]);
    w->tv_slot = reinterpret_cast<float *>(p + off[3]);
    w->seg_tot = reinterpret_cast<double *>(p + off[4]);
    w->slot_mass = reinterpret_cast<double *>(p + off[5]);
  }
  return total;
}

// ------------------------------------------------------------------ arithmetic

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Exponent reference of a maximum m: fl(m k), floored so that a slice of -inf
// logits keeps finite arithmetic (its sum is 0).
__device__ __forceinline__ float ref_of(float m, float k) { return fmaxf(__fmul_rn(m, k), -1e30f); }

// Residual weight of one token of a pair: S_q max(0, p - q) = max(0, 2^{b + c} - 2^a).
__device__ __forceinline__ float res_weight(float yq, float yp, float k, float Rq, float Rp, float c) {
  const float a = fmaf(yq, k, -Rq), b = fmaf(yp, k, -Rp);
  return fmaxf(0.0f, ex2(__fadd_rn(b, c)) - ex2(a));
}

// ------------------------------------------------------------------ loads

// Eight logits of a row as raw registers, loaded before they are converted so
// that all of a thread's loads are in flight together.
template <typename E>
struct Raw8;
template <>
struct Raw8<uint16_t> {  // bf16 bit patterns
  uint4 v;
  __device__ __forceinline__ void load(const uint16_t *s) { v = __ldg(reinterpret_cast<const uint4 *>(s)); }
  __device__ __forceinline__ void to_float(float (&y)[8]) const {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      y[2 * i] = __uint_as_float(w[i] << 16);
      y[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
  __device__ __forceinline__ static float at(const uint16_t *g, long long i) {
    return __uint_as_float(static_cast<uint32_t>(g[i]) << 16);
  }
};
template <>
struct Raw8<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float *s) {
    a = __ldg(reinterpret_cast<const float4 *>(s));
    b = __ldg(reinterpret_cast<const float4 *>(s + 4));
  }
  __device__ __forceinline__ void to_float(float (&y)[8]) const {
    y[0] = a.x; y[1] = a.y; y[2] = a.z; y[3] = a.w;
    y[4] = b.x; y[5] = b.y; y[6] = b.z; y[7] = b.w;
  }
  __device__ __forceinline__ static float at(const float *g, long long i) { return g[i]; }
};

// The 8 logits at positions [e, e + 8) of a slice of n valid tokens starting at
// `row`; positions at or past n read as -inf (probability 0).  kVec: the row
// start is 16-byte aligned, so whole groups are read as vectors.
template <typename E, bool kVec>
struct Group {
  Raw8<E> raw;
  bool whole;
  __device__ __forceinline__ void load(const E *row, int e, int n) {
    whole = kVec && e + 8 <= n;
    if (whole) raw.load(row + e);
  }
  __device__ __forceinline__ void get(const E *row, int e, int n, float (&y)[8]) const {
    if (whole) {
      raw.to_float(y);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) y[i] = e + i < n ? Raw8<E>::at(row, e + i) : -INFINITY;
    }
  }
};

// Position in its slice of the group of 8 tokens that lane `lane` of warp
// `warp` handles in round i: segment i * kWarps + warp, lane-th group of it.
__device__ __forceinline__ int group_pos(int i, int warp, int lane) { return (i * kWarps + warp) * kSeg + lane * 8; }

// ------------------------------------------------------------------ reductions

// (max, sum) pairs: every lane ends with the warp's (M, S), S relative to ref_of(M).
__device__ __forceinline__ void warp_ms(float &m, float &s, float k) {
  float M = m;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
  float t = s * ex2(ref_of(m, k) - ref_of(M, k));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t = __fadd_rn(t, __shfl_xor_sync(0xFFFFFFFFu, t, o));
  m = M;
  s = t;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Inclusive prefix over the warp's lanes, in double.
__device__ __forceinline__ double warp_scan_d(double v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double t = __shfl_up_sync(0xFFFFFFFFu, v, o);
    if (lane >= o) v += t;
  }
  return v;
}

// The 8 weights of one lane's group of the row a sequence draws from: the
// residual S_q max(0, p - q) of a rejected pair, or 2^{b} (proportional to p)
// of the bonus row, and their sum in f32, left to right.
template <typename E, bool kVec>
__device__ __forceinline__ float lane_weights(const E *rq, const E *rp, bool pair, int e, int n,
                                              const Geom &G, float Rq, float Rp, float c,
                                              float (&w)[8]) {
  float yp[8];
  Group<E, kVec> gp;
  gp.load(rp, e, n);
  gp.get(rp, e, n, yp);
  if (pair) {
    float yq[8];
    Group<E, kVec> gq;
    gq.load(rq, e, n);
    gq.get(rq, e, n, yq);
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = res_weight(yq[i], yp[i], G.k, Rq, Rp, c);
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = ex2(fmaf(yp[i], G.k, -Rp));
  }
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < 8; ++i) s = __fadd_rn(s, w[i]);
  return s;
}

__device__ __forceinline__ int unit_b(int u, int gamma) { return u / (gamma + 1); }
__device__ __forceinline__ int unit_j(int u, int gamma) { return u % (gamma + 1); }

template <typename E>
__device__ __forceinline__ const E *q_row(const E *q, const Geom &G, int b, int j, int lo) {
  return q + (static_cast<long long>(b) * G.gamma + j) * G.ld + lo;
}
template <typename E>
__device__ __forceinline__ const E *p_row(const E *p, const Geom &G, int b, int j, int lo) {
  return p + (static_cast<long long>(b) * (G.gamma + 1) + j) * G.ld + lo;
}

// ------------------------------------------------------------------ pass 1

// One CTA per (unit, slice): the slice's (m_q, s_q, m_p, s_p); the CTA holding
// a pair's draft token also records the token's two logits.
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_pass1_kernel(const E *__restrict__ q, const E *__restrict__ p,
                                                         const int32_t *__restrict__ tokens, Geom G,
                                                         float4 *__restrict__ slot_rec, float2 *__restrict__ xrec) {
  const int slot = blockIdx.x % G.slots, u = blockIdx.x / G.slots;
  const int b = unit_b(u, G.gamma), j = unit_j(u, G.gamma);
  const bool pair = j < G.gamma;
  const int lo = slot * kL, n = min(kL, G.width - lo);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const E *rp = p_row(p, G, b, j, lo);
  const E *rq = pair ? q_row(q, G, b, j, lo) : rp;

  Group<E, kVec> gq[kRounds], gp[kRounds];
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gp[i].load(rp, group_pos(i, warp, lane), n);
    if (pair) gq[i].load(rq, group_pos(i, warp, lane), n);
  }
  float mq = -INFINITY, mp = -INFINITY;
  float y[8];
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gp[i].get(rp, group_pos(i, warp, lane), n, y);
#pragma unroll
    for (int t = 0; t < 8; ++t) mp = fmaxf(mp, y[t]);
    if (pair) {
      gq[i].get(rq, group_pos(i, warp, lane), n, y);
#pragma unroll
      for (int t = 0; t < 8; ++t) mq = fmaxf(mq, y[t]);
    }
  }
  const float Rq = ref_of(mq, G.k), Rp = ref_of(mp, G.k);
  float sq = 0.0f, sp = 0.0f;
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gp[i].get(rp, group_pos(i, warp, lane), n, y);
#pragma unroll
    for (int t = 0; t < 8; ++t) sp = __fadd_rn(sp, ex2(fmaf(y[t], G.k, -Rp)));
    if (pair) {
      gq[i].get(rq, group_pos(i, warp, lane), n, y);
#pragma unroll
      for (int t = 0; t < 8; ++t) sq = __fadd_rn(sq, ex2(fmaf(y[t], G.k, -Rq)));
    }
  }
  warp_ms(mq, sq, G.k);
  warp_ms(mp, sp, G.k);
  __shared__ float4 red[kWarps];
  if (lane == 0) red[warp] = make_float4(mq, sq, mp, sp);
  __syncthreads();
  if (threadIdx.x == 0) {
    float Mq = -INFINITY, Mp = -INFINITY;
    for (int w = 0; w < kWarps; ++w) {
      Mq = fmaxf(Mq, red[w].x);
      Mp = fmaxf(Mp, red[w].z);
    }
    const float RQ = ref_of(Mq, G.k), RP = ref_of(Mp, G.k);
    float Sq = 0.0f, Sp = 0.0f;
    for (int w = 0; w < kWarps; ++w) {
      Sq = fmaf(red[w].y, ex2(ref_of(red[w].x, G.k) - RQ), Sq);
      Sp = fmaf(red[w].w, ex2(ref_of(red[w].z, G.k) - RP), Sp);
    }
    slot_rec[static_cast<size_t>(u) * G.slots + slot] = make_float4(Mq, Sq, Mp, Sp);
    if (pair) {
      const int x = tokens[b * G.gamma + j] - G.begin[G.rank] - lo;
      if (x >= 0 && x < n) xrec[b * G.gamma + j] = make_float2(Raw8<E>::at(rq, x), Raw8<E>::at(rp, x));
    }
  }
}

// One thread per unit: the rank's (m, s) over its slices, in slice order.
__global__ void shard_merge1_kernel(Geom G, const float4 *__restrict__ slot_rec, float4 *__restrict__ rec) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= G.B * (G.gamma + 1)) return;
  const float4 *r = slot_rec + static_cast<size_t>(u) * G.slots;
  float Mq = -INFINITY, Mp = -INFINITY;
  for (int s = 0; s < G.slots; ++s) {
    Mq = fmaxf(Mq, r[s].x);
    Mp = fmaxf(Mp, r[s].z);
  }
  const float RQ = ref_of(Mq, G.k), RP = ref_of(Mp, G.k);
  float Sq = 0.0f, Sp = 0.0f;
  for (int s = 0; s < G.slots; ++s) {
    Sq = fmaf(r[s].y, ex2(ref_of(r[s].x, G.k) - RQ), Sq);
    Sp = fmaf(r[s].w, ex2(ref_of(r[s].z, G.k) - RP), Sp);
  }
  rec[u] = make_float4(Mq, Sq, Mp, Sp);
}

// ------------------------------------------------------------------ decide

__device__ __forceinline__ int owner_of(const Geom &G, int x) {
  int r = 0;
  while (r + 1 < G.W && x >= G.begin[r + 1]) ++r;
  return r;
}

// Merge of the W ranks' (m, s) of one row, in rank order: R = fl(M k) and
// S = sum_r s_r 2^{fl(m_r k) - R} in double.
__device__ __forceinline__ void merge_ranks(const float4 *const *recs, int W, size_t u, bool p_row_,
                                            float k, float &M, float &R, double &S) {
  M = -INFINITY;
  for (int r = 0; r < W; ++r) M = fmaxf(M, p_row_ ? recs[r][u].z : recs[r][u].x);
  R = ref_of(M, k);
  S = 0.0;
  for (int r = 0; r < W; ++r) {
    const float m = p_row_ ? recs[r][u].z : recs[r][u].x, s = p_row_ ? recs[r][u].w : recs[r][u].y;
    S += static_cast<double>(s) * exp2(static_cast<double>(ref_of(m, k)) - static_cast<double>(R));
  }
}

// log2 of the softmax probability of logit y in a row of maximum M, reference R
// and sum S (of 2^{fma(y_v, k, -R)}, k the f32 factor):
//   log2 p(y) = y kd - M (kd - k) - R - log2 S,
// the exponents' f32 factor corrected to kd = log2(e) / T for the row's
// dominant terms (those with y_v near M).
__device__ __forceinline__ double log2_prob(float y, float M, float R, double S, const Geom &G) {
  const double kl = G.kd - static_cast<double>(G.k);
  return static_cast<double>(y) * G.kd - static_cast<double>(M) * kl - static_cast<double>(R) - log2(S);
}

// Acceptance of the draft token when delta = 1 (pi = p): [u < min(1, p(x)/q(x))];
// q(x) = 0 accepts, p(x) = 0 < q(x) rejects.
__device__ __forceinline__ bool accept_deferred(const UnitState &s, float u) {
  if (s.xq0) return true;
  if (s.xp0) return false;
  return s.L >= 0.0 || static_cast<double>(u) < exp2(s.L);
}

__global__ void shard_decide_kernel(Geom G, const void *__restrict__ gathered1, size_t msg1,
                                    const int32_t *__restrict__ tokens, const float *__restrict__ uniforms,
                                    UnitState *__restrict__ unit, int32_t *status) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= G.B * (G.gamma + 1)) return;
  const int b = unit_b(u, G.gamma), j = unit_j(u, G.gamma);
  const bool pair = j < G.gamma;
  const float4 *recs[SC_SHARD_MAX];
  for (int r = 0; r < G.W; ++r)
    recs[r] = msg1_at(const_cast<char *>(static_cast<const char *>(gathered1)) + r * msg1, G.B, G.gamma).rec;
  UnitState s{};
  float Mq = 0.0f, Mp, Rq = 0.0f, Rp;
  double Sq = 1.0, Sp;
  merge_ranks(recs, G.W, u, true, G.k, Mp, Rp, Sp);
  if (pair) merge_ranks(recs, G.W, u, false, G.k, Mq, Rq, Sq);
  int err = 0;
  const float uj = uniforms[b * (G.gamma + 1) + j];
  if (!(uj >= 0.0f && uj < 1.0f)) err |= SC_DEV_BAD_UNIFORM;
  if (!(isfinite(Sp) && Sp > 0.0 && Mp < INFINITY) || (pair && !(isfinite(Sq) && Sq > 0.0 && Mq < INFINITY)))
    err |= SC_DEV_BAD_LOGIT;
  int x = -1;
  if (pair) {
    x = tokens[b * G.gamma + j];
    if (x < 0 || x >= G.begin[G.W]) err |= SC_DEV_BAD_TOKEN;
  }
  s.Rq = Rq;
  s.Rp = Rp;
  s.Sq = Sq;
  s.Sp = Sp;
  if (err) {
    s.kind = kBad;
    if (status) atomicOr(status, err);
    unit[u] = s;
    return;
  }
  s.maxp = exp2(static_cast<double>(Mp) * G.k - Rp) / Sp;
  if (!pair) {
    s.kind = kBonus;
    unit[u] = s;
    return;
  }
  s.maxq = exp2(static_cast<double>(Mq) * G.k - Rq) / Sq;
  s.c = static_cast<float>(log2(Sq) - log2(Sp));
  const float2 xl = msg1_at(const_cast<char *>(static_cast<const char *>(gathered1)) + owner_of(G, x) * msg1,
                            G.B, G.gamma).x[b * G.gamma + j];
  s.xq0 = !(xl.x > -INFINITY);
  s.xp0 = !(xl.y > -INFINITY);
  if (!s.xq0 && !s.xp0) s.L = log2_prob(xl.y, Mp, Rp, Sp, G) - log2_prob(xl.x, Mq, Rq, Sq, G);
  int delta;
  switch (G.rule) {
    case SC_RULE_CHOW: delta = s.maxq < 1.0 - G.alpha; break;
    case SC_RULE_DIFF: delta = s.maxq < s.maxp - G.alpha; break;
    case SC_RULE_ALWAYS_DEFER: delta = 1; break;
    case SC_RULE_NEVER_DEFER: delta = 0; break;
    default:  // OPT (Eq. 10), D_TV in [0, 1]: decided outside the band
      if (s.maxq >= s.maxp) delta = 0;
      else if (s.maxq < s.maxp - G.alpha) delta = 1;
      else delta = -1;
  }
  if (delta < 0) s.kind = kNeedTV;
  else s.kind = !delta || accept_deferred(s, uj) ? kAccepted : kRejected;
  unit[u] = s;
}

// One CTA per (pair, slice) of a pair that needs D_TV: the slice's sum of
// S_q max(0, p - q).
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_tv_kernel(const E *__restrict__ q, const E *__restrict__ p, Geom G,
                                                      const UnitState *__restrict__ unit, float *__restrict__ tv_slot) {
  const int slot = blockIdx.x % G.slots, pr = blockIdx.x / G.slots;
  const int b = pr / G.gamma, j = pr % G.gamma;
  const UnitState &s = unit[b * (G.gamma + 1) + j];
  if (s.kind != kNeedTV) return;
  const int lo = slot * kL, n = min(kL, G.width - lo);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const E *rq = q_row(q, G, b, j, lo), *rp = p_row(p, G, b, j, lo);
  Group<E, kVec> gq[kRounds], gp[kRounds];
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gq[i].load(rq, group_pos(i, warp, lane), n);
    gp[i].load(rp, group_pos(i, warp, lane), n);
  }
  float acc = 0.0f, yq[8], yp[8];
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gq[i].get(rq, group_pos(i, warp, lane), n, yq);
    gp[i].get(rp, group_pos(i, warp, lane), n, yp);
#pragma unroll
    for (int t = 0; t < 8; ++t) acc = __fadd_rn(acc, res_weight(yq[t], yp[t], G.k, s.Rq, s.Rp, s.c));
  }
  acc = warp_sum(acc);
  __shared__ float red[kWarps];
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < kWarps; ++w) t = __fadd_rn(t, red[w]);
    tv_slot[static_cast<size_t>(pr) * G.slots + slot] = t;
  }
}

// One thread per pair: the rank's part of S_q D_TV, in slice order (0 for a
// pair that does not need it).
__global__ void shard_merge2_kernel(Geom G, const UnitState *__restrict__ unit, const float *__restrict__ tv_slot,
                                    double *__restrict__ send2) {
  const int pr = blockIdx.x * blockDim.x + threadIdx.x;
  if (pr >= G.B * G.gamma) return;
  const int b = pr / G.gamma, j = pr % G.gamma;
  double t = 0.0;
  if (unit[b * (G.gamma + 1) + j].kind == kNeedTV)
    for (int s = 0; s < G.slots; ++s) t += static_cast<double>(tv_slot[static_cast<size_t>(pr) * G.slots + s]);
  send2[pr] = t;
}

// ------------------------------------------------------------------ accept

// One thread per sequence: delta of the band pairs from D_TV (Eq. 10),
// acceptance, and j* = min{j : a_j = 0}.
__global__ void shard_accept_kernel(Geom G, const double *__restrict__ gathered2, size_t msg2_doubles,
                                    const float *__restrict__ uniforms, const UnitState *__restrict__ unit,
                                    SeqState *__restrict__ seq) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= G.B) return;
  SeqState st{G.gamma, 0};
  for (int j = 0; j <= G.gamma; ++j)
    if (unit[b * (G.gamma + 1) + j].kind == kBad) st.bad = 1;
  if (st.bad) {
    st.jstar = 0;
  } else {
    for (int j = 0; j < G.gamma; ++j) {
      const UnitState &s = unit[b * (G.gamma + 1) + j];
      bool acc = s.kind == kAccepted;
      if (s.kind == kNeedTV) {
        if (gathered2 == nullptr) {  // decided with OPT, accepted with another rule
          st.bad = 1;
          st.jstar = 0;
          break;
        }
        double R = 0.0;
        for (int r = 0; r < G.W; ++r) R += gathered2[r * msg2_doubles + b * G.gamma + j];
        const double tv = R / s.Sq;
        acc = !(s.maxq < s.maxp - G.alpha * tv) || accept_deferred(s, uniforms[b * (G.gamma + 1) + j]);
      }
      if (!acc) {
        st.jstar = j;
        break;
      }
    }
  }
  seq[b] = st;
}

// One CTA per (sequence, slice): the weights of the row the sequence draws
// from, per segment (lane sums left to right in f32, warp prefix in double),
// and the slice's total, in segment order.
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_mass_kernel(const E *__restrict__ q, const E *__restrict__ p, Geom G,
                                                        const UnitState *__restrict__ unit,
                                                        const SeqState *__restrict__ seq,
                                                        double *__restrict__ seg_tot, double *__restrict__ slot_mass) {
  const int slot = blockIdx.x % G.slots, b = blockIdx.x / G.slots;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const SeqState st = seq[b];
  __shared__ double seg[kSegs];
  double *out = seg_tot + (static_cast<size_t>(b) * G.slots + slot) * kSegs;
  if (st.bad) {
    if (threadIdx.x < kSegs) out[threadIdx.x] = 0.0;
    if (threadIdx.x == 0) slot_mass[static_cast<size_t>(b) * G.slots + slot] = 0.0;
    return;
  }
  const int j = st.jstar;
  const bool pair = j < G.gamma;
  const UnitState &s = unit[b * (G.gamma + 1) + j];
  const int lo = slot * kL, n = min(kL, G.width - lo);
  const E *rp = p_row(p, G, b, j, lo);
  const E *rq = pair ? q_row(q, G, b, j, lo) : rp;
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    float w[8];
    const float ls = lane_weights<E, kVec>(rq, rp, pair, group_pos(i, warp, lane), n, G, s.Rq, s.Rp, s.c, w);
    const double incl = warp_scan_d(static_cast<double>(ls), lane);
    if (lane == 31) seg[i * kWarps + warp] = incl;
  }
  __syncthreads();
  if (threadIdx.x < kSegs) out[threadIdx.x] = seg[threadIdx.x];
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int g = 0; g < kSegs; ++g) t += seg[g];
    slot_mass[static_cast<size_t>(b) * G.slots + slot] = t;
  }
}

// One thread per sequence: the rank's total weight, in slice order.
__global__ void shard_merge3_kernel(Geom G, const double *__restrict__ slot_mass, double *__restrict__ send3) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= G.B) return;
  double t = 0.0;
  for (int s = 0; s < G.slots; ++s) t += slot_mass[static_cast<size_t>(b) * G.slots + s];
  send3[b] = t;
}

// ------------------------------------------------------------------ draw

// First index i of a running sum of v[0..n) (in order, from 0) that exceeds t;
// -1 if none.  *before receives the running sum before it.
__device__ __forceinline__ int crossing(const double *v, int n, double t, double *before) {
  double acc = 0.0;
  for (int i = 0; i < n; ++i) {
    const double nx = acc + v[i];
    if (t < nx) {
      *before = acc;
      return i;
    }
    acc = nx;
  }
  *before = acc;
  return -1;
}
__device__ __forceinline__ int last_positive(const double *v, int n) {
  for (int i = n - 1; i >= 0; --i)
    if (v[i] > 0.0) return i;
  return -1;
}

// One warp per sequence: the rank holding u R (R the total weight over all
// ranks, u = uniforms[b][gamma]) draws the token; the others send -1.
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_draw_kernel(const E *__restrict__ q, const E *__restrict__ p, Geom G,
                                                        const double *__restrict__ gathered3, size_t msg3_doubles,
                                                        const float *__restrict__ uniforms,
                                                        const UnitState *__restrict__ unit,
                                                        const SeqState *__restrict__ seq,
                                                        const double *__restrict__ seg_tot,
                                                        const double *__restrict__ slot_mass,
                                                        int32_t *__restrict__ send4) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * kWarps + warp;
  if (b >= G.B) return;
  const SeqState st = seq[b];
  int slot = -1, sg = -1;
  double t = 0.0;
  if (lane == 0 && !st.bad) {
    double tot[SC_SHARD_MAX], R = 0.0;
    for (int r = 0; r < G.W; ++r) {
      tot[r] = gathered3[r * msg3_doubles + b];
      R += tot[r];
    }
    if (R > 0.0) {
      // t is u R relative to the start of the part searched next; +inf once
      // rounding has put u R past the end of a part, which then resolves to
      // the last positive weight of every level below
      const double target = static_cast<double>(uniforms[b * (G.gamma + 1) + G.gamma]) * R;
      double before;
      int r = crossing(tot, G.W, target, &before);
      if (r < 0) {
        r = last_positive(tot, G.W);
        t = INFINITY;
      } else {
        t = target - before;
      }
      if (r == G.rank) {
        const double *sm = slot_mass + static_cast<size_t>(b) * G.slots;
        slot = crossing(sm, G.slots, t, &before);
        if (slot < 0) {
          slot = last_positive(sm, G.slots);
          t = INFINITY;
        } else {
          t -= before;
        }
        if (slot >= 0) {
          const double *seg = seg_tot + (static_cast<size_t>(b) * G.slots + slot) * kSegs;
          sg = crossing(seg, kSegs, t, &before);
          if (sg < 0) {
            sg = last_positive(seg, kSegs);
            t = INFINITY;
          } else {
            t -= before;
          }
        }
      }
    }
  }
  slot = __shfl_sync(0xFFFFFFFFu, slot, 0);
  sg = __shfl_sync(0xFFFFFFFFu, sg, 0);
  t = __shfl_sync(0xFFFFFFFFu, t, 0);
  if (slot < 0 || sg < 0) {
    if (lane == 0) send4[b] = -1;
    return;
  }
  const int j = st.jstar;
  const bool pair = j < G.gamma;
  const UnitState &s = unit[b * (G.gamma + 1) + j];
  const int lo = slot * kL, n = min(kL, G.width - lo);
  const E *rp = p_row(p, G, b, j, lo);
  const E *rq = pair ? q_row(q, G, b, j, lo) : rp;
  float w[8];
  const int e = sg * kSeg + lane * 8;
  const float ls = lane_weights<E, kVec>(rq, rp, pair, e, n, G, s.Rq, s.Rp, s.c, w);
  const double incl = warp_scan_d(static_cast<double>(ls), lane);
  double excl = __shfl_up_sync(0xFFFFFFFFu, incl, 1);
  if (lane == 0) excl = 0.0;
  const unsigned hit = __ballot_sync(0xFFFFFFFFu, t < incl);
  int tok = -1;
  if (hit != 0u) {
    const int l = __ffs(hit) - 1;
    if (lane == l) {
      double acc = excl;
      int last = -1;
      for (int i = 0; i < 8; ++i) {
        if (w[i] > 0.0f) last = i;
        acc += static_cast<double>(w[i]);
        if (t < acc && w[i] > 0.0f) {
          last = i;
          break;
        }
      }
      tok = last >= 0 ? e + last : -1;
    }
    tok = __shfl_sync(0xFFFFFFFFu, tok, l);
  }
  if (tok < 0) {  // rounding past the segment's end: its last positive weight
    int last = -1;
    for (int i = 0; i < 8; ++i)
      if (w[i] > 0.0f) last = e + i;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xFFFFFFFFu, last, o));
    tok = last;
  }
  if (lane == 0) send4[b] = tok >= 0 ? G.begin[G.rank] + lo + tok : -1;
}

// One thread per sequence: the token of the rank that drew it.
__global__ void shard_finish_kernel(int B, int W, const int32_t *__restrict__ gathered4, size_t msg4_ints,
                                    const SeqState *__restrict__ seq, int32_t *__restrict__ num_accepted,
                                    int32_t *__restrict__ next_token) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const SeqState st = seq[b];
  int tok = -1;
  for (int r = 0; r < W; ++r) tok = max(tok, gathered4[r * msg4_ints + b]);
  num_accepted[b] = st.bad ? 0 : st.jstar;
  next_token[b] = st.bad ? -1 : tok;
}

// ------------------------------------------------------------------ host

bool device_accessible(const void *p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

int slots_of(int width) { return (width + kL - 1) / kL; }

// Checks shared by every phase; fills the geometry.
int make_geom(int B, int gamma, int W, int rank, const int *shard_begin, float temperature, int rule,
              float alpha, long long ld, Geom *G) {
  if (B < 1 || gamma < 1 || gamma > SC_MAX_GAMMA || W < 1 || W > SC_SHARD_MAX || rank < 0 || rank >= W ||
      shard_begin == nullptr)
    return SC_ERR_INVALID_ARG;
  if (shard_begin[0] != 0) return SC_ERR_INVALID_ARG;
  for (int r = 0; r < W; ++r)
    if (!(shard_begin[r + 1] > shard_begin[r])) return SC_ERR_INVALID_ARG;
  if (!(temperature > 0.0f) || !std::isfinite(temperature)) return SC_ERR_INVALID_ARG;
  if (rule < SC_RULE_CHOW || rule > SC_RULE_NEVER_DEFER) return SC_ERR_INVALID_ARG;
  if (!(alpha >= 0.0f && alpha <= 1.0f)) return SC_ERR_INVALID_ARG;
  G->B = B;
  G->gamma = gamma;
  G->W = W;
  G->rank = rank;
  for (int r = 0; r <= SC_SHARD_MAX; ++r) G->begin[r] = r <= W ? shard_begin[r] : shard_begin[W];
  G->width = shard_begin[rank + 1] - shard_begin[rank];
  if (ld < G->width) return SC_ERR_INVALID_ARG;
  G->slots = slots_of(G->width);
  G->ld = ld;
  G->kd = 1.4426950408889634 / static_cast<double>(temperature);
  G->k = static_cast<float>(G->kd);
  G->rule = rule;
  G->alpha = alpha;
  return SC_OK;
}

size_t elt_size(sc_dtype d) { return d == SC_BF16 ? 2 : 4; }

bool vec_ok(const void *base, sc_dtype d, long long ld) {
  return (reinterpret_cast<uintptr_t>(base) & 15u) == 0 && (static_cast<size_t>(ld) * elt_size(d)) % 16 == 0;
}

int check_work(const Geom &G, void *ws, size_t ws_bytes) {
  if (ws == nullptr || !device_accessible(ws)) return SC_ERR_WORKSPACE;
  if (ws_bytes < work_layout(G.B, G.gamma, G.slots, nullptr, nullptr)) return SC_ERR_WORKSPACE;
  return SC_OK;
}

int launched() { return cudaGetLastError() == cudaSuccess ? SC_OK : SC_ERR_CUDA; }

// Launch kernel template K<E, kVec> for the logit type and alignment.
#define SC_SHARD_DISPATCH(KERNEL, GRID, ...)                                                          \
  do {                                                                                                \
    if (dtype == SC_BF16) {                                                                           \
      const uint16_t *q_ = static_cast<const uint16_t *>(draft), *p_ = static_cast<const uint16_t *>(target); \
      if (vec) KERNEL<uint16_t, true><<<GRID, kT, 0, stream>>>(q_, p_, __VA_ARGS__);                   \
      else KERNEL<uint16_t, false><<<GRID, kT, 0, stream>>>(q_, p_, __VA_ARGS__);                      \
    } else {                                                                                          \
      const float *q_ = static_cast<const float *>(draft), *p_ = static_cast<const float *>(target);  \
      if (vec) KERNEL<float, true><<<GRID, kT, 0, stream>>>(q_, p_, __VA_ARGS__);                      \
      else KERNEL<float, false><<<GRID, kT, 0, stream>>>(q_, p_, __VA_ARGS__);                         \
    }                                                                                                 \
  } while (0)

int check_logits(const void *draft, const void *target, sc_dtype dtype) {
  if (dtype != SC_F32 && dtype != SC_BF16) return SC_ERR_INVALID_ARG;
  if (!draft || !target || !device_accessible(draft) || !device_accessible(target)) return SC_ERR_INVALID_ARG;
  return SC_OK;
}

}  // namespace

extern "C" {

size_t sc_shard_message_bytes(int B, int gamma, int message) {
  if (B < 1 || gamma < 1) return 0;
  return msg_bytes(B, gamma, message);
}

size_t sc_shard_workspace_bytes(int B, int gamma, int width, sc_dtype dtype) {
  (void)dtype;
  if (B < 1 || gamma < 1 || width < 1) return 0;
  return work_layout(B, gamma, slots_of(width), nullptr, nullptr);
}

int sc_shard_pass1(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                   const int32_t *draft_tokens, int B, int gamma, int W, int rank,
                   const int *shard_begin, float temperature, void *workspace,
                   size_t workspace_bytes, void *send1, cudaStream_t stream) {
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, SC_RULE_CHOW, 0.0f, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!draft_tokens || !send1 || !device_accessible(draft_tokens) || !device_accessible(send1)))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  const Msg1 m = msg1_at(send1, B, gamma);
  const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
  const int units = B * (gamma + 1);
  SC_SHARD_DISPATCH(shard_pass1_kernel, units * G.slots, draft_tokens, G, w.slot_rec, m.x);
  shard_merge1_kernel<<<(units + kT - 1) / kT, kT, 0, stream>>>(G, w.slot_rec, m.rec);
  return launched();
}

int sc_shard_decide(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                    const void *gathered1, const int32_t *draft_tokens, const float *uniforms,
                    int B, int gamma, int W, int rank, const int *shard_begin, sc_rule rule,
                    float alpha, float temperature, void *workspace, size_t workspace_bytes,
                    void *send2, int32_t *device_status, cudaStream_t stream) {
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, rule, alpha, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!gathered1 || !draft_tokens || !uniforms || !send2 || !device_accessible(gathered1) ||
                      !device_accessible(draft_tokens) || !device_accessible(uniforms) ||
                      !device_accessible(send2) || (device_status && !device_accessible(device_status))))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  const int units = B * (gamma + 1), pairs = B * gamma;
  shard_decide_kernel<<<(units + 127) / 128, 128, 0, stream>>>(G, gathered1, msg_bytes(B, gamma, 1), draft_tokens,
                                                               uniforms, w.unit, device_status);
  if (rule == SC_RULE_OPT) {
    const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
    SC_SHARD_DISPATCH(shard_tv_kernel, pairs * G.slots, G, w.unit, w.tv_slot);
    shard_merge2_kernel<<<(pairs + kT - 1) / kT, kT, 0, stream>>>(G, w.unit, w.tv_slot,
                                                                  static_cast<double *>(send2));
  }
  return launched();
}

int sc_shard_accept(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                    const void *gathered2, const float *uniforms, int B, int gamma, int W,
                    int rank, const int *shard_begin, sc_rule rule, float alpha,
                    float temperature, void *workspace, size_t workspace_bytes, void *send3,
                    cudaStream_t stream) {
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, rule, alpha, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!uniforms || !send3 || !device_accessible(uniforms) || !device_accessible(send3)))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK && rule == SC_RULE_OPT && (!gathered2 || !device_accessible(gathered2))) rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  shard_accept_kernel<<<(B + 127) / 128, 128, 0, stream>>>(
      G, rule == SC_RULE_OPT ? static_cast<const double *>(gathered2) : nullptr,
      msg_bytes(B, gamma, 2) / sizeof(double), uniforms, w.unit, w.seq);
  const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
  SC_SHARD_DISPATCH(shard_mass_kernel, B * G.slots, G, w.unit, w.seq, w.seg_tot, w.slot_mass);
  shard_merge3_kernel<<<(B + kT - 1) / kT, kT, 0, stream>>>(G, w.slot_mass, static_cast<double *>(send3));
  return launched();
}

int sc_shard_draw(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                  const void *gathered3, const float *uniforms, int B, int gamma, int W, int rank,
                  const int *shard_begin, float temperature, void *workspace,
                  size_t workspace_bytes, void *send4, cudaStream_t stream) {
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, SC_RULE_CHOW, 0.0f, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!gathered3 || !uniforms || !send4 || !device_accessible(gathered3) ||
                      !device_accessible(uniforms) || !device_accessible(send4)))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
  SC_SHARD_DISPATCH(shard_draw_kernel, (B + kWarps - 1) / kWarps, G, static_cast<const double *>(gathered3),
                    msg_bytes(B, gamma, 3) / sizeof(double), uniforms, w.unit, w.seq, w.seg_tot, w.slot_mass,
                    static_cast<int32_t *>(send4));
  return launched();
}

int sc_shard_finish(const void *gathered4, int B, int gamma, int W, const void *workspace,
                    size_t workspace_bytes, int32_t *num_accepted, int32_t *next_token,
                    cudaStream_t stream) {
  if (B < 1 || gamma < 1 || gamma > SC_MAX_GAMMA || W < 1 || W > SC_SHARD_MAX) return SC_ERR_INVALID_ARG;
  if (!gathered4 || !num_accepted || !next_token || !device_accessible(gathered4) ||
      !device_accessible(num_accepted) || !device_accessible(next_token))
    return SC_ERR_INVALID_ARG;
  // the sequence states sit at the same offset for every shard width
  if (workspace == nullptr || !device_accessible(workspace)) return SC_ERR_WORKSPACE;
  if (workspace_bytes < work_layout(B, gamma, 1, nullptr, nullptr)) return SC_ERR_WORKSPACE;
  Work w;
  work_layout(B, gamma, 1, const_cast<void *>(workspace), &w);
  shard_finish_kernel<<<(B + kT - 1) / kT, kT, 0, stream>>>(B, W, static_cast<const int32_t *>(gathered4),
                                                            msg_bytes(B, gamma, 4) / sizeof(int32_t), w.seq,
                                                            num_accepted, next_token);
  return launched();
}

}  // extern "C"
