// GB300 (sm_103a) verification step of speculative cascades with the
// vocabulary split across W GPUs (include/sc_shard.h).
//
// Each rank holds the logits of a contiguous range of tokens of every row.
// The step is Algorithm 4 with Algorithm 5's target, for the deferral rules of
// Table 1 (and delta = 1, delta = 0), written as phases with an all-gather of
// a small message between consecutive phases:
//
//   pass 1   grid (unit, slice): every CTA reads one slice of kL logits of a
//            row pair (or of the bonus target row) with coalesced 16-byte
//            loads, all of them in flight before any arithmetic, takes the
//            slice's maxima (packed bf16x2 max trees), and sums
//            2^{fma(y, k, -fl(max k))} per row (packed f32x2 arithmetic) --
//            per warp, kept for the lower bound on D_TV below, and per slice;
//            OPT pairs also sum the Bhattacharyya terms 2^{(a + b)/2}; a
//            second kernel merges the rank's slices per unit   -> message 1
//   decide   one warp per unit merges the W ranks' partials in rank order
//            (identical on every rank): M, S, max q, max p, delta by the rule,
//            and the acceptance test.  OPT pairs in the band
//            max p - alpha <= max q < max p need D_TV (Eq. 10): every rank
//            settles delta = 1 where the Hellinger bound D_TV <= (1 - BC^2)^{1/2}
//            decides; for the rest the rank sends its part of the lower bound
//            sum_t max(0, P_t - Q_t) over its warps' token sets -> message 2
//   tv       (OPT) the summed lower bound settles delta = 0 where it decides;
//            the rest take a TV pass, a grid walking the work list of
//            (pair, slice) items, summing max(0, 2^{b + c} - 2^a) =
//            S_q max(0, p - q) over the rank's part of the row -> message 3
//   accept   one warp per sequence finishes the band pairs (Eq. 10) and
//            settles j*; a grid (sequence, slice) sums the residual weights of
//            row j* of rejected sequences; a sequence that reaches the bonus
//            row takes p's slice sums from pass 1             -> message 4
//   draw     one CTA per sequence: the rank holding u R finds the slice, the
//            segment and the token in ascending token order; the other ranks
//            send -1                                          -> message 5
//   finish   one thread per sequence takes the drawing rank's token.
//
// Every sum that a later phase splits again (rank totals into slices, slices
// into segments, segments into lanes) is formed in the same order by the
// same code in both places, so a search never falls between two levels; a
// rounding gap at the bottom level falls back to the last positive weight of
// the segment.

#include "sc_shard.h"

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cfloat>
#include <cmath>
#include <cstdint>

namespace {

#ifndef SC_SHARD_THREADS
#define SC_SHARD_THREADS 128
#endif

constexpr int kT = SC_SHARD_THREADS;    // threads per CTA
constexpr int kWarps = kT / 32;         // warps per CTA
constexpr int kSeg = 256;               // tokens per segment: one warp, 8 per lane
constexpr int kRounds = 4;              // segments per warp per slice
constexpr int kSegs = kRounds * kWarps; // segments per slice
constexpr int kL = kSeg * kSegs;        // tokens per slice (4096 at 128 threads)

enum UnitKind : int { kAccepted = 0, kRejected = 1, kNeedTV = 2, kBonus = 3, kBad = 4 };

// Decision state of one unit (row pair (b, j < gamma) or bonus row (b, gamma)).
struct UnitState {
  double Sq, Sp;      // sums of 2^{fma(y, k, -R)} over the whole row
  double maxq, maxp;  // max_v q(v), max_v p(v)
  float Lhi, Llo;     // log2 p(x) - log2 q(x) (both finite) as a double-float hi + lo
  float Rq, Rp;       // exponent references fl(M k)
  float c;            // log2(S_q / S_p) rounded to f32: the residual weights' shift
  int kind;           // UnitKind
  int xq0, xp0;       // q(x) = 0, p(x) = 0 (masked logits at the draft token)
  int settled0;       // kNeedTV: the lower bound on D_TV (every rank's part) settles delta = 0
};

// Pass-1 record of one (unit, slice), every sum relative to the references
// fl(m_q k) and fl(m_p k) of the slice's maxima.
struct SlotRec {
  float4 ms;             // (m_q, s_q, m_p, s_p)
  float bc;              // OPT pairs: sum of 2^{(a + b)/2}, a and b the exponents of q and p
  float pad[3];
  float2 set[kWarps];    // (s_q, s_p) over the tokens of each warp (the lower bound's sets)
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
  float kl;   // log2(e) / T - k: with k, log2(e) / T to twice f32 precision
  double kd;  // log2(e) / T in double
  int rule;
  double alpha;
};
static_assert(sizeof(SlotRec) % 16 == 0, "SlotRec layout");

__host__ __device__ inline size_t align16(size_t n) { return (n + 15) & ~static_cast<size_t>(15); }

struct Msg1 {
  float4 *rec;  // [units] (m_q, s_q, m_p, s_p) of this rank
  float2 *x;    // [pairs] the draft token's logits (q, p), from the rank holding it
  float *bc;    // [pairs] OPT: the rank's sum of 2^{(a + b)/2}, relative to its references
};
__host__ __device__ inline Msg1 msg1_at(void *base, int B, int gamma) {
  const size_t units = static_cast<size_t>(B) * (gamma + 1), pairs = static_cast<size_t>(B) * gamma;
  char *p = static_cast<char *>(base);
  const size_t o1 = align16(units * sizeof(float4)), o2 = o1 + align16(pairs * sizeof(float2));
  return Msg1{reinterpret_cast<float4 *>(p), reinterpret_cast<float2 *>(p + o1), reinterpret_cast<float *>(p + o2)};
}
size_t msg_bytes(int B, int gamma, int k) {
  const size_t units = static_cast<size_t>(B) * (gamma + 1), pairs = static_cast<size_t>(B) * gamma;
  switch (k) {
    case 1: return align16(units * sizeof(float4)) + align16(pairs * sizeof(float2)) + align16(pairs * sizeof(float));
    case 2: return align16(pairs * sizeof(float));
    case 3: return align16(pairs * sizeof(double));
    case 4: return align16(static_cast<size_t>(B) * sizeof(double));
    case 5: return align16(static_cast<size_t>(B) * sizeof(int32_t));
    default: return 0;
  }
}

// Workspace of one rank.  The per-sequence and per-unit states come first, at
// offsets that do not depend on the shard's width (sc_shard_finish does not know it).
struct Work {
  SeqState *seq;       // [B]
  UnitState *unit;     // [units]
  int *tv_count;       // [1] pairs in tv_list
  int *tv_list;        // [pairs] the pairs that take the TV pass (any order)
  SlotRec *slot_rec;   // [units][slots]
  float *tv_slot;      // [pairs][slots]
  double *slot_mass;   // [B][slots]
};
__host__ __device__ inline size_t work_layout(int B, int gamma, int slots, void *base, Work *w) {
  const size_t units = static_cast<size_t>(B) * (gamma + 1), pairs = static_cast<size_t>(B) * gamma;
  const size_t sizes[7] = {static_cast<size_t>(B) * sizeof(SeqState), units * sizeof(UnitState), sizeof(int),
                           pairs * sizeof(int), units * slots * sizeof(SlotRec), pairs * slots * sizeof(float),
                           static_cast<size_t>(B) * slots * sizeof(double)};
  size_t off[7], total = 0;
  for (int i = 0; i < 7; ++i) {
    off[i] = total;
    total += (sizes[i] + 255) & ~static_cast<size_t>(255);
  }
  if (w != nullptr) {
    char *p = static_cast<char *>(base);
    w->seq = reinterpret_cast<SeqState *>(p + off[0]);
    w->unit = reinterpret_cast<UnitState *>(p + off[1]);
    w->tv_count = reinterpret_cast<int *>(p + off[2]);
    w->tv_list = reinterpret_cast<int *>(p + off[3]);
    w->slot_rec = reinterpret_cast<SlotRec *>(p + off[4]);
    w->tv_slot = reinterpret_cast<float *>(p + off[5]);
    w->slot_mass = reinterpret_cast<double *>(p + off[6]);
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
  // streaming loads (evict first): the slice is read once here
  __device__ __forceinline__ void load(const uint16_t *s) { v = __ldcs(reinterpret_cast<const uint4 *>(s)); }
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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Inclusive prefix over the warp's lanes (f32, Hillis-Steele: the same
// additions in the same order wherever it runs).
__device__ __forceinline__ float warp_scan(float v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xFFFFFFFFu, v, o);
    if (lane >= o) v = __fadd_rn(v, t);
  }
  return v;
}

// The 8 weights of one lane's group of the row a sequence draws from -- the
// residual S_q max(0, p - q) of a rejected pair, or 2^{b} (proportional to p)
// of the bonus row -- from its loaded groups, and their sum in f32, left to
// right.  The mass pass and the draw both take a segment's weights from here.
template <typename E, bool kVec>
__device__ __forceinline__ float lane_weights(const Group<E, kVec> &gq, const Group<E, kVec> &gp, const E *rq,
                                              const E *rp, bool pair, int e, int n, const Geom &G, float Rq, float Rp,
                                              float c, float (&w)[8]) {
  float yp[8];
  gp.get(rp, e, n, yp);
  if (pair) {
    float yq[8];
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

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

__device__ __forceinline__ __nv_bfloat162 as_bf162(uint32_t w) { return *reinterpret_cast<__nv_bfloat162 *>(&w); }
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

// This thread's sums over its groups (kRounds groups of 8 logits per row):
// sq = sum 2^a, sp = sum 2^b, bc = sum 2^{(a + b)/2}, a = fma(y_q, k, -Rq),
// b = fma(y_p, k, -Rp).  Any logit type and slice; the bf16 full-slice case
// has its own packed version below.
template <typename E, bool kVec>
__device__ __forceinline__ void thread_sums(const Group<E, kVec> (&gq)[kRounds], const Group<E, kVec> (&gp)[kRounds],
                                            const E *rq, const E *rp, int n, int warp, int lane, bool pair,
                                            bool bcw, float k, float Rq, float Rp, float &sq, float &sp, float &bc) {
  sq = sp = bc = 0.0f;
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    float yp[8];
    gp[i].get(rp, group_pos(i, warp, lane), n, yp);
    if (pair) {
      float yq[8];
      gq[i].get(rq, group_pos(i, warp, lane), n, yq);
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const float a = fmaf(yq[t], k, -Rq), b = fmaf(yp[t], k, -Rp);
        sq = __fadd_rn(sq, ex2(a));
        sp = __fadd_rn(sp, ex2(b));
        if (bcw) bc = __fadd_rn(bc, ex2(0.5f * __fadd_rn(a, b)));
      }
    } else {
#pragma unroll
      for (int t = 0; t < 8; ++t) sp = __fadd_rn(sp, ex2(fmaf(yp[t], k, -Rp)));
    }
  }
}

// bf16 rows, every group whole: the maximum by packed bf16x2 max trees over
// the raw words, the exponent arguments by packed f32x2 FMAs, the sums by
// packed f32x2 adds.
__device__ __forceinline__ float bf16_max(const Group<uint16_t, true> (&g)[kRounds]) {
  __nv_bfloat162 m = __hmax2(as_bf162(g[0].raw.v.x), as_bf162(g[0].raw.v.y));
  m = __hmax2(m, __hmax2(as_bf162(g[0].raw.v.z), as_bf162(g[0].raw.v.w)));
#pragma unroll
  for (int i = 1; i < kRounds; ++i) {
    m = __hmax2(m, __hmax2(as_bf162(g[i].raw.v.x), as_bf162(g[i].raw.v.y)));
    m = __hmax2(m, __hmax2(as_bf162(g[i].raw.v.z), as_bf162(g[i].raw.v.w)));
  }
  return fmaxf(__low2float(m), __high2float(m));
}

template <bool kPair, bool kBC>
__device__ __forceinline__ void bf16_sums(const Group<uint16_t, true> (&gq)[kRounds],
                                          const Group<uint16_t, true> (&gp)[kRounds], float k, float Rq, float Rp,
                                          float &sq, float &sp, float &bc) {
  const float2 kk = make_float2(k, k), nq = make_float2(-Rq, -Rq), np = make_float2(-Rp, -Rp);
  const float2 half = make_float2(0.5f, 0.5f);
  float2 aq = make_float2(0.0f, 0.0f), ap = aq, ab = aq;
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    const uint32_t wp[4] = {gp[i].raw.v.x, gp[i].raw.v.y, gp[i].raw.v.z, gp[i].raw.v.w};
    uint32_t wq[4] = {0u, 0u, 0u, 0u};
    if (kPair) {
      wq[0] = gq[i].raw.v.x; wq[1] = gq[i].raw.v.y; wq[2] = gq[i].raw.v.z; wq[3] = gq[i].raw.v.w;
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const float2 b = __ffma2_rn(bf16x2_to_float2(wp[t]), kk, np);
      ap = __fadd2_rn(ap, make_float2(ex2(b.x), ex2(b.y)));
      if (kPair) {
        const float2 a = __ffma2_rn(bf16x2_to_float2(wq[t]), kk, nq);
        aq = __fadd2_rn(aq, make_float2(ex2(a.x), ex2(a.y)));
        if (kBC) {
          const float2 h = __fmul2_rn(__fadd2_rn(a, b), half);
          ab = __fadd2_rn(ab, make_float2(ex2(h.x), ex2(h.y)));
        }
      }
    }
  }
  sq = __fadd_rn(aq.x, aq.y);
  sp = __fadd_rn(ap.x, ap.y);
  bc = __fadd_rn(ab.x, ab.y);
}

// One CTA per (unit, slice): the slice's maxima, its sums relative to their
// references, per warp and in total, and for OPT pairs the Bhattacharyya sum;
// the CTA holding a pair's draft token also records the token's two logits.
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_pass1_kernel(const E *__restrict__ q, const E *__restrict__ p,
                                                         const int32_t *__restrict__ tokens, Geom G,
                                                         SlotRec *__restrict__ slot_rec, float2 *__restrict__ xrec) {
  const int slot = blockIdx.x % G.slots, u = blockIdx.x / G.slots;
  const int b = unit_b(u, G.gamma), j = unit_j(u, G.gamma);
  const bool pair = j < G.gamma, bcw = pair && G.rule == SC_RULE_OPT;
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
  constexpr bool kPacked = kVec && sizeof(E) == 2;
  const bool packed = kPacked && n == kL;  // every group whole
  float mq = -INFINITY, mp = -INFINITY;
  if constexpr (kPacked) {
    if (packed) {
      mp = bf16_max(gp);
      if (pair) mq = bf16_max(gq);
    }
  }
  if (!packed) {
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
  }
  // the slice's maxima: one reference per row for every sum of the CTA
  __shared__ float smax[2][kWarps];
  __shared__ float3 ssum[kWarps];
  mq = warp_max(mq);
  mp = warp_max(mp);
  if (lane == 0) {
    smax[0][warp] = mq;
    smax[1][warp] = mp;
  }
  __syncthreads();
  float Mq = smax[0][0], Mp = smax[1][0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) {
    Mq = fmaxf(Mq, smax[0][w]);
    Mp = fmaxf(Mp, smax[1][w]);
  }
  const float Rq = ref_of(Mq, G.k), Rp = ref_of(Mp, G.k);
  float sq, sp, bc;
  bool done = false;
  if constexpr (kPacked) {
    if (packed) {
      if (!pair) bf16_sums<false, false>(gq, gp, G.k, Rq, Rp, sq, sp, bc);
      else if (bcw) bf16_sums<true, true>(gq, gp, G.k, Rq, Rp, sq, sp, bc);
      else bf16_sums<true, false>(gq, gp, G.k, Rq, Rp, sq, sp, bc);
      done = true;
    }
  }
  if (!done) thread_sums<E, kVec>(gq, gp, rq, rp, n, warp, lane, pair, bcw, G.k, Rq, Rp, sq, sp, bc);
  sq = warp_sum(sq);
  sp = warp_sum(sp);
  if (bcw) bc = warp_sum(bc);
  SlotRec *rec = slot_rec + static_cast<size_t>(u) * G.slots + slot;
  if (lane == 0) {
    rec->set[warp] = make_float2(sq, sp);
    ssum[warp] = make_float3(sq, sp, bc);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float Sq = 0.0f, Sp = 0.0f, BC = 0.0f;
    for (int w = 0; w < kWarps; ++w) {
      Sq = __fadd_rn(Sq, ssum[w].x);
      Sp = __fadd_rn(Sp, ssum[w].y);
      BC = __fadd_rn(BC, ssum[w].z);
    }
    rec->ms = make_float4(Mq, Sq, Mp, Sp);
    rec->bc = bcw ? BC : 0.0f;
    if (pair) {
      const int x = tokens[b * G.gamma + j] - G.begin[G.rank] - lo;
      if (x >= 0 && x < n) xrec[b * G.gamma + j] = make_float2(Raw8<E>::at(rq, x), Raw8<E>::at(rp, x));
    }
  }
}

// One warp per unit: the rank's (m, s) over its slices and, for OPT pairs, its
// Bhattacharyya sum relative to the rank's references (lanes over slices).
__global__ void shard_merge1_kernel(Geom G, const SlotRec *__restrict__ slot_rec, float4 *__restrict__ rec,
                                    float *__restrict__ bcm) {
  const int lane = threadIdx.x & 31;
  const int u = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (u >= G.B * (G.gamma + 1)) return;
  const SlotRec *r = slot_rec + static_cast<size_t>(u) * G.slots;
  float mq = -INFINITY, mp = -INFINITY;
  for (int s = lane; s < G.slots; s += 32) {
    mq = fmaxf(mq, r[s].ms.x);
    mp = fmaxf(mp, r[s].ms.z);
  }
  const float Mq = warp_max(mq), Mp = warp_max(mp);
  const float RQ = ref_of(Mq, G.k), RP = ref_of(Mp, G.k);
  float Sq = 0.0f, Sp = 0.0f, BC = 0.0f;
  for (int s = lane; s < G.slots; s += 32) {
    const float dq = ref_of(r[s].ms.x, G.k) - RQ, dp = ref_of(r[s].ms.z, G.k) - RP;
    Sq = fmaf(r[s].ms.y, ex2(dq), Sq);
    Sp = fmaf(r[s].ms.w, ex2(dp), Sp);
    BC = fmaf(r[s].bc, ex2(0.5f * (dq + dp)), BC);
  }
  Sq = warp_sum(Sq);
  Sp = warp_sum(Sp);
  BC = warp_sum(BC);
  if (lane == 0) {
    rec[u] = make_float4(Mq, Sq, Mp, Sp);
    const int b = unit_b(u, G.gamma), j = unit_j(u, G.gamma);
    if (j < G.gamma) bcm[b * G.gamma + j] = BC;
  }
}

// ------------------------------------------------------------------ decide

__device__ __forceinline__ int owner_of(const Geom &G, int x) {
  int r = 0;
  while (r + 1 < G.W && x >= G.begin[r + 1]) ++r;
  return r;
}

// Merge of the W ranks' (m, s) of one row, in rank order: R = fl(M k) and
// S = sum_r s_r 2^{fl(m_r k) - R}, as pass 1 merges its warps and slices.
__device__ __forceinline__ void merge_ranks(const float4 *const *recs, int W, size_t u, bool p_row_,
                                            float k, float &M, float &R, float &S) {
  M = -INFINITY;
  for (int r = 0; r < W; ++r) M = fmaxf(M, p_row_ ? recs[r][u].z : recs[r][u].x);
  R = ref_of(M, k);
  S = 0.0f;
  for (int r = 0; r < W; ++r) {
    const float m = p_row_ ? recs[r][u].z : recs[r][u].x, s = p_row_ ? recs[r][u].w : recs[r][u].y;
    S = fmaf(s, ex2(ref_of(m, k) - R), S);
  }
}

// Double-float f32 arithmetic (a value is hi + lo, |lo| <= ulp(hi) / 2): the
// precision of the acceptance ratio at f32 speed (this GPU's f64 rate is low).
// two_sum: a + b = s + e exactly (Knuth); an FMA gives a product's rounding error.
__device__ __forceinline__ float2 two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return make_float2(s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb)));
}
__device__ __forceinline__ float2 quick_norm(float hi, float lo) {
  const float s = __fadd_rn(hi, lo);
  return make_float2(s, __fsub_rn(lo, __fsub_rn(s, hi)));
}

// log2 p(x) - log2 q(x) for logits yp, yq of rows with maxima Mp, Mq, references
// Rp, Rq and sums Sp, Sq (of 2^{fma(y, k, -R)}):
//   log2 p(y) = y (k + kl) - R - log2 S - M kl = y k - R + (y - M) kl - log2 S,
// the f32 factor k of the sums' exponents corrected to log2(e) / T = k + kl for
// each row's dominant terms (y near M).  The difference of the two is formed
// from exact pieces: yp - yq by two_sum, its product with k by an FMA.
__device__ __forceinline__ float2 log_ratio(float yp, float yq, float Mp, float Mq, float Rp, float Rq, float Sp,
                                            float Sq, float k, float kl) {
  const float2 d = two_sum(yp, -yq);                      // yp - yq = d.x + d.y
  const float dk = __fmul_rn(d.x, k), dke = fmaf(d.x, k, -dk);  // d.x k = dk + dke
  const float2 r = two_sum(Rp, -Rq);                      // Rp - Rq
  const float2 t = two_sum(dk, -r.x);
  const float corr = __fmul_rn(__fsub_rn(__fsub_rn(yp, Mp), __fsub_rn(yq, Mq)), kl);
  const float lo = __fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(t.y, dke), __fsub_rn(__fmul_rn(d.y, k), r.y)), corr),
                             log2f(Sq / Sp));
  return quick_norm(t.x, lo);
}

// Acceptance of the draft token when delta = 1 (pi = p): [u < min(1, p(x)/q(x))];
// q(x) = 0 accepts, p(x) = 0 < q(x) rejects.  2^L = 2^hi (1 + lo ln 2).
__device__ __forceinline__ bool accept_deferred(const UnitState &s, float u) {
  if (s.xq0) return true;
  if (s.xp0) return false;
  if (s.Lhi > 0.0f || (s.Lhi == 0.0f && s.Llo >= 0.0f)) return true;
  return u < exp2f(s.Lhi) * fmaf(s.Llo, 0.69314718f, 1.0f);
}

// Margin by which a bound on D_TV must clear the OPT threshold to settle delta
// without the exact value (far above the bounds' rounding, ~1e-6).
constexpr double kBoundMargin = 1e-4;

// This rank's part of the lower bound D_TV >= sum_t max(0, P_t - Q_t), the sets
// t its warps' tokens of every slice, P_t and Q_t their masses under p and q
// (the lanes of a warp take the slices in turn; every lane returns the total).
__device__ __forceinline__ float rank_lower_bound(const Geom &G, const SlotRec *r, float Rq, float Rp, float Sq,
                                                  float Sp, int lane) {
  float lb = 0.0f;
  for (int s = lane; s < G.slots; s += 32) {
    const float fq = ex2(ref_of(r[s].ms.x, G.k) - Rq) / Sq;
    const float fp = ex2(ref_of(r[s].ms.z, G.k) - Rp) / Sp;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) lb += fmaxf(0.0f, r[s].set[w].y * fp - r[s].set[w].x * fq);
  }
  return warp_sum(lb);
}

__global__ void shard_decide_kernel(Geom G, const void *__restrict__ gathered1, size_t msg1,
                                    const int32_t *__restrict__ tokens, const float *__restrict__ uniforms,
                                    const SlotRec *__restrict__ slot_rec, UnitState *__restrict__ unit,
                                    float *__restrict__ send2, int32_t *status) {
  // one warp per unit: every lane merges the ranks' records (the same values);
  // the lanes share the lower bound's slices; lane 0 writes
  const int lane = threadIdx.x & 31;
  const int u = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (u >= G.B * (G.gamma + 1)) return;
  const int b = unit_b(u, G.gamma), j = unit_j(u, G.gamma);
  const bool pair = j < G.gamma;
  const float4 *recs[SC_SHARD_MAX];
  for (int r = 0; r < G.W; ++r)
    recs[r] = msg1_at(const_cast<char *>(static_cast<const char *>(gathered1)) + r * msg1, G.B, G.gamma).rec;
  UnitState s{};
  float Mq = 0.0f, Mp, Rq = 0.0f, Rp, Sq = 1.0f, Sp;
  merge_ranks(recs, G.W, u, true, G.k, Mp, Rp, Sp);
  if (pair) merge_ranks(recs, G.W, u, false, G.k, Mq, Rq, Sq);
  int err = 0;
  const float uj = uniforms[b * (G.gamma + 1) + j];
  if (!(uj >= 0.0f && uj < 1.0f)) err |= SC_DEV_BAD_UNIFORM;
  if (!(isfinite(Sp) && Sp > 0.0f && Mp < INFINITY) || (pair && !(isfinite(Sq) && Sq > 0.0f && Mq < INFINITY)))
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
    if (lane == 0) {
      if (status) atomicOr(status, err);
      unit[u] = s;
    }
    return;
  }
  s.maxp = ex2(fmaf(Mp, G.k, -Rp)) / Sp;
  if (!pair) {
    s.kind = kBonus;
    if (lane == 0) unit[u] = s;
    return;
  }
  s.maxq = ex2(fmaf(Mq, G.k, -Rq)) / Sq;
  s.c = log2f(Sq / Sp);
  const float2 xl = msg1_at(const_cast<char *>(static_cast<const char *>(gathered1)) + owner_of(G, x) * msg1,
                            G.B, G.gamma).x[b * G.gamma + j];
  s.xq0 = !(xl.x > -INFINITY);
  s.xp0 = !(xl.y > -INFINITY);
  if (!s.xq0 && !s.xp0) {
    const float2 L = log_ratio(xl.y, xl.x, Mp, Mq, Rp, Rq, Sp, Sq, G.k, G.kl);
    s.Lhi = L.x;
    s.Llo = L.y;
  }
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
  if (delta < 0) {
    // Hellinger: D_TV <= (1 - BC^2)^{1/2}, BC = sum_v (q p)^{1/2} from every
    // rank's Bhattacharyya sum (the same on every rank), BC taken 2e-4 low
    // against the rounding of its f32 sums
    float bcs = 0.0f;
    for (int r = 0; r < G.W; ++r) {
      const char *m = static_cast<const char *>(gathered1) + r * msg1;
      const Msg1 mr = msg1_at(const_cast<char *>(m), G.B, G.gamma);
      const float4 v = mr.rec[u];
      bcs = fmaf(mr.bc[b * G.gamma + j], ex2(0.5f * ((ref_of(v.x, G.k) - Rq) + (ref_of(v.z, G.k) - Rp))), bcs);
    }
    const float bcl = bcs * rsqrtf(Sq) * rsqrtf(Sp) * (1.0f - 2e-4f);
    const float ub = sqrtf(fmaxf(0.0f, 1.0f - bcl * bcl)) * (1.0f + 1e-6f);
    if (s.maxq < s.maxp - G.alpha * ub - kBoundMargin) {
      delta = 1;
    } else {
      // this rank's part of the lower bound, summed over the ranks by sc_shard_tv
      const float lb = rank_lower_bound(G, slot_rec + static_cast<size_t>(u) * G.slots, Rq, Rp, Sq, Sp, lane);
      if (lane == 0) send2[b * G.gamma + j] = lb;
    }
  }
  if (delta < 0) {
    s.kind = kNeedTV;
  } else if (lane == 0) {
    s.kind = !delta || accept_deferred(s, uj) ? kAccepted : kRejected;
  }
  if (lane == 0) unit[u] = s;
}

// The TV pass: a grid of CTAs walks the work list of (pair, slice) items of the
// pairs no bound settled, each item the slice's sum of S_q max(0, p - q).
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_tv_kernel(const E *__restrict__ q, const E *__restrict__ p, Geom G,
                                                      const UnitState *__restrict__ unit,
                                                      const int *__restrict__ tv_count, const int *__restrict__ tv_list,
                                                      float *__restrict__ tv_slot) {
  const int items = *tv_count * G.slots;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ float red[kWarps];
  for (int it = blockIdx.x; it < items; it += gridDim.x) {
    const int pr = tv_list[it / G.slots], slot = it % G.slots;
    const int b = pr / G.gamma, j = pr % G.gamma;
    const UnitState &s = unit[b * (G.gamma + 1) + j];
    const int lo = slot * kL, n = min(kL, G.width - lo);
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
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      float t = 0.0f;
      for (int w = 0; w < kWarps; ++w) t = __fadd_rn(t, red[w]);
      tv_slot[static_cast<size_t>(pr) * G.slots + slot] = t;
    }
    __syncthreads();
  }
}

// One thread per pair (OPT): the lower bound on D_TV summed over the ranks'
// parts (rank order, the same on every rank) settles delta = 0 where it
// decides; the other band pairs join the TV pass's work list.
__global__ void shard_settle_kernel(Geom G, const float *__restrict__ gathered2, size_t msg2_floats,
                                    UnitState *__restrict__ unit, int *__restrict__ tv_count,
                                    int *__restrict__ tv_list) {
  const int pr = blockIdx.x * blockDim.x + threadIdx.x;
  if (pr >= G.B * G.gamma) return;
  const int b = pr / G.gamma, j = pr % G.gamma;
  UnitState &st = unit[b * (G.gamma + 1) + j];
  if (st.kind != kNeedTV) return;
  float lb = 0.0f;
  for (int r = 0; r < G.W; ++r) lb += gathered2[r * msg2_floats + pr];
  st.settled0 = st.maxq >= st.maxp - G.alpha * lb + kBoundMargin;
  if (!st.settled0) tv_list[atomicAdd(tv_count, 1)] = pr;
}

// One thread per pair: the rank's part of S_q D_TV, in slice order (0 for a
// pair that takes no TV pass).
__global__ void shard_merge_tv_kernel(Geom G, const UnitState *__restrict__ unit, const float *__restrict__ tv_slot,
                                      double *__restrict__ send3) {
  const int pr = blockIdx.x * blockDim.x + threadIdx.x;
  if (pr >= G.B * G.gamma) return;
  const int b = pr / G.gamma, j = pr % G.gamma;
  const UnitState &st = unit[b * (G.gamma + 1) + j];
  double t = 0.0;
  if (st.kind == kNeedTV && !st.settled0)
    for (int s = 0; s < G.slots; ++s) t += static_cast<double>(tv_slot[static_cast<size_t>(pr) * G.slots + s]);
  send3[pr] = t;
}

// ------------------------------------------------------------------ accept

// One warp per sequence (lane j takes position j): delta of the band pairs
// from D_TV (Eq. 10), acceptance, and j* = min{j : a_j = 0}.
__global__ void shard_accept_kernel(Geom G, const double *__restrict__ gathered3, size_t msg3_doubles,
                                    const float *__restrict__ uniforms, const UnitState *__restrict__ unit,
                                    SeqState *__restrict__ seq) {
  const int lane = threadIdx.x & 31;
  const int b = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (b >= G.B) return;
  const UnitState *us = unit + static_cast<size_t>(b) * (G.gamma + 1);
  int bad = 0;
  for (int j = lane; j <= G.gamma; j += 32)
    bad |= us[j].kind == kBad || (us[j].kind == kNeedTV && gathered3 == nullptr);  // (decided as OPT, accepted as not)
  bad = __any_sync(0xFFFFFFFFu, bad);
  int jstar = G.gamma;
  for (int j0 = 0; !bad && j0 < G.gamma; j0 += 32) {
    const int j = j0 + lane;
    bool rej = false;
    if (j < G.gamma) {
      const UnitState &s = us[j];
      bool acc = s.kind == kAccepted;
      if (s.kind == kNeedTV) {
        double R = 0.0;
        if (!s.settled0)
          for (int r = 0; r < G.W; ++r) R += gathered3[r * msg3_doubles + b * G.gamma + j];
        const double tv = static_cast<float>(R) / static_cast<float>(s.Sq);  // (f32 division: f64 is slow here)
        acc = s.settled0 || !(s.maxq < s.maxp - G.alpha * tv) || accept_deferred(s, uniforms[b * (G.gamma + 1) + j]);
      }
      rej = !acc;
    }
    const unsigned r = __ballot_sync(0xFFFFFFFFu, rej);
    if (r != 0u) {
      jstar = j0 + __ffs(r) - 1;
      break;
    }
  }
  if (lane == 0) seq[b] = SeqState{bad ? 0 : jstar, bad};
}

// One CTA per (sequence, slice) of a sequence rejected at j* < gamma: the
// slice's total residual weight S_q max(0, p - q) of row j*.  (A sequence that
// reaches the bonus row draws from p, whose slice sums pass 1 already holds.)
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_mass_kernel(const E *__restrict__ q, const E *__restrict__ p, Geom G,
                                                        const UnitState *__restrict__ unit,
                                                        const SeqState *__restrict__ seq,
                                                        double *__restrict__ slot_mass) {
  const int slot = blockIdx.x % G.slots, b = blockIdx.x / G.slots;
  const SeqState st = seq[b];
  if (st.bad || st.jstar >= G.gamma) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = st.jstar;
  const UnitState &s = unit[b * (G.gamma + 1) + j];
  const int lo = slot * kL, n = min(kL, G.width - lo);
  const E *rq = q_row(q, G, b, j, lo), *rp = p_row(p, G, b, j, lo);
  Group<E, kVec> gq[kRounds], gp[kRounds];
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gq[i].load(rq, group_pos(i, warp, lane), n);
    gp[i].load(rp, group_pos(i, warp, lane), n);
  }
  float acc = 0.0f;
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    float w[8];
    acc = __fadd_rn(acc, lane_weights<E, kVec>(gq[i], gp[i], rq, rp, true, group_pos(i, warp, lane), n, G, s.Rq,
                                               s.Rp, s.c, w));
  }
  acc = warp_sum(acc);
  __shared__ float red[kWarps];
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < kWarps; ++w) t = __fadd_rn(t, red[w]);
    slot_mass[static_cast<size_t>(b) * G.slots + slot] = t;
  }
}

// The weight of slice `slot` of the row sequence b draws from, in the row's
// frame (the residual S_q max(0, p - q), or 2^{fma(y, k, -R_p)} of the bonus
// row, R_p its global reference); the rank's totals and the draw's search add
// these in slice order.  *frame receives the slice's own scale: its weights are
// computed as frame * (the value above); 1 for a residual, 2^{R_p - r_slot} for
// the bonus row, whose pass-1 sum is relative to the slice's reference r_slot.
__device__ __forceinline__ double slice_weight(const Geom &G, int b, int slot, int jstar, const UnitState *unit,
                                               const SlotRec *slot_rec, const double *slot_mass, float *ref) {
  if (jstar < G.gamma) {
    *ref = 0.0f;
    return slot_mass[static_cast<size_t>(b) * G.slots + slot];
  }
  const int u = b * (G.gamma + 1) + G.gamma;
  const SlotRec &r = slot_rec[static_cast<size_t>(u) * G.slots + slot];
  *ref = ref_of(r.ms.z, G.k);
  return static_cast<double>(r.ms.w) * static_cast<double>(ex2(*ref - unit[u].Rp));
}

// The slice weights of sequence b (slice_weight), computed by a warp's lanes
// and added in slice order (every lane forms the same sums): the total, the
// first slice whose running sum exceeds t (-1: none) with the sum before it,
// and the last slice with weight.
struct SliceSearch {
  int slot;
  double before;
  double total;
  int last;
};
__device__ __forceinline__ SliceSearch search_slices(const Geom &G, int b, int jstar, const UnitState *unit,
                                                     const SlotRec *slot_rec, const double *slot_mass, double t,
                                                     int lane) {
  SliceSearch r{-1, 0.0, 0.0, -1};
  for (int base = 0; base < G.slots; base += 32) {
    float ref;
    const double m = base + lane < G.slots ? slice_weight(G, b, base + lane, jstar, unit, slot_rec, slot_mass, &ref)
                                           : 0.0;
    const int n = min(32, G.slots - base);
    for (int i = 0; i < n; ++i) {
      const double mi = __shfl_sync(0xFFFFFFFFu, m, i);
      if (mi > 0.0) r.last = base + i;
      if (r.slot < 0 && t < r.total + mi) {
        r.slot = base + i;
        r.before = r.total;
      }
      r.total += mi;
    }
  }
  return r;
}

// One warp per sequence: the rank's total weight, in slice order.
__global__ void shard_merge3_kernel(Geom G, const UnitState *__restrict__ unit, const SeqState *__restrict__ seq,
                                    const SlotRec *__restrict__ slot_rec, const double *__restrict__ slot_mass,
                                    double *__restrict__ send3) {
  const int lane = threadIdx.x & 31;
  const int b = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (b >= G.B) return;
  const SeqState st = seq[b];
  const double t = st.bad ? 0.0 : search_slices(G, b, st.jstar, unit, slot_rec, slot_mass, INFINITY, lane).total;
  if (lane == 0) send3[b] = t;
}

// ------------------------------------------------------------------ draw

// One CTA per sequence: the rank holding u R (R the total weight over all
// ranks, u = uniforms[b][gamma]) draws the token.  Warp 0 finds the rank and
// then the slice holding u R; every warp computes the weights of its segments
// of that slice (the pass-1 layout) and their warp scans; thread 0 finds the
// segment holding u R from the segment totals in order, and the warp that holds
// the segment finds the token.  The other ranks send -1.
template <typename E, bool kVec>
__global__ void __launch_bounds__(kT) shard_draw_kernel(const E *__restrict__ q, const E *__restrict__ p, Geom G,
                                                        const double *__restrict__ gathered3, size_t msg3_doubles,
                                                        const float *__restrict__ uniforms,
                                                        const UnitState *__restrict__ unit,
                                                        const SeqState *__restrict__ seq,
                                                        const SlotRec *__restrict__ slot_rec,
                                                        const double *__restrict__ slot_mass,
                                                        int32_t *__restrict__ send4) {
  const int b = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const SeqState st = seq[b];
  __shared__ int s_slot, s_seg, s_tok;
  __shared__ float s_ref;
  __shared__ double s_t;
  __shared__ float segw[kSegs];
  __shared__ int lastw[kWarps];
  if (warp == 0) {
    int slot = -1;
    float sref = 0.0f;
    double t = 0.0;  // u R past the start of the part searched next (+inf: past the end of a part)
    if (!st.bad) {
      double R = 0.0, before = 0.0;
      int r = -1, rlast = -1;
      const double mine = lane < G.W ? gathered3[lane * msg3_doubles + b] : 0.0;
      double tot[SC_SHARD_MAX];
      for (int i = 0; i < G.W; ++i) {
        tot[i] = __shfl_sync(0xFFFFFFFFu, mine, i);
        R += tot[i];
      }
      const double target = static_cast<double>(uniforms[b * (G.gamma + 1) + G.gamma]) * R;
      double acc = 0.0;
      for (int i = 0; i < G.W; ++i) {
        if (tot[i] > 0.0) rlast = i;
        if (r < 0 && target < acc + tot[i]) {
          r = i;
          before = acc;
        }
        acc += tot[i];
      }
      if (R > 0.0) {
        if (r < 0) {
          r = rlast;
          t = INFINITY;
        } else {
          t = target - before;
        }
        if (r == G.rank) {
          const SliceSearch ss = search_slices(G, b, st.jstar, unit, slot_rec, slot_mass, t, lane);
          if (ss.slot >= 0) {
            slot = ss.slot;
            t -= ss.before;
          } else {
            slot = ss.last;
            t = INFINITY;
          }
          if (slot >= 0) slice_weight(G, b, slot, st.jstar, unit, slot_rec, slot_mass, &sref);
        }
      }
    }
    if (lane == 0) {
      s_slot = slot;
      s_ref = sref;
      s_t = t;
    }
  }
  __syncthreads();
  const int slot = s_slot;
  if (slot < 0) {
    if (threadIdx.x == 0) send4[b] = -1;
    return;
  }
  const int j = st.jstar;
  const bool pair = j < G.gamma;
  const UnitState &s = unit[b * (G.gamma + 1) + j];
  // the bonus row's weights in its slice's own frame, 2^{fma(y, k, -r_slot)}
  const float Rw = pair ? s.Rp : s_ref;
  double t = s_t;
  if (!pair && t < INFINITY) t /= static_cast<double>(ex2(s_ref - s.Rp));
  const int lo = slot * kL, n = min(kL, G.width - lo);
  const E *rp = p_row(p, G, b, j, lo);
  const E *rq = pair ? q_row(q, G, b, j, lo) : rp;
  Group<E, kVec> gq[kRounds], gp[kRounds];
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    gp[i].load(rp, group_pos(i, warp, lane), n);
    if (pair) gq[i].load(rq, group_pos(i, warp, lane), n);
  }
  float w[kRounds][8], incl[kRounds];
  int lastpos = -1;
#pragma unroll
  for (int i = 0; i < kRounds; ++i) {
    const int e = group_pos(i, warp, lane);
    const float ls = lane_weights<E, kVec>(gq[i], gp[i], rq, rp, pair, e, n, G, s.Rq, Rw, s.c, w[i]);
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (w[i][k] > 0.0f) lastpos = max(lastpos, e + k);
    incl[i] = warp_scan(ls, lane);
    if (lane == 31) segw[i * kWarps + warp] = incl[i];
  }
  lastpos = __reduce_max_sync(0xFFFFFFFFu, lastpos);
  if (lane == 0) lastw[warp] = lastpos;
  __syncthreads();
  if (threadIdx.x == 0) {
    int g = -1;
    double acc = 0.0;
    for (int i = 0; i < kSegs; ++i) {
      if (t < acc + static_cast<double>(segw[i])) {
        g = i;
        break;
      }
      acc += static_cast<double>(segw[i]);
    }
    s_seg = g;
    s_t = t - acc;
    int last = -1;
    for (int i = 0; i < kWarps; ++i) last = max(last, lastw[i]);
    s_tok = last;  // rounding past the slice's end: its last positive weight
  }
  __syncthreads();
  const int g = s_seg;
  if (g >= 0 && warp == g % kWarps) {
    const double ts = s_t;
    const int round = g / kWarps;
    int cand = -1;
#pragma unroll
    for (int i = 0; i < kRounds; ++i) {
      if (i != round) continue;
      const unsigned hit = __ballot_sync(0xFFFFFFFFu, ts < static_cast<double>(incl[i]));
      if (hit != 0u) {
        const int l = __ffs(hit) - 1;
        float excl = __shfl_up_sync(0xFFFFFFFFu, incl[i], 1);
        if (lane == 0) excl = 0.0f;
        if (lane == l) {
          double acc = excl;
          int lk = -1;
          for (int k = 0; k < 8; ++k) {
            if (w[i][k] > 0.0f) lk = k;
            acc += static_cast<double>(w[i][k]);
            if (ts < acc && w[i][k] > 0.0f) {
              lk = k;
              break;
            }
          }
          cand = lk >= 0 ? group_pos(i, warp, lane) + lk : -1;
        }
        cand = __shfl_sync(0xFFFFFFFFu, cand, l);
      }
    }
    if (lane == 0 && cand >= 0) s_tok = cand;
  }
  __syncthreads();
  if (threadIdx.x == 0) send4[b] = s_tok >= 0 ? G.begin[G.rank] + lo + s_tok : -1;
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

// Set by each entry point: its stream is being captured into a CUDA graph; the
// pointer checks then reject only null pointers, so that nothing but the
// launches happens inside the capture sequence.
thread_local bool t_capturing = false;

bool capturing(cudaStream_t stream) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(stream, &st) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return st != cudaStreamCaptureStatusNone;
}

bool device_accessible(const void *p) {
  if (!p) return false;
  if (t_capturing) return true;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

int slots_of(int width) { return (width + kL - 1) / kL; }

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return 132;
  }
  return n;
}

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
  // grids: B (gamma + 1) slices for pass 1, a warp per unit for the merges
  if (static_cast<double>(B) * (gamma + 1) * std::max(G->slots, 32) > 2147483647.0) return SC_ERR_INVALID_ARG;
  G->ld = ld;
  G->kd = 1.4426950408889634 / static_cast<double>(temperature);
  G->k = static_cast<float>(G->kd);
  G->kl = static_cast<float>(G->kd - static_cast<double>(G->k));
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
                   const int *shard_begin, float temperature, sc_rule rule, void *workspace,
                   size_t workspace_bytes, void *send1, cudaStream_t stream) {
  t_capturing = capturing(stream);
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, rule, 0.0f, ld, &G);
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
  shard_merge1_kernel<<<(units * 32 + kT - 1) / kT, kT, 0, stream>>>(G, w.slot_rec, m.rec, m.bc);
  return launched();
}

int sc_shard_decide(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                    const void *gathered1, const int32_t *draft_tokens, const float *uniforms,
                    int B, int gamma, int W, int rank, const int *shard_begin, sc_rule rule,
                    float alpha, float temperature, void *workspace, size_t workspace_bytes,
                    void *send2, int32_t *device_status, cudaStream_t stream) {
  t_capturing = capturing(stream);
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, rule, alpha, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!gathered1 || !draft_tokens || !uniforms || !device_accessible(gathered1) ||
                      !device_accessible(draft_tokens) || !device_accessible(uniforms) ||
                      (rule == SC_RULE_OPT && (!send2 || !device_accessible(send2))) ||
                      (device_status && !device_accessible(device_status))))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  const int units = B * (gamma + 1);
  shard_decide_kernel<<<(units * 32 + kT - 1) / kT, kT, 0, stream>>>(G, gathered1, msg_bytes(B, gamma, 1), draft_tokens,
                                                               uniforms, w.slot_rec, w.unit,
                                                               static_cast<float *>(send2), device_status);
  return launched();
}

int sc_shard_tv(const void *draft, const void *target, sc_dtype dtype, int64_t ld, const void *gathered2,
                int B, int gamma, int W, int rank, const int *shard_begin, sc_rule rule, float alpha,
                float temperature, void *workspace, size_t workspace_bytes, void *send3, cudaStream_t stream) {
  t_capturing = capturing(stream);
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, rule, alpha, ld, &G);
  if (rc == SC_OK && rule != SC_RULE_OPT) rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!gathered2 || !send3 || !device_accessible(gathered2) || !device_accessible(send3)))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  const int pairs = B * gamma;
  if (cudaMemsetAsync(w.tv_count, 0, sizeof(int), stream) != cudaSuccess) return SC_ERR_CUDA;
  shard_settle_kernel<<<(pairs + kT - 1) / kT, kT, 0, stream>>>(G, static_cast<const float *>(gathered2),
                                                                msg_bytes(B, gamma, 2) / sizeof(float), w.unit,
                                                                w.tv_count, w.tv_list);
  const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
  const int grid = std::min(pairs * G.slots, 8 * sm_count());  // CTAs walking the TV work list
  SC_SHARD_DISPATCH(shard_tv_kernel, grid, G, w.unit, w.tv_count, w.tv_list, w.tv_slot);
  shard_merge_tv_kernel<<<(pairs + kT - 1) / kT, kT, 0, stream>>>(G, w.unit, w.tv_slot, static_cast<double *>(send3));
  return launched();
}

int sc_shard_accept(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                    const void *gathered3, const float *uniforms, int B, int gamma, int W,
                    int rank, const int *shard_begin, sc_rule rule, float alpha,
                    float temperature, void *workspace, size_t workspace_bytes, void *send4,
                    cudaStream_t stream) {
  t_capturing = capturing(stream);
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, rule, alpha, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!uniforms || !send4 || !device_accessible(uniforms) || !device_accessible(send4)))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK && rule == SC_RULE_OPT && (!gathered3 || !device_accessible(gathered3))) rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  shard_accept_kernel<<<(B * 32 + kT - 1) / kT, kT, 0, stream>>>(
      G, rule == SC_RULE_OPT ? static_cast<const double *>(gathered3) : nullptr,
      msg_bytes(B, gamma, 3) / sizeof(double), uniforms, w.unit, w.seq);
  const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
  SC_SHARD_DISPATCH(shard_mass_kernel, B * G.slots, G, w.unit, w.seq, w.slot_mass);
  shard_merge3_kernel<<<(B * 32 + kT - 1) / kT, kT, 0, stream>>>(G, w.unit, w.seq, w.slot_rec, w.slot_mass,
                                                                 static_cast<double *>(send4));
  return launched();
}

int sc_shard_draw(const void *draft, const void *target, sc_dtype dtype, int64_t ld,
                  const void *gathered4, const float *uniforms, int B, int gamma, int W, int rank,
                  const int *shard_begin, float temperature, void *workspace,
                  size_t workspace_bytes, void *send5, cudaStream_t stream) {
  t_capturing = capturing(stream);
  Geom G;
  int rc = make_geom(B, gamma, W, rank, shard_begin, temperature, SC_RULE_CHOW, 0.0f, ld, &G);
  if (rc == SC_OK) rc = check_logits(draft, target, dtype);
  if (rc == SC_OK && (!gathered4 || !uniforms || !send5 || !device_accessible(gathered4) ||
                      !device_accessible(uniforms) || !device_accessible(send5)))
    rc = SC_ERR_INVALID_ARG;
  if (rc == SC_OK) rc = check_work(G, workspace, workspace_bytes);
  if (rc != SC_OK) return rc;
  Work w;
  work_layout(B, gamma, G.slots, workspace, &w);
  const bool vec = vec_ok(draft, dtype, ld) && vec_ok(target, dtype, ld);
  SC_SHARD_DISPATCH(shard_draw_kernel, B, G, static_cast<const double *>(gathered4),
                    msg_bytes(B, gamma, 4) / sizeof(double), uniforms, w.unit, w.seq, w.slot_rec, w.slot_mass,
                    static_cast<int32_t *>(send5));
  return launched();
}

int sc_shard_finish(const void *gathered5, int B, int gamma, int W, const void *workspace,
                    size_t workspace_bytes, int32_t *num_accepted, int32_t *next_token,
                    cudaStream_t stream) {
  t_capturing = capturing(stream);
  if (B < 1 || gamma < 1 || gamma > SC_MAX_GAMMA || W < 1 || W > SC_SHARD_MAX) return SC_ERR_INVALID_ARG;
  if (!gathered5 || !num_accepted || !next_token || !device_accessible(gathered5) ||
      !device_accessible(num_accepted) || !device_accessible(next_token))
    return SC_ERR_INVALID_ARG;
  // the sequence states sit at the same offset for every shard width
  if (workspace == nullptr || !device_accessible(workspace)) return SC_ERR_WORKSPACE;
  if (workspace_bytes < work_layout(B, gamma, 1, nullptr, nullptr)) return SC_ERR_WORKSPACE;
  Work w;
  work_layout(B, gamma, 1, const_cast<void *>(workspace), &w);
  shard_finish_kernel<<<(B + kT - 1) / kT, kT, 0, stream>>>(B, W, static_cast<const int32_t *>(gathered5),
                                                            msg_bytes(B, gamma, 5) / sizeof(int32_t), w.seq,
                                                            num_accepted, next_token);
  return launched();
}

}  // extern "C"
