// GB300 (sm_103a) verification step of speculative cascades.
//
// One call of sc_verify runs GenSpecSample's verification phase (Algorithm 4)
// with the SpecCascade target pi = (1 - delta) q + delta p (Algorithm 5, Eq. 6)
// for B sequences of gamma drafted positions over a V-token vocabulary, in ONE
// kernel launch:
//
//   unit  = one (b, j < gamma) row pair (draft row q_j, target row p_j), or the
//           bonus target row (b, gamma);
//   grid  = one thread-block cluster of C CTAs per unit; CTA r of the cluster
//           owns the vocabulary slice [r L, (r+1) L) of both rows;
//   HBM   = each logit is read once, by TMA bulk copies (cp.async.bulk) into the
//           owning CTA's shared memory, in chunks that each have an mbarrier;
//   pass1 = online max / sum-of-exp per thread while the chunks land, reduced
//           over warps, then over the cluster through distributed shared memory;
//   TV    = only when needed (sc_row_stats, or the OPT rule when the TV term can
//           change the decision): sum_v min(p_v, q_v) from shared memory,
//           D_TV = 1 - sum_v min(p_v, q_v) (Lemma 3);
//   accept= delta (Table 1) and the Bernoulli test u < pi(x)/q(x) on two
//           scalars, in fp64;
//   sample= a rejecting pair (residual max(0, p - q)) or the bonus row (p)
//           draws its token by inverse CDF: per-thread contiguous partial sums,
//           a block scan, a cluster scan of CTA totals, then one thread finds
//           the crossing element;
//   scan  = the last unit of a sequence to finish (atomic ticket, no waiting)
//           finds j* = min{j : a_j = 0} and writes the outputs.
//
// Exponentials use ex2.approx on (y - M) * log2(e)/T; (y - M) is exact for bf16
// logits.  Nothing in the kernel waits on another cluster; mbarrier waits are
// bounded and report SC_DEV_TIMEOUT instead of hanging.

#include "sc.h"

#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <cfloat>
#include <cmath>
#include <cstdint>
#include <algorithm>
#include <cstdlib>
#include <mutex>

namespace cg = cooperative_groups;

namespace {

constexpr int kNT = 256;                      // threads per CTA
constexpr int kNW = kNT / 32;                 // warps per CTA
constexpr int kVPT = 2;                       // 8-element vectors per thread per chunk
constexpr int kVecPerChunk = kNT * kVPT;      // 512 vectors = 4096 elements per chunk
constexpr int kChunkElems = kVecPerChunk * 8;
constexpr int kMaxChunks = 32;
constexpr int kMaxCluster = 16;
constexpr uint32_t kWaitLimit = 1u << 22;     // bounded mbarrier waits (~seconds)

enum Mode : int { kVerify = 0, kStats = 1 };

struct Params {
  const void *draft;
  const void *target;
  const int32_t *tokens;
  const float *uniforms;
  int B, gamma, V;
  int rule;
  float alpha;
  float temperature;
  float k;        // log2(e) / T
  double inv_t;   // 1 / T
  int L;          // slice length per CTA (multiple of 8 elements)
  int cluster;    // CTAs per unit
  int bulk;       // 1: TMA bulk copies, 0: per-thread loads (unaligned rows)
  int mode;
  int32_t *num_accepted;
  int32_t *next_token;
  float *row_info;
  float *max_q;
  float *max_p;
  float *tv;
  uint32_t *tickets;
  int32_t *unit_flags;
  int32_t *unit_cand;
  int32_t *status;
};

// ------------------------------------------------------------------ PTX helpers

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// Bounded wait for phase `parity` of an mbarrier; false on timeout.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  for (uint32_t i = 0; i < kWaitLimit; ++i) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(a), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}

// 1-D TMA bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// ------------------------------------------------------------------ logit types

template <typename E>
struct Elt;

template <>
struct Elt<uint16_t> {  // bf16 bit patterns
  static constexpr uint16_t kNegInf = 0xFF80u;
  __device__ __forceinline__ static void load8(const uint16_t *s, float (&y)[8]) {
    const uint4 v = *reinterpret_cast<const uint4 *>(s);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      y[2 * i] = __uint_as_float(w[i] << 16);
      y[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
  __device__ __forceinline__ static float at(const void *g, size_t i) {
    return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(g)[i]) << 16);
  }
};

template <>
struct Elt<float> {
  static constexpr float kNegInf = -INFINITY;
  __device__ __forceinline__ static void load8(const float *s, float (&y)[8]) {
    const float4 a = *reinterpret_cast<const float4 *>(s);
    const float4 b = *reinterpret_cast<const float4 *>(s + 4);
    y[0] = a.x; y[1] = a.y; y[2] = a.z; y[3] = a.w;
    y[4] = b.x; y[5] = b.y; y[6] = b.z; y[7] = b.w;
  }
  __device__ __forceinline__ static float at(const void *g, size_t i) {
    return static_cast<const float *>(g)[i];
  }
};

// ------------------------------------------------------------------ shared state

struct __align__(16) Shared {
  uint64_t bar[kMaxChunks];
  float4 part_ms;        // this CTA's (m_q, s_q, m_p, s_p), read by the cluster
  float part_tv;         // this CTA's sum of 2^min(a, b + c)
  float part_r;          // this CTA's total sampling weight
  int cand;              // sampled token (written remotely into rank 0)
  int timeout;
  float red[kNW][4];
  float wtot[kNW + 1];
  // row statistics, identical in every CTA of the cluster
  float Mq, Sq, Mp, Sp;
  float c;               // log2(S_q / S_p)
  float tv;
  int err, delta, need_tv, need_sample, accept;
  float qx, pix;
  double t_local;        // u * R minus the weight of the CTAs before the crossing one
  float ug;              // u[b][gamma], the residual / bonus draw
  int sample_here;       // 1: crossing inside this CTA, 2: take its last positive weight
};

__device__ __forceinline__ void ms_combine(float &m, float &s, float m2, float s2, float k) {
  const float mn = fmaxf(m, m2);
  s = s * ex2((m - mn) * k) + s2 * ex2((m2 - mn) * k);
  m = mn;
}

// Per-thread online max / sum of exp2((y - m) k) over this thread's vectors of
// one chunk (vectors vbeg + tid + i * kNT).
template <typename E>
__device__ __forceinline__ void online_chunk(const E *row, int vbeg, int vend, float k, float &m,
                                             float &s) {
  float y[kVPT][8];
  bool act[kVPT];
  float vmax = -FLT_MAX;
#pragma unroll
  for (int i = 0; i < kVPT; ++i) {
    const int v = vbeg + static_cast<int>(threadIdx.x) + i * kNT;
    act[i] = v < vend;
    if (act[i]) {
      Elt<E>::load8(row + 8 * v, y[i]);
#pragma unroll
      for (int e = 0; e < 8; ++e) vmax = fmaxf(vmax, y[i][e]);
    }
  }
  const float mn = fmaxf(m, vmax);
  float acc = s * ex2((m - mn) * k);
#pragma unroll
  for (int i = 0; i < kVPT; ++i)
    if (act[i]) {
#pragma unroll
      for (int e = 0; e < 8; ++e) acc += ex2((y[i][e] - mn) * k);
    }
  m = mn;
  s = acc;
}

// Row scalars in registers for the shared-memory passes.  With
// a_v = (y^q_v - M_q) k and b_v = (y^p_v - M_p) k (k = log2(e)/T):
//   q_v = 2^{a_v} / S_q,   p_v = 2^{b_v} / S_p = 2^{b_v + c} / S_q,   c = log2(S_q / S_p).
struct RowScalars {
  float Mq, Mp, k, c;
};

// Sampling weight of one element, up to the common factor 1/S_q:
// residual max(0, p - q) of a pair, or p of the bonus row.
template <bool kPair>
__device__ __forceinline__ float weight(float yq, float yp, const RowScalars &r) {
  if constexpr (kPair) {
    const float a = (yq - r.Mq) * r.k;
    const float b = fmaf(yp - r.Mp, r.k, r.c);
    return fmaxf(0.0f, ex2(b) - ex2(a));
  } else {
    return ex2((yp - r.Mp) * r.k);
  }
}

// f32 a, f64 t: (a > t) == (a > round_down_to_f32(t)).
__device__ __forceinline__ float f32_floor(double t) { return __double2float_rd(t); }

// Inverse-CDF draw over the cluster's slices.  Every thread of every CTA calls
// it; the chosen token is written into rank 0's Shared::cand, visible there
// after the caller's next cluster barrier.
template <typename E, bool kPair>
__device__ void sample_unit(const E *sq, const E *sp, int nv, int v0, Shared &sh,
                            const RowScalars &rs, float u, cg::cluster_group &cluster, int rank,
                            int C) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // contiguous ownership with an odd stride: conflict-free 16-byte shared loads
  const int G = ((nv + kNT - 1) / kNT) | 1;
  const int vb = tid * G, ve = min(nv, vb + G);
  float gt = 0.0f;
  for (int v = vb; v < ve; ++v) {
    float yq[8], yp[8];
    if constexpr (kPair) Elt<E>::load8(sq + 8 * v, yq);
    Elt<E>::load8(sp + 8 * v, yp);
#pragma unroll
    for (int e = 0; e < 8; ++e) gt += weight<kPair>(kPair ? yq[e] : 0.0f, yp[e], rs);
  }
  // block scan of the thread totals: warp inclusive scan, then warp offsets
  float incl = gt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += t;
  }
  const float prev = __shfl_up_sync(0xFFFFFFFFu, incl, 1);
  if (lane == 31) sh.wtot[warp] = incl;
  __syncthreads();
  if (tid == 0) {
    float acc = 0.0f;
    for (int w = 0; w < kNW; ++w) {
      const float t = sh.wtot[w];
      sh.wtot[w] = acc;  // becomes the warp offset
      acc = acc + t;
    }
    sh.wtot[kNW] = acc;
    sh.part_r = acc;
  }
  __syncthreads();
  const float woff = sh.wtot[warp];
  const float excl = lane == 0 ? woff : woff + prev;  // == previous thread's inclusive prefix
  const float inc = woff + incl;
  cluster.sync();  // totals of every CTA are published

  if (warp == 0) {
    float tot = 0.0f;
    if (lane < C) tot = *cluster.map_shared_rank(&sh.part_r, lane);
    // inclusive prefix over ranks in rank order (lane r: ranks 0..r)
    float pre = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xFFFFFFFFu, pre, o);
      if (lane >= o) pre += t;
    }
    const float R = __shfl_sync(0xFFFFFFFFu, pre, C - 1);
    float before = __shfl_up_sync(0xFFFFFFFFu, pre, 1);  // previous rank's inclusive prefix
    if (lane == 0) before = 0.0f;
    const double t = static_cast<double>(u) * static_cast<double>(R);
    const bool cross = lane < C && tot > 0.0f && t >= static_cast<double>(before) &&
                       t < static_cast<double>(pre);
    const unsigned cm = __ballot_sync(0xFFFFFFFFu, cross);
    const unsigned pm = __ballot_sync(0xFFFFFFFFu, lane < C && tot > 0.0f);
    const int cr = cm ? __ffs(cm) - 1 : -1;
    const float bcr = __shfl_sync(0xFFFFFFFFu, before, cr >= 0 ? cr : 0);
    if (lane == 0) {
      int here = 0;
      double tl = 0.0;
      if (R > 0.0f) {
        if (cr >= 0) {
          if (cr == rank) {
            here = 1;
            tl = t - static_cast<double>(bcr);
          }
        } else if (pm && 31 - __clz(pm) == rank) {
          here = 2;  // rounding left u R at the top: take the last positive weight
        }
      }
      sh.sample_here = here;
      sh.t_local = tl;
    }
  }
  __syncthreads();
  if (sh.sample_here == 1) {
    const double tl = sh.t_local;
    const int mine = (tl >= static_cast<double>(excl) && tl < static_cast<double>(inc)) ? 1 : 0;
    const int any = __syncthreads_or(mine);
    if (mine) {
      const float tf = f32_floor(tl - static_cast<double>(excl));
      float acc = 0.0f;
      int token = -1, lastpos = -1;
      for (int v = vb; v < ve && token < 0; ++v) {
        float yq[8], yp[8];
        if constexpr (kPair) Elt<E>::load8(sq + 8 * v, yq);
        Elt<E>::load8(sp + 8 * v, yp);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float w = weight<kPair>(kPair ? yq[e] : 0.0f, yp[e], rs);
          acc += w;
          if (w > 0.0f) lastpos = 8 * v + e;
          if (token < 0 && acc > tf) token = 8 * v + e;
        }
      }
      if (token < 0) token = lastpos;
      if (token >= 0) *cluster.map_shared_rank(&sh.cand, 0) = v0 + token;
    }
    if (!any && tid == 0) sh.sample_here = 2;  // rounding gap between the two scan levels
    __syncthreads();
  }
  if (sh.sample_here == 2) {
    // last positive weight of this CTA: the highest thread with gt > 0 scans
    const int mine = gt > 0.0f ? tid : -1;
    int best = mine;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) best = max(best, __shfl_xor_sync(0xFFFFFFFFu, best, o));
    if (lane == 0) sh.red[warp][0] = __int_as_float(best);
    __syncthreads();
    int top = -1;
    for (int w = 0; w < kNW; ++w) top = max(top, __float_as_int(sh.red[w][0]));
    if (tid == top) {
      int lastpos = -1;
      for (int v = vb; v < ve; ++v) {
        float yq[8], yp[8];
        if constexpr (kPair) Elt<E>::load8(sq + 8 * v, yq);
        Elt<E>::load8(sp + 8 * v, yp);
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (weight<kPair>(kPair ? yq[e] : 0.0f, yp[e], rs) > 0.0f) lastpos = 8 * v + e;
      }
      if (lastpos >= 0) *cluster.map_shared_rank(&sh.cand, 0) = v0 + lastpos;
    }
  }
}

// exp(a) for an f64 argument, to f32 accuracy without f64 transcendentals:
// a = hi + lo with hi = f32(a), exp(a) ~= expf(hi) (1 + lo).
__device__ __forceinline__ float exp_split(double a) {
  const float hi = static_cast<float>(a);
  const float lo = static_cast<float>(a - static_cast<double>(hi));
  return expf(hi) * (1.0f + lo);
}

// Acceptance of draft x (Algorithm 4): a = 1 when delta = 0 or q(x) <= pi(x),
// else a = [u < pi(x)/q(x)].  ln p(x) - ln q(x) is formed in f64 from exact
// logit differences, so the ratio carries only the f32 error of S_q / S_p.
__device__ __forceinline__ void accept_test(Shared &sh, float yqx, float ypx, float u,
                                            double invT) {
  const double dq = static_cast<double>(yqx) - static_cast<double>(sh.Mq);
  const double dp = static_cast<double>(ypx) - static_cast<double>(sh.Mp);
  const double lq = static_cast<double>(logf(sh.Sq)), lp = static_cast<double>(logf(sh.Sp));
  const float qx = exp_split(dq * invT - lq);
  const float px = exp_split(dp * invT - lp);
  int accept = 1;
  if (sh.delta) {
    const double L = (dp - dq) * invT + static_cast<double>(logf(sh.Sq / sh.Sp));
    if (L < 0.0) accept = u < exp_split(L);
  }
  sh.accept = accept;
  sh.qx = qx;
  sh.pix = sh.delta ? px : qx;
  sh.need_sample = !accept;
}

// ------------------------------------------------------------------ the kernel

template <typename E>
__global__ void __launch_bounds__(kNT, 3) sc_unit_kernel(const Params P) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  cg::cluster_group cluster = cg::this_cluster();
  const int C = P.cluster;
  const int rank = static_cast<int>(cluster.block_rank());
  const int unit = static_cast<int>(blockIdx.x) / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G1 = P.gamma + 1;

  int b, j;
  bool pair;
  if (P.mode == kVerify) {
    b = unit / G1;
    j = unit % G1;
    pair = j < P.gamma;
  } else {
    b = unit / P.gamma;
    j = unit % P.gamma;
    pair = true;
  }
  const size_t qoff = (static_cast<size_t>(b) * P.gamma + j) * P.V;
  const size_t poff = (static_cast<size_t>(b) * G1 + j) * P.V;
  const E *gq = static_cast<const E *>(P.draft) + qoff;
  const E *gp = static_cast<const E *>(P.target) + poff;
  const int v0 = rank * P.L;
  const int len = max(0, min(P.L, P.V - v0));
  const int lenp = (len + 7) & ~7;
  const int nv = lenp >> 3;
  const int nchunks = (len + kChunkElems - 1) / kChunkElems;

  E *sq = reinterpret_cast<E *>(smem_raw);
  E *sp = sq + P.L;
  Shared &sh = *reinterpret_cast<Shared *>(
      smem_raw + ((2 * static_cast<size_t>(P.L) * sizeof(E) + 15) & ~size_t(15)));

  // ---- stage the slices; thread 0 then prefetches the row's scalars
  float uj = 0.0f, ug = 0.0f, yqx = 0.0f, ypx = 0.0f;
  int x = 0;
  if (tid == 0) {
    sh.cand = -1;
    sh.timeout = 0;
    if (P.bulk) {
      for (int c = 0; c < nchunks; ++c) mbar_init(&sh.bar[c], 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      for (int c = 0; c < nchunks; ++c) {
        const int e0 = c * kChunkElems, e1 = min(len, e0 + kChunkElems);
        const uint32_t bytes = static_cast<uint32_t>(e1 - e0) * sizeof(E);
        mbar_expect_tx(&sh.bar[c], pair ? 2 * bytes : bytes);
        if (pair) bulk_g2s(sq + e0, gq + v0 + e0, bytes, &sh.bar[c]);
        bulk_g2s(sp + e0, gp + v0 + e0, bytes, &sh.bar[c]);
      }
    }
    if (P.mode == kVerify) {
      uj = P.uniforms[static_cast<size_t>(b) * G1 + j];
      ug = P.uniforms[static_cast<size_t>(b) * G1 + P.gamma];
      if (pair) {
        x = P.tokens[static_cast<size_t>(b) * P.gamma + j];
        if (x >= 0 && x < P.V) {
          yqx = Elt<E>::at(P.draft, qoff + x);
          ypx = Elt<E>::at(P.target, poff + x);
        }
      }
    }
  }
  if (!P.bulk) {
    for (int i = tid; i < len; i += kNT) {
      if (pair) sq[i] = gq[v0 + i];
      sp[i] = gp[v0 + i];
    }
  }
  for (int i = len + tid; i < lenp; i += kNT) {  // -inf padding: weight 0 everywhere
    sq[i] = Elt<E>::kNegInf;
    sp[i] = Elt<E>::kNegInf;
  }
  __syncthreads();

  // ---- pass 1: online max and sum of exponentials while the chunks land
  const float k = P.k;
  float mq = -FLT_MAX, s_q = 0.0f, mp = -FLT_MAX, s_p = 0.0f;
  int tmo = 0;
  const int nchunk_loop = P.bulk ? nchunks : (nv + kVecPerChunk - 1) / kVecPerChunk;
  for (int c = 0; c < nchunk_loop; ++c) {
    if (P.bulk && !mbar_wait(&sh.bar[c], 0)) tmo = 1;
    const int vbeg = c * kVecPerChunk, vend = min(nv, vbeg + kVecPerChunk);
    if (pair) online_chunk<E>(sq, vbeg, vend, k, mq, s_q);
    online_chunk<E>(sp, vbeg, vend, k, mp, s_p);
  }
  tmo = __syncthreads_or(tmo);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2q = __shfl_down_sync(0xFFFFFFFFu, mq, o), s2q = __shfl_down_sync(0xFFFFFFFFu, s_q, o);
    const float m2p = __shfl_down_sync(0xFFFFFFFFu, mp, o), s2p = __shfl_down_sync(0xFFFFFFFFu, s_p, o);
    ms_combine(mq, s_q, m2q, s2q, k);
    ms_combine(mp, s_p, m2p, s2p, k);
  }
  if (lane == 0) {
    sh.red[warp][0] = mq; sh.red[warp][1] = s_q;
    sh.red[warp][2] = mp; sh.red[warp][3] = s_p;
  }
  __syncthreads();
  if (tid == 0) {
    float a = sh.red[0][0], as = sh.red[0][1], c = sh.red[0][2], cs = sh.red[0][3];
    for (int w = 1; w < kNW; ++w) {
      ms_combine(a, as, sh.red[w][0], sh.red[w][1], k);
      ms_combine(c, cs, sh.red[w][2], sh.red[w][3], k);
    }
    if (tmo) {
      as = NAN;
      cs = NAN;
      sh.timeout = 1;
      if (P.status) atomicOr(P.status, static_cast<int32_t>(SC_DEV_TIMEOUT));
    }
    sh.part_ms = make_float4(a, as, c, cs);
  }
  cluster.sync();  // #1: partials published

  if (warp == 0) {
    float4 v = make_float4(-FLT_MAX, 0.0f, -FLT_MAX, 0.0f);
    if (lane < C) v = *cluster.map_shared_rank(&sh.part_ms, lane);
    float a = v.x, as = v.y, c = v.z, cs = v.w;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float a2 = __shfl_down_sync(0xFFFFFFFFu, a, o), as2 = __shfl_down_sync(0xFFFFFFFFu, as, o);
      const float c2 = __shfl_down_sync(0xFFFFFFFFu, c, o), cs2 = __shfl_down_sync(0xFFFFFFFFu, cs, o);
      ms_combine(a, as, a2, as2, k);
      ms_combine(c, cs, c2, cs2, k);
    }
    if (lane == 0) {  // thread 0: it holds the prefetched scalars
      sh.Mq = a; sh.Sq = as; sh.Mp = c; sh.Sp = cs;
      int err = 0;
      const bool okq = !pair || (isfinite(a) && isfinite(as) && as > 0.0f);
      const bool okp = isfinite(c) && isfinite(cs) && cs > 0.0f;
      if (!(okq && okp)) err |= SC_DEV_BAD_LOGIT;
      if (P.mode == kVerify) {
        if (!(uj >= 0.0f && uj < 1.0f)) err |= SC_DEV_BAD_UNIFORM;
        if (pair && (x < 0 || x >= P.V)) err |= SC_DEV_BAD_TOKEN;
      }
      if (err && P.status) atomicOr(P.status, err);
      sh.err = err;
      sh.delta = 0;
      sh.need_tv = 0;
      sh.need_sample = 0;
      sh.accept = 0;
      sh.tv = -1.0f;
      sh.qx = 0.0f;
      sh.pix = 0.0f;
      sh.c = pair && !err ? log2f(as / cs) : 0.0f;
      sh.ug = ug;
      if (!err) {
        if (!pair) {
          sh.need_sample = P.mode == kVerify;  // bonus row: drawn speculatively
        } else if (P.mode == kStats) {
          sh.need_tv = 1;
        } else {
          // deferral rule (Table 1); max q = 1/S_q, max p = 1/S_p
          const float maxq = 1.0f / as, maxp = 1.0f / cs, al = P.alpha;
          switch (P.rule) {
            case SC_RULE_CHOW: sh.delta = maxq < 1.0f - al; break;  // Eq. 2
            case SC_RULE_DIFF: sh.delta = maxq < maxp - al; break;  // Eq. 5
            case SC_RULE_OPT:                                       // Eq. 10
              // alpha * TV lies in [0, alpha]: the TV term decides only inside that band
              if (!(maxq < maxp)) sh.delta = 0;
              else if (maxq < maxp - al) sh.delta = 1;
              else sh.need_tv = 1;
              break;
            case SC_RULE_ALWAYS_DEFER: sh.delta = 1; break;
            default: sh.delta = 0; break;
          }
          if (!sh.need_tv) accept_test(sh, yqx, ypx, uj, P.inv_t);
        }
      }
    }
  }
  __syncthreads();
  const RowScalars rs = {sh.Mq, sh.Mp, k, sh.c};

  // ---- TV pass (shared memory only): sum_v min(p_v, q_v) = (1/S_q) sum_v 2^min(a_v, b_v + c)
  if (sh.need_tv) {
    float acc = 0.0f;
    for (int v = tid; v < nv; v += kNT) {
      float yq[8], yp[8];
      Elt<E>::load8(sq + 8 * v, yq);
      Elt<E>::load8(sp + 8 * v, yp);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        acc += ex2(fminf((yq[e] - rs.Mq) * k, fmaf(yp[e] - rs.Mp, k, rs.c)));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(0xFFFFFFFFu, acc, o);
    if (lane == 0) sh.red[warp][0] = acc;
    __syncthreads();
    if (tid == 0) {
      float t = 0.0f;
      for (int w = 0; w < kNW; ++w) t += sh.red[w][0];
      sh.part_tv = t;
    }
    cluster.sync();  // #2
    if (warp == 0) {
      float t = 0.0f;
      if (lane < C) t = *cluster.map_shared_rank(&sh.part_tv, lane);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) t += __shfl_down_sync(0xFFFFFFFFu, t, o);
      if (lane == 0) {
        const float tv = fminf(1.0f, fmaxf(0.0f, 1.0f - t / sh.Sq));  // Lemma 3
        sh.tv = tv;
        if (P.mode == kVerify) {
          sh.delta = 1.0f / sh.Sq < 1.0f / sh.Sp - P.alpha * tv;  // Eq. 10
          accept_test(sh, yqx, ypx, uj, P.inv_t);
        }
      }
    }
    __syncthreads();
  }

  if (sh.need_sample) {
    const float u = sh.ug;  // thread 0 prefetched it
    if (pair) sample_unit<E, true>(sq, sp, nv, v0, sh, rs, u, cluster, rank, C);
    else sample_unit<E, false>(sq, sp, nv, v0, sh, rs, u, cluster, rank, C);
  }
  if (sh.timeout && tid == 0 && P.bulk) {
    // let copies still in flight land before this CTA's shared memory is released
    for (int c = 0; c < nchunks; ++c) mbar_wait(&sh.bar[c], 0);
  }
  cluster.sync();  // candidate visible in rank 0; no peer reads this CTA's shared memory after

  // ---- publish this unit; the last unit of the sequence finishes it
  if (rank == 0 && tid == 0) {
    if (P.mode == kStats) {
      const size_t r = static_cast<size_t>(b) * P.gamma + j;
      const bool bad = sh.err != 0;
      P.max_q[r] = bad ? NAN : 1.0f / sh.Sq;
      P.max_p[r] = bad ? NAN : 1.0f / sh.Sp;
      P.tv[r] = bad ? NAN : sh.tv;
    } else {
      const size_t r = static_cast<size_t>(b) * G1 + j;
      const int cand = sh.need_sample ? sh.cand : -1;
      if (P.row_info) {
        float *ri = P.row_info + r * SC_ROW_FIELDS;
        ri[SC_ROW_MAXQ] = pair && !sh.err ? 1.0f / sh.Sq : NAN;
        ri[SC_ROW_MAXP] = !sh.err ? 1.0f / sh.Sp : NAN;
        ri[SC_ROW_TV] = sh.tv;
        ri[SC_ROW_DELTA] = static_cast<float>(sh.delta);
        ri[SC_ROW_ACCEPT] = static_cast<float>(sh.accept);
        ri[SC_ROW_QX] = sh.qx;
        ri[SC_ROW_PIX] = sh.pix;
        ri[SC_ROW_CAND] = static_cast<float>(cand);
      }
      P.unit_flags[r] = (sh.accept ? 1 : 0) | (sh.err ? 2 : 0);
      P.unit_cand[r] = cand;
      uint32_t ticket;
      asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;"
                   : "=r"(ticket)
                   : "l"(P.tickets + b)
                   : "memory");
      if (ticket == static_cast<uint32_t>(P.gamma)) {
        int jstar = P.gamma, bad = 0;
        const size_t base = static_cast<size_t>(b) * G1;
        for (int jj = 0; jj <= P.gamma; ++jj) {
          const int f = __ldcg(P.unit_flags + base + jj);
          bad |= f & 2;
          if (jj < P.gamma && !(f & 1) && jstar == P.gamma) jstar = jj;
        }
        const int tok = __ldcg(P.unit_cand + base + jstar);
        P.num_accepted[b] = bad ? 0 : jstar;
        P.next_token[b] = bad ? -1 : tok;
        P.tickets[b] = 0u;
      }
    }
  }
}

// ------------------------------------------------------------------ host side

struct DeviceInfo {
  int smem_optin = 0;
  bool configured[2] = {false, false};
};

DeviceInfo g_dev[64];
std::mutex g_mu;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

template <typename E>
size_t smem_bytes(int L) {
  return align_up(2 * static_cast<size_t>(L) * sizeof(E), 16) + sizeof(Shared);
}

// Slice length L (multiple of 8) and cluster size C for a row of V elements.
template <typename E>
int pick_layout(int V, int smem_optin, int *C_out, int *L_out) {
  const size_t row_bytes = static_cast<size_t>(V) * sizeof(E);
  size_t target = 32768;  // bytes per row per CTA: 64 KB of staging per CTA for a pair
  if (const char *s = getenv("SC_SLICE_BYTES")) {
    const long t = atol(s);
    if (t >= 1024) target = static_cast<size_t>(t);
  }
  int C = static_cast<int>((row_bytes + target - 1) / target);
  C = C < 1 ? 1 : C;
  for (; C <= kMaxCluster; ++C) {
    int L = static_cast<int>(align_up((static_cast<size_t>(V) + C - 1) / C, 8));
    const int Ceff = (V + L - 1) / L;
    if ((L + kChunkElems - 1) / kChunkElems > kMaxChunks) continue;
    if (smem_bytes<E>(L) > static_cast<size_t>(smem_optin)) continue;
    *C_out = Ceff;
    *L_out = L;
    return 0;
  }
  return -1;
}

bool device_accessible(const void *p) {
  if (!p) return false;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

template <typename E>
int launch(Params P, cudaStream_t stream, int units) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SC_ERR_CUDA;
  DeviceInfo &di = g_dev[dev];
  const int ti = sizeof(E) == 2 ? 1 : 0;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!di.smem_optin &&
        cudaDeviceGetAttribute(&di.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
      return SC_ERR_CUDA;
    if (!di.configured[ti]) {
      if (cudaFuncSetAttribute(sc_unit_kernel<E>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               di.smem_optin) != cudaSuccess ||
          cudaFuncSetAttribute(sc_unit_kernel<E>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
              cudaSuccess)
        return SC_ERR_CUDA;
      di.configured[ti] = true;
    }
  }
  int C = 1, L = 8;
  if (pick_layout<E>(P.V, di.smem_optin, &C, &L) != 0) return SC_ERR_UNSUPPORTED;
  if (const char *s = getenv("SC_CLUSTER")) {  // tuning override (must still fit)
    const int c = atoi(s);
    if (c >= 1 && c <= kMaxCluster) {
      const int Lc = static_cast<int>(align_up((static_cast<size_t>(P.V) + c - 1) / c, 8));
      if (smem_bytes<E>(Lc) <= static_cast<size_t>(di.smem_optin) &&
          (Lc + kChunkElems - 1) / kChunkElems <= kMaxChunks) {
        L = Lc;
        C = (P.V + L - 1) / L;
      }
    }
  }
  P.L = L;
  P.cluster = C;
  const size_t row_bytes = static_cast<size_t>(P.V) * sizeof(E);
  P.bulk = (row_bytes % 16 == 0) && (reinterpret_cast<uintptr_t>(P.draft) % 16 == 0) &&
           (reinterpret_cast<uintptr_t>(P.target) % 16 == 0);
  if (units == 0) return SC_OK;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(units) * static_cast<unsigned>(C), 1, 1);
  cfg.blockDim = dim3(kNT, 1, 1);
  cfg.dynamicSmemBytes = smem_bytes<E>(L);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(C);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, sc_unit_kernel<E>, P) != cudaSuccess) return SC_ERR_CUDA;
  return SC_OK;
}

int common_checks(const void *draft, const void *target, int dtype, int B, int gamma, int V,
                  float temperature) {
  if (dtype != SC_F32 && dtype != SC_BF16) return SC_ERR_INVALID_ARG;
  if (B < 1 || gamma < 1 || gamma > SC_MAX_GAMMA || V < 1) return SC_ERR_INVALID_ARG;
  if (V > sc_max_vocab(static_cast<sc_dtype>(dtype))) return SC_ERR_UNSUPPORTED;
  if (!(temperature > 0.0f) || !std::isfinite(temperature)) return SC_ERR_INVALID_ARG;
  if (static_cast<double>(B) * (gamma + 1) * kMaxCluster > 2147483647.0) return SC_ERR_INVALID_ARG;
  if (!device_accessible(draft) || !device_accessible(target)) return SC_ERR_INVALID_ARG;
  return SC_OK;
}

}  // namespace

// ------------------------------------------------------------------ C ABI

extern "C" {

size_t sc_workspace_bytes(int B, int gamma, int V) {
  (void)V;
  if (B < 1 || gamma < 1) return 0;
  const size_t n = static_cast<size_t>(B) * (gamma + 1);
  return align_up(4 * static_cast<size_t>(B), 256) + 2 * align_up(4 * n, 256);
}

int sc_workspace_init(void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  if (!workspace) return SC_ERR_INVALID_ARG;
  return cudaMemsetAsync(workspace, 0, workspace_bytes, stream) == cudaSuccess ? SC_OK : SC_ERR_CUDA;
}

int sc_max_vocab(sc_dtype dtype) {
  // one cluster of kMaxCluster CTAs, each staging both rows of its slice
  const size_t budget = 227 * 1024 - sizeof(Shared) - 64;
  const size_t elt = dtype == SC_F32 ? 4 : 2;
  const size_t per_cta = std::min(budget / (2 * elt), static_cast<size_t>(kMaxChunks) * kChunkElems) & ~size_t(7);
  return static_cast<int>(per_cta * kMaxCluster);
}

int sc_verify_rows(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                   const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                   sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
                   int32_t *next_token, void *workspace, size_t workspace_bytes,
                   int32_t *device_status, float *row_info, cudaStream_t stream) {
  int rc = common_checks(draft_logits, target_logits, dtype, B, gamma, V, temperature);
  if (rc != SC_OK) return rc;
  if (static_cast<int>(rule) < 0 || static_cast<int>(rule) > 4) return SC_ERR_INVALID_ARG;
  if (!(alpha >= 0.0f && alpha <= 1.0f)) return SC_ERR_INVALID_ARG;
  if (!device_accessible(draft_tokens) || !device_accessible(uniforms) ||
      !device_accessible(num_accepted) || !device_accessible(next_token))
    return SC_ERR_INVALID_ARG;
  if (device_status && !device_accessible(device_status)) return SC_ERR_INVALID_ARG;
  if (row_info && !device_accessible(row_info)) return SC_ERR_INVALID_ARG;
  if (!workspace || workspace_bytes < sc_workspace_bytes(B, gamma, V)) return SC_ERR_WORKSPACE;
  if (!device_accessible(workspace)) return SC_ERR_WORKSPACE;

  Params P = {};
  P.draft = draft_logits;
  P.target = target_logits;
  P.tokens = draft_tokens;
  P.uniforms = uniforms;
  P.B = B;
  P.gamma = gamma;
  P.V = V;
  P.rule = static_cast<int>(rule);
  P.alpha = alpha;
  P.temperature = temperature;
  P.k = static_cast<float>(1.4426950408889634 / static_cast<double>(temperature));
  P.inv_t = 1.0 / static_cast<double>(temperature);
  P.mode = kVerify;
  P.num_accepted = num_accepted;
  P.next_token = next_token;
  P.row_info = row_info;
  P.status = device_status;
  unsigned char *ws = static_cast<unsigned char *>(workspace);
  const size_t n = static_cast<size_t>(B) * (gamma + 1);
  P.tickets = reinterpret_cast<uint32_t *>(ws);
  P.unit_flags = reinterpret_cast<int32_t *>(ws + align_up(4 * static_cast<size_t>(B), 256));
  P.unit_cand = reinterpret_cast<int32_t *>(ws + align_up(4 * static_cast<size_t>(B), 256) + align_up(4 * n, 256));
  const int units = B * (gamma + 1);
  return dtype == SC_BF16 ? launch<uint16_t>(P, stream, units) : launch<float>(P, stream, units);
}

int sc_verify(const void *draft_logits, const void *target_logits, sc_dtype dtype,
              const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
              sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
              int32_t *next_token, void *workspace, size_t workspace_bytes,
              int32_t *device_status, cudaStream_t stream) {
  return sc_verify_rows(draft_logits, target_logits, dtype, draft_tokens, uniforms, B, gamma, V,
                        rule, alpha, temperature, num_accepted, next_token, workspace,
                        workspace_bytes, device_status, nullptr, stream);
}

int sc_row_stats(const void *draft_logits, const void *target_logits, sc_dtype dtype, int B,
                 int gamma, int V, float temperature, float *max_q, float *max_p, float *tv,
                 cudaStream_t stream) {
  int rc = common_checks(draft_logits, target_logits, dtype, B, gamma, V, temperature);
  if (rc != SC_OK) return rc;
  if (!device_accessible(max_q) || !device_accessible(max_p) || !device_accessible(tv))
    return SC_ERR_INVALID_ARG;
  Params P = {};
  P.draft = draft_logits;
  P.target = target_logits;
  P.B = B;
  P.gamma = gamma;
  P.V = V;
  P.temperature = temperature;
  P.k = static_cast<float>(1.4426950408889634 / static_cast<double>(temperature));
  P.inv_t = 1.0 / static_cast<double>(temperature);
  P.mode = kStats;
  P.max_q = max_q;
  P.max_p = max_p;
  P.tv = tv;
  const int units = B * gamma;
  return dtype == SC_BF16 ? launch<uint16_t>(P, stream, units) : launch<float>(P, stream, units);
}

const char *sc_status_string(int code) {
  switch (code) {
    case SC_OK: return "ok";
    case SC_ERR_INVALID_ARG: return "invalid argument";
    case SC_ERR_CUDA: return "CUDA launch error";
    case SC_ERR_WORKSPACE: return "workspace missing or too small";
    case SC_ERR_UNSUPPORTED: return "vocabulary too large for one cluster per row";
    default: return "unknown status";
  }
}

}  // extern "C"
