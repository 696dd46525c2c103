// GB300 (sm_103a) verification step of speculative cascades.
//
// One call of sc_verify runs GenSpecSample's verification phase (Algorithm 4)
// with the SpecCascade target pi = (1 - delta) q + delta p (Algorithm 5, Eq. 6)
// -- or another target: the token-specific rules of Section 4.4, lossy
// speculative decoding and BiLD* (Table 3), the log-loss rules, greedy
// decoding -- for B sequences of gamma drafted positions over a V-token
// vocabulary, in ONE kernel launch:
//
//   unit    one (b, j < gamma) row pair (draft row q_j, target row p_j), or the
//           bonus target row (b, gamma); units in position-major order (every
//           sequence's position j before any position j + 1);
//   grid    one thread-block cluster of C CTAs per unit; CTA r of the cluster
//           owns the vocabulary slice [r L, (r+1) L) of both rows;
//   pass 1  the slice streams from HBM through a two-stage shared-memory ring
//           filled by TMA bulk copies (cp.async.bulk + mbarrier), 4096 logits
//           per row per stage, the older chunks with the L2 evict-first
//           policy; each thread keeps an online (max, sum of exp) in four
//           lanes; thread 0 merges the warp partials and pushes the CTA partial
//           into every CTA of the cluster (st.shared::cluster) before one
//           cluster barrier, after which every read is local: M and S of both
//           rows, max q and max p, the deferral decision and the acceptance
//           test of the draft token;
//   token   a token-specific rule evaluates r(v) per token; eta = sum r(v) q(v)
//           comes from a pass-1 screen of each thread's two largest tested
//           logits, or, where the screen cannot settle it, from a second pass;
//   TV      only inside the OPT (or OPTLog) band, where the TV term of Eq. 10
//           decides: lower and upper bounds on D_TV from the pass-1 partials
//           settle most such rows; the rest, and sc_row_stats, sum the
//           residual weights max(0, p - q) over the slice again (newest chunk
//           first) and over the cluster: D_TV(p, q) S_q (Lemma 3);
//   finish  every CTA writes its unit's decision record and reports its
//           arrival (and rejection) on the ticket of its slice rank r in the
//           sequence.  A rejected pair that is certainly row j* (every earlier
//           position of its rank reported without a rejection) stores its own
//           residual's chunk prefixes at once; otherwise the CTA whose report
//           settles j* = min{j : a_j = 0} streams its slice of row j*.  The
//           bonus row's prefixes come from its pass 1.  The last of a
//           sequence's C owners does the inverse-CDF draw: it finds the slice
//           and chunk holding u R, copies that chunk in and one warp scans the
//           segment holding it.  Only row j* of each sequence is sampled, and
//           no CTA ever waits on another cluster.
//
// Exponentials are ex2.approx of fma(y, log2(e)/T, -R), R = fl(M log2(e)/T):
// one rounding per logit.  Every mbarrier wait is bounded and reports
// SC_DEV_TIMEOUT instead of hanging.

#include "sc.h"

#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cfloat>
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <mutex>

namespace cg = cooperative_groups;

namespace {

#ifndef SC_RING_STAGES
#define SC_RING_STAGES 2
#endif
#ifndef SC_CHUNK
#define SC_CHUNK 4096
#endif
#ifndef SC_MIN_BLOCKS
#define SC_MIN_BLOCKS 6
#endif
#ifndef SC_DEBUG
#define SC_DEBUG 0  // 1: check computed indices and copy sizes, skip and record a failing access
#endif
#ifndef SC_OPT_UB
#define SC_OPT_UB 1  // OPT and OPTLog band rows: settle delta = 1 by an upper bound on D_TV
#endif
#ifndef SC_L2_PREFETCH
#define SC_L2_PREFETCH 1  // second passes prefetch their slice into L2 before streaming it
#endif

constexpr int kNT = 128;                   // threads per CTA
constexpr int kNW = kNT / 32;              // warps per CTA
constexpr int kCH = SC_CHUNK;              // logits per row per ring stage
constexpr int kVPC = kCH / 8;              // 8-element vectors per chunk
constexpr int kRounds = kVPC / kNT;        // vectors per thread per chunk
constexpr int kStages = SC_RING_STAGES;    // ring depth
#ifndef SC_MAX_SLICE
#define SC_MAX_SLICE 65536
#endif
constexpr int kMaxChunks = SC_MAX_SLICE / kCH;  // slice <= SC_MAX_SLICE logits per row
constexpr int kMaxCluster = 16;
constexpr int kEntries = kMaxChunks * kRounds * kNW;  // (chunk, round, warp) segments
constexpr uint32_t kWaitLimit = 1u << 21;  // bounded mbarrier waits (~seconds)
constexpr uint32_t kSuspendNs = 1000;      // try_wait suspend hint
constexpr int kMinBlocksPerSM = SC_MIN_BLOCKS;

enum Mode : int { kVerify = 0, kStats = 1 };

// The kernel is compiled once per rule family.  kFamCascade: the deferral
// rules of Table 1 and lossy speculative decoding (Table 3); kFamToken: the
// token-specific rules of Section 4.4, whose weight passes evaluate r(v) per
// logit; kFamExt: the rules that read entropies or a cross entropy (BiLD*, the
// log-loss rules) and greedy decoding (T = 0), whose pass 1 also accumulates
// first moments of the exponents and the rows' argmaxes.
enum Family : int { kFamCascade = 0, kFamToken = 1, kFamExt = 2 };

struct Params {
  const void *draft;
  const void *target;
  const int32_t *tokens;
  const float *uniforms;
  int B, gamma, V;
  int rule;
  float alpha;
  float temperature;
  float k;        // log2(e) / T, the f32 factor of every exponent of pass 1
  float kl;       // log2(e) / T - k: with k, log2(e) / T to twice f32 precision
  int units;      // units of the call: B (gamma + 1) row pairs and bonus rows, or B gamma pairs
  int L;          // slice length per CTA (multiple of 8 logits)
  int cluster;    // CTAs per unit
  int bulk;       // 1: TMA bulk copies, 0: per-thread loads (rows not 16-byte aligned)
  int mode;
  int greedy;     // T = 0: greedy decoding; the rules' statistics use T = 1 (k = log2(e))
  float lossy_l;  // lossy speculative decoding: -log2(1 - alpha) as lossy_l + lossy_ll,
  float lossy_ll; // the shift of log2 of the acceptance ratio (+inf: alpha = 1)
  float lossy_c;  // -log2(beta): the residual max(0, p / beta - q) is 2^{b + c + lossy_c} - 2^a
  float beta;     // lossy speculative decoding's beta (Table 3), >= 1 - alpha
  int32_t *num_accepted;
  int32_t *next_token;
  float *row_info;
  float *max_q;
  float *max_p;
  float *tv;
  // workspace (verification only)
  unsigned long long *rank_tickets;  // [B][kMaxCluster] arrivals of the rank-r CTAs; zero at rest
  uint32_t *seq_tickets;   // [B] finished sample passes (+1 for rank 0's last arrival); zero at rest
  float4 *records;         // [B][kMaxCluster][gamma+1] (R_q, R_p, c, flags) as seen by rank r
  float4 *records2;        // [B][kMaxCluster][gamma+1] (eta, thr, token, on_q) of token rules
  int spec_res;            // a rejected pair that is certainly row j* stores its residual's chunk
                           // prefixes itself (row_pre); 0: the owners always sample
  int pos_major;           // units in position-major order: (b, j) is unit j B + b
  int opt_ub;              // OPT pairs accumulate sqrt(q p) in pass 1 for an upper bound on D_TV
  int l2_hint;             // all but the newest l2_hint chunks of a pair's slice (all of a bonus row)
                           // are copied evict-first (0: no hints)
  float *row_pre;          // [B][gamma+1][kMaxCluster][kMaxChunks + 1] those prefixes, per row
  float *bonus_pre;        // [B][kMaxCluster][kMaxChunks + 1] the same for the bonus row p_gamma,
                           // written by the bonus unit from its pass-1 chunk totals
  float *chunk_pre;        // [B][kMaxCluster][kMaxChunks + 1] exclusive prefix of slice r of the
                           // sampled row at each chunk start, then the slice total
  int32_t *status;
};

// ------------------------------------------------------------------ debug checks

// First source line whose check failed (SC_DEBUG builds; 0: none).
__device__ int g_sc_debug_line;

// In SC_DEBUG builds, false for a failed check (its line recorded, the access
// skipped by the caller); always true otherwise, and compiled away.
__device__ __forceinline__ bool sc_check(bool cond, int line) {
  if (!SC_DEBUG || cond) return true;
  atomicCAS(&g_sc_debug_line, 0, line);
  return false;
}
#define SC_CHECK(cond) sc_check((cond), __LINE__)

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

// Bounded wait for the phase of parity `parity` of an mbarrier; false on timeout.
// Each try_wait suspends the thread for up to kSuspendNs (it resumes as soon as
// the phase completes), so a waiting warp issues a few instructions per
// microsecond instead of spinning.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  for (uint32_t i = 0; i < kWaitLimit; ++i) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(a), "r"(parity), "n"(kSuspendNs)
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

// bulk_g2s with an L2 cache policy (createpolicy): here evict-first, for data
// that no later pass is likely to read from L2.
__device__ __forceinline__ void bulk_g2s_hint(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                              uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}

__device__ __forceinline__ uint64_t evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// Hint: bring [src, src + bytes) into L2 (16-byte aligned, a multiple of 16 bytes).
__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Stores into the shared memory of the cluster's CTA `rank` (same offset as p here).
__device__ __forceinline__ uint32_t peer_addr(const void *p, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_peer(uint32_t a, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(a), "f"(v.x), "f"(v.y), "f"(v.z),
               "f"(v.w)
               : "memory");
}
__device__ __forceinline__ void st_peer(uint32_t a, float2 v) {
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(a), "f"(v.x), "f"(v.y) : "memory");
}
__device__ __forceinline__ void st_peer(uint32_t a, int2 v) {
  asm volatile("st.shared::cluster.v2.s32 [%0], {%1, %2};" ::"r"(a), "r"(v.x), "r"(v.y) : "memory");
}
__device__ __forceinline__ void st_peer(uint32_t a, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(a), "f"(v) : "memory");
}

// ------------------------------------------------------------------ logit types

template <typename E>
struct Elt;

template <>
struct Elt<uint16_t> {  // bf16 bit patterns
  __device__ __forceinline__ static void unpack(const uint4 v, float (&y)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      y[2 * i] = __uint_as_float(w[i] << 16);
      y[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
  __device__ __forceinline__ static void load8(const uint16_t *s, float (&y)[8]) {
    unpack(*reinterpret_cast<const uint4 *>(s), y);
  }
  __device__ __forceinline__ static float at(const uint16_t *g, size_t i) {
    return __uint_as_float(static_cast<uint32_t>(g[i]) << 16);
  }
};

template <>
struct Elt<float> {
  __device__ __forceinline__ static void load8(const float *s, float (&y)[8]) {
    const float4 a = *reinterpret_cast<const float4 *>(s);
    const float4 b = *reinterpret_cast<const float4 *>(s + 4);
    y[0] = a.x; y[1] = a.y; y[2] = a.z; y[3] = a.w;
    y[4] = b.x; y[5] = b.y; y[6] = b.z; y[7] = b.w;
  }
  __device__ __forceinline__ static float at(const float *g, size_t i) { return g[i]; }
};

// Eight logits starting at element e of a row slice of n valid logits; the
// ones at or past n read as -inf (probability 0).
template <typename E>
__device__ __forceinline__ void load8_smem(const E *s, int e, int n, float (&y)[8]) {
  if (e + 8 <= n) {
    Elt<E>::load8(s + e, y);
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) y[i] = e + i < n ? Elt<E>::at(s, e + i) : -INFINITY;
  }
}

// ------------------------------------------------------------------ shared state

struct __align__(16) Shared {
  uint64_t full[kStages];
  // cluster exchanges, written by every CTA of the cluster into slot [its rank]:
  float4 all_ms[kMaxCluster];  // 1: (m_q, s_q, m_p, s_p) of the slice
  float2 all_x[kMaxCluster];   // 1: raw logits at the draft token, if in the slice
  float all_r[kMaxCluster];    // 2 (TV pass): the slice's total residual weight
  float2 all_lb[kMaxCluster];  // OPT band: the slice's parts of the lower and upper bounds on D_TV
  float2 all_scr[kMaxCluster]; // token rules: the slice's sum of q over its undeferred tokens, and
                               // whether its screen is exact (1) or not (0)
  float4 all_ext[kMaxCluster];  // 1 (kFamExt): (A_q, A_p, X, -) of the slice, see ExtState
  int2 all_idx[kMaxCluster];    // 1 (kFamExt): the slice's argmax of q and of p
  int timeout;
  float4 red[kNW];          // (m_q, s_q, m_p, s_p) of each warp
  float4 ext_red[kNW];      // (kFamExt) (A_q, A_p, X, -) of each warp
  int2 idx_red[kNW];        // (kFamExt) argmax of q and of p of each warp
  float seg[kEntries + 1];  // per-(chunk, round, warp) weights, then exclusive prefixes
  float xq, xp;             // raw logits at the draft token, when in this slice
  // row state, identical in every CTA of the cluster
  float Mq, Sq, Mp, Sp, Rq, Rp, maxq, maxp, c, tv, qx, pix;
  int err, delta, accept, need_p2, band;
  int tok, on_q;            // a token rule (Section 4.4) and its r(v) test's variable
  float dl, dr;             // OPT and OPTLog: delta = [dl < dr - alpha D_TV]
  float nhq, nhp;           // (kFamExt) sum_v q log q and sum_v p log p, in nats
  float klqp;               // (kFamExt) KL(q || p) = sum_v q log q - sum_v q log p, in nats
  int iq, ip;               // (kFamExt) argmax q and argmax p, lowest index on ties
  float thr, eta;           // its r(v) threshold (exponent domain) and eta = sum_v r(v) q(v)
  // sequence finish
  int self_res;             // this rejected pair stores its residual's chunk prefixes (row_pre)
  int owner;                // this CTA runs its rank's sample pass of row j*
  int scan_records;         // j* must be read from the records (gamma + 1 > 32)
  int seq_last;             // the sequence's last finisher: draws the token
  int jstar, bad, sample_ok;
  float4 rj;                // (R_q, R_p, c, flags) of row j*
  float4 rj2;               // (eta, thr, token, on_q) of row j*
  int cross_rank;           // slice holding u * R_tot
  int cross_chunk;          // chunk of that slice holding it (else its last chunk with weight)
  int have_t;               // u * R_tot lies inside that chunk (not past a rounding gap)
  float chunk_lo;           // exclusive prefix of the slice at the start of that chunk
  int cross_seg;            // segment of that chunk holding it (-1: none)
  int token;                // the drawn token
  float2 t_slice;           // u * R_tot minus the weight before the crossing slice (hi + lo)
  float t_seg;              // ... minus the weight before the crossing segment
};

__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Exponent reference of a running maximum m: r = fl(m k), floored at -1e30 so
// that a slice of -inf logits keeps finite arithmetic.  Every exponential of
// pass 1 is 2^{fma(y, k, -r)}: one rounding, no systematic error (the max
// logit's own term is 2^{fma(M, k, -R)}, not exactly 1, and is treated so).
__device__ __forceinline__ float refk(float m, float k) { return fmaxf(__fmul_rn(m, k), -1e30f); }

// Merge the (max, sum) partials held by the 32 lanes of a warp (each sum is
// relative to refk of its own max): the largest max M by a shuffle tree, then
// every lane's sum rescaled to refk(M) by ONE exponential, then a butterfly
// sum -- a short dependent chain, which matters when this warp shares its SM
// with streaming warps.  Every lane ends with (M, S); identical inputs give
// identical results in every CTA.  A lane with s = 0 contributes 0.
__device__ __forceinline__ void warp_ms_merge(float &m, float &s, float k) {
  float M = m;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, o));
  float t = s * ex2(refk(m, k) - refk(M, k));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t = __fadd_rn(t, __shfl_xor_sync(0xFFFFFFFFu, t, o));
  m = M;
  s = t;
}

// Merge n (m_q, s_q, m_p, s_p) partials in index order, in one thread: the
// largest maxima first, then every sum rescaled to refk of its row's maximum
// by one exponential (all independent).  Shared-memory reads and arithmetic
// only: no shuffles, which queue behind the streaming warps' shared-memory
// loads on the same SM.
__device__ __forceinline__ float4 merge_partials(const float4 *v, int n, float k) {
  float Mq = -FLT_MAX, Mp = -FLT_MAX;
  for (int i = 0; i < n; ++i) {
    Mq = fmaxf(Mq, v[i].x);
    Mp = fmaxf(Mp, v[i].z);
  }
  const float Rq = refk(Mq, k), Rp = refk(Mp, k);
  float Sq = 0.0f, Sp = 0.0f;
  for (int i = 0; i < n; ++i) {
    Sq = fmaf(v[i].y, ex2(refk(v[i].x, k) - Rq), Sq);
    Sp = fmaf(v[i].w, ex2(refk(v[i].z, k) - Rp), Sp);
  }
  return make_float4(Mq, Sq, Mp, Sp);
}

// Pass 1 on one row of one chunk: this thread's kRounds vectors, online
// (max m, sum s of 2^{y k - refk(m)}), s kept as four partial sums, over the logits 0, 1, 2, 3 (mod 4).
// kFull: the chunk holds kCH logits.
template <typename E, bool kFull>
__device__ __forceinline__ void online_row(const E *src, int n, float k, float &m, float4 &s) {
  float y[kRounds][8];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    if constexpr (kFull) {
      Elt<E>::load8(src + e, y[r]);
    } else {
      load8_smem(src, e, n, y[r]);
    }
  }
  float mn = m;
#pragma unroll
  for (int r = 0; r < kRounds; ++r)
#pragma unroll
    for (int i = 0; i < 8; i += 2) mn = max3(mn, y[r][i], y[r][i + 1]);
  const float rn = refk(mn, k);
  const float sc = ex2(refk(m, k) - rn);
  float s0 = s.x * sc, s1 = s.y * sc, s2 = s.z * sc, s3 = s.w * sc;
#pragma unroll
  for (int r = 0; r < kRounds; ++r)
#pragma unroll
    for (int i = 0; i < 8; i += 4) {
      s0 += ex2(fmaf(y[r][i], k, -rn));
      s1 += ex2(fmaf(y[r][i + 1], k, -rn));
      s2 += ex2(fmaf(y[r][i + 2], k, -rn));
      s3 += ex2(fmaf(y[r][i + 3], k, -rn));
    }
  m = mn;
  s = make_float4(s0, s1, s2, s3);
}

__device__ __forceinline__ __nv_bfloat162 as_bf162(uint32_t w) {
  return *reinterpret_cast<__nv_bfloat162 *>(&w);
}

// bf16 full chunk: the exact maximum from a packed bf16x2 max tree over the raw
// words, then one packed f32x2 FMA per two logits for the exponent arguments
// and packed f32x2 adds for the four partial sums (two packed pairs).
template <>
__device__ __forceinline__ void online_row<uint16_t, true>(const uint16_t *src, int n, float k,
                                                           float &m, float4 &s) {
  (void)n;
  uint32_t w[kRounds * 4];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const uint4 v = *reinterpret_cast<const uint4 *>(src + 8 * (r * kNT + static_cast<int>(threadIdx.x)));
    w[4 * r] = v.x; w[4 * r + 1] = v.y; w[4 * r + 2] = v.z; w[4 * r + 3] = v.w;
  }
  __nv_bfloat162 mx = as_bf162(w[0]);
#pragma unroll
  for (int i = 1; i < kRounds * 4; ++i) mx = __hmax2(mx, as_bf162(w[i]));
  const float mn = fmaxf(m, fmaxf(__low2float(mx), __high2float(mx)));
  const float rn = refk(mn, k);
  const float sc = ex2(refk(m, k) - rn);
  float2 acc = __fmul2_rn(make_float2(s.x, s.y), make_float2(sc, sc));
  float2 acb = __fmul2_rn(make_float2(s.z, s.w), make_float2(sc, sc));
  const float2 kk = make_float2(k, k), nr = make_float2(-rn, -rn);
#pragma unroll
  for (int i = 0; i < kRounds * 4; i += 2) {  // words 2j' hold logits 0, 1 (mod 4), words 2j' + 1 logits 2, 3
    const float2 y = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u));
    const float2 t = __ffma2_rn(y, kk, nr);
    acc = __fadd2_rn(acc, make_float2(ex2(t.x), ex2(t.y)));
    const float2 y2 = make_float2(__uint_as_float(w[i + 1] << 16), __uint_as_float(w[i + 1] & 0xFFFF0000u));
    const float2 t2 = __ffma2_rn(y2, kk, nr);
    acb = __fadd2_rn(acb, make_float2(ex2(t2.x), ex2(t2.y)));
  }
  m = mn;
  s = make_float4(acc.x, acc.y, acb.x, acb.y);
}

// online_row<uint16_t, true> for the row a token rule screens: the chunk's two
// largest logits of this thread (y1 >= y2, a tie giving y1 == y2) from packed
// bf16x2 max/min over the raw words, in the sweep that takes the maximum.
__device__ __forceinline__ void online_row_top2(const uint16_t *src, float k, float &m, float4 &s, float &y1,
                                                float &y2) {
  uint32_t w[kRounds * 4];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const uint4 v = *reinterpret_cast<const uint4 *>(src + 8 * (r * kNT + static_cast<int>(threadIdx.x)));
    w[4 * r] = v.x; w[4 * r + 1] = v.y; w[4 * r + 2] = v.z; w[4 * r + 3] = v.w;
  }
  __nv_bfloat162 m1 = as_bf162(w[0]), m2 = as_bf162(0xFF80FF80u);  // (-inf, -inf)
#pragma unroll
  for (int i = 1; i < kRounds * 4; ++i) {
    const __nv_bfloat162 v = as_bf162(w[i]);
    m2 = __hmax2(m2, __hmin2(m1, v));
    m1 = __hmax2(m1, v);
  }
  const float a = __low2float(m1), b = __high2float(m1);
  y1 = fmaxf(a, b);
  y2 = fmaxf(fminf(a, b), fmaxf(__low2float(m2), __high2float(m2)));
  const float mn = fmaxf(m, y1);
  const float rn = refk(mn, k);
  const float sc = ex2(refk(m, k) - rn);
  float2 acc = __fmul2_rn(make_float2(s.x, s.y), make_float2(sc, sc));
  float2 acb = __fmul2_rn(make_float2(s.z, s.w), make_float2(sc, sc));
  const float2 kk = make_float2(k, k), nr = make_float2(-rn, -rn);
#pragma unroll
  for (int i = 0; i < kRounds * 4; i += 2) {
    const float2 y = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u));
    const float2 t = __ffma2_rn(y, kk, nr);
    acc = __fadd2_rn(acc, make_float2(ex2(t.x), ex2(t.y)));
    const float2 y3 = make_float2(__uint_as_float(w[i + 1] << 16), __uint_as_float(w[i + 1] & 0xFFFF0000u));
    const float2 t2 = __ffma2_rn(y3, kk, nr);
    acb = __fadd2_rn(acb, make_float2(ex2(t2.x), ex2(t2.y)));
  }
  m = mn;
  s = make_float4(acc.x, acc.y, acb.x, acb.y);
}

// Pass-1 state of the kFamExt rules.  With a_v = y^q_v k - r_q and
// b_v = y^p_v k - r_p relative to the references r = refk(m) of the running
// maxima m:
//   sq = sum 2^a,  aq = sum 2^a a,  sp = sum 2^b,  ap = sum 2^b b,  x = sum 2^a b,
// so that, for the row's final references and sums (log2 q_v = a_v - log2 S_q),
//   sum_v q log2 q = A_q / S_q - log2 S_q,   sum_v q log2 p = X / S_q - log2 S_p.
// iq and ip are the lowest indices of the largest q and p logits seen (-1: none).
// A term whose exponential is 0 contributes 0 to the moments.
struct ExtState {
  float mq, sq, aq, mp, sp, ap, x;
  int iq, ip;
};

__device__ __forceinline__ ExtState ext_empty() {
  return {-FLT_MAX, 0.0f, 0.0f, -FLT_MAX, 0.0f, 0.0f, 0.0f, -1, -1};
}

// Re-reference a partial by dq = r_q - r_q' <= 0 and dp = r_p - r_p' <= 0:
// a' = a + dq and 2^{a'} = 2^{dq} 2^a, so A' = 2^{dq} (A + dq S) and
// X' = 2^{dq} (X + dp S_q).  (A reference floored at -1e30 comes with S = 0.)
__device__ __forceinline__ void ext_rebase(ExtState &e, float dq, float dp) {
  const float fq = ex2(dq), fp = ex2(dp);
  e.x = e.x == -INFINITY ? e.x : fq * fmaf(dp, e.sq, e.x);  // (-inf: D(q, p) = +inf, kept)
  e.aq = fq * fmaf(dq, e.sq, e.aq);
  e.sq = fq * e.sq;
  e.ap = fp * fmaf(dp, e.sp, e.ap);
  e.sp = fp * e.sp;
}

// The index of the larger of two maxima, the lower index on a tie (-1: none).
__device__ __forceinline__ int pick_index(float ma, int ia, float mb, int ib) {
  if (ma > mb) return ia;
  if (mb > ma) return ib;
  if (ia < 0) return ib;
  if (ib < 0) return ia;
  return min(ia, ib);
}

// b += a: both re-referenced to the larger maxima, then summed.
__device__ __forceinline__ void ext_merge(ExtState &b, ExtState a, float k) {
  const float Mq = fmaxf(a.mq, b.mq), Mp = fmaxf(a.mp, b.mp);
  const float Rq = refk(Mq, k), Rp = refk(Mp, k);
  ext_rebase(a, refk(a.mq, k) - Rq, refk(a.mp, k) - Rp);
  ext_rebase(b, refk(b.mq, k) - Rq, refk(b.mp, k) - Rp);
  b.iq = pick_index(b.mq, b.iq, a.mq, a.iq);
  b.ip = pick_index(b.mp, b.ip, a.mp, a.ip);
  b.mq = Mq;
  b.mp = Mp;
  b.sq = __fadd_rn(b.sq, a.sq);
  b.aq = __fadd_rn(b.aq, a.aq);
  b.sp = __fadd_rn(b.sp, a.sp);
  b.ap = __fadd_rn(b.ap, a.ap);
  b.x = __fadd_rn(b.x, a.x);
}

// Merge the partials of the 32 lanes of a warp (butterfly); lane 0 ends with
// the warp's partial.
// The first of this thread's logits equal to m in the chunk starting at token
// vc (the order of the sweep), as a token index; row = the slice's row in global
// memory, v0 its first token.  -1 if none (cannot happen for a recorded maximum).
// Greedy decoding's argmaxes in packed chunks are not located during the
// sweep: a thread whose running maximum rises in the chunk starting at token
// vc records the code -2 - vc, and ext_resolve_index finds the position later
// for the threads that hold their warp's maximum.
__device__ __forceinline__ int lazy_code(int vc) { return -2 - vc; }

// Greedy decoding's bonus row (p only), full bf16 chunk: the maximum by a
// packed max tree (its position recorded as a chunk code) and the sum of
// exponentials by packed arithmetic; the bonus row needs no moments.
__device__ __forceinline__ void ext_bonus_bf16(const uint16_t *srcp, int v0, float k, ExtState &st) {
  uint32_t wp[kRounds * 4];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const uint4 v = *reinterpret_cast<const uint4 *>(srcp + 8 * (r * kNT + static_cast<int>(threadIdx.x)));
    wp[4 * r] = v.x; wp[4 * r + 1] = v.y; wp[4 * r + 2] = v.z; wp[4 * r + 3] = v.w;
  }
  __nv_bfloat162 xp = as_bf162(wp[0]);
#pragma unroll
  for (int i = 1; i < kRounds * 4; ++i) xp = __hmax2(xp, as_bf162(wp[i]));
  const float cp = fmaxf(__low2float(xp), __high2float(xp));
  float mp = st.mp;
  int ip = st.ip;
  if (cp > mp) {
    mp = cp;
    ip = lazy_code(v0);
  }
  const float rp = refk(mp, k);
  const float sc = ex2(refk(st.mp, k) - rp);
  const float2 kk = make_float2(k, k), nrp = make_float2(-rp, -rp);
  float2 sp = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int i = 0; i < kRounds * 4; ++i) {
    const float2 b = __ffma2_rn(make_float2(__uint_as_float(wp[i] << 16), __uint_as_float(wp[i] & 0xFFFF0000u)), kk, nrp);
    sp = __fadd2_rn(sp, make_float2(ex2(b.x), ex2(b.y)));
  }
  st.mp = mp;
  st.ip = ip;
  st.sp = fmaf(st.sp, sc, sp.x + sp.y);
}

template <typename E>
__device__ __forceinline__ int ext_resolve_index(const E *row, int v0, int vc, float m) {
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    for (int i = 0; i < 8; ++i)
      if (Elt<E>::at(row, static_cast<size_t>(vc - v0 + e + i)) == m) return vc + e + i;
  }
  return -1;
}

__device__ __forceinline__ void ext_warp_merge(ExtState &e, float k) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ExtState t;
    t.mq = __shfl_xor_sync(0xFFFFFFFFu, e.mq, o);
    t.sq = __shfl_xor_sync(0xFFFFFFFFu, e.sq, o);
    t.aq = __shfl_xor_sync(0xFFFFFFFFu, e.aq, o);
    t.mp = __shfl_xor_sync(0xFFFFFFFFu, e.mp, o);
    t.sp = __shfl_xor_sync(0xFFFFFFFFu, e.sp, o);
    t.ap = __shfl_xor_sync(0xFFFFFFFFu, e.ap, o);
    t.x = __shfl_xor_sync(0xFFFFFFFFu, e.x, o);
    t.iq = __shfl_xor_sync(0xFFFFFFFFu, e.iq, o);
    t.ip = __shfl_xor_sync(0xFFFFFFFFu, e.ip, o);
    ext_merge(e, t, k);
  }
}

__device__ __forceinline__ ExtState ext_load(float4 ms, float4 m1, int2 idx) {
  return {ms.x, ms.y, m1.x, ms.z, ms.w, m1.y, m1.z, idx.x, idx.y};
}

// Pass 1 of kFamExt on one chunk of the slice (both rows at once, or the bonus
// row's p alone): this thread's kRounds vectors, in increasing vocabulary
// order, so that a strict comparison keeps the lowest index of a maximum.  v0
// is the vocabulary index of the chunk start.  Two reads of shared memory (the
// maxima, then the terms) keep few logits live; the chunk's terms are summed
// apart and then added, which keeps the f32 sums short.
template <typename E, bool kFull>
__device__ __forceinline__ void load8_chunk(const E *src, int e, int n, float (&y)[8]) {
  if constexpr (kFull) {
    Elt<E>::load8(src + e, y);
  } else {
    load8_smem(src, e, n, y);
  }
}

template <typename E, bool kFull, bool kPair>
__device__ __forceinline__ void ext_chunk(const E *srcq, const E *srcp, int n, int v0, float k,
                                          ExtState &st) {
  float mq = st.mq, mp = st.mp;
  int iq = st.iq, ip = st.ip;
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    float yq[8], yp[8];
    if constexpr (kPair) load8_chunk<E, kFull>(srcq, e, n, yq);
    load8_chunk<E, kFull>(srcp, e, n, yp);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if constexpr (kPair) {
        if (yq[i] > mq) {
          mq = yq[i];
          iq = v0 + e + i;
        }
      }
      if (yp[i] > mp) {
        mp = yp[i];
        ip = v0 + e + i;
      }
    }
  }
  const float rq = refk(mq, k), rp = refk(mp, k);
  ext_rebase(st, refk(st.mq, k) - rq, refk(st.mp, k) - rp);
  float sq = 0.0f, aq = 0.0f, sp = 0.0f, ap = 0.0f, x = 0.0f;
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    float yq[8], yp[8];
    if constexpr (kPair) load8_chunk<E, kFull>(srcq, e, n, yq);
    load8_chunk<E, kFull>(srcp, e, n, yp);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float b = fmaf(yp[i], k, -rp);
      const float eb = ex2(b);
      sp += eb;
      ap += eb > 0.0f ? eb * b : 0.0f;
      if constexpr (kPair) {
        const float a = fmaf(yq[i], k, -rq);
        const float ea = ex2(a);
        sq += ea;
        aq += ea > 0.0f ? ea * a : 0.0f;
        // a finite draft logit with a masked target logit (q(v) > 0 = p(v)) makes
        // D(q, p) = +inf even where 2^a underflows: X = -inf, kept by every merge
        x += yq[i] > -INFINITY && !(yp[i] > -INFINITY) ? -INFINITY : (ea > 0.0f ? ea * b : 0.0f);
      }
    }
  }
  st.mq = mq;
  st.mp = mp;
  st.iq = iq;
  st.ip = ip;
  st.sq = __fadd_rn(st.sq, sq);
  st.aq = __fadd_rn(st.aq, aq);
  st.sp = __fadd_rn(st.sp, sp);
  st.ap = __fadd_rn(st.ap, ap);
  st.x = __fadd_rn(st.x, x);
}

// kFamExt pass 1 of a pair, full bf16 chunk: ext_chunk's maxima, argmaxes,
// sums and moments in one read of shared memory, two logits at a time.  The
// maxima come from packed bf16x2 max trees; only a chunk that raises a running
// maximum is scanned for the lowest index holding it (later chunks hold higher
// indices, so an equal maximum keeps the earlier one).  The moments take the
// logits clamped at -1e30, so that a masked (-inf) logit gives 2^a = 0 and a
// finite product 0 * a = 0 where ext_chunk skips the term; a finite draft logit
// with a masked target logit still makes X = -inf (D(q, p) = +inf), found by a
// scan of the chunks whose target minimum is -inf.
__device__ __forceinline__ void ext_pair_bf16(const uint16_t *srcq, const uint16_t *srcp, int v0, float k,
                                              ExtState &st, bool argmax) {
  // two sweeps over the chunk in shared memory, one round (4 words per row) at
  // a time and not unrolled across rounds: the maxima, then the sums and
  // moments (the same order of additions as one sweep over all 16 words)
  __nv_bfloat162 xq = as_bf162(0xFF80FF80u), xp = xq, np = as_bf162(0x7F807F80u);  // -inf, -inf, +inf
#pragma unroll 1
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    const uint4 vq = *reinterpret_cast<const uint4 *>(srcq + e);
    const uint4 vp = *reinterpret_cast<const uint4 *>(srcp + e);
    const uint32_t wq[4] = {vq.x, vq.y, vq.z, vq.w}, wp[4] = {vp.x, vp.y, vp.z, vp.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      xq = __hmax2(xq, as_bf162(wq[i]));
      xp = __hmax2(xp, as_bf162(wp[i]));
      np = __hmin2(np, as_bf162(wp[i]));
    }
  }
  const float cq = fmaxf(__low2float(xq), __high2float(xq));
  const float cp = fmaxf(__low2float(xp), __high2float(xp));
  float mq = st.mq, mp = st.mp;
  int iq = st.iq, ip = st.ip;
  // (the argmaxes are read only by greedy decoding, located after pass 1)
  if (cq > mq) {
    mq = cq;
    if (argmax) iq = lazy_code(v0);
  }
  if (cp > mp) {
    mp = cp;
    if (argmax) ip = lazy_code(v0);
  }
  const float rq = refk(mq, k), rp = refk(mp, k);
  ext_rebase(st, refk(st.mq, k) - rq, refk(st.mp, k) - rp);
  const __nv_bfloat162 lo = __float2bfloat162_rn(-1e30f);
  const float2 kk = make_float2(k, k), nrq = make_float2(-rq, -rq), nrp = make_float2(-rp, -rp);
  const bool check_inf = !(fminf(__low2float(np), __high2float(np)) > -INFINITY);
  float2 sq = make_float2(0.0f, 0.0f), aq = sq, sp = sq, ap = sq, x = sq;
  bool inf_x = false;
#pragma unroll 1
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    const uint4 vq = *reinterpret_cast<const uint4 *>(srcq + e);
    const uint4 vp = *reinterpret_cast<const uint4 *>(srcp + e);
    const uint32_t wq[4] = {vq.x, vq.y, vq.z, vq.w}, wp[4] = {vp.x, vp.y, vp.z, vp.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 q2 = __hmax2(as_bf162(wq[i]), lo), p2 = __hmax2(as_bf162(wp[i]), lo);
      const float2 a = __ffma2_rn(__bfloat1622float2(q2), kk, nrq);
      const float2 b = __ffma2_rn(__bfloat1622float2(p2), kk, nrp);
      const float2 ea = make_float2(ex2(a.x), ex2(a.y)), eb = make_float2(ex2(b.x), ex2(b.y));
      sq = __fadd2_rn(sq, ea);
      sp = __fadd2_rn(sp, eb);
      aq = __ffma2_rn(ea, a, aq);
      ap = __ffma2_rn(eb, b, ap);
      x = __ffma2_rn(ea, b, x);
    }
    if (check_inf) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float q0 = __uint_as_float(wq[i] << 16), q1 = __uint_as_float(wq[i] & 0xFFFF0000u);
        const float p0 = __uint_as_float(wp[i] << 16), p1 = __uint_as_float(wp[i] & 0xFFFF0000u);
        inf_x |= (q0 > -INFINITY && !(p0 > -INFINITY)) || (q1 > -INFINITY && !(p1 > -INFINITY));
      }
    }
  }
  st.mq = mq;
  st.mp = mp;
  st.iq = iq;
  st.ip = ip;
  st.sq = __fadd_rn(st.sq, sq.x + sq.y);
  st.aq = __fadd_rn(st.aq, aq.x + aq.y);
  st.sp = __fadd_rn(st.sp, sp.x + sp.y);
  st.ap = __fadd_rn(st.ap, ap.x + ap.y);
  st.x = inf_x ? -INFINITY : __fadd_rn(st.x, x.x + x.y);
}

// Pass-1 screen of a token rule: per thread, the two largest logits of the row
// that r(v) tests (q for TokenV1, p otherwise) and the draft logit at the
// largest.  When every thread's second largest turns out deferred (r = 1), the
// tokens that are not deferred are exactly the threads' largest ones that pass
// the test, so eta = 1 - (their q) needs no pass over the row.
struct Top2 {
  float y1, y2, z1;
  int c1;      // chunk holding y1 (packed chunks: z1 not kept, looked up when needed)
  bool known;  // z1 holds the draft logit at y1
};

template <typename E, bool kFull>
__device__ __forceinline__ void screen_chunk(const E *ssrc, const E *qsrc, int n, Top2 &t) {
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    float y[8], z[8];
    load8_chunk<E, kFull>(ssrc, e, n, y);
    load8_chunk<E, kFull>(qsrc, e, n, z);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (y[i] > t.y2) {
        if (y[i] > t.y1) {
          t.y2 = t.y1;
          t.y1 = y[i];
          t.z1 = z[i];
          t.known = true;
        } else {
          t.y2 = y[i];
        }
      }
    }
  }
}

// Row scalars of the weight formulas.  With a_v = y^q_v k - R_q, b_v = y^p_v k - R_p
// (R = refk(M)) and c = log2(S_q / S_p):
//   q_v = 2^{a_v} / S_q,   p_v = 2^{b_v} / S_p = 2^{b_v + c} / S_q,
// and, up to the common factor 1/S_q, the weight of logit v is
//   kResidual  max(0, p - q) = max(0, 2^{b + c} - 2^a)   a rejected draft (Eq. 6 with
//              delta = 1), or the D_TV pass (Lemma 3)
//   kEta       r(v) q(v)                                eta = sum_v r(v) q(v) of a token rule
//   kTokenRes  max(0, eta p - r(v) q(v))                a rejected draft, token rule
// where r(v) = [a_v < thr] (TokenV1) or [b_v < thr] (TokenV2, TokenV3).
enum WeightKind : int { kResidual = 0, kEta = 1, kTokenRes = 2 };

struct RowScalars {
  float Rq, Rp, k, c;
  int kind;   // WeightKind
  int on_q;   // r(v) compares a_v (TokenV1) rather than b_v
  float thr;  // r(v) threshold, in the exponent domain of a or b
  float eta;  // eta of the row (kTokenRes)
};

// The sampling weights' scalars of a row from its records (R_q, R_p, c, flags)
// and (eta, thr, token, on_q): the residual max(0, pi - q) of a rejected draft
// under either target, or p of the bonus row.
__device__ __forceinline__ RowScalars sample_scalars(float4 r1, float4 r2, float k) {
  return {r1.x, r1.y, k, r1.z, __float_as_int(r2.z) ? kTokenRes : kResidual, __float_as_int(r2.w),
          r2.y, r2.x};
}

// Sampling weights of eight logits (see RowScalars), computed two at a time in
// packed f32x2; the bonus row (kPair = false) weighs p.  Returns their sum in
// index order.  Every pass and the search call exactly this, so the same logit
// always gets the same weight and the same prefix sums.
template <bool kPair, bool kTok>
__device__ __forceinline__ float vec_weights(const float (&yq)[8], const float (&yp)[8],
                                             const RowScalars &r, float (&w)[8]) {
  const float2 kk = make_float2(r.k, r.k);
  const float2 nrp = make_float2(-r.Rp, -r.Rp);
#pragma unroll
  for (int e = 0; e < 8; e += 2) {
    const float2 b = __ffma2_rn(make_float2(yp[e], yp[e + 1]), kk, nrp);
    if constexpr (kPair) {
      const float2 a = __ffma2_rn(make_float2(yq[e], yq[e + 1]), kk, make_float2(-r.Rq, -r.Rq));
      const float2 bc = __fadd2_rn(b, make_float2(r.c, r.c));
      if (!kTok || r.kind == kResidual) {  // (kTok: the kernel serves a token rule)
        const float2 d = __ffma2_rn(make_float2(ex2(a.x), ex2(a.y)), make_float2(-1.0f, -1.0f),
                                    make_float2(ex2(bc.x), ex2(bc.y)));
        w[e] = fmaxf(0.0f, d.x);
        w[e + 1] = fmaxf(0.0f, d.y);
      } else {
        const bool r0 = (r.on_q ? a.x : b.x) < r.thr, r1 = (r.on_q ? a.y : b.y) < r.thr;
        const float q0 = r0 ? ex2(a.x) : 0.0f, q1 = r1 ? ex2(a.y) : 0.0f;
        if (r.kind == kEta) {
          w[e] = q0;
          w[e + 1] = q1;
        } else {
          w[e] = fmaxf(0.0f, fmaf(r.eta, ex2(bc.x), -q0));
          w[e + 1] = fmaxf(0.0f, fmaf(r.eta, ex2(bc.y), -q1));
        }
      }
    } else {
      w[e] = ex2(b.x);
      w[e + 1] = ex2(b.y);
    }
  }
  float s = 0.0f;
#pragma unroll
  for (int e = 0; e < 8; ++e) s = __fadd_rn(s, w[e]);
  return s;
}

__device__ __forceinline__ float warp_incl_scan(float v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xFFFFFFFFu, v, o);
    if (lane >= o) v = __fadd_rn(v, t);
  }
  return v;
}

// Sum over a warp (butterfly, the same order in every lane and every call).
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Pass 1 on a chunk of the bonus row p_gamma: online_row's running (max, sum)
// and, per warp, the chunk's total weight sum_v 2^{y_v k - refk(W)}, W the
// warp's largest logit of the chunk, in seg[c kNW + warp] (W in
// seg[kBonusRef + c kNW + warp]).  After exchange 1 these give the chunk
// prefixes of p_gamma's inverse CDF, so a sequence that accepts every draft
// needs no second pass over its bonus row.
constexpr int kBonusRef = kMaxChunks * kNW;
static_assert(2 * kMaxChunks * kNW <= kEntries, "bonus chunk totals live in seg");
static_assert(kMaxChunks <= 32, "one lane per chunk of a slice");

template <typename E, bool kFull>
__device__ __forceinline__ void bonus_row(const E *src, int n, float k, float &m, float4 &s, int c,
                                          float *seg, int lane, int warp) {
  float y[kRounds][8];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    if constexpr (kFull) {
      Elt<E>::load8(src + e, y[r]);
    } else {
      load8_smem(src, e, n, y[r]);
    }
  }
  float W = -FLT_MAX;
#pragma unroll
  for (int r = 0; r < kRounds; ++r)
#pragma unroll
    for (int i = 0; i < 8; i += 2) W = max3(W, y[r][i], y[r][i + 1]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) W = fmaxf(W, __shfl_xor_sync(0xFFFFFFFFu, W, o));
  const float rw = refk(W, k);
  float c0 = 0.0f, c1 = 0.0f;
#pragma unroll
  for (int r = 0; r < kRounds; ++r)
#pragma unroll
    for (int i = 0; i < 8; i += 2) {
      c0 += ex2(fmaf(y[r][i], k, -rw));
      c1 += ex2(fmaf(y[r][i + 1], k, -rw));
    }
  const float cs = c0 + c1;
  // fold the chunk into the running sum, referenced to refk(max(m, W))
  const float mn = fmaxf(m, W), rn = refk(mn, k);
  const float so = ex2(refk(m, k) - rn);
  s = make_float4(fmaf(cs, ex2(rw - rn), s.x * so), s.y * so, s.z * so, s.w * so);
  m = mn;
  const float tot = warp_sum(cs);
  if (lane == 0 && SC_CHECK(c >= 0 && c < kMaxChunks)) {
    seg[c * kNW + warp] = tot;
    seg[kBonusRef + c * kNW + warp] = W;
  }
}

// OPT: this thread's sum over a chunk of 2^{(a_v + b_v)/2} = 2^{((y^q_v + y^p_v) k - r_q - r_p)/2},
// sqrt(q_v p_v) up to the rows' normalisers: the Bhattacharyya coefficient
// BC = sum_v sqrt(q_v p_v) bounds D_TV from above, D_TV <= sqrt(1 - BC^2).
template <typename E, bool kFull>
__device__ __forceinline__ float4 bc_chunk(const E *srcq, const E *srcp, int n, float hk, float hr) {
  float acc0 = 0.0f, acc1 = 0.0f, acc2 = 0.0f, acc3 = 0.0f;
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    float yq[8], yp[8];
    load8_chunk<E, kFull>(srcq, e, n, yq);
    load8_chunk<E, kFull>(srcp, e, n, yp);
#pragma unroll
    for (int i = 0; i < 8; i += 4) {
      acc0 += ex2(fmaf(yq[i] + yp[i], hk, -hr));
      acc1 += ex2(fmaf(yq[i + 1] + yp[i + 1], hk, -hr));
      acc2 += ex2(fmaf(yq[i + 2] + yp[i + 2], hk, -hr));
      acc3 += ex2(fmaf(yq[i + 3] + yp[i + 3], hk, -hr));
    }
  }
  return make_float4(acc0, acc1, acc2, acc3);  // (logits 0, 1, 2, 3 mod 4)
}

// OPT pair, full bf16 chunk: online_row of both rows and the chunk's
// 2^{(a_v + b_v)/2} terms (bc_chunk) in one sweep over the registers, so the
// logits are read from shared memory and unpacked once.  a_v and b_v are
// relative to the rows' updated references, as in bc_chunk, and the running
// sums are rescaled as online_row rescales its sums.
__device__ __forceinline__ void online_pair_bc(const uint16_t *srcq, const uint16_t *srcp, float k,
                                               float &mq, float4 &sq, float &mp, float4 &sp, float4 &bc) {
  uint32_t wq[kRounds * 4], wp[kRounds * 4];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    const uint4 vq = *reinterpret_cast<const uint4 *>(srcq + e);
    const uint4 vp = *reinterpret_cast<const uint4 *>(srcp + e);
    wq[4 * r] = vq.x; wq[4 * r + 1] = vq.y; wq[4 * r + 2] = vq.z; wq[4 * r + 3] = vq.w;
    wp[4 * r] = vp.x; wp[4 * r + 1] = vp.y; wp[4 * r + 2] = vp.z; wp[4 * r + 3] = vp.w;
  }
  __nv_bfloat162 xq = as_bf162(wq[0]), xp = as_bf162(wp[0]);
#pragma unroll
  for (int i = 1; i < kRounds * 4; ++i) {
    xq = __hmax2(xq, as_bf162(wq[i]));
    xp = __hmax2(xp, as_bf162(wp[i]));
  }
  const float mqn = fmaxf(mq, fmaxf(__low2float(xq), __high2float(xq)));
  const float mpn = fmaxf(mp, fmaxf(__low2float(xp), __high2float(xp)));
  const float rq = refk(mqn, k), rp = refk(mpn, k);
  const float dq = refk(mq, k) - rq, dp = refk(mp, k) - rp;
  const float fq = ex2(dq), fp = ex2(dp);
  float2 aq = __fmul2_rn(make_float2(sq.x, sq.y), make_float2(fq, fq));
  float2 ap = __fmul2_rn(make_float2(sp.x, sp.y), make_float2(fp, fp));
  float2 aq2 = __fmul2_rn(make_float2(sq.z, sq.w), make_float2(fq, fq));
  float2 ap2 = __fmul2_rn(make_float2(sp.z, sp.w), make_float2(fp, fp));
  const float fb = ex2(0.5f * (dq + dp));
  float2 h = __fmul2_rn(make_float2(bc.x, bc.y), make_float2(fb, fb));
  float2 h2 = __fmul2_rn(make_float2(bc.z, bc.w), make_float2(fb, fb));
  const float2 kk = make_float2(k, k), nrq = make_float2(-rq, -rq), nrp = make_float2(-rp, -rp);
  const float2 half = make_float2(0.5f, 0.5f);
#pragma unroll
  for (int i = 0; i < kRounds * 4; ++i) {
    const float2 yq = make_float2(__uint_as_float(wq[i] << 16), __uint_as_float(wq[i] & 0xFFFF0000u));
    const float2 yp = make_float2(__uint_as_float(wp[i] << 16), __uint_as_float(wp[i] & 0xFFFF0000u));
    const float2 a = __ffma2_rn(yq, kk, nrq);
    const float2 b = __ffma2_rn(yp, kk, nrp);
    const float2 ea = make_float2(ex2(a.x), ex2(a.y)), eb = make_float2(ex2(b.x), ex2(b.y));
    const float2 hh = __fmul2_rn(__fadd2_rn(a, b), half);
    const float2 eh = make_float2(ex2(hh.x), ex2(hh.y));
    if (i & 1) {  // logits 2, 3 (mod 4)
      aq2 = __fadd2_rn(aq2, ea);
      ap2 = __fadd2_rn(ap2, eb);
      h2 = __fadd2_rn(h2, eh);
    } else {      // logits 0, 1 (mod 4)
      aq = __fadd2_rn(aq, ea);
      ap = __fadd2_rn(ap, eb);
      h = __fadd2_rn(h, eh);
    }
  }
  mq = mqn;
  mp = mpn;
  sq = make_float4(aq.x, aq.y, aq2.x, aq2.y);
  sp = make_float4(ap.x, ap.y, ap2.x, ap2.y);
  bc = make_float4(h.x, h.y, h2.x, h2.y);
}

// Weights of one chunk in the ring: per round, the warp's total weight (the
// segment total) lands in seg[(c, round, warp)].  Every round's weights come
// before any reduction or store, so the rounds' shared-memory loads and
// exponentials overlap (a store to seg between rounds would order the next
// round's loads after it), and the rounds' warp sums run interleaved, each in
// warp_sum's butterfly order (the same totals as one warp_sum per round).
template <typename E, bool kPair, bool kFull, bool kTok>
__device__ __forceinline__ void weights_chunk(const E *sq, const E *sp, int n, int c,
                                              const RowScalars &rs, Shared &sh, int lane,
                                              int warp) {
  float tot[kRounds];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int e = 8 * (r * kNT + static_cast<int>(threadIdx.x));
    float yq[8], yp[8], w[8];
    if constexpr (kFull) {
      if constexpr (kPair) Elt<E>::load8(sq + e, yq);
      Elt<E>::load8(sp + e, yp);
    } else {
      if constexpr (kPair) load8_smem(sq, e, n, yq);
      load8_smem(sp, e, n, yp);
    }
    tot[r] = vec_weights<kPair, kTok>(yq, yp, rs, w);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int r = 0; r < kRounds; ++r) tot[r] = __fadd_rn(tot[r], __shfl_xor_sync(0xFFFFFFFFu, tot[r], o));
  }
  if (lane == 0 && SC_CHECK(c >= 0 && c < kMaxChunks)) {
#pragma unroll
    for (int r = 0; r < kRounds; ++r) sh.seg[(c * kRounds + r) * kNW + warp] = tot[r];
  }
}

// Double-float arithmetic in f32 (the GPU's f64 rate is a small fraction of
// its f32 rate): a value is hi + lo with |lo| <= ulp(hi) / 2.  two_sum is
// Knuth's error-free sum, a + b = s + e exactly; an FMA gives a product's
// rounding error exactly.
__device__ __forceinline__ float2 two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return make_float2(s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb)));
}
__device__ __forceinline__ float2 df_norm(float hi, float lo) {
  const float s = __fadd_rn(hi, lo);
  return make_float2(s, __fsub_rn(lo, __fsub_rn(s, hi)));
}
// y (k + kl) as hi + lo
__device__ __forceinline__ float2 df_mul_k(float y, float k, float kl) {
  const float p = __fmul_rn(y, k);
  return make_float2(p, fmaf(y, kl, fmaf(y, k, -p)));
}
// a - b, and comparisons with a float
__device__ __forceinline__ float2 df_sub(float2 a, float b) {
  const float2 s = two_sum(a.x, -b);
  return df_norm(s.x, __fadd_rn(s.y, a.y));
}
__device__ __forceinline__ bool df_ge(float2 a, float b) { return a.x > b || (a.x == b && a.y >= 0.0f); }
__device__ __forceinline__ bool df_lt(float2 a, float b) { return a.x < b || (a.x == b && a.y < 0.0f); }
// the largest float <= a
__device__ __forceinline__ float df_floor(float2 a) { return a.y < 0.0f ? nextafterf(a.x, -INFINITY) : a.x; }
// 2^a to f32 accuracy: 2^hi (1 + lo ln 2)
__device__ __forceinline__ float df_exp2(float2 a) { return exp2f(a.x) * fmaf(a.y, 0.69314718f, 1.0f); }

// log2 of a softmax probability of the row with maximum M, reference R and
// pass-1 sum S, as hi + lo.  S sums 2^{fma(y_v, k, -R)}: its exponents use the
// f32 factor k, and differ from the exact y_v (k + kl) - R by -y_v kl =
// -M kl - (y_v - M) kl.  For every term that S holds to f32 accuracy, (y_v - M) kl
// is below ~1e-6 (y_v - M >= -24 / k there, |kl| <= ulp(k) / 2), so the exact
// sum is 2^{M kl} S to that accuracy, and
//   log2 p(y) = y (k + kl) - R - log2 S - M kl = y k - R + (y - M) kl - log2 S.
// (M kl alone reaches 1e-3 for logits near 3e4 at T = 1, or 3e3 at T = 0.1.)
__device__ __forceinline__ float2 log2_prob(float y, float M, float R, float S, float k, float kl) {
  const float p = __fmul_rn(y, k);
  const float e = fmaf(y, k, -p);  // y k = p + e exactly
  const float2 t = two_sum(p, -R);
  const float lo = __fadd_rn(__fadd_rn(t.y, e), __fmul_rn(__fsub_rn(y, M), kl));
  return df_norm(t.x, __fadd_rn(lo, -log2f(S)));
}

// A softmax probability from its logit; 0 for a masked (-inf) logit.
__device__ __forceinline__ float prob_of(float y, float M, float R, float S, float k, float kl) {
  return y > -INFINITY ? df_exp2(log2_prob(y, M, R, S, k, kl)) : 0.0f;
}

// Acceptance of the draft token x (Algorithm 4): a = 1 when delta = 0 or
// q(x) <= pi(x), else a = [u < pi(x)/q(x)].  L = log2 p(x) - log2 q(x)
//   = (y_p(x) - y_q(x)) k - (R_p - R_q) + ((y_p(x) - M_p) - (y_q(x) - M_q)) kl
//     + log2(S_q / S_p)
// (see log2_prob) is formed in double-float from the logits, so the ratio 2^L
// carries essentially only the f32 error of log2(S_q / S_p).  With a token rule
// (Section 4.4) the draft token's own deferral r(x) takes delta's place and
// pi(x)/q(x) = (1 - r(x)) + eta p(x)/q(x): accepted outright when r(x) = 0,
// else [u < eta 2^L].  With lossy speculative decoding (Table 3, delta = 1)
// the ratio is min(1, p(x) / ((1 - alpha) q(x))) (Lemma 2): L shifted by
// -log2(1 - alpha).  Greedy decoding compares indices only.  A masked logit
// (-inf) is handled before L, whose double-float terms it would turn into NaN:
// q(x) = 0 accepts, and p(x) = 0 < q(x) makes the ratio 1 - delta.  q(x) and
// pi(x) themselves are evaluated only for the diagnostics output.
template <int kFam>
__device__ __forceinline__ void accept_test(Shared &sh, const Params &P, int x, float yqx, float ypx,
                                            float u, float k) {
  constexpr bool kTok = kFam == kFamToken;
  const float kl = P.kl;
  if constexpr (kFam == kFamExt) {
    if (P.greedy) {
      // one-hot q~ and p~ at the argmaxes: pi(x)/q~(x) is 1 unless delta = 1 and
      // x is not p's argmax (then 0); a draft with q~(x) = 0 is accepted
      const bool on_q = x == sh.iq, on_p = x == sh.ip;
      sh.accept = !(on_q && sh.delta && !on_p);
      sh.qx = on_q ? 1.0f : 0.0f;
      sh.pix = sh.delta ? (on_p ? 1.0f : 0.0f) : sh.qx;
      return;
    }
  }
  const bool lossy = kFam == kFamCascade && P.rule == SC_RULE_LOSSY;
  if (kTok && sh.tok) {
    const float ax = fmaf(yqx, k, -sh.Rq), bx = fmaf(ypx, k, -sh.Rp);  // as vec_weights forms them
    sh.delta = (sh.on_q ? ax : bx) < sh.thr;                           // reported: r(x)
  }
  int accept = 1;
  if (!(yqx > -INFINITY)) {
    // q(x) = 0: accepted
  } else if (!(ypx > -INFINITY)) {
    accept = !sh.delta;  // p(x) = 0 < q(x): pi(x)/q(x) = 1 - delta (also eta p/q = 0 for a token rule)
  } else if (sh.delta) {
    const float2 d = two_sum(ypx, -yqx);  // y_p(x) - y_q(x), exactly
    const float2 dk = df_mul_k(d.x, k, 0.0f);  // d.x k, exactly
    const float2 r = two_sum(sh.Rp, -sh.Rq);
    const float2 s = two_sum(dk.x, -r.x);
    const float corr = __fmul_rn(__fsub_rn(__fsub_rn(ypx, sh.Mp), __fsub_rn(yqx, sh.Mq)), kl);
    const float lo = __fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(s.y, dk.y), __fsub_rn(__fmul_rn(d.y, k), r.y)), corr),
                               log2f(sh.Sq / sh.Sp));
    float2 L = df_norm(s.x, lo);
    if (kTok && sh.tok) {
      if (L.x < INFINITY) accept = u < sh.eta * df_exp2(L);  // (q(x) = 0 accepts)
    } else {
      if (lossy) {
        if (P.lossy_l < INFINITY) {
          const float2 t = two_sum(L.x, P.lossy_l);
          L = df_norm(t.x, __fadd_rn(__fadd_rn(t.y, L.y), P.lossy_ll));
        } else {
          L = make_float2(0.0f, 0.0f);  // alpha = 1 and p(x) > 0 here: the ratio is 1
        }
      }
      if (df_lt(L, 0.0f)) accept = u < df_exp2(L);
    }
  }
  sh.accept = accept;
  if (P.row_info != nullptr) {
    const float qx = prob_of(yqx, sh.Mq, sh.Rq, sh.Sq, k, kl);
    const float px = prob_of(ypx, sh.Mp, sh.Rp, sh.Sp, k, kl);
    sh.qx = qx;
    if (kTok && sh.tok) sh.pix = fmaf(sh.eta, px, sh.delta ? 0.0f : qx);
    else if (lossy)  // (alpha = 1: the limit alpha -> 1-, p / (1 - alpha) = +inf where p > 0, 0 where p = 0)
      sh.pix = fmaxf(fminf(qx, P.alpha < 1.0f ? px / (1.0f - P.alpha) : (px > 0.0f ? INFINITY : 0.0f)), px / P.beta);
    else sh.pix = sh.delta ? px : qx;
  }
}

// ------------------------------------------------------------------ chunk ring

template <typename E>
struct Ring {
  E *base;        // kStages stages of [2][kCH] logits (q then p)
  const E *gq;    // slice start in global memory
  const E *gp;
  int len;        // valid logits in the slice
  int nch;        // chunks in the slice
  int first;      // chunks c < first are copied with the L2 evict-first policy
  bool pair;
  bool bulk;
  __device__ E *q(int s) const { return base + static_cast<size_t>(s) * 2 * kCH; }
  __device__ E *p(int s) const { return q(s) + kCH; }
  __device__ int chunk_len(int c) const { return min(kCH, len - c * kCH); }
  // thread 0, bulk mode: start the copies of chunk c into stage s
  __device__ void issue(Shared &sh, int c, int s) const {
    const uint32_t bytes = static_cast<uint32_t>(chunk_len(c)) * sizeof(E);
    if (!SC_CHECK(c >= 0 && c < nch && s >= 0 && s < kStages && bytes > 0 && bytes % 16 == 0 &&
                  reinterpret_cast<uintptr_t>(gp + static_cast<size_t>(c) * kCH) % 16 == 0 &&
                  (!pair || reinterpret_cast<uintptr_t>(gq + static_cast<size_t>(c) * kCH) % 16 == 0)))
      return;
    mbar_expect_tx(&sh.full[s], pair ? 2 * bytes : bytes);
    if (c < first) {
      const uint64_t pol = evict_first_policy();
      if (pair) bulk_g2s_hint(q(s), gq + static_cast<size_t>(c) * kCH, bytes, &sh.full[s], pol);
      bulk_g2s_hint(p(s), gp + static_cast<size_t>(c) * kCH, bytes, &sh.full[s], pol);
    } else {
      if (pair) bulk_g2s(q(s), gq + static_cast<size_t>(c) * kCH, bytes, &sh.full[s]);
      bulk_g2s(p(s), gp + static_cast<size_t>(c) * kCH, bytes, &sh.full[s]);
    }
  }
  // thread 0, bulk mode: hint chunk c into L2
  __device__ void prefetch(int c) const {
    const uint32_t bytes = static_cast<uint32_t>(chunk_len(c)) * sizeof(E);
    if (!SC_CHECK(c >= 0 && c < nch && bytes > 0 && bytes % 16 == 0 &&
                  reinterpret_cast<uintptr_t>(gp + static_cast<size_t>(c) * kCH) % 16 == 0 &&
                  (!pair || reinterpret_cast<uintptr_t>(gq + static_cast<size_t>(c) * kCH) % 16 == 0)))
      return;
    if (pair) prefetch_l2(gq + static_cast<size_t>(c) * kCH, bytes);
    prefetch_l2(gp + static_cast<size_t>(c) * kCH, bytes);
  }
  // all threads, per-thread mode: copy chunk c into stage s
  __device__ void load_sync(int c, int s) const {
    if (!SC_CHECK(c >= 0 && c < nch && s >= 0 && s < kStages)) return;
    const int n = chunk_len(c);
    const size_t o = static_cast<size_t>(c) * kCH;
    for (int i = threadIdx.x; i < n; i += kNT) {
      if (pair) q(s)[i] = gq[o + i];
      p(s)[i] = gp[o + i];
    }
  }
};

// A ring over slice `rank` of row pair (b, j) -- only the target row when j is
// the bonus position gamma.
template <typename E>
__device__ __forceinline__ Ring<E> make_ring(const Params &P, unsigned char *smem, int b, int j,
                                             int rank) {
  const int v0 = rank * P.L;
  Ring<E> R;
  R.base = reinterpret_cast<E *>(smem);
  R.pair = j < P.gamma;
  R.gq = static_cast<const E *>(P.draft) +
         (static_cast<size_t>(b) * P.gamma + (R.pair ? j : 0)) * P.V + v0;
  R.gp = static_cast<const E *>(P.target) + (static_cast<size_t>(b) * (P.gamma + 1) + j) * P.V + v0;
  R.len = max(0, min(P.L, P.V - v0));
  R.nch = (R.len + kCH - 1) / kCH;
  R.bulk = P.bulk != 0;
  // a second pass over a pair (TV, residual) streams newest chunk first: it finds
  // more of its slice in L2 when every slice's older chunks, which it would miss
  // anyway, leave L2 first; a bonus row is never read again
  R.first = !P.l2_hint || P.mode != kVerify ? 0 : (R.pair ? max(0, R.nch - P.l2_hint) : R.nch);
  return R;
}

// Every pass starts with all stages free and puts chunk c in stage c % kStages.
// Bit s of `ph` is the parity of the next completion of stage s's mbarrier;
// all threads keep identical copies.
template <typename E>
__device__ __forceinline__ void prime(const Ring<E> &R, Shared &sh) {
  if (R.bulk && threadIdx.x == 0)
    for (int c = 0; c < min(kStages, R.nch); ++c) R.issue(sh, c, c);
}

__device__ __forceinline__ int wait_stage(Shared &sh, int s, uint32_t &ph) {
  const bool ok = mbar_wait(&sh.full[s], (ph >> s) & 1u);
  ph ^= 1u << s;
  return ok ? 0 : 1;
}

// Stream every chunk of the slice through the ring (primed by prime()) and call
// body(c, stage) on each.  Returns 1 if a copy did not land within the wait limit.
template <typename E, typename Body>
__device__ __forceinline__ int stream(const Ring<E> &R, Shared &sh, uint32_t &ph, Body &&body) {
  int tmo = 0;
  for (int c = 0; c < R.nch; ++c) {
    const int s = c % kStages;
    if (R.bulk) {
      tmo |= wait_stage(sh, s, ph);
    } else {
      R.load_sync(c, s);
      __syncthreads();
    }
    body(c, s);
    __syncthreads();  // every thread is done with stage s
    if (R.bulk && threadIdx.x == 0 && c + kStages < R.nch) R.issue(sh, c + kStages, s);
  }
  return tmo;
}

// A pass over the slice in reverse chunk order, newest first: a row streamed a
// moment ago has its last chunks in L2 (and, with `resident`, its last
// min(kStages, nch) chunks still in the ring in stages c % kStages, which
// need no copy), while its first chunks may already have been evicted.
template <typename E, typename Body>
__device__ __forceinline__ int stream_rev(const Ring<E> &R, Shared &sh, uint32_t &ph, bool resident,
                                          Body &&body) {
  const int nch = R.nch;
  const int nres = resident ? min(kStages, nch) : 0;
  if (!resident && R.bulk && threadIdx.x == 0)
    for (int c = nch - 1; c >= max(0, nch - kStages); --c) R.issue(sh, c, c % kStages);
  // a second pass finds its older chunks mostly gone from L2 and streams them with
  // only the ring in flight: ask for all of them at once, in the order they are used
  if (SC_L2_PREFETCH && R.bulk && threadIdx.x == 0)
    for (int c = nch - 1 - kStages; c >= 0; --c) R.prefetch(c);
  int tmo = 0;
  for (int i = 0; i < nch; ++i) {
    const int c = nch - 1 - i, s = c % kStages;
    if (i >= nres) {
      if (R.bulk) {
        tmo |= wait_stage(sh, s, ph);
      } else {
        R.load_sync(c, s);
        __syncthreads();
      }
    }
    body(c, s);
    __syncthreads();  // every thread is done with stage s
    if (R.bulk && threadIdx.x == 0 && c - kStages >= 0) R.issue(sh, c - kStages, s);
  }
  return tmo;
}

// Residual weights of one slice: per-(chunk, round, warp) totals in sh.seg.
enum SliceOrder { kNewestFirst, kNewestFirstResident };

template <bool kTok, typename E>
__device__ __forceinline__ int slice_weights(const Ring<E> &R, Shared &sh, uint32_t &ph,
                                             const RowScalars &rs, SliceOrder order, int lane, int warp) {
  auto body = [&](int c, int s) {
    const int n = R.chunk_len(c);
    if (R.pair) {
      if (n == kCH) weights_chunk<E, true, true, kTok>(R.q(s), R.p(s), n, c, rs, sh, lane, warp);
      else weights_chunk<E, true, false, kTok>(R.q(s), R.p(s), n, c, rs, sh, lane, warp);
    } else {
      if (n == kCH) weights_chunk<E, false, true, kTok>(R.q(s), R.p(s), n, c, rs, sh, lane, warp);
      else weights_chunk<E, false, false, kTok>(R.q(s), R.p(s), n, c, rs, sh, lane, warp);
    }
  };
  return stream_rev(R, sh, ph, order == kNewestFirstResident, body);
}

// One warp: turn sh.seg[0, nseg) into exclusive prefixes in vocabulary order
// (chunk, round, warp); returns the slice total (in every lane), also left in
// sh.seg[nseg].  Lane l sums its run of ceil(nseg / 32) entries in order, a warp
// scan gives each run's start, and each lane writes its run's prefixes.
__device__ __forceinline__ float seg_prefix(Shared &sh, int nseg, int lane) {
  const int per = (nseg + 31) >> 5;
  const int i0 = min(nseg, lane * per), i1 = min(nseg, i0 + per);
  float t = 0.0f;
  for (int i = i0; i < i1; ++i) t = __fadd_rn(t, sh.seg[i]);
  const float incl = warp_incl_scan(t, lane);
  float acc = __shfl_up_sync(0xFFFFFFFFu, incl, 1);
  if (lane == 0) acc = 0.0f;
  for (int i = i0; i < i1; ++i) {
    const float v = sh.seg[i];
    sh.seg[i] = acc;
    acc = __fadd_rn(acc, v);
  }
  const float tot = __shfl_sync(0xFFFFFFFFu, incl, 31);
  if (lane == 0) sh.seg[nseg] = tot;
  return tot;
}

__device__ __forceinline__ void flag_timeout(Shared &sh, const Params &P) {
  sh.timeout = 1;
  if (P.status) atomicOr(P.status, static_cast<int32_t>(SC_DEV_TIMEOUT));
}

// ------------------------------------------------------------------ the kernel

__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t *p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ unsigned long long atom_or_acq_rel(unsigned long long *p, unsigned long long v) {
  unsigned long long old;
  asm volatile("atom.acq_rel.gpu.global.or.b64 %0, [%1], %2;" : "=l"(old) : "l"(p), "l"(v) : "memory");
  return old;
}
__device__ __forceinline__ unsigned long long atom_add_acq_rel(unsigned long long *p, unsigned long long v) {
  unsigned long long old;
  asm volatile("atom.acq_rel.gpu.global.add.u64 %0, [%1], %2;" : "=l"(old) : "l"(p), "l"(v) : "memory");
  return old;
}

// With arrivals (bits 0..31) and rejections (bits 32..63) of one slice rank's
// units, is j* = min{j : a_j = 0} settled -- the first rejection with every
// earlier position in, or all gamma + 1 positions in without one?  Sets js.
__device__ __forceinline__ bool jstar_settled(unsigned long long m, int G1, int &js) {
  const uint32_t arr = static_cast<uint32_t>(m), rej = static_cast<uint32_t>(m >> 32);
  if (rej) {
    js = __ffs(rej) - 1;
    const uint32_t need = js == 31 ? 0xFFFFFFFFu : (2u << js) - 1u;
    return (arr & need) == need;
  }
  js = G1 - 1;
  return arr == (G1 == 32 ? 0xFFFFFFFFu : (1u << G1) - 1u);
}

// The token inside segment (round r, this warp) of a chunk held in shared
// memory (sq, sp; n valid logits): its weights are recomputed with vec_weights
// -- the values weights_chunk summed -- and the smallest k whose running sum
// passes t is taken (the smallest k with C_k > u R).  Without t (u R fell past
// the last boundary by rounding), the segment's last positive weight.  v0 is
// the vocabulary index of the chunk start.
template <bool kTok, typename E>
__device__ __forceinline__ int search_segment(const E *sq, const E *sp, int n, bool pair,
                                              const RowScalars &rs, int v0, int r, bool have_t,
                                              float t, int lane, int warp) {
  const int e = 8 * (r * kNT + warp * 32 + lane);
  float yq[8], yp[8], w[8];
  if (pair) load8_smem(sq, e, n, yq);
  load8_smem(sp, e, n, yp);
  const float vs = pair ? vec_weights<true, kTok>(yq, yp, rs, w) : vec_weights<false, kTok>(yq, yp, rs, w);
  const float incl = warp_incl_scan(vs, lane);
  float excl = __shfl_up_sync(0xFFFFFFFFu, incl, 1);
  if (lane == 0) excl = 0.0f;
  const float tt0 = have_t ? t : FLT_MAX;
  int tok = -1;
  const unsigned mm = __ballot_sync(0xFFFFFFFFu, tt0 >= excl && tt0 < incl && vs > 0.0f);
  if (mm) {
    const int src = __ffs(mm) - 1;
    if (lane == src) {
      const float tt = __fsub_rn(tt0, excl);
      float acc = 0.0f;
      int last = -1;
      for (int i = 0; i < 8; ++i) {
        acc = __fadd_rn(acc, w[i]);
        if (w[i] > 0.0f) last = i;
        if (tok < 0 && acc > tt) tok = i;
      }
      if (tok < 0) tok = last;
      tok = v0 + e + tok;
    }
    tok = __shfl_sync(0xFFFFFFFFu, tok, src);
  } else {
    int last = -1;
    for (int i = 0; i < 8; ++i)
      if (w[i] > 0.0f) last = i;
    const unsigned lm = __ballot_sync(0xFFFFFFFFu, last >= 0);
    if (lm) {
      const int ln = 31 - __clz(lm);
      const int li = __shfl_sync(0xFFFFFFFFu, last, ln);
      tok = v0 + 8 * (r * kNT + warp * 32 + ln) + li;
    }
  }
  return tok;
}

// Row pair (b, j < gamma) or bonus row (b, gamma) of a unit (pairs only for sc_row_stats).
__device__ __forceinline__ void unit_coords(const Params &P, int unit, int &b, int &j) {
  const int G1 = P.gamma + 1;
  if (P.mode == kVerify && P.pos_major) {
    // every sequence's position j before any sequence's position j + 1: a
    // rejected pair then mostly finds an earlier rejection of its sequence
    // already reported, and skips the residual pass of a row that is not j*
    b = unit % P.B;
    j = unit / P.B;
  } else if (P.mode == kVerify) {
    b = unit / G1;
    j = unit % G1;
  } else {
    b = unit / P.gamma;
    j = unit % P.gamma;
  }
}

template <typename E, int kFam>
__global__ void __launch_bounds__(kNT, kMinBlocksPerSM) sc_unit_kernel(const Params P) {
  constexpr bool kTok = kFam == kFamToken;
  constexpr bool kExt = kFam == kFamExt;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  cg::cluster_group cluster = cg::this_cluster();
  const int C = P.cluster;
  const int rank = static_cast<int>(cluster.block_rank());
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G1 = P.gamma + 1;
  const bool verify = P.mode == kVerify;
  Shared &sh = *reinterpret_cast<Shared *>(smem_raw + static_cast<size_t>(kStages) * 2 * kCH * sizeof(E));
  if (tid == 0) {
    sh.timeout = 0;
    if (P.bulk) {
      for (int s = 0; s < kStages; ++s) mbar_init(&sh.full[s], 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
  }
  uint32_t ph = 0;  // phase bits of the ring's stages (see wait_stage)

  // one cluster per unit: every CTA of the cluster works on unit blockIdx / C
  const int unit = static_cast<int>(blockIdx.x) / C;
  int b, j;
  unit_coords(P, unit, b, j);
  const int v0 = rank * P.L;
  const Ring<E> R = make_ring<E>(P, smem_raw, b, j, rank);
  const bool pair = R.pair;

  // ---- start the stream; prefetch the row's scalars
  if (tid == 0) {
    sh.xq = NAN;
    sh.xp = NAN;
  }
  prime(R, sh);
  float uj = 0.0f, ug = 0.0f;
  int x = -1;
  if (verify && tid == 0) {
    uj = P.uniforms[static_cast<size_t>(b) * G1 + j];
    ug = P.uniforms[static_cast<size_t>(b) * G1 + P.gamma];
    if (pair) x = P.tokens[static_cast<size_t>(b) * P.gamma + j];
  }
  __syncthreads();
  cluster_arrive_relaxed();  // this CTA has started (peers may store into it after their wait)

  // ---- pass 1: online max and sum of exponentials
  const float k = P.k;
  float mq = -FLT_MAX, mp = -FLT_MAX;
  float4 s2q = make_float4(0.0f, 0.0f, 0.0f, 0.0f), s2p = s2q;
  ExtState ex = ext_empty();  // (kFamExt) moments and argmaxes
  Top2 top = {-FLT_MAX, -FLT_MAX, -FLT_MAX, -1, false};  // (kFamToken) the eta screen
  const bool scr_q = P.rule == SC_RULE_TOKEN_V1;
  // OPT: the pair's running sum of sqrt(q p) terms, relative to (r_q + r_p) / 2
  const bool opt_bc = SC_OPT_UB && P.opt_ub && !kTok && !kExt && verify && pair && P.rule == SC_RULE_OPT;
  // the pair's running sums of sqrt(q p) terms over this thread's logits 0, 1, 2, 3
  // (mod 4), relative to (r_q + r_p) / 2
  float4 bc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  // the bonus row also leaves its per-(chunk, warp) totals for the sampler
  const bool bonus_tot = verify && !pair && !P.greedy;
  const int lx = x - v0;  // draft token's offset in this slice (thread 0 only)
  int tmo = stream(R, sh, ph, [&](int c, int s) {
    const int n = R.chunk_len(c);
    if (bonus_tot) {
      if (n == kCH) bonus_row<E, true>(R.p(s), n, k, mp, s2p, c, sh.seg, lane, warp);
      else bonus_row<E, false>(R.p(s), n, k, mp, s2p, c, sh.seg, lane, warp);
    } else if constexpr (kExt) {
      const int vc = v0 + c * kCH;
      if (pair) {
        bool done = false;
        if constexpr (sizeof(E) == 2) {
          if (n == kCH) {
            ext_pair_bf16(reinterpret_cast<const uint16_t *>(R.q(s)), reinterpret_cast<const uint16_t *>(R.p(s)),
                          vc, k, ex, P.greedy != 0);
            done = true;
          }
        }
        if (!done) {
          if (n == kCH) ext_chunk<E, true, true>(R.q(s), R.p(s), n, vc, k, ex);
          else ext_chunk<E, false, true>(R.q(s), R.p(s), n, vc, k, ex);
        }
      } else {
        bool done = false;
        if constexpr (sizeof(E) == 2) {
          if (n == kCH && P.greedy) {
            ext_bonus_bf16(reinterpret_cast<const uint16_t *>(R.p(s)), vc, k, ex);
            done = true;
          }
        }
        if (!done) {
          if (n == kCH) ext_chunk<E, true, false>(R.q(s), R.p(s), n, vc, k, ex);
          else ext_chunk<E, false, false>(R.q(s), R.p(s), n, vc, k, ex);
        }
      }
    } else {
      bool fused = false;
      if constexpr (sizeof(E) == 2) {
        if (opt_bc && n == kCH) {
          online_pair_bc(reinterpret_cast<const uint16_t *>(R.q(s)), reinterpret_cast<const uint16_t *>(R.p(s)),
                         k, mq, s2q, mp, s2p, bc);
          fused = true;
        }
      }
      if (!fused) {
        const float mq0 = mq, mp0 = mp;
        bool screened = false;
        if constexpr (kTok && sizeof(E) == 2) {
          if (pair && n == kCH) {
            // the screened row's top two come out of its max sweep; the draft
            // logit at the largest is looked up only if the screen needs it
            const uint16_t *sq16 = reinterpret_cast<const uint16_t *>(R.q(s));
            const uint16_t *sp16 = reinterpret_cast<const uint16_t *>(R.p(s));
            float c1, c2;
            if (scr_q) {
              online_row_top2(sq16, k, mq, s2q, c1, c2);
              online_row<uint16_t, true>(sp16, n, k, mp, s2p);
            } else {
              online_row<uint16_t, true>(sq16, n, k, mq, s2q);
              online_row_top2(sp16, k, mp, s2p, c1, c2);
            }
            if (c1 > top.y1) {
              top.y2 = fmaxf(top.y1, c2);
              top.y1 = c1;
              top.c1 = c;
              top.known = false;
            } else {
              top.y2 = fmaxf(top.y2, c1);
            }
            screened = true;
          }
        }
        if (screened) {
        } else if (n == kCH) {
          if (pair) online_row<E, true>(R.q(s), n, k, mq, s2q);
          online_row<E, true>(R.p(s), n, k, mp, s2p);
          if (kTok && pair) screen_chunk<E, true>(scr_q ? R.q(s) : R.p(s), R.q(s), n, top);
        } else {
          if (pair) online_row<E, false>(R.q(s), n, k, mq, s2q);
          online_row<E, false>(R.p(s), n, k, mp, s2p);
          if (kTok && pair) screen_chunk<E, false>(scr_q ? R.q(s) : R.p(s), R.q(s), n, top);
        }
        if (opt_bc) {
          const float rq = refk(mq, k), rp = refk(mp, k);
          const float sc = ex2(0.5f * ((refk(mq0, k) - rq) + (refk(mp0, k) - rp)));
          const float4 add = n == kCH ? bc_chunk<E, true>(R.q(s), R.p(s), n, 0.5f * k, 0.5f * (rq + rp))
                                      : bc_chunk<E, false>(R.q(s), R.p(s), n, 0.5f * k, 0.5f * (rq + rp));
          bc = make_float4(fmaf(bc.x, sc, add.x), fmaf(bc.y, sc, add.y), fmaf(bc.z, sc, add.z), fmaf(bc.w, sc, add.w));
        }
      }
    }
    if (tid == 0 && static_cast<unsigned>(lx - c * kCH) < static_cast<unsigned>(n)) {
      sh.xq = Elt<E>::at(R.q(s), lx - c * kCH);
      sh.xp = Elt<E>::at(R.p(s), lx - c * kCH);
    }
  });
  if constexpr (kExt) {
    if (bonus_tot) {
      ex.mp = mp;
      ex.sp = (s2p.x + s2p.y) + (s2p.z + s2p.w);
    }
    mq = ex.mq;
    mp = ex.mp;
    s2q = make_float4(ex.sq, 0.0f, 0.0f, 0.0f);
    s2p = make_float4(ex.sp, 0.0f, 0.0f, 0.0f);
  }
  float s_q = (s2q.x + s2q.y) + (s2q.z + s2q.w), s_p = (s2p.x + s2p.y) + (s2p.z + s2p.w);
  const float4 mine = make_float4(mq, s_q, mp, s_p);  // this thread's partial, kept for the D_TV bounds
  const float4 mq4 = s2q, mp4 = s2p;  // ... split over its logits 0, 1, 2, 3 (mod 4)
  tmo = __syncthreads_or(tmo);
  if constexpr (kExt) {
    if (P.greedy) {
      // locate the argmaxes recorded as chunk codes, for the threads holding their
      // warp's maximum (the others cannot win the merge)
      float wq = ex.mq, wp = ex.mp;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        wq = fmaxf(wq, __shfl_xor_sync(0xFFFFFFFFu, wq, o));
        wp = fmaxf(wp, __shfl_xor_sync(0xFFFFFFFFu, wp, o));
      }
      if (ex.iq <= -2 && ex.mq == wq) ex.iq = ext_resolve_index(R.gq, v0, -2 - ex.iq, ex.mq);
      if (ex.ip <= -2 && ex.mp == wp) ex.ip = ext_resolve_index(R.gp, v0, -2 - ex.ip, ex.mp);
    }
    ext_warp_merge(ex, k);
    if (lane == 0) {
      sh.red[warp] = make_float4(ex.mq, ex.sq, ex.mp, ex.sp);
      sh.ext_red[warp] = make_float4(ex.aq, ex.ap, ex.x, 0.0f);
      sh.idx_red[warp] = make_int2(ex.iq, ex.ip);
    }
  } else {
    warp_ms_merge(mq, s_q, k);
    warp_ms_merge(mp, s_p, k);
    if (lane == 0) sh.red[warp] = make_float4(mq, s_q, mp, s_p);
  }
  __syncthreads();
  // ---- exchange 1: thread 0 merges the warp partials into the slice partial
  // and pushes it into every CTA of the cluster; one barrier; then every read
  // is local, and thread 0 decides
  float4 part = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  float4 part_ext = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  int2 part_idx = make_int2(-1, -1);
  if (tid == 0) {
    if constexpr (kExt) {
      ExtState e = ext_load(sh.red[0], sh.ext_red[0], sh.idx_red[0]);
      for (int w = 1; w < kNW; ++w) ext_merge(e, ext_load(sh.red[w], sh.ext_red[w], sh.idx_red[w]), k);
      part = make_float4(e.mq, e.sq, e.mp, e.sp);
      part_ext = make_float4(e.aq, e.ap, e.x, 0.0f);
      part_idx = make_int2(e.iq, e.ip);
    } else {
      part = merge_partials(sh.red, kNW, k);
    }
    if (tmo || sh.timeout) {  // (a copy of an earlier unit that never landed may land now)
      part.y = NAN;
      part.w = NAN;
      flag_timeout(sh, P);
    }
  }
  cluster_wait();  // every CTA of the cluster has started
  if (tid == 0) {
    const float2 xv = make_float2(sh.xq, sh.xp);
    for (int r = 0; r < C; ++r) {
      st_peer(peer_addr(&sh.all_ms[rank], r), part);
      st_peer(peer_addr(&sh.all_x[rank], r), xv);
      if constexpr (kExt) {
        st_peer(peer_addr(&sh.all_ext[rank], r), part_ext);
        st_peer(peer_addr(&sh.all_idx[rank], r), part_idx);
      }
    }
  }
  cluster_arrive();
  cluster_wait();

  if (tid == 0) {  // thread 0 also holds the prefetched scalars
    // the row's M and S over the cluster (and, for kFamExt, its moments and argmaxes)
    ExtState g = ext_empty();
    float4 v;
    if constexpr (kExt) {
      g = ext_load(sh.all_ms[0], sh.all_ext[0], sh.all_idx[0]);
      for (int r = 1; r < C; ++r)
        ext_merge(g, ext_load(sh.all_ms[r], sh.all_ext[r], sh.all_idx[r]), k);
      v = make_float4(g.mq, g.sq, g.mp, g.sp);
    } else {
      v = merge_partials(sh.all_ms, C, k);
    }
    const float a = v.x, as = v.y, c = v.z, cs = v.w;
    const float2 xv = sh.all_x[(x >= 0 && x < P.V) ? x / P.L : 0];
    const float yqx = xv.x, ypx = xv.y;
    // S = sum_v 2^{y_v k - R} with R = fl(M k); the max logit's own term is
    // 2^{fma(M, k, -R)}, so max_v q(v) = 2^{fma(M, k, -R)} / S.
    const float Rq = refk(a, k), Rp = refk(c, k);
    sh.Mq = a; sh.Sq = as; sh.Mp = c; sh.Sp = cs;
    sh.Rq = Rq;
    sh.Rp = Rp;
    sh.maxq = ex2(fmaf(a, k, -Rq)) / as;
    sh.maxp = ex2(fmaf(c, k, -Rp)) / cs;
    int err = 0;
    const bool okq = !pair || (isfinite(a) && isfinite(as) && as > 0.0f);
    const bool okp = isfinite(c) && isfinite(cs) && cs > 0.0f;
    if (!(okq && okp)) err |= SC_DEV_BAD_LOGIT;
    if (verify) {
      if (!(uj >= 0.0f && uj < 1.0f)) err |= SC_DEV_BAD_UNIFORM;
      if (pair && (x < 0 || x >= P.V)) err |= SC_DEV_BAD_TOKEN;
    }
    if (err && P.status && rank == 0) atomicOr(P.status, err);
    sh.err = err;
    sh.delta = 0;
    sh.need_p2 = 0;
    sh.band = 0;
    sh.tok = 0;
    sh.on_q = 0;
    sh.thr = -INFINITY;
    sh.eta = 0.0f;
    sh.accept = 0;
    sh.self_res = 0;
    sh.tv = -1.0f;
    sh.qx = 0.0f;
    sh.pix = 0.0f;
    sh.c = pair && !err ? log2f(as / cs) : 0.0f;
    sh.dl = sh.maxq;
    sh.dr = sh.maxp;
    float xent = 0.0f;  // (kFamExt) BiLD*'s discrepancy D(q, p) = -sum_v q log p, in nats
    if constexpr (kExt) {
      // sum q ln q = ln 2 (A_q / S_q - log2 S_q), sum q ln p = ln 2 (X / S_q - log2 S_p)
      constexpr float kLn2 = 0.69314718f;
      sh.iq = g.iq;
      sh.ip = g.ip;
      sh.nhq = kLn2 * (g.aq / as - log2f(as));
      sh.nhp = kLn2 * (g.ap / cs - log2f(cs));
      xent = kLn2 * (log2f(cs) - g.x / as);
      sh.klqp = sh.nhq + xent;
      if (P.greedy && pair && P.rule == SC_RULE_BILD && g.iq >= 0 && g.iq < P.V) {
        // greedy decoding: the BiLD baseline's D = -log p(argmax q), from the target
        // logit at q's argmax (one load; every CTA of the cluster reads the same value)
        const E *prow = static_cast<const E *>(P.target) + (static_cast<size_t>(b) * G1 + j) * P.V;
        const float y = Elt<E>::at(prow, static_cast<size_t>(g.iq));
        const float2 lp = log2_prob(y, c, Rp, cs, k, P.kl);
        xent = y > -INFINITY ? -kLn2 * (lp.x + lp.y) : INFINITY;
      }
      if (P.greedy && pair) sh.tv = g.iq != g.ip ? 1.0f : 0.0f;  // D_TV of the one-hot q~, p~
    }
    if (!err && pair) {
      if (!verify) {
        sh.need_p2 = 1;  // sc_row_stats: TV of every pair
      } else {
        // deferral rule (Table 1)
        const float maxq = sh.maxq, maxp = sh.maxp, al = P.alpha;
        bool pending = false;
        switch (P.rule) {
          case SC_RULE_CHOW: sh.delta = maxq < 1.0f - al; break;  // Eq. 2
          case SC_RULE_DIFF: sh.delta = maxq < maxp - al; break;  // Eq. 5
          case SC_RULE_OPT:                                       // Eq. 10
            if (kExt) {  // greedy decoding: the one-hot D_TV is known
              sh.delta = maxq < maxp - al * sh.tv;
              break;
            }
            // alpha * TV lies in [0, alpha]: TV decides only inside that band
            if (!(maxq < maxp)) sh.delta = 0;
            else if (maxq < maxp - al) sh.delta = 1;
            else pending = true;
            break;
          case SC_RULE_ALWAYS_DEFER: sh.delta = 1; break;
          case SC_RULE_LOSSY: sh.delta = 1; break;  // Table 3: the target min/max of q, p
          // Table 3 and the log-loss rules
          case SC_RULE_BILD: sh.delta = xent > al; break;              // D(q, p) > alpha
          case SC_RULE_CHOW_LOG: sh.delta = -sh.nhq > al; break;       // H(q) > alpha
          case SC_RULE_DIFF_LOG: sh.delta = sh.nhq < sh.nhp - al; break;
          case SC_RULE_OPT_LOG:  // sum q log q < sum p log p - alpha D_TV
            sh.dl = sh.nhq;
            sh.dr = sh.nhp;
            if (P.greedy) sh.delta = sh.nhq < sh.nhp - al * sh.tv;
            else if (!(sh.nhq < sh.nhp)) sh.delta = 0;
            else if (sh.nhq < sh.nhp - al) sh.delta = 1;
            else pending = true;
            break;
          case SC_RULE_TOKEN_V1:
          case SC_RULE_TOKEN_V2:
          case SC_RULE_TOKEN_V3: {
            // token-specific target (Section 4.4): r(v) compares a_v or b_v with a
            // threshold; eta = sum_v r(v) q(v) needs a pass over the row
            const float bM = fmaf(c, k, -Rp);  // b of the mode of p: max p = 2^bM / S_p
            sh.tok = 1;
            pending = true;
            if (P.rule == SC_RULE_TOKEN_V3) {  // p(v) < max p (1 - alpha)  <=>  b_v < bM + log2(1 - alpha)
              sh.thr = al < 1.0f ? bM + log2f(1.0f - al) : -INFINITY;
            } else {                           // p(v) or q(v) < max p - alpha
              const float m = maxp - al;
              sh.on_q = P.rule == SC_RULE_TOKEN_V1;
              sh.thr = m > 0.0f ? log2f(m * (sh.on_q ? as : cs)) : -INFINITY;
            }
            if (sh.thr == -INFINITY) pending = false;  // r = 0 everywhere: eta = 0, pi = q
            break;
          }
          default: sh.delta = 0; break;
        }
        if (pending) sh.need_p2 = 1;
        if (pending && !sh.tok) sh.band = 1;
        if (!pending) accept_test<kFam>(sh, P, x, yqx, ypx, uj, k);
      }
    }
    // keep the draft-token logits for a decision after the TV pass
    sh.xq = yqx;
    sh.xp = ypx;
  }
  __syncthreads();
  if (bonus_tot && warp == 0) {
    // p_gamma's chunk prefixes over this slice from pass 1's per-(chunk, warp)
    // totals, re-referenced to R_p: what a sampling pass over the row would store
    // (lane c: chunk c; a warp scan in chunk order)
    float t = 0.0f;
    if (lane < R.nch)
      for (int w = 0; w < kNW; ++w)
        t = fmaf(sh.seg[lane * kNW + w], ex2(refk(sh.seg[kBonusRef + lane * kNW + w], k) - sh.Rp), t);
    const float incl = warp_incl_scan(t, lane);
    float excl = __shfl_up_sync(0xFFFFFFFFu, incl, 1);
    if (lane == 0) excl = 0.0f;
    float *cp = P.bonus_pre + (static_cast<size_t>(b) * kMaxCluster + rank) * (kMaxChunks + 1);
    if (lane < R.nch && SC_CHECK(b < P.B && rank < kMaxCluster && lane < kMaxChunks)) cp[lane] = excl;
    if (lane == max(R.nch - 1, 0) && SC_CHECK(b < P.B && rank < kMaxCluster && R.nch <= kMaxChunks))
      cp[R.nch] = sh.err || tmo ? NAN : (R.nch > 0 ? incl : 0.0f);
  }

  // ---- token rules: eta without a pass when the pass-1 screen settles it.  A
  // thread whose second-largest screened logit is deferred holds at most one
  // undeferred token, its largest; if that holds in every thread of the
  // cluster, eta = (S_q - sum of 2^a over those tokens) / S_q.
  if (kTok && sh.tok && sh.need_p2) {
    const float Rs = sh.on_q ? sh.Rq : sh.Rp;  // r(v) tests a_v or b_v, formed as vec_weights forms them
    bool ok = !(fmaf(top.y2, k, -Rs) >= sh.thr);
    float h = 0.0f;
    if (fmaf(top.y1, k, -Rs) >= sh.thr) {
      float z1 = top.z1;
      bool have = top.known;
      if (!have && SC_CHECK(top.c1 >= 0 && top.c1 < R.nch && R.chunk_len(top.c1) == kCH)) {
        // y1 came from a full chunk swept in packed form: this thread's first
        // logit equal to y1 in that chunk (the sweep's order) and the draft
        // logit there, read element by element from the slice in global memory
        const size_t c0 = static_cast<size_t>(top.c1) * kCH;
        const E *ts = scr_q ? R.gq : R.gp;
        for (int r = 0; r < kRounds && !have; ++r) {
          const int e = 8 * (r * kNT + tid);
          for (int i = 0; i < 8; ++i)
            if (Elt<E>::at(ts, c0 + e + i) == top.y1) {
              z1 = Elt<E>::at(R.gq, c0 + e + i);
              have = true;
              break;
            }
        }
      }
      ok = ok && have;  // (not found cannot happen; it would take the eta pass)
      if (have) h = ex2(fmaf(z1, k, -sh.Rq));
    }
    const bool wok = __all_sync(0xFFFFFFFFu, ok);
    const float hs = warp_sum(h);
    if (lane == 0) sh.red[warp] = make_float4(hs, wok ? 1.0f : 0.0f, 0.0f, 0.0f);
    __syncthreads();
    if (tid == 0) {
      float acc = 0.0f, okc = 1.0f;
      for (int w = 0; w < kNW; ++w) {
        acc = __fadd_rn(acc, sh.red[w].x);
        okc = fminf(okc, sh.red[w].y);
      }
      for (int r = 0; r < C; ++r) st_peer(peer_addr(&sh.all_scr[rank], r), make_float2(acc, okc));
    }
    cluster_arrive();
    cluster_wait();
    if (tid == 0) {
      float H = 0.0f, okc = 1.0f;  // in rank order
      for (int r = 0; r < C; ++r) {
        H = __fadd_rn(H, sh.all_scr[r].x);
        okc = fminf(okc, sh.all_scr[r].y);
      }
      if (okc > 0.0f) {
        sh.need_p2 = 0;
        sh.eta = fmaxf(0.0f, sh.Sq - H) / sh.Sq;  // eta = sum_v r(v) q(v) = 1 - sum over undeferred
        accept_test<kFam>(sh, P, x, sh.xq, sh.xp, uj, k);
      }
    }
    __syncthreads();
  }

  // ---- OPT band: bounds on D_TV from the pass-1 partials.  Each thread's logits
  // 0, 1, 2 and 3 (mod 4) form four sets t (the lanes of its two packed sums),
  // with masses P_t, Q_t; the sets partition the vocabulary, so
  // sum_t max(0, P_t - Q_t) <= D_TV.  From above, OPT takes Cauchy-Schwarz on
  // sum |sqrt p - sqrt q| (sqrt p + sqrt q) within each set,
  //   sum_{v in t} max(0, p - q) <= (((P_t + Q_t)^2 - 4 BC_t^2)^(1/2) + P_t - Q_t) / 2,
  // BC_t = sum_{v in t} sqrt(q p) from pass 1, summed over t (never above the
  // Hellinger bound (1 - BC^2)^(1/2)); OPTLog takes Pinsker's (KL(q || p) / 2)^(1/2)
  // from its entropy and cross entropy.  When alpha times the lower bound already
  // reaches dr - dl (max p - max q for OPT, Eq. 10; the negative-entropy gap for
  // OPTLog), delta = 0 for the exact D_TV too; when alpha times the upper bound
  // stays below it, delta = 1; either way the TV pass is skipped.  The bounds
  // carry ~1e-6 of f32 rounding over their 512 C terms, BC_t is deflated and KL
  // inflated well past their f32 errors: only a clear 1e-4 margin settles the row.
  if (sh.band) {
    const float dq = refk(mine.x, k) - sh.Rq, dp = refk(mine.z, k) - sh.Rp;
    const float fq = ex2(dq) / sh.Sq, fp = ex2(dp) / sh.Sp;
    const float qs[4] = {mq4.x * fq, mq4.y * fq, mq4.z * fq, mq4.w * fq};
    const float ps[4] = {mp4.x * fp, mp4.y * fp, mp4.z * fp, mp4.w * fp};
    const float bs[4] = {bc.x, bc.y, bc.z, bc.w};
    const float fb = opt_bc ? ex2(0.5f * (dq + dp)) / sqrtf(sh.Sq * sh.Sp) * (1.0f - 2e-4f) : 0.0f;
    float lbt = 0.0f, ubt = 0.0f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      lbt += fmaxf(0.0f, ps[i] - qs[i]);
      const float m = ps[i] + qs[i], bt = bs[i] * fb;
      ubt += 0.5f * (sqrtf(fmaxf(0.0f, fmaf(m, m, -4.0f * bt * bt))) + (ps[i] - qs[i]));
    }
    const float lb = warp_sum(lbt);
    const float bcw = warp_sum(ubt);
    if (lane == 0) sh.red[warp] = make_float4(lb, bcw, 0.0f, 0.0f);
    __syncthreads();
    if (tid == 0) {
      float acc = 0.0f, accb = 0.0f;
      for (int w = 0; w < kNW; ++w) {
        acc = __fadd_rn(acc, sh.red[w].x);
        accb = __fadd_rn(accb, sh.red[w].y);
      }
      for (int r = 0; r < C; ++r) st_peer(peer_addr(&sh.all_lb[rank], r), make_float2(acc, accb));
    }
    cluster_arrive();
    cluster_wait();
    if (tid == 0) {
      float LB = 0.0f, UBs = 0.0f;  // in rank order
      for (int r = 0; r < C; ++r) {
        LB = __fadd_rn(LB, sh.all_lb[r].x);
        UBs = __fadd_rn(UBs, sh.all_lb[r].y);
      }
      const float gap = sh.dr - sh.dl;
      float ub = INFINITY;
      if (opt_bc) {
        ub = UBs;
      } else if (kExt && SC_OPT_UB) {
        const float kv = sh.klqp;  // NaN or +inf (masked logits) settle nothing
        if (kv == kv)
          ub = sqrtf(0.5f * fmaf(fmaxf(kv, 0.0f), 1.001f, 1e-5f * (1.0f + fabsf(sh.nhq) + fabsf(sh.nhq - kv))));
      }
      if (P.alpha * LB - gap >= 1e-4f) {
        sh.need_p2 = 0;
        sh.delta = 0;
        accept_test<kFam>(sh, P, x, sh.xq, sh.xp, uj, k);
      } else if (ub < INFINITY && gap - P.alpha * ub >= 1e-4f) {
        sh.need_p2 = 0;
        sh.delta = 1;
        accept_test<kFam>(sh, P, x, sh.xq, sh.xp, uj, k);
      }
    }
    __syncthreads();
  }

  // ---- TV pass (sc_row_stats, or the OPT band): residual weights of this row;
  // for a token rule the same pass sums r(v) q(v) instead (eta)
  if (sh.need_p2) {
    const RowScalars rs = {sh.Rq, sh.Rp, k, sh.c, sh.tok ? kEta : kResidual, sh.on_q, sh.thr, 0.0f};
    tmo = slice_weights<kTok>(R, sh, ph, rs, kNewestFirstResident, lane, warp);
    tmo = __syncthreads_or(tmo);
    // exchange 2: push the slice total, one barrier, local reads
    if (warp == 0) {
      float acc = seg_prefix(sh, R.nch * kRounds * kNW, lane);
      if (lane == 0) {
        if (tmo) {
          acc = NAN;
          flag_timeout(sh, P);
        }
        for (int r = 0; r < C; ++r) st_peer(peer_addr(&sh.all_r[rank], r), acc);
      }
    }
    cluster_arrive();
    cluster_wait();
    if (tid == 0) {
      float Rtot = 0.0f;  // in rank order
      for (int r = 0; r < C; ++r) Rtot = __fadd_rn(Rtot, sh.all_r[r]);
      if (!isfinite(Rtot)) {
        sh.err |= SC_DEV_TIMEOUT;
      } else if (sh.tok) {
        sh.eta = Rtot / sh.Sq;  // eta = sum_v r(v) q(v)
        accept_test<kFam>(sh, P, x, sh.xq, sh.xp, uj, k);
      } else {
        sh.tv = fminf(1.0f, fmaxf(0.0f, Rtot / sh.Sq));  // Lemma 3: R = S_q D_TV(p, q)
        if (verify) {
          sh.delta = sh.dl < sh.dr - P.alpha * sh.tv;  // Eq. 10 (or OPTLog)
          accept_test<kFam>(sh, P, x, sh.xq, sh.xp, uj, k);
        }
      }
    }
    __syncthreads();
  }

  // ---- a rejected pair that is certainly row j* of its sequence stores its own
  // residual's chunk prefixes now, while its slice is in the ring and in L2, so
  // that no sampling pass is left for the end of the sequence's chain: certain
  // when every earlier position of this slice rank has reported without a
  // rejection.  A rejected pair whose rank shows an earlier rejection is not j*;
  // one whose earlier positions have not all reported leaves the pass to the
  // owner that settles j* (so no row but j* is ever sampled).  An OPT band row's
  // TV pass has summed exactly these weights already: it always stores them.
  // Drafts longer than 32 positions (an arrival count, no bits) leave it to the owner.
  if (P.spec_res && verify && pair && !sh.accept && !sh.err && !(kExt && P.greedy)) {
    if (tid == 0) {
      int self = sh.need_p2 && !sh.tok;
      if (!self && G1 <= 32) {
        const unsigned long long t = __ldcg(P.rank_tickets + static_cast<size_t>(b) * kMaxCluster + rank);
        const unsigned long long earlier = (1ull << j) - 1ull;
        self = ((t >> 32) & earlier) == 0ull && (t & earlier) == earlier;
      }
      sh.self_res = self;
    }
    __syncthreads();
  }
  if (sh.self_res) {
    if (!(sh.need_p2 && !sh.tok)) {
      const bool lossy = kFam == kFamCascade && P.rule == SC_RULE_LOSSY;
      const RowScalars rs = {sh.Rq, sh.Rp, k, lossy ? sh.c + P.lossy_c : sh.c,
                             sh.tok ? kTokenRes : kResidual, sh.on_q, sh.thr, sh.eta};
      tmo = slice_weights<kTok>(R, sh, ph, rs, sh.need_p2 ? kNewestFirst : kNewestFirstResident, lane, warp);
      tmo = __syncthreads_or(tmo);
      if (warp == 0) {
        seg_prefix(sh, R.nch * kRounds * kNW, lane);
        if (lane == 0 && tmo) flag_timeout(sh, P);
      }
      __syncthreads();
    }
    if (tid == 0) {
      float *cp = P.row_pre + ((static_cast<size_t>(b) * G1 + j) * kMaxCluster + rank) * (kMaxChunks + 1);
      if (SC_CHECK(b < P.B && j < G1 && rank < kMaxCluster && R.nch <= kMaxChunks)) {
        for (int c = 0; c < R.nch; ++c) cp[c] = sh.seg[c * kRounds * kNW];
        cp[R.nch] = sh.timeout ? NAN : sh.seg[R.nch * kRounds * kNW];
      }
    }
    __syncthreads();
  }

  if (!verify) {
    if (tid == 0 && rank == 0) {
      const size_t r = static_cast<size_t>(b) * P.gamma + j;
      const bool bad = sh.err != 0;
      P.max_q[r] = bad ? NAN : sh.maxq;
      P.max_p[r] = bad ? NAN : sh.maxp;
      P.tv[r] = bad ? NAN : sh.tv;
    }
  } else {
    // ---- record the decision and report it on this slice rank's ticket; the
    // CTA whose report settles j* samples this rank's slice of row j*
    float4 *rec = P.records + (static_cast<size_t>(b) * kMaxCluster + rank) * G1;
    float4 *rec2 = P.records2 + (static_cast<size_t>(b) * kMaxCluster + rank) * G1;
    if (tid == 0) {
      // flags: 1 accepted, 2 invalid, 4 this rank's residual prefixes are in row_pre
      const int flags = (sh.accept ? 1 : 0) | (sh.err ? 2 : 0) | (sh.self_res ? 4 : 0);
      float4 r1 = make_float4(sh.Rq, sh.Rp, sh.c, __int_as_float(flags));
      if (kFam == kFamCascade && P.rule == SC_RULE_LOSSY)
        r1.z = sh.c + P.lossy_c;  // the residual max(0, p / beta - q) (Lemma 2)
      if (kExt && P.greedy) r1.x = __int_as_float(sh.ip);  // greedy: the token emitted at row j*
      if (SC_CHECK(b < P.B && rank < kMaxCluster && j < G1)) rec[j] = r1;
      if (kTok)  // (only token rules read the second record)
        if (SC_CHECK(b < P.B && rank < kMaxCluster && j < G1))
          rec2[j] = make_float4(sh.eta, sh.thr, __int_as_float(sh.tok), __int_as_float(sh.on_q));
      if (rank == 0 && P.row_info) {
        float *ri = P.row_info + (static_cast<size_t>(b) * G1 + j) * SC_ROW_FIELDS;
        ri[SC_ROW_MAXQ] = pair && !sh.err ? sh.maxq : NAN;
        ri[SC_ROW_MAXP] = !sh.err ? sh.maxp : NAN;
        ri[SC_ROW_TV] = sh.tv;
        ri[SC_ROW_DELTA] = static_cast<float>(sh.delta);
        ri[SC_ROW_ACCEPT] = static_cast<float>(sh.accept);
        ri[SC_ROW_QX] = sh.qx;
        ri[SC_ROW_PIX] = sh.pix;
        ri[SC_ROW_CAND] = -1.0f;  // the sequence's finisher fills in row j*
      }
      unsigned long long *tk = P.rank_tickets + static_cast<size_t>(b) * kMaxCluster + rank;
      int owner, all_in, js = P.gamma;
      sh.scan_records = 0;
      if (G1 <= 32) {
        // arrival bit j, and rejection bit 32 + j (a_j = 0; the bonus row never rejects)
        const unsigned long long mine = (1ull << j) | (pair && !sh.accept ? 1ull << (32 + j) : 0ull);
        const unsigned long long old = atom_or_acq_rel(tk, mine);
        int js_old;
        owner = jstar_settled(old | mine, G1, js) && !jstar_settled(old, G1, js_old);
        all_in = static_cast<uint32_t>(old | mine) == (G1 == 32 ? 0xFFFFFFFFu : (1u << G1) - 1u);
      } else {
        // long drafts: the last arrival settles j* and reads it from the records
        owner = all_in = atom_add_acq_rel(tk, 1ull) == static_cast<unsigned long long>(P.gamma);
        sh.scan_records = owner;
      }
      if (all_in) *tk = 0ull;  // every unit of the sequence has reported on this rank
      sh.owner = owner;
      sh.jstar = js;
      // the finisher needs every sample pass and all of rank 0's records
      sh.seq_last = all_in && rank == 0 &&
                    atom_add_acq_rel(P.seq_tickets + b, 1u) == static_cast<uint32_t>(C);
    }
    __syncthreads();
    if (sh.scan_records && warp == 0) {
      int js = P.gamma;
      for (int base = 0; base < P.gamma; base += 32) {
        const int jj = base + lane;
        const int f = jj < P.gamma ? __float_as_int(__ldcg(&rec[jj].w)) : 1;
        const unsigned m = __ballot_sync(0xFFFFFFFFu, !(f & 1));
        if (m) {
          js = base + __ffs(m) - 1;
          break;
        }
      }
      if (lane == 0) sh.jstar = js;
    }
    if (sh.owner && tid == 0) {  // row j*'s records (they are in)
      sh.rj = __ldcg(&rec[sh.jstar]);
      sh.rj2 = kTok ? __ldcg(&rec2[sh.jstar]) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    }
    __syncthreads();

    if (sh.owner && ((kExt && P.greedy) || sh.jstar == P.gamma || (__float_as_int(sh.rj.w) & 4))) {
      // nothing to sample: greedy decoding emits row j*'s argmax p (in the
      // records), the bonus row's chunk prefixes came from its pass 1, or row
      // j* stored this rank's prefixes itself (flag 4 of its record)
      if (tid == 0) sh.seq_last = atom_add_acq_rel(P.seq_tickets + b, 1u) == static_cast<uint32_t>(C);
      __syncthreads();
    } else if (sh.owner) {
      // ---- sample pass: weights of this rank's slice of row j* -- the residual
      // max(0, p - q) of a rejected pair (Algorithm 4), or p of the bonus row
      const int js = sh.jstar;
      const RowScalars rs = sample_scalars(sh.rj, sh.rj2, k);
      const Ring<E> Rj = make_ring<E>(P, smem_raw, b, js, rank);
      // this unit's own row, untouched since pass 1, still has its last chunks in the ring
      const bool resident = js == j && !sh.need_p2;
      tmo = slice_weights<kTok>(Rj, sh, ph, rs, resident ? kNewestFirstResident : kNewestFirst, lane, warp);
      tmo = __syncthreads_or(tmo);
      if (warp == 0) seg_prefix(sh, Rj.nch * kRounds * kNW, lane);
      __syncthreads();
      if (tid == 0) {
        float tot_r = sh.seg[Rj.nch * kRounds * kNW];
        if (tmo) {
          tot_r = NAN;
          flag_timeout(sh, P);
        }
        float *cp = P.chunk_pre + (static_cast<size_t>(b) * kMaxCluster + rank) * (kMaxChunks + 1);
        if (SC_CHECK(b < P.B && rank < kMaxCluster && Rj.nch <= kMaxChunks)) {
          for (int c = 0; c < Rj.nch; ++c) cp[c] = sh.seg[c * kRounds * kNW];
          cp[Rj.nch] = tot_r;  // the slice total
        }
        sh.seq_last = atom_add_acq_rel(P.seq_tickets + b, 1u) == static_cast<uint32_t>(C);
      }
      __syncthreads();
    }

    if (sh.seq_last) {
      // ---- the draw (the ring is idle: stage 0 holds the chunk prefixes of
      // every slice, the last stage the chunk searched)
      constexpr int kCP = kMaxChunks + 1;
      float *cpall = reinterpret_cast<float *>(smem_raw);  // [C][kCP]
      if (tid == 0) P.seq_tickets[b] = 0u;  // every report of the sequence is in
      // warp 0: j* and the error flags from rank 0's records
      if (warp == 0) {
        const float4 *rec0 = P.records + static_cast<size_t>(b) * kMaxCluster * G1;
        int js = P.gamma, bad = 0;
        float4 rj = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        for (int base = 0; base <= P.gamma; base += 32) {
          const int jj = base + lane;
          const float4 rv = jj <= P.gamma ? __ldcg(&rec0[jj]) : make_float4(0.0f, 0.0f, 0.0f, __int_as_float(1));
          const int f = __float_as_int(rv.w);
          bad |= __any_sync(0xFFFFFFFFu, f & 2);
          const unsigned m = __ballot_sync(0xFFFFFFFFu, jj < P.gamma && !(f & 1));
          const int hit = js == P.gamma ? (m ? base + __ffs(m) - 1 : (P.gamma - base < 32 ? P.gamma : -1)) : -1;
          if (hit >= 0) {
            js = hit;
            const int src = hit - base;
            rj = make_float4(__shfl_sync(0xFFFFFFFFu, rv.x, src), __shfl_sync(0xFFFFFFFFu, rv.y, src),
                             __shfl_sync(0xFFFFFFFFu, rv.z, src), __shfl_sync(0xFFFFFFFFu, rv.w, src));
          }
        }
        if (lane == 0) {
          sh.jstar = js;
          sh.bad = bad;
          sh.rj = rj;
          sh.rj2 = kTok ? __ldcg(P.records2 + static_cast<size_t>(b) * kMaxCluster * G1 + js)
                                              : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        }
      }
      __syncthreads();
      const int js = sh.jstar;
      // one round of loads: every slice's chunk prefixes of row j* (ending in its
      // total), from the bonus row's pass 1, from row j* itself (flag 4 of that
      // rank's record) or from that rank's owner
      const float *bonus = P.bonus_pre + static_cast<size_t>(b) * kMaxCluster * kCP;
      const float *self = P.row_pre + (static_cast<size_t>(b) * G1 + js) * kMaxCluster * kCP;
      const float *owned = P.chunk_pre + static_cast<size_t>(b) * kMaxCluster * kCP;
      for (int i = tid; i < C * kCP && !(kExt && P.greedy); i += kNT) {
        const int r = i / kCP, c = i % kCP;
        const int len = max(0, min(P.L, P.V - r * P.L));
        if (c <= (len + kCH - 1) / kCH && SC_CHECK(b < P.B && js <= P.gamma && C <= kMaxCluster)) {
          const float *src = bonus;
          if (js < P.gamma) {
            const int f = __float_as_int(__ldcg(&P.records[(static_cast<size_t>(b) * kMaxCluster + r) * G1 + js].w));
            src = (f & 4) ? self : owned;
          }
          cpall[i] = __ldcg(src + i);
        }
      }
      __syncthreads();
      if (kExt && P.greedy) {
        // greedy decoding: the argmax p of row j*, from rank 0's record
        if (tid == 0 && SC_CHECK(b < P.B && js >= 0 && js <= P.gamma)) {
          const bool ok = !sh.bad;
          const int tok = __float_as_int(sh.rj.x);
          P.num_accepted[b] = ok ? js : 0;
          P.next_token[b] = ok ? tok : -1;
          if (ok && P.row_info)
            P.row_info[(static_cast<size_t>(b) * G1 + js) * SC_ROW_FIELDS + SC_ROW_CAND] = static_cast<float>(tok);
        }
      } else {
        const RowScalars rs = sample_scalars(sh.rj, sh.rj2, k);
        // ---- inverse CDF over the slices in rank order, u = u[b][gamma], then
        // over the chunks of the crossing slice
        if (warp == 0) {
          auto nch_of = [&](int r) {
            const int len = max(0, min(P.L, P.V - r * P.L));
            return (len + kCH - 1) / kCH;
          };
          const float tot = lane < C ? cpall[lane * kCP + nch_of(lane)] : 0.0f;
          const float pre = warp_incl_scan(tot, lane);  // through rank `lane`
          const float Rtot = __shfl_sync(0xFFFFFFFFu, pre, C - 1);
          float before = __shfl_up_sync(0xFFFFFFFFu, pre, 1);
          if (lane == 0) before = 0.0f;
          const float u = __shfl_sync(0xFFFFFFFFu, ug, 0);
          const bool ok = !sh.bad && isfinite(Rtot);
          int cr = -1, cc = -1, clast = -1;
          float2 tl = make_float2(-1.0f, 0.0f);  // (negative: u R fell past the last boundary)
          if (ok && Rtot > 0.0f) {
            const float th = __fmul_rn(u, Rtot);
            const float2 t = make_float2(th, fmaf(u, Rtot, -th));  // u R_tot, exactly
            const bool cross = lane < C && tot > 0.0f && df_ge(t, before) && df_lt(t, pre);
            const unsigned cm = __ballot_sync(0xFFFFFFFFu, cross);
            const unsigned pm = __ballot_sync(0xFFFFFFFFu, lane < C && tot > 0.0f);
            cr = cm ? __ffs(cm) - 1 : 31 - __clz(pm);
            const float bcr = __shfl_sync(0xFFFFFFFFu, before, cr);
            if (cm) tl = df_sub(t, bcr);
            // the chunk of slice cr holding tl (or, past a rounding gap, its last chunk with weight)
            const float *cp = cpall + cr * kCP;
            const int nch = nch_of(cr);
            for (int base = 0; base < nch; base += 32) {
              const int c = base + lane;
              const float lo = c < nch ? cp[c] : 0.0f, hi = c < nch ? cp[c + 1] : 0.0f;
              const bool pos = c < nch && hi > lo;
              const unsigned mi = __ballot_sync(0xFFFFFFFFu, pos && df_ge(tl, lo) && df_lt(tl, hi));
              const unsigned mp = __ballot_sync(0xFFFFFFFFu, pos);
              if (cc < 0 && mi) cc = base + __ffs(mi) - 1;
              if (mp) clast = base + 31 - __clz(mp);
            }
          }
          if (lane == 0) {
            sh.sample_ok = ok;
            sh.cross_rank = cr;
            sh.t_slice = tl;
            sh.token = -1;
            sh.cross_chunk = cc >= 0 ? cc : clast;
            sh.have_t = cc >= 0;
            sh.chunk_lo = sh.cross_chunk >= 0 ? cpall[cr * kCP + sh.cross_chunk] : 0.0f;
          }
        }
        __syncthreads();
        const int cr = sh.cross_rank, cc = sh.cross_chunk;
        if (cr >= 0 && cc >= 0) {
          // the chunk's weights again, by the code the sample pass ran (the same values)
          const Ring<E> Rc = make_ring<E>(P, smem_raw, b, js, cr);
          const int sl = kStages - 1, n = Rc.chunk_len(cc);
          if (Rc.bulk) {
            if (tid == 0) Rc.issue(sh, cc, sl);
            tmo = wait_stage(sh, sl, ph);
          } else {
            tmo = 0;
            Rc.load_sync(cc, sl);
          }
          tmo = __syncthreads_or(tmo);
          if (Rc.pair) {
            if (n == kCH) weights_chunk<E, true, true, kTok>(Rc.q(sl), Rc.p(sl), n, 0, rs, sh, lane, warp);
            else weights_chunk<E, true, false, kTok>(Rc.q(sl), Rc.p(sl), n, 0, rs, sh, lane, warp);
          } else {
            if (n == kCH) weights_chunk<E, false, true, kTok>(Rc.q(sl), Rc.p(sl), n, 0, rs, sh, lane, warp);
            else weights_chunk<E, false, false, kTok>(Rc.q(sl), Rc.p(sl), n, 0, rs, sh, lane, warp);
          }
          if (tmo && tid == 0) {
            flag_timeout(sh, P);
            sh.sample_ok = 0;
          }
          __syncthreads();
          constexpr int kSegC = kRounds * kNW;  // segments per chunk
          if (tid == 0) {
            // exclusive prefixes continue from the chunk's stored start, as in the sample pass
            float acc = sh.chunk_lo;
            for (int i = 0; i < kSegC; ++i) {
              const float t = sh.seg[i];
              sh.seg[i] = acc;
              acc = __fadd_rn(acc, t);
            }
            sh.seg[kSegC] = acc;
            const float2 tl = sh.t_slice;
            int sgi = -1;
            if (sh.have_t)
              for (int i = 0; i < kSegC; ++i)
                if (df_ge(tl, sh.seg[i]) && df_lt(tl, sh.seg[i + 1]) && sh.seg[i + 1] > sh.seg[i]) {
                  sgi = i;
                  break;
                }
            sh.cross_seg = sgi;
            sh.t_seg = sgi >= 0 ? df_floor(df_sub(tl, sh.seg[sgi])) : 0.0f;
          }
          __syncthreads();
          int sgi = sh.cross_seg;
          if (sgi < 0) {
            // no t inside the chunk: its last segment with weight
            for (int i = kSegC - 1; i >= 0; --i)
              if (sh.seg[i + 1] > sh.seg[i]) { sgi = i; break; }
          }
          if (sgi >= 0 && warp == sgi % kNW) {
            const int tok = search_segment<kTok>(Rc.q(sl), Rc.p(sl), n, Rc.pair, rs, cr * P.L + cc * kCH,
                                           sgi / kNW, sh.cross_seg >= 0, sh.t_seg, lane, warp);
            if (lane == 0) sh.token = tok;
          }
          __syncthreads();
        }
        if (tid == 0 && SC_CHECK(b < P.B && js >= 0 && js <= P.gamma)) {
          const bool ok = sh.sample_ok != 0;
          P.num_accepted[b] = ok ? js : 0;
          P.next_token[b] = ok ? sh.token : -1;
          if (ok && P.row_info)
            P.row_info[(static_cast<size_t>(b) * G1 + js) * SC_ROW_FIELDS + SC_ROW_CAND] =
                static_cast<float>(sh.token);
        }
      }
    }
  }
  if (sh.timeout && tid == 0 && P.bulk) {
    // let copies still in flight land before this CTA's shared memory is released
    for (int s = 0; s < kStages; ++s) mbar_wait(&sh.full[s], 0), mbar_wait(&sh.full[s], 1);
  }
  // (no CTA touches a peer's shared memory after its last exchange barrier)
}

// ------------------------------------------------------------------ host side

struct DeviceInfo {
  int smem_optin = 0;
  int sms = 0;
  bool configured[6] = {};  // [dtype][rule family]
};

DeviceInfo g_dev[64];
std::mutex g_mu;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace of sc_verify for B sequences of gamma drafts: slice-rank tickets,
// sequence tickets (both zero between calls), then unit records and chunk
// prefixes (written before they are read).
struct WsLayout {
  size_t rank_tickets, seq_tickets, zeroed, records, records2, chunk_pre, bonus_pre, row_pre, total;
};

constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }

constexpr WsLayout ws_layout(size_t B, size_t units) {
  WsLayout w = {};
  w.rank_tickets = 0;
  w.seq_tickets = align256(8 * kMaxCluster * B);
  w.zeroed = w.seq_tickets + align256(4 * B);
  w.records = w.zeroed;
  w.records2 = w.records + align256(16 * kMaxCluster * units);
  w.chunk_pre = w.records2 + align256(16 * kMaxCluster * units);
  w.bonus_pre = w.chunk_pre + align256(4 * kMaxCluster * (kMaxChunks + 1) * B);
  w.row_pre = w.bonus_pre + align256(4 * kMaxCluster * (kMaxChunks + 1) * B);
  w.total = w.row_pre + align256(4 * kMaxCluster * (kMaxChunks + 1) * units);
  return w;
}


template <typename E>
size_t smem_bytes() {
  return static_cast<size_t>(kStages) * 2 * kCH * sizeof(E) + sizeof(Shared);
}

// Cluster size C and slice length L (multiple of 8) for a row of V logits.
// Long slices amortise each unit's cluster exchange, decision and ticket over
// more streamed bytes and wait on fewer peers; short ones give small batches
// enough CTAs to cover the GPU.  65536 logits per CTA once that still fills
// the resident CTA slots one and a half times over, else 32768, else (small
// batches) 8192.  V = 256000, gamma = 8 (OPT / Diff, us): B = 48 121 -> 116 /
// 97 -> 89, B = 64 142 -> 131 / 119 -> 115 with 65536; below 1.5 waves it
// loses (B = 64, gamma = 4: 89 -> 97 / 82 -> 88; B = 32, gamma = 5: 69 -> 70).
int pick_layout(int V, int units, int sms, int *C_out, int *L_out) {
  const long resident = static_cast<long>(kMinBlocksPerSM) * sms;
  auto ctas = [&](long t) { return static_cast<long>(units) * ((V + t - 1) / t); };
  long target = 32768;  // logits per row per CTA
  if (2 * ctas(65536) >= 3 * resident) target = 65536;
  else if (ctas(32768) < 4L * sms) target = 8192;
  if (const char *s = getenv("SC_SLICE")) {
    const long t = atol(s);
    if (t >= 64) target = t;
  }
  int C = static_cast<int>((V + target - 1) / target);
  if (const char *s = getenv("SC_CLUSTER")) {
    const int c = atoi(s);
    if (c >= 1 && c <= kMaxCluster) C = c;
  }
  C = std::max(1, std::min(C, kMaxCluster));
  for (; C <= kMaxCluster; ++C) {
    const int L = static_cast<int>(align_up((static_cast<size_t>(V) + C - 1) / C, 8));
    if ((L + kCH - 1) / kCH > kMaxChunks) continue;
    *C_out = (V + L - 1) / L;
    *L_out = L;
    return 0;
  }
  return -1;
}

// k = log2(e) / T as an f32 value plus its f32 remainder.
void set_k(Params &P, float temperature) {
  const double kd = 1.4426950408889634 / static_cast<double>(temperature);
  P.k = static_cast<float>(kd);
  P.kl = static_cast<float>(kd - static_cast<double>(P.k));
}

// Set by each entry point: its stream is being captured into a CUDA graph.  The
// pointer checks then only reject null pointers, so that nothing but the launch
// itself happens inside the capture sequence.
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

// The rule family of a call (see Family): each family is its own kernel, so
// the SpecCascade rules run without the per-logit branches of the others.
int family_of(const Params &P) {
  if (P.greedy || P.rule >= SC_RULE_BILD) return kFamExt;
  if (P.rule >= SC_RULE_TOKEN_V1 && P.rule <= SC_RULE_TOKEN_V3) return kFamToken;
  return kFamCascade;
}

template <typename E>
int launch(Params P, cudaStream_t stream, int units) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SC_ERR_CUDA;
  DeviceInfo &di = g_dev[dev];
  const int fam = family_of(P);
  const auto kernel = fam == kFamExt     ? sc_unit_kernel<E, kFamExt>
                      : fam == kFamToken ? sc_unit_kernel<E, kFamToken>
                                         : sc_unit_kernel<E, kFamCascade>;
  const int ti = (sizeof(E) == 2 ? 3 : 0) + fam;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!di.smem_optin &&
        (cudaDeviceGetAttribute(&di.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
         cudaDeviceGetAttribute(&di.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess))
      return SC_ERR_CUDA;
    if (!di.configured[ti]) {
      if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(smem_bytes<E>())) != cudaSuccess ||
          cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
              cudaSuccess ||
          cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                               cudaSharedmemCarveoutMaxShared) != cudaSuccess)
        return SC_ERR_CUDA;
      di.configured[ti] = true;
    }
  }
  int C = 1, L = 8;
  if (pick_layout(P.V, units, di.sms, &C, &L) != 0) return SC_ERR_UNSUPPORTED;
  P.L = L;
  P.cluster = C;
  // Rejected pairs store their residual's prefixes themselves, right after their
  // decision and from their ring and L2, unless their rank already shows an
  // earlier rejection; the owners then never stream a second pass.
  P.spec_res = 1;
  if (const char *e = getenv("SC_SPEC_RES")) P.spec_res = atoi(e) != 0;
  // Position-major unit order (every sequence's position j before any position
  // j + 1): a rejected pair then mostly sees its sequence's earlier rejection
  // already reported and skips its residual pass (B=512, gamma=8: Chow 834 ->
  // 738 us, OPT 874 -> 837 us; Diff unchanged).
  P.pos_major = 1;
  if (const char *e = getenv("SC_POS_MAJOR")) P.pos_major = atoi(e) != 0;
  // The upper bound on D_TV costs OPT pairs one more exponential per logit pair
  // in pass 1 and saves the TV pass of the band rows it settles.  With slices of
  // up to 64000 logits (C <= 4, large batches) that pass mostly re-reads HBM and
  // the bound pays (B=512, gamma=8: 873 -> 809 us); with the shorter slices of
  // C = 8 the bound costs more than it saves (B=64, gamma=8 held at C = 8:
  // 143 -> 155 us; at its C = 4, with the bound, 131 us).
  P.opt_ub = C <= 4;
  if (const char *e = getenv("SC_OPT_UB")) P.opt_ub = atoi(e) != 0;
  // L2 eviction priorities (cp.async.bulk with an evict-first cache policy): a
  // pair's slice except its newest 4 chunks, and every bonus row, leave L2
  // first, so the second passes (TV, residual), which stream newest first, hit
  // L2 more often (B=512, gamma=8: OPT 795 -> 776 us, Chow 749 -> 722 us;
  // cfg3 196 -> 189 us; keeping 2 to 6 chunks, or evict-last on them, alike).
  P.l2_hint = 4;
  if (const char *e = getenv("SC_L2_HINT")) P.l2_hint = atoi(e);
  const size_t row_bytes = static_cast<size_t>(P.V) * sizeof(E);
  P.bulk = (row_bytes % 16 == 0) && (reinterpret_cast<uintptr_t>(P.draft) % 16 == 0) &&
           (reinterpret_cast<uintptr_t>(P.target) % 16 == 0);
  P.units = units;
  if (units == 0) return SC_OK;

  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kNT, 1, 1);
  cfg.dynamicSmemBytes = smem_bytes<E>();
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(C);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // one cluster per unit; no cluster ever waits on another
  cfg.gridDim = dim3(static_cast<unsigned>(units) * static_cast<unsigned>(C), 1, 1);
  if (cudaLaunchKernelEx(&cfg, kernel, P) != cudaSuccess) return SC_ERR_CUDA;
  return SC_OK;
}

// greedy_ok: T = 0 (greedy decoding) is accepted.
int common_checks(const void *draft, const void *target, int dtype, int B, int gamma, int V,
                  float temperature, bool greedy_ok) {
  if (dtype != SC_F32 && dtype != SC_BF16) return SC_ERR_INVALID_ARG;
  if (B < 1 || gamma < 1 || gamma > SC_MAX_GAMMA || V < 1) return SC_ERR_INVALID_ARG;
  if (V > sc_max_vocab(static_cast<sc_dtype>(dtype))) return SC_ERR_UNSUPPORTED;
  if (!(temperature > 0.0f || (greedy_ok && temperature == 0.0f)) || !std::isfinite(temperature))
    return SC_ERR_INVALID_ARG;
  if (static_cast<double>(B) * (gamma + 1) * kMaxCluster > 2147483647.0) return SC_ERR_INVALID_ARG;
  if (!device_accessible(draft) || !device_accessible(target)) return SC_ERR_INVALID_ARG;
  return SC_OK;
}

// Every argument check of sc_verify_ex except the workspace's, in its order;
// SC_OK or the status the entry point returns without queueing work.
int verify_checks(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                  const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                  sc_rule rule, float alpha, float beta, float temperature,
                  const int32_t *num_accepted, const int32_t *next_token,
                  const int32_t *device_status, const float *row_info, cudaStream_t stream) {
  t_capturing = capturing(stream);
  int rc = common_checks(draft_logits, target_logits, dtype, B, gamma, V, temperature, true);
  if (rc != SC_OK) return rc;
  const int ri = static_cast<int>(rule);
  if (ri < 0 || ri > SC_RULE_OPT_LOG) return SC_ERR_INVALID_ARG;
  // alpha: a probability-scale cost for Table 1, lossy and token rules, a
  // threshold on a (cross) entropy for BiLD* and the log-loss rules
  if (ri <= SC_RULE_LOSSY ? !(alpha >= 0.0f && alpha <= 1.0f) : !(alpha >= 0.0f && std::isfinite(alpha)))
    return SC_ERR_INVALID_ARG;
  const bool greedy = temperature == 0.0f;
  // greedy decoding is defined for the scalar deferral rules only
  if (greedy && ((ri >= SC_RULE_TOKEN_V1 && ri <= SC_RULE_TOKEN_V3) || ri == SC_RULE_LOSSY))
    return SC_ERR_INVALID_ARG;
  if (ri == SC_RULE_LOSSY && !(beta > 0.0f && std::isfinite(beta) && beta >= 1.0f - alpha))
    return SC_ERR_INVALID_ARG;
  if (!device_accessible(draft_tokens) || !device_accessible(uniforms) ||
      !device_accessible(num_accepted) || !device_accessible(next_token))
    return SC_ERR_INVALID_ARG;
  if (device_status && !device_accessible(device_status)) return SC_ERR_INVALID_ARG;
  if (row_info && !device_accessible(row_info)) return SC_ERR_INVALID_ARG;
  return SC_OK;
}

// ------------------------------------------------------------------ fixed scratch

// Workspace of sc_verify_static: sc_verify's layout for the largest accepted
// batch -- SC_STATIC_MAX_UNITS units, and at most half as many sequences since
// gamma >= 1 (SC_STATIC_MAX_B is that half).  One copy per device, zeroed when
// the module loads.
static_assert(2 * SC_STATIC_MAX_B <= SC_STATIC_MAX_UNITS, "gamma >= 1 gives each sequence two units");
constexpr size_t kStaticMaxSeqs = SC_STATIC_MAX_B;
constexpr size_t kStaticScratchBytes = ws_layout(kStaticMaxSeqs, SC_STATIC_MAX_UNITS).total;
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Device address of g_static_scratch in the current device's context.  The
// host-side name is only a stand-in and must never reach a kernel.  It is looked
// up on every call (a host-side table lookup once the module is loaded), so a
// context torn down and recreated (cudaDeviceReset) never leaves a stale address.
int static_scratch(void **out) {
  void *p = nullptr;
  if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) {
    cudaGetLastError();
    return SC_ERR_CUDA;
  }
  *out = p;
  return SC_OK;
}

}  // namespace

// ------------------------------------------------------------------ C ABI

extern "C" {

size_t sc_workspace_bytes(int B, int gamma, int V) {
  (void)V;
  if (B < 1 || gamma < 1) return 0;
  return ws_layout(static_cast<size_t>(B), static_cast<size_t>(B) * (gamma + 1)).total;
}

int sc_workspace_init(void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  if (!workspace) return SC_ERR_INVALID_ARG;
  return cudaMemsetAsync(workspace, 0, workspace_bytes, stream) == cudaSuccess ? SC_OK : SC_ERR_CUDA;
}

int sc_debug_line(int reset) {
  if (!SC_DEBUG) return -1;
  int line = 0;
  if (cudaMemcpyFromSymbol(&line, g_sc_debug_line, sizeof(int)) != cudaSuccess) return SC_ERR_CUDA;
  if (reset) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(g_sc_debug_line, &zero, sizeof(int)) != cudaSuccess) return SC_ERR_CUDA;
  }
  return line;
}

int sc_max_vocab(sc_dtype dtype) {
  (void)dtype;  // the ring does not depend on V: one cluster covers kMaxCluster slices
  return kMaxCluster * kMaxChunks * kCH;
}

int sc_verify_ex(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                 const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                 sc_rule rule, float alpha, float beta, float temperature, int32_t *num_accepted,
                 int32_t *next_token, void *workspace, size_t workspace_bytes,
                 int32_t *device_status, float *row_info, cudaStream_t stream) {
  int rc = verify_checks(draft_logits, target_logits, dtype, draft_tokens, uniforms, B, gamma, V, rule,
                         alpha, beta, temperature, num_accepted, next_token, device_status, row_info,
                         stream);
  if (rc != SC_OK) return rc;
  const int ri = static_cast<int>(rule);
  const bool greedy = temperature == 0.0f;
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
  P.rule = ri;
  P.alpha = alpha;
  P.temperature = temperature;
  P.greedy = greedy ? 1 : 0;
  set_k(P, greedy ? 1.0f : temperature);  // greedy: the rules' statistics at T = 1
  if (ri == SC_RULE_LOSSY) {
    // -log2(1 - alpha) as hi + lo, and -log2(beta)
    const double l = alpha < 1.0f ? -std::log2(1.0 - static_cast<double>(alpha)) : HUGE_VAL;
    P.lossy_l = static_cast<float>(l);
    P.lossy_ll = std::isfinite(l) ? static_cast<float>(l - static_cast<double>(P.lossy_l)) : 0.0f;
    P.lossy_c = static_cast<float>(-std::log2(static_cast<double>(beta)));
    P.beta = beta;
  }
  P.mode = kVerify;
  P.num_accepted = num_accepted;
  P.next_token = next_token;
  P.row_info = row_info;
  P.status = device_status;
  unsigned char *ws = static_cast<unsigned char *>(workspace);
  const WsLayout wl = ws_layout(static_cast<size_t>(B), static_cast<size_t>(B) * (gamma + 1));
  P.rank_tickets = reinterpret_cast<unsigned long long *>(ws + wl.rank_tickets);
  P.seq_tickets = reinterpret_cast<uint32_t *>(ws + wl.seq_tickets);
  P.records = reinterpret_cast<float4 *>(ws + wl.records);
  P.records2 = reinterpret_cast<float4 *>(ws + wl.records2);
  P.chunk_pre = reinterpret_cast<float *>(ws + wl.chunk_pre);
  P.bonus_pre = reinterpret_cast<float *>(ws + wl.bonus_pre);
  P.row_pre = reinterpret_cast<float *>(ws + wl.row_pre);
  const int units = B * (gamma + 1);
  return dtype == SC_BF16 ? launch<uint16_t>(P, stream, units) : launch<float>(P, stream, units);
}

int sc_verify_rows(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                   const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                   sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
                   int32_t *next_token, void *workspace, size_t workspace_bytes,
                   int32_t *device_status, float *row_info, cudaStream_t stream) {
  return sc_verify_ex(draft_logits, target_logits, dtype, draft_tokens, uniforms, B, gamma, V, rule,
                      alpha, 1.0f, temperature, num_accepted, next_token, workspace, workspace_bytes,
                      device_status, row_info, stream);
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
  t_capturing = capturing(stream);
  int rc = common_checks(draft_logits, target_logits, dtype, B, gamma, V, temperature, false);
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
  set_k(P, temperature);
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
    case SC_ERR_SCRATCH_LIMIT: return "batch exceeds the fixed scratch of sc_verify_static";
    default: return "unknown status";
  }
}

// Same verification kernel, with its workspace in g_static_scratch instead of
// caller memory.  No allocation: after the argument checks the tickets are
// cleared with a memset on the caller's stream and sc_verify_rows runs on the
// fixed array.
int sc_verify_static(const void *draft_logits, const void *target_logits, sc_dtype dtype,
                     const int32_t *draft_tokens, const float *uniforms, int B, int gamma, int V,
                     sc_rule rule, float alpha, float temperature, int32_t *num_accepted,
                     int32_t *next_token, int32_t *device_status, cudaStream_t stream) {
  if (B < 1 || gamma < 1) return SC_ERR_INVALID_ARG;
  if (B > SC_STATIC_MAX_B || static_cast<long>(B) * (static_cast<long>(gamma) + 1) > SC_STATIC_MAX_UNITS)
    return SC_ERR_SCRATCH_LIMIT;
  const size_t need = sc_workspace_bytes(B, gamma, V);
  if (need > kStaticScratchBytes) return SC_ERR_SCRATCH_LIMIT;
  // every other argument is checked before the scratch is touched: a refused
  // call queues nothing
  int rc = verify_checks(draft_logits, target_logits, dtype, draft_tokens, uniforms, B, gamma, V, rule,
                         alpha, 1.0f, temperature, num_accepted, next_token, device_status, nullptr,
                         stream);
  if (rc != SC_OK) return rc;
  void *ws = nullptr;
  rc = static_scratch(&ws);
  if (rc != SC_OK) return rc;
  // the previous call left the tickets at zero unless it was cut short: clear them
  const size_t zeroed = ws_layout(static_cast<size_t>(B), static_cast<size_t>(B) * (gamma + 1)).zeroed;
  if (cudaMemsetAsync(ws, 0, zeroed, stream) != cudaSuccess) return SC_ERR_CUDA;
  return sc_verify_rows(draft_logits, target_logits, dtype, draft_tokens, uniforms, B, gamma, V,
                        rule, alpha, temperature, num_accepted, next_token, ws, need,
                        device_status, nullptr, stream);
}

}  // extern "C"
