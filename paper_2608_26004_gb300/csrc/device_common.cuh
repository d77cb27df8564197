// Device helpers shared by the fuse-and-verify kernels (sm_103a).
#pragma once

#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cmath>
#include <cstdint>

#include "asymspec.h"

namespace cg = cooperative_groups;

namespace asymspec_impl {


constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.69314718055994531f;
constexpr float kMinNormal = 1.17549435e-38f;  // 2^-126
constexpr int kMaxSmem = 227 * 1024;
constexpr int kPreferredSliceBytes = 96 * 1024;

// ----------------------------------------------------------- device helpers

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gmem) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;" ::: "memory");
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// The fused score t + beta delta of one entry (Eq. 2) for delta source ds
// (ASYMSPEC_DELTA_*: a - b, a, or t - b).
__device__ __forceinline__ float fuse1(float beta, float a, float b, float t, int ds) {
  return ds == ASYMSPEC_DELTA_A    ? fmaf(beta, a, t)
         : ds == ASYMSPEC_DELTA_TB ? fmaf(beta, t - b, t)
                                   : fmaf(beta, a - b, t);
}

// Vector of VE consecutive elements from shared memory, widened to fp32.
__device__ __forceinline__ void load_vec(const float* p, float (&x)[4]) {
  const float4 v = *reinterpret_cast<const float4*>(p);
  x[0] = v.x;
  x[1] = v.y;
  x[2] = v.z;
  x[3] = v.w;
}
__device__ __forceinline__ void load_vec(const float* p, float (&x)[1]) { x[0] = *p; }
__device__ __forceinline__ void load_vec(const __nv_bfloat16* p, float (&x)[8]) {
  const uint4 v = *reinterpret_cast<const uint4*>(p);
  const unsigned w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    x[2 * h] = __uint_as_float(w[h] << 16);
    x[2 * h + 1] = __uint_as_float(w[h] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void load_vec(const __nv_bfloat16* p, float (&x)[1]) {
  x[0] = __bfloat162float(*p);
}

template <int N>
__device__ __forceinline__ float vmax(const float (&x)[N]) {
  float m = x[0];
#pragma unroll
  for (int e = 1; e < N; ++e) m = fmaxf(m, x[e]);
  return m;
}

// Adds a chunk to a running (max m, sum of 2^((x - m) log2 e)) pair and
// returns the chunk maximum.  The running sum is rescaled only when the chunk
// raises the maximum.
template <int N>
__device__ __forceinline__ float online_add(float& m, float& s, const float (&x)[N]) {
  const float cm = vmax(x);
  if (cm > m) {
    s *= ex2((m - cm) * kLog2e);
    m = cm;
  }
  const float mL = m * kLog2e;
  float acc = 0.f;
#pragma unroll
  for (int e = 0; e < N; ++e) acc += ex2(fmaf(x[e], kLog2e, -mL));
  s += acc;
  return cm;
}

// (m, s) pairs combine into (max, rescaled sum).  The operation is
// commutative bit for bit, so a butterfly leaves every lane with the same
// value.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  const float f1 = (m == M) ? 1.f : ex2((m - M) * kLog2e);
  const float f2 = (m2 == M) ? 1.f : ex2((m2 - M) * kLog2e);
  s = s * f1 + s2 * f2;
  m = M;
}

// Larger value wins; the lower index wins a tie; NaN never wins.
__device__ __forceinline__ void arg_merge(float& v, int& i, float v2, int i2) {
  if (v2 > v || (v2 == v && i2 < i)) {
    v = v2;
    i = i2;
  }
}

struct Stats1 {
  float m[4];  // running maxima of a, b, t, s
  float s[4];  // sums of 2^((x - m) log2 e)
  float vs;    // max of s and its lowest index
  int is;
  float vt;    // max of t and its lowest index
  int it;
};

struct Stats2 {
  float j;     // sum of p (log2 p - log2(p+q)) + q (log2 q - log2(p+q))
  float msum;  // sum of p + q
  float kl;    // sum of p (log2 p - log2 q)
  float R;     // residual mass sum max(0, q_fused - p)
  float Q;     // fused mass sum q_fused
};

__device__ __forceinline__ Stats1 stats1_neutral() {
  Stats1 r;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    r.m[q] = -INFINITY;
    r.s[q] = 0.f;
  }
  r.vs = -INFINITY;
  r.is = INT_MAX;
  r.vt = -INFINITY;
  r.it = INT_MAX;
  return r;
}

__device__ __forceinline__ void stats1_merge(Stats1& r, const Stats1& o) {
#pragma unroll
  for (int q = 0; q < 4; ++q) lse_merge(r.m[q], r.s[q], o.m[q], o.s[q]);
  arg_merge(r.vs, r.is, o.vs, o.is);
  arg_merge(r.vt, r.it, o.vt, o.it);
}

__device__ __forceinline__ Stats1 stats1_shfl(const Stats1& r, int off) {
  Stats1 o;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    o.m[q] = __shfl_xor_sync(0xffffffffu, r.m[q], off);
    o.s[q] = __shfl_xor_sync(0xffffffffu, r.s[q], off);
  }
  o.vs = __shfl_xor_sync(0xffffffffu, r.vs, off);
  o.is = __shfl_xor_sync(0xffffffffu, r.is, off);
  o.vt = __shfl_xor_sync(0xffffffffu, r.vt, off);
  o.it = __shfl_xor_sync(0xffffffffu, r.it, off);
  return o;
}

__device__ __forceinline__ void stats1_warp_reduce(Stats1& r) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) stats1_merge(r, stats1_shfl(r, off));
}

__device__ __forceinline__ void stats2_warp_reduce(Stats2& r) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    r.j += __shfl_xor_sync(0xffffffffu, r.j, off);
    r.msum += __shfl_xor_sync(0xffffffffu, r.msum, off);
    r.kl += __shfl_xor_sync(0xffffffffu, r.kl, off);
    r.R += __shfl_xor_sync(0xffffffffu, r.R, off);
    r.Q += __shfl_xor_sync(0xffffffffu, r.Q, off);
  }
}


// ----------------------------------------------------------- packed fp32 pairs
// sm_100+ executes add/sub/mul/fma on two fp32 lanes per instruction; a
// 64-bit register holds the pair (low half = first element).

using f2 = unsigned long long;

__device__ __forceinline__ f2 pk(float lo, float hi) {
  f2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void upk(f2 v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ float lo_of(f2 v) {
  float lo, hi;
  upk(v, lo, hi);
  return lo;
}
__device__ __forceinline__ float hi_of(f2 v) {
  float lo, hi;
  upk(v, lo, hi);
  return hi;
}
__device__ __forceinline__ f2 add2(f2 a, f2 b) {
  f2 r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ f2 sub2(f2 a, f2 b) {
  f2 r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ f2 mul2(f2 a, f2 b) {
  f2 r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ f2 fma2(f2 a, f2 b, f2 c) {
  f2 r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ f2 ex2_2(f2 x) {
  float a, b;
  upk(x, a, b);
  return pk(ex2(a), ex2(b));
}
__device__ __forceinline__ f2 lg2_2(f2 x) {
  float a, b;
  upk(x, a, b);
  return pk(lg2(a), lg2(b));
}
__device__ __forceinline__ f2 relu2(f2 x) {
  float a, b;
  upk(x, a, b);
  return pk(fmaxf(a, 0.f), fmaxf(b, 0.f));
}
__device__ __forceinline__ float hsum2(f2 x) {
  float a, b;
  upk(x, a, b);
  return a + b;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
// NaN-propagating maximum (flags non-finite data in argmax-only streams).
__device__ __forceinline__ float max_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Pairs of a 16-byte vector held in shared memory.
__device__ __forceinline__ void load_pairs(const float* p, f2 (&x)[2]) {
  const float4 v = *reinterpret_cast<const float4*>(p);
  x[0] = pk(v.x, v.y);
  x[1] = pk(v.z, v.w);
}
__device__ __forceinline__ void load_pairs(const __nv_bfloat16* p, f2 (&x)[4]) {
  const uint4 v = *reinterpret_cast<const uint4*>(p);
  const unsigned w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int h = 0; h < 4; ++h) x[h] = pk(__uint_as_float(w[h] << 16), __uint_as_float(w[h] & 0xFFFF0000u));
}

// ----------------------------------------------------------- mbarrier and bulk copies

__device__ __forceinline__ unsigned smem_u32(const void* p) {
  return static_cast<unsigned>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(unsigned long long* bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(unsigned long long* bar, unsigned bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(unsigned long long* bar, unsigned parity) {
  unsigned ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking test of the phase with the given parity (try_wait may suspend
// the thread for a while; test_wait returns at once).
__device__ __forceinline__ bool mbar_test_wait(unsigned long long* bar, unsigned parity) {
  unsigned ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// As mbar_try_wait, suspending the thread for up to hint_ns while the phase
// is incomplete (the thread resumes as soon as it completes), so a waiting
// warp takes no issue slots.
__device__ __forceinline__ bool mbar_try_wait_hint(unsigned long long* bar, unsigned parity,
                                                   unsigned hint_ns) {
  unsigned ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3; "
      "selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}
constexpr unsigned kSuspendHintNs = 100000;  // 0.1 ms per suspension

// Waits for the phase with the given parity, giving up after limit_ns.  A
// limit of 0 gives up at once, without looking at the barrier (the test hook
// ASYMSPEC_TEST_COPY_GIVE_UP: a wait that times out, with no fault needed).
__device__ __forceinline__ bool mbar_wait_bounded(unsigned long long* bar, unsigned parity,
                                                  unsigned long long limit_ns) {
  if (limit_ns == 0) return false;
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  while (!mbar_try_wait_hint(bar, parity, kSuspendHintNs)) {
    if (global_ns() - t0 > limit_ns) return false;
  }
  return true;
}
// Cluster-scope acquire wait (sees stores another CTA released before its
// remote arrive on this barrier), bounded like mbar_wait_bounded.
__device__ __forceinline__ bool mbar_try_wait_cluster(unsigned long long* bar, unsigned parity) {
  unsigned ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2; "
      "selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_cluster_bounded(unsigned long long* bar, unsigned parity,
                                                          unsigned long long limit_ns) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  while (!mbar_try_wait_cluster(bar, parity)) {
    if (global_ns() - t0 > limit_ns) return false;
  }
  return true;
}
// Arrive, with cluster-scope release, on an mbarrier of CTA `rank` of this
// cluster (the local address of the same variable names it in every CTA).
__device__ __forceinline__ void mbar_arrive_remote(unsigned long long* bar, unsigned rank) {
  unsigned remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote)
               : "memory");
}

// Orders this thread's earlier generic-proxy accesses to shared memory before
// later async-proxy ones (a bulk copy into a buffer that was just read).
__device__ __forceinline__ void fence_proxy_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 1-D bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, unsigned bytes,
                                          unsigned long long* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Plain arrive (one count) on an mbarrier of this CTA.
__device__ __forceinline__ void mbar_arrive(unsigned long long* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

struct KParams {
  const void* a;
  const void* b;
  const void* t;
  const int32_t* tokens;
  const float* dprobs;
  const float* unif;
  int B, K, V;
  int C, W, sh_off;
  float gamma, beta, lambda, ln_gamma;
  int divergence, fuse_bonus;
  int delta_src;               // ASYMSPEC_DELTA_*: the signal fused into the emission (Eq. 1)
  int need_lse_s, need_pass2;  // generic kernel: compute LSE(s); run pass 2
  int full;                    // compute every row quantity (debug outputs)
  int want_tokens;             // also track argmax(s) in stochastic rows (per-row tokens)
  long long rows;              // B (K+1)
  int32_t* out_len;
  int32_t* out_next;
  float* row_stats;
  int32_t* row_tokens;
  float* logprobs;
  uint32_t* err_word;
  int4* recs;
  unsigned int* tickets;
  // cluster TMA kernel: what its rows leave for the decision kernel
  void* row_stat;       // [B(K+1)] RowStat (rank 0 of the row's cluster)
  float* pass2_rec;     // [B(K+1)][C] X2 records (8 floats), one per CTA
  float* group_mass;    // [B(K+1)][C][group_stride] inverse-CDF group masses (stochastic)
  int group_stride;     // floats per row and CTA in group_mass (one per warp and round)
  int tma_threads;      // threads per CTA of the row kernel (its group layout)
  int row_blocks;       // 1: fuse_verify_row's layout, one inverse-CDF group per warp block
  unsigned long long copy_wait_ns;  // limit of each bulk-copy wait (0: give up at once)
  int walk_stage;       // decide_rows on fuse_verify_row's rows: staging bytes per warp
};

// What pass 1 leaves for the decision of a row: the normalisers, the
// argmaxes, the data-error bits and the draft token's three logits.
struct __align__(16) RowStat {
  float lse[4];
  int is, it;
  unsigned bad;
  int dtok;
  float da, db, dt;
  float pad;
};


// ----------------------------------------------------------- row epilogue

constexpr unsigned kBadS = 1u;        // non-finite fused score seen by an argmax-only stream
constexpr unsigned kBadT = 2u;        // non-finite verifier logit seen by an argmax-only stream
constexpr unsigned kBadTimeout = 4u;  // a bulk copy did not complete in time

// Everything a row contributes to the scan, as combined over its cluster.
struct RowResult {
  float lse_a, lse_b, lse_t, lse_s;  // NaN when not computed
  float D;                           // JSD or KL in nats (0 when the gate has none)
  int is, it;                        // argmax of s and of t (INT_MAX if not computed)
  int sample;                        // stochastic inverse-CDF draw (-1 if none)
  float mass;                        // stochastic inverse-CDF mass (NaN in greedy mode)
  unsigned bad;                      // kBad* bits
  bool have_lse_t;                   // lse_t was computed (greedy bonus rows may skip it)
};

// The stochastic inputs of one row: the drafter's probability of the draft
// token, the uniform of its test, and the element's one non-draft uniform.
struct RowScalars {
  float dprob, u, u_last;
};

__device__ __forceinline__ RowScalars load_row_scalars(const KParams& P, int bi, int k) {
  RowScalars sc{0.f, 0.f, 0.f};
  const int K1 = P.K + 1;
  sc.u_last = P.unif[static_cast<size_t>(bi) * K1 + P.K];
  if (k < P.K) {
    sc.dprob = P.dprobs[static_cast<size_t>(bi) * P.K + k];
    sc.u = P.unif[static_cast<size_t>(bi) * K1 + k];
  }
  return sc;
}

// The decision of one complete row, on one thread: data checks, the
// acceptance test of Eq. 4 (or its stochastic counterpart), the emitted
// candidate, and the optional per-row outputs.  Returns the 16-byte row
// record (accept bit, candidate, ASYMSPEC_DATA_* bits).
// dtok/ad/bd/td: the draft token of this row and its three logits.
template <bool STOCH>
__device__ int4 row_record(const KParams& P, long long row, int k, const RowResult& r, int dtok,
                           float ad, float bd, float td, const RowScalars& sc) {
  const int V = P.V, K = P.K;
  const bool bonus = (k == K);
  unsigned err = 0;
  if (r.bad & kBadTimeout) err |= ASYMSPEC_DATA_TIMEOUT;
  float D = r.D;
  const bool div_sum = (P.divergence == ASYMSPEC_DIV_JSD || P.divergence == ASYMSPEC_DIV_KL);
  if (!bonus || STOCH) {
    if (!bonus || !STOCH) {
      if (!isfinite(r.lse_a) || !isfinite(r.lse_b)) err |= ASYMSPEC_DATA_NONFINITE;
      if (div_sum && !isfinite(D)) err |= ASYMSPEC_DATA_NONFINITE;
    }
    if (STOCH) {
      if (!isfinite(r.lse_s)) err |= ASYMSPEC_DATA_NONFINITE;
    } else {
      if (!isfinite(r.lse_t)) err |= ASYMSPEC_DATA_NONFINITE;
      if (r.is == INT_MAX || (r.bad & kBadS)) err |= ASYMSPEC_DATA_NONFINITE;
    }
  } else if (P.fuse_bonus) {  // greedy bonus, fused
    if (r.is == INT_MAX || (r.bad & kBadS)) err |= ASYMSPEC_DATA_NONFINITE;
  } else {                    // greedy bonus: only t is used
    if (r.it == INT_MAX || (r.bad & kBadT) || (r.have_lse_t && !isfinite(r.lse_t)))
      err |= ASYMSPEC_DATA_NONFINITE;
  }
  if (P.divergence == ASYMSPEC_DIV_JSD) D = fminf(fmaxf(D, 0.f), kLn2);
  if (P.divergence == ASYMSPEC_DIV_KL) D = fmaxf(D, 0.f);
  if (STOCH && !(sc.u_last >= 0.f && sc.u_last < 1.f)) err |= ASYMSPEC_DATA_BAD_UNIFORM;
  int accept = 1;
  float margin = NAN;
  float gamma_eff = P.gamma;
  if (!bonus) {
    if (dtok < 0 || dtok >= V) {
      err |= ASYMSPEC_DATA_BAD_TOKEN;
    } else {
      const float la_d = ad - r.lse_a, lb_d = bd - r.lse_b;
      if (P.divergence == ASYMSPEC_DIV_LAMBDA) D = P.lambda * (la_d - lb_d);
      const float ln_geff = P.ln_gamma - D;
      gamma_eff = expf(ln_geff);
      if (!STOCH) {
        const float lr = (td - r.lse_t) - lb_d;  // log(softmax(t)[d] / softmax(b)[d])
        accept = lr > ln_geff;                   // Eq. 4
        margin = 1.f - expf(lr - ln_geff);
      } else {
        const float pd = sc.dprob, u = sc.u;
        if (!(pd > 0.f && pd <= 1.f)) err |= ASYMSPEC_DATA_BAD_PROB;
        if (!(u >= 0.f && u < 1.f)) err |= ASYMSPEC_DATA_BAD_UNIFORM;
        // the draft token's fused score, for the delta source in use
        const float sd = P.delta_src == ASYMSPEC_DELTA_A    ? fmaf(P.beta, ad, td)
                         : P.delta_src == ASYMSPEC_DELTA_TB ? fmaf(P.beta, td - bd, td)
                                                            : fmaf(P.beta, ad - bd, td);
        const float qd = expf(sd - r.lse_s);
        accept = qd > u * gamma_eff * pd;
        margin = u - (qd / pd) / gamma_eff;
      }
    }
  } else if (P.divergence != ASYMSPEC_DIV_LAMBDA) {
    gamma_eff = expf(P.ln_gamma - D);
  } else {
    D = 0.f;
  }
  int cand;
  if (STOCH) cand = r.sample;
  else cand = (!bonus || P.fuse_bonus) ? r.is : r.it;
  if (cand < 0 || cand >= V) err |= ASYMSPEC_DATA_NONFINITE;

  if (P.row_stats) {
    float* rs = P.row_stats + static_cast<size_t>(row) * 8;
    rs[0] = r.lse_a;
    rs[1] = r.lse_b;
    rs[2] = r.lse_t;
    rs[3] = r.lse_s;
    rs[4] = D;
    rs[5] = gamma_eff;
    rs[6] = margin;
    rs[7] = r.mass;
  }
  if (P.row_tokens) {
    P.row_tokens[static_cast<size_t>(row) * 2] = (r.is == INT_MAX) ? -1 : r.is;
    P.row_tokens[static_cast<size_t>(row) * 2 + 1] = cand;
  }
  if (err && P.err_word) atomicOr(P.err_word, err);
  return make_int4(accept, cand, static_cast<int>(err), 0);
}

// Runs on one thread per row once the row is complete: the row record and
// the batch element's ticket.  The last row of a batch element to arrive
// runs Algorithm 1's scan.
template <bool STOCH>
__device__ void finish_row(const KParams& P, long long row, int bi, int k, const RowResult& r,
                           int dtok, float ad, float bd, float td) {
  const int K = P.K, K1 = K + 1;
  const RowScalars sc = STOCH ? load_row_scalars(P, bi, k) : RowScalars{0.f, 0.f, 0.f};
  P.recs[row] = row_record<STOCH>(P, row, k, r, dtok, ad, bd, td, sc);
  __threadfence();
  const unsigned ticket = atomicAdd(&P.tickets[bi], 1u);
  if (ticket != static_cast<unsigned>(K)) return;

  // last row of batch element bi: Algorithm 1's sequential scan
  __threadfence();
  const int4* recs = P.recs + static_cast<size_t>(bi) * K1;
  int any_err = 0;
  for (int j = 0; j < K1; ++j) any_err |= __ldcg(&recs[j].z);
  int len = K;
  for (int j = 0; j < K; ++j) {
    if (!__ldcg(&recs[j].x)) {
      len = j;
      break;
    }
  }
  const int next = __ldcg(&recs[len].y);
  P.out_len[bi] = any_err ? -1 : len;
  P.out_next[bi] = any_err ? -1 : next;
  P.tickets[bi] = 0u;
}

__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v)
               : "memory");
  return old;
}

// As finish_row, executed by a whole warp (lane 0 decides the row).  The
// ticket's read-modify-write has acquire-release semantics, which orders this
// row's record before it and every other row's record after it; the last
// row reads the K+1 records 32 at a time, one per lane, and takes Algorithm
// 1's first rejection with a ballot.
template <bool STOCH>
__device__ void finish_row_warp(const KParams& P, long long row, int bi, int k,
                                const RowResult& r, int dtok, float ad, float bd, float td,
                                const RowScalars& sc) {
  const int lane = threadIdx.x & 31;
  const int K = P.K, K1 = K + 1;
  unsigned ticket = 0;
  if (lane == 0) {
    P.recs[row] = row_record<STOCH>(P, row, k, r, dtok, ad, bd, td, sc);
    ticket = atom_add_acq_rel(&P.tickets[bi], 1u);
  }
  ticket = __shfl_sync(0xffffffffu, ticket, 0);
  if (ticket != static_cast<unsigned>(K)) return;
  __syncwarp();
  const int4* recs = P.recs + static_cast<size_t>(bi) * K1;
  bool any_err = false;
  int len = -1, next = -1;
  for (int base = 0; base < K1; base += 32) {
    const int j = base + lane;
    int4 v = make_int4(1, -1, 0, 0);
    if (j < K1) v = __ldcg(&recs[j]);
    any_err |= __any_sync(0xffffffffu, v.z != 0);
    if (len < 0) {
      const unsigned rej = __ballot_sync(0xffffffffu, j < K && v.x == 0);
      if (rej) len = base + __ffs(rej) - 1;
      else if (K < base + 32) len = K;
      if (len >= 0) next = __shfl_sync(0xffffffffu, v.y, len - base);
    }
  }
  if (lane == 0) {
    P.out_len[bi] = any_err ? -1 : len;
    P.out_next[bi] = any_err ? -1 : next;
    P.tickets[bi] = 0u;
  }
}

// The draft token of row (bi, k) and its three logits (rank 0, thread 0).
template <typename T>
__device__ __forceinline__ void fetch_draft(const KParams& P, long long row, int bi, int k,
                                            int& dtok, float& ad, float& bd, float& td) {
  dtok = -1;
  ad = bd = td = 0.f;
  if (k >= P.K) return;
  dtok = P.tokens[static_cast<size_t>(bi) * P.K + k];
  if (dtok >= 0 && dtok < P.V) {
    const size_t o = static_cast<size_t>(row) * P.V + dtok;
    ad = to_f32(static_cast<const T*>(P.a)[o]);
    bd = to_f32(static_cast<const T*>(P.b)[o]);
    td = to_f32(static_cast<const T*>(P.t)[o]);
  }
}

}  // namespace asymspec_impl
