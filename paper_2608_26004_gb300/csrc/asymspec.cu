// AsymSpec per-step fuse-and-verify on GB300 (sm_103a): kernels and the C ABI
// declared in include/asymspec.h.
//
// One thread-block cluster of C CTAs handles one row triple (a, b, t) of one
// position.  Each CTA copies a disjoint slice of the vocabulary of the three
// rows from HBM into shared memory with 16-byte asynchronous copies (the only
// HBM read of the logits) and then works from shared memory:
//   pass 1  online (max, sum of exponentials) of a, b, t and of the fused
//           scores s = t + beta (a - b) (Eqs. 1-2), argmax of s and of t;
//   DSMEM   the C partial results are combined in every CTA (same order in
//           each, so every CTA holds bit-identical row normalisers);
//   pass 2  Jensen-Shannon (or KL) divergence of softmax(a) and softmax(b)
//           (Eq. 3), and, in stochastic mode, the residual mass
//           max(0, q - softmax(a)) and the fused mass q = softmax(s);
//   DSMEM   partial sums combined again; a prefix over the cluster ranks picks
//           the CTA that owns the inverse-CDF target, and that CTA locates the
//           index with a block-wide prefix scan over its slice;
//   epilogue  rank 0 evaluates the acceptance test of Eq. 4 for the row's draft
//           token, writes a 16-byte row record and takes a ticket; the last
//           row of a batch element to finish runs Algorithm 1's sequential
//           scan over the K+1 records and writes the outputs.
// There are no spin-waits: hardware cluster barriers are reached by every CTA
// of a cluster, and the cross-cluster hand-off is a fetch-and-add ticket.
#include "asymspec.h"

#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cmath>
#include <cstdint>
#include <mutex>

namespace cg = cooperative_groups;

namespace {

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

struct Shared {
  Stats1 warp1[kWarps];
  Stats2 warp2[kWarps];
  Stats1 cta1;  // this CTA's pass-1 totals (read by the cluster)
  Stats2 cta2;  // this CTA's pass-2 totals (read by the cluster)
  float lse[4];
  int is, it;
  float D;
  float mass_total;  // inverse-CDF mass of the row (stochastic)
  float tau_local;   // target relative to the owning CTA's start
  int owner;         // rank owning the inverse-CDF target, -1 if none
  int use_r;         // 1: residual mass, 0: fused mass
  int sample;        // drawn token (written into rank 0 by the owner)
  int found;
  float scan[kWarps];
};

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
  int need_lse_s, need_pass2;
  int32_t* out_len;
  int32_t* out_next;
  float* row_stats;
  int32_t* row_tokens;
  float* logprobs;
  uint32_t* err_word;
  int4* recs;
  unsigned int* tickets;
};

// The residual / fused mass of one element (stochastic mode).  Pass 2 and the
// inverse-CDF walk both call this, so they see identical values.
__device__ __forceinline__ float sample_mass(float xa, float xb, float xt, float beta, float A2,
                                             float S2, bool use_r) {
  const float xs = fmaf(beta, xa - xb, xt);
  const float qf = ex2(fmaf(xs, kLog2e, -S2));
  if (!use_r) return qf;
  const float p = ex2(fmaf(xa, kLog2e, -A2));
  return fmaxf(qf - p, 0.f);
}

template <typename T, int VE, bool STOCH>
__global__ void __launch_bounds__(kThreads, 1) fuse_verify_kernel(const KParams P) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int C = P.C;
  const long long row = blockIdx.x / C;
  const int K1 = P.K + 1;
  const int bi = static_cast<int>(row / K1);
  const int k = static_cast<int>(row % K1);
  const int V = P.V;
  const int lo = rank * P.W;
  const int n = max(0, min(P.W, V - lo));
  const int nv = n / VE;

  T* sa = reinterpret_cast<T*>(smem_raw);
  T* sb = sa + P.W;
  T* st = sb + P.W;
  Shared* sh = reinterpret_cast<Shared*>(smem_raw + P.sh_off);

  const size_t roff = static_cast<size_t>(row) * V + lo;
  const T* ga = static_cast<const T*>(P.a) + roff;
  const T* gb = static_cast<const T*>(P.b) + roff;
  const T* gt = static_cast<const T*>(P.t) + roff;

  // ---- stage the slice: the single HBM read of the three rows
  if constexpr (VE > 1) {
    for (int i = tid; i < nv; i += kThreads) {
      cp_async16(sa + i * VE, ga + i * VE);
      cp_async16(sb + i * VE, gb + i * VE);
      cp_async16(st + i * VE, gt + i * VE);
    }
    cp_async_wait_all();
  } else {
    for (int i = tid; i < n; i += kThreads) {
      sa[i] = ga[i];
      sb[i] = gb[i];
      st[i] = gt[i];
    }
  }

  // set before the first cluster barrier, so a remote owner's write lands after it
  if (tid == 0) sh->sample = -1;

  // rank 0 fetches the draft token and its three logits meanwhile
  const bool leader = (rank == 0 && tid == 0);
  int dtok = -1;
  float ad = 0.f, bd = 0.f, td = 0.f;
  if (leader && k < P.K) {
    dtok = P.tokens[static_cast<size_t>(bi) * P.K + k];
    if (dtok >= 0 && dtok < V) {
      const size_t o = static_cast<size_t>(row) * V + dtok;
      ad = to_f32(static_cast<const T*>(P.a)[o]);
      bd = to_f32(static_cast<const T*>(P.b)[o]);
      td = to_f32(static_cast<const T*>(P.t)[o]);
    }
  }
  __syncthreads();

  // ---- pass 1: normalisers and argmaxes
  const float beta = P.beta;
  Stats1 r1 = stats1_neutral();
  for (int i = tid; i < nv; i += kThreads) {
    float xa[VE], xb[VE], xt[VE], xs[VE];
    load_vec(sa + i * VE, xa);
    load_vec(sb + i * VE, xb);
    load_vec(st + i * VE, xt);
#pragma unroll
    for (int e = 0; e < VE; ++e) xs[e] = fmaf(beta, xa[e] - xb[e], xt[e]);
    online_add(r1.m[0], r1.s[0], xa);
    online_add(r1.m[1], r1.s[1], xb);
    const float ct = online_add(r1.m[2], r1.s[2], xt);
    const float cs = P.need_lse_s ? online_add(r1.m[3], r1.s[3], xs) : vmax(xs);
    const int base = lo + i * VE;
    if (cs > r1.vs) {
      r1.vs = cs;
#pragma unroll
      for (int e = VE - 1; e >= 0; --e)
        if (xs[e] == cs) r1.is = base + e;
    }
    if (ct > r1.vt) {
      r1.vt = ct;
#pragma unroll
      for (int e = VE - 1; e >= 0; --e)
        if (xt[e] == ct) r1.it = base + e;
    }
  }
  stats1_warp_reduce(r1);
  if (lane == 0) sh->warp1[warp] = r1;
  __syncthreads();
  if (warp == 0) {
    Stats1 w = (lane < kWarps) ? sh->warp1[lane] : stats1_neutral();
    stats1_warp_reduce(w);
    if (lane == 0) sh->cta1 = w;
  }
  cluster.sync();  // #1: every CTA's pass-1 totals are in place
  if (warp == 0) {
    Stats1 w = stats1_neutral();
    if (lane < C) w = *cluster.map_shared_rank(&sh->cta1, lane);
    stats1_warp_reduce(w);
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < 4; ++q) sh->lse[q] = w.m[q] + logf(w.s[q]);
      sh->is = w.is;
      sh->it = w.it;
    }
  }
  __syncthreads();

  // ---- pass 2: divergence, residual and fused masses
  const float lse_a = sh->lse[0], lse_b = sh->lse[1], lse_s = sh->lse[3];
  const float A2 = lse_a * kLog2e, B2 = lse_b * kLog2e, S2 = lse_s * kLog2e;
  const bool do_jsd = P.divergence == ASYMSPEC_DIV_JSD;
  const bool do_kl = P.divergence == ASYMSPEC_DIV_KL;
  float* lp = P.logprobs ? P.logprobs + static_cast<size_t>(row) * V + lo : nullptr;
  Stats2 r2 = {0.f, 0.f, 0.f, 0.f, 0.f};
  if (P.need_pass2) {
    for (int i = tid; i < nv; i += kThreads) {
      float xa[VE], xb[VE], xt[VE];
      load_vec(sa + i * VE, xa);
      load_vec(sb + i * VE, xb);
      if (STOCH || lp) load_vec(st + i * VE, xt);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const float la2 = fmaf(xa[e], kLog2e, -A2);
        const float lb2 = fmaf(xb[e], kLog2e, -B2);
        const float p = ex2(la2);
        if (do_jsd) {
          const float q = ex2(lb2);
          const float mm = fmaxf(p + q, kMinNormal);
          const float lg = lg2(mm);
          r2.j += p * (la2 - lg) + q * (lb2 - lg);
          r2.msum += mm;
        }
        if (do_kl) r2.kl += p * (la2 - lb2);
        if (STOCH) {
          const float xs = fmaf(beta, xa[e] - xb[e], xt[e]);
          const float qf = ex2(fmaf(xs, kLog2e, -S2));
          r2.R += fmaxf(qf - p, 0.f);
          r2.Q += qf;
        }
        if (lp) lp[i * VE + e] = fmaf(beta, xa[e] - xb[e], xt[e]) - lse_s;
      }
    }
  }
  stats2_warp_reduce(r2);
  if (lane == 0) sh->warp2[warp] = r2;
  __syncthreads();
  if (warp == 0) {
    Stats2 w = {0.f, 0.f, 0.f, 0.f, 0.f};
    if (lane < kWarps) w = sh->warp2[lane];
    stats2_warp_reduce(w);
    if (lane == 0) sh->cta2 = w;
  }
  cluster.sync();  // #2: every CTA's pass-2 totals are in place
  if (warp == 0) {
    Stats2 w = {0.f, 0.f, 0.f, 0.f, 0.f};
    if (lane < C) w = *cluster.map_shared_rank(&sh->cta2, lane);
    // inclusive prefix of the inverse-CDF mass over ranks, in rank order
    const bool use_r = STOCH && (k < P.K);
    float mass = 0.f;
    float tot_R = w.R, tot_Q = w.Q;
    Stats2 tot = w;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      tot.j += __shfl_xor_sync(0xffffffffu, tot.j, off);
      tot.msum += __shfl_xor_sync(0xffffffffu, tot.msum, off);
      tot.kl += __shfl_xor_sync(0xffffffffu, tot.kl, off);
    }
    // sequential-in-rank totals of R and Q (every lane ends with the same)
    float incl_R = tot_R, incl_Q = tot_Q;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float vr = __shfl_up_sync(0xffffffffu, incl_R, off);
      const float vq = __shfl_up_sync(0xffffffffu, incl_Q, off);
      if (lane >= off) {
        incl_R += vr;
        incl_Q += vq;
      }
    }
    const float R_all = __shfl_sync(0xffffffffu, incl_R, 31);
    const float Q_all = __shfl_sync(0xffffffffu, incl_Q, 31);
    const bool r_ok = use_r && (R_all > 0.f);
    const float incl = r_ok ? incl_R : incl_Q;
    mass = r_ok ? tot_R : tot_Q;
    const float total = r_ok ? R_all : Q_all;
    float u = 0.f;
    if (STOCH) u = P.unif[static_cast<size_t>(bi) * K1 + P.K];
    const float tau = u * total;
    const unsigned over = __ballot_sync(0xffffffffu, lane < C && incl > tau);
    const unsigned pos = __ballot_sync(0xffffffffu, lane < C && mass > 0.f);
    int owner = -1;
    if (over) owner = __ffs(over) - 1;
    else if (pos) owner = 31 - __clz(pos);
    const float incl_owner = __shfl_sync(0xffffffffu, incl, owner < 0 ? 0 : owner);
    const float mass_owner = __shfl_sync(0xffffffffu, mass, owner < 0 ? 0 : owner);
    if (lane == 0) {
      float D = 0.f;
      if (do_jsd) D = 0.5f * kLn2 * (tot.j + tot.msum);
      else if (do_kl) D = kLn2 * tot.kl;
      sh->D = D;
      sh->mass_total = total;
      sh->use_r = r_ok ? 1 : 0;
      sh->owner = STOCH ? owner : -1;
      sh->tau_local = fmaxf(tau - (incl_owner - mass_owner), 0.f);
    }
  }
  __syncthreads();

  // ---- inverse-CDF walk in the CTA that owns the target (stochastic)
  if (STOCH && rank == sh->owner) {
    const bool use_r = sh->use_r != 0;
    const float tau = sh->tau_local;
    const int seg = (nv + kThreads - 1) / kThreads;
    const int v0 = tid * seg, v1 = min(nv, v0 + seg);
    float tsum = 0.f;
    int last_pos = -1;
    for (int i = v0; i < v1; ++i) {
      float xa[VE], xb[VE], xt[VE];
      load_vec(sa + i * VE, xa);
      load_vec(sb + i * VE, xb);
      load_vec(st + i * VE, xt);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const float mm = sample_mass(xa[e], xb[e], xt[e], beta, A2, S2, use_r);
        tsum += mm;
        if (mm > 0.f) last_pos = i * VE + e;
      }
    }
    // block-wide inclusive scan of the per-thread segment masses
    float incl = tsum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    if (lane == 31) sh->scan[warp] = incl;
    if (tid == 0) sh->found = -1;
    __syncthreads();
    float woff = 0.f;
    for (int w = 0; w < warp; ++w) woff += sh->scan[w];
    incl += woff;
    const float excl = incl - tsum;
    if (excl <= tau && tau < incl) {
      float cum = excl;
      int pick = -1;
      for (int i = v0; i < v1 && pick < 0; ++i) {
        float xa[VE], xb[VE], xt[VE];
        load_vec(sa + i * VE, xa);
        load_vec(sb + i * VE, xb);
        load_vec(st + i * VE, xt);
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float mm = sample_mass(xa[e], xb[e], xt[e], beta, A2, S2, use_r);
          cum += mm;
          if (pick < 0 && cum > tau) pick = i * VE + e;
        }
      }
      if (pick < 0) pick = last_pos;
      atomicMax(&sh->found, pick);
    }
    __syncthreads();
    const int found0 = sh->found;
    __syncthreads();
    if (found0 < 0) {
      // the target fell in the rounding gap at the end: last positive element
      if (last_pos >= 0) atomicMax(&sh->found, last_pos);
      __syncthreads();
    }
    if (tid == 0) {
      const int pick = sh->found >= 0 ? lo + sh->found : -1;
      *cluster.map_shared_rank(&sh->sample, 0) = pick;
    }
  }
  cluster.sync();  // #3: the sample is in rank 0; no CTA's shared memory is read after this

  // ---- epilogue: acceptance test, row record, ticket, scan
  if (!leader) return;
  const float lse_t = sh->lse[2];
  unsigned err = 0;
  if (!isfinite(lse_a) || !isfinite(lse_b) || !isfinite(lse_t)) err |= ASYMSPEC_DATA_NONFINITE;
  if ((STOCH || P.need_lse_s) && !isfinite(lse_s)) err |= ASYMSPEC_DATA_NONFINITE;
  float D = sh->D;
  if (!isfinite(D)) err |= ASYMSPEC_DATA_NONFINITE;
  if (P.divergence == ASYMSPEC_DIV_JSD) D = fminf(fmaxf(D, 0.f), kLn2);
  if (P.divergence == ASYMSPEC_DIV_KL) D = fmaxf(D, 0.f);
  if (sh->is == INT_MAX || sh->it == INT_MAX) err |= ASYMSPEC_DATA_NONFINITE;
  float u_last = 0.f;
  if (STOCH) {
    u_last = P.unif[static_cast<size_t>(bi) * K1 + P.K];
    if (!(u_last >= 0.f && u_last < 1.f)) err |= ASYMSPEC_DATA_BAD_UNIFORM;
  }
  int accept = 1;
  float margin = NAN;
  float gamma_eff = P.gamma;
  if (k < P.K) {
    if (dtok < 0 || dtok >= V) {
      err |= ASYMSPEC_DATA_BAD_TOKEN;
    } else {
      const float la_d = ad - lse_a, lb_d = bd - lse_b;
      if (P.divergence == ASYMSPEC_DIV_LAMBDA) D = P.lambda * (la_d - lb_d);
      const float ln_geff = P.ln_gamma - D;
      gamma_eff = expf(ln_geff);
      if (!STOCH) {
        const float lr = (td - lse_t) - lb_d;  // log(softmax(t)[d] / softmax(b)[d])
        accept = lr > ln_geff;                 // Eq. 4
        margin = 1.f - expf(lr - ln_geff);
      } else {
        const float pd = P.dprobs[static_cast<size_t>(bi) * P.K + k];
        const float u = P.unif[static_cast<size_t>(bi) * K1 + k];
        if (!(pd > 0.f && pd <= 1.f)) err |= ASYMSPEC_DATA_BAD_PROB;
        if (!(u >= 0.f && u < 1.f)) err |= ASYMSPEC_DATA_BAD_UNIFORM;
        const float sd = fmaf(beta, ad - bd, td);
        const float qd = expf(sd - lse_s);
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
  if (STOCH) cand = sh->sample;
  else cand = (k < P.K || P.fuse_bonus) ? sh->is : sh->it;
  if (cand < 0 || cand >= V) err |= ASYMSPEC_DATA_NONFINITE;

  if (P.row_stats) {
    float* rs = P.row_stats + static_cast<size_t>(row) * 8;
    rs[0] = lse_a;
    rs[1] = lse_b;
    rs[2] = lse_t;
    rs[3] = (STOCH || P.need_lse_s) ? lse_s : NAN;
    rs[4] = D;
    rs[5] = gamma_eff;
    rs[6] = margin;
    rs[7] = STOCH ? sh->mass_total : NAN;
  }
  if (P.row_tokens) {
    P.row_tokens[static_cast<size_t>(row) * 2] = sh->is;
    P.row_tokens[static_cast<size_t>(row) * 2 + 1] = cand;
  }
  if (err && P.err_word) atomicOr(P.err_word, err);
  P.recs[row] = make_int4(accept, cand, static_cast<int>(err), 0);
  __threadfence();
  const unsigned ticket = atomicAdd(&P.tickets[bi], 1u);
  if (ticket != static_cast<unsigned>(P.K)) return;

  // last row of batch element bi: Algorithm 1's sequential scan
  __threadfence();
  const int4* recs = P.recs + static_cast<size_t>(bi) * K1;
  int any_err = 0;
  for (int j = 0; j < K1; ++j) any_err |= __ldcg(&recs[j].z);
  int len = P.K;
  for (int j = 0; j < P.K; ++j) {
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

// ----------------------------------------------------------- host side

thread_local int g_last_cuda_error = 0;

int cuda_fail(cudaError_t e) {
  g_last_cuda_error = static_cast<int>(e);
  return ASYMSPEC_ERR_CUDA;
}

struct Plan {
  int C, W, VE, sh_off, smem;
  long long ctas;
  bool vector_path;
};

int elt_size(int dtype) { return dtype == ASYMSPEC_FP32 ? 4 : 2; }

int make_plan(int B, int K, int V, int dtype, const asymspec_launch_opts* opts, bool vec_ok,
              Plan* pl) {
  const int elt = elt_size(dtype);
  const int VE = vec_ok ? 16 / elt : 1;
  const int shared_bytes = static_cast<int>(sizeof(Shared));
  auto fill = [&](int C) {
    const long long per = (static_cast<long long>(V) + C - 1) / C;
    const long long W = ((per + VE - 1) / VE) * VE;
    const long long sh_off = ((3 * W * elt) + 15) / 16 * 16;
    pl->C = C;
    pl->W = static_cast<int>(W);
    pl->VE = VE;
    pl->sh_off = static_cast<int>(sh_off);
    pl->smem = static_cast<int>(sh_off + shared_bytes);
    pl->ctas = static_cast<long long>(B) * (K + 1) * C;
    pl->vector_path = vec_ok;
    return sh_off + shared_bytes <= kMaxSmem;
  };
  if (opts && opts->cluster_size > 0) {
    const int C = opts->cluster_size;
    if (C != 1 && C != 2 && C != 4 && C != 8 && C != 16) return ASYMSPEC_ERR_INVALID_ARG;
    if (!fill(C)) return ASYMSPEC_ERR_TOO_LARGE;
  } else {
    bool ok = false;
    for (int C = 1; C <= 16 && !ok; C *= 2) {
      ok = fill(C) && pl->sh_off <= kPreferredSliceBytes;
    }
    if (!ok) ok = fill(16);  // widest split when no slice fits the preferred size
    if (!ok) return ASYMSPEC_ERR_TOO_LARGE;
  }
  if (pl->ctas > INT_MAX) return ASYMSPEC_ERR_TOO_LARGE;
  return ASYMSPEC_OK;
}

using KernelFn = void (*)(KParams);

KernelFn pick_kernel(int dtype, bool vec, bool stoch) {
  if (dtype == ASYMSPEC_FP32) {
    if (vec) return stoch ? fuse_verify_kernel<float, 4, true> : fuse_verify_kernel<float, 4, false>;
    return stoch ? fuse_verify_kernel<float, 1, true> : fuse_verify_kernel<float, 1, false>;
  }
  if (vec)
    return stoch ? fuse_verify_kernel<__nv_bfloat16, 8, true>
                 : fuse_verify_kernel<__nv_bfloat16, 8, false>;
  return stoch ? fuse_verify_kernel<__nv_bfloat16, 1, true>
               : fuse_verify_kernel<__nv_bfloat16, 1, false>;
}

// cudaFuncSetAttribute once per (kernel, device), under a lock.
std::mutex g_attr_mu;
struct AttrEntry {
  const void* fn;
  int device;
};
AttrEntry g_attr_done[256];
int g_attr_count = 0;

cudaError_t prepare_kernel(KernelFn fn, int device) {
  std::lock_guard<std::mutex> lock(g_attr_mu);
  for (int i = 0; i < g_attr_count; ++i)
    if (g_attr_done[i].fn == reinterpret_cast<const void*>(fn) && g_attr_done[i].device == device)
      return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  if (g_attr_count < 256) g_attr_done[g_attr_count++] = {reinterpret_cast<const void*>(fn), device};
  return cudaSuccess;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

size_t ws_records_bytes(int B, int K) {
  return round_up(static_cast<size_t>(B) * (K + 1) * sizeof(int4), 256);
}

int check_params(const asymspec_gate_params* gp) {
  if (!(gp->gamma > 0.f && gp->gamma <= 1.f)) return ASYMSPEC_ERR_INVALID_ARG;
  if (!(std::isfinite(gp->beta) && gp->beta >= 0.f)) return ASYMSPEC_ERR_INVALID_ARG;
  if (gp->mode != ASYMSPEC_MODE_GREEDY && gp->mode != ASYMSPEC_MODE_STOCHASTIC)
    return ASYMSPEC_ERR_UNSUPPORTED;
  if (gp->divergence < ASYMSPEC_DIV_JSD || gp->divergence > ASYMSPEC_DIV_LAMBDA)
    return ASYMSPEC_ERR_UNSUPPORTED;
  if (gp->divergence == ASYMSPEC_DIV_LAMBDA && !std::isfinite(gp->lambda))
    return ASYMSPEC_ERR_INVALID_ARG;
  if (gp->flags != 0) return ASYMSPEC_ERR_INVALID_ARG;
  return ASYMSPEC_OK;
}

}  // namespace

extern "C" {

void asymspec_default_gate_params(asymspec_gate_params* p) {
  if (!p) return;
  p->gamma = 0.5f;
  p->beta = 1.0f;
  p->lambda = 0.1f;
  p->mode = ASYMSPEC_MODE_GREEDY;
  p->divergence = ASYMSPEC_DIV_JSD;
  p->fuse_bonus = 0;
  p->flags = 0;
}

size_t asymspec_workspace_bytes(int B, int K, int V) {
  (void)V;
  if (B < 1 || K < 1) return 0;
  return ws_records_bytes(B, K) + round_up(static_cast<size_t>(B) * sizeof(unsigned), 256);
}

int asymspec_workspace_reset(void* workspace, size_t workspace_bytes, void* stream) {
  if (!workspace) return ASYMSPEC_ERR_INVALID_ARG;
  const cudaError_t e =
      cudaMemsetAsync(workspace, 0, workspace_bytes, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ASYMSPEC_OK : cuda_fail(e);
}

int asymspec_plan(int B, int K, int V, int dtype, const asymspec_gate_params* gate_params,
                  const asymspec_launch_opts* opts, asymspec_launch_info* out) {
  if (!out || B < 1 || K < 1 || V < 2) return ASYMSPEC_ERR_INVALID_ARG;
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return ASYMSPEC_ERR_UNSUPPORTED;
  if (opts && opts->block_threads != 0 && opts->block_threads != kThreads)
    return ASYMSPEC_ERR_INVALID_ARG;
  asymspec_gate_params gp;
  asymspec_default_gate_params(&gp);
  if (gate_params) gp = *gate_params;
  int st = check_params(&gp);
  if (st) return st;
  const bool vec_ok = (static_cast<long long>(V) * elt_size(dtype)) % 16 == 0;
  Plan pl;
  st = make_plan(B, K, V, dtype, opts, vec_ok, &pl);
  if (st) return st;
  out->cluster_size = pl.C;
  out->block_threads = kThreads;
  out->slice_elems = pl.W;
  out->smem_bytes = pl.smem;
  out->ctas = pl.ctas;
  out->vector_path = vec_ok ? 1 : 0;
  out->max_active_clusters = 0;
  int device = 0;
  if (cudaGetDevice(&device) == cudaSuccess) {
    KernelFn fn = pick_kernel(dtype, vec_ok, gp.mode == ASYMSPEC_MODE_STOCHASTIC);
    if (prepare_kernel(fn, device) == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = pl.C;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(static_cast<unsigned>(pl.ctas));
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = pl.smem;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int nclusters = 0;
      if (cudaOccupancyMaxActiveClusters(&nclusters, fn, &cfg) == cudaSuccess)
        out->max_active_clusters = nclusters;
    }
    cudaGetLastError();
  } else {
    cudaGetLastError();
  }
  return ASYMSPEC_OK;
}

int asymspec_fuse_verify_ex(const void* logits_full, const void* logits_comp,
                            const void* logits_ver, const int32_t* draft_tokens,
                            const float* draft_probs, const float* uniforms, int B, int K,
                            int V, int dtype, const asymspec_gate_params* gate_params,
                            int32_t* out_accept_len, int32_t* out_next_token,
                            void* workspace, size_t workspace_bytes, float* out_row_stats,
                            int32_t* out_row_tokens, float* out_fused_logprobs,
                            uint32_t* out_error_word, const asymspec_launch_opts* opts,
                            void* stream) {
  if (B < 1 || K < 1 || V < 2) return ASYMSPEC_ERR_INVALID_ARG;
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return ASYMSPEC_ERR_UNSUPPORTED;
  asymspec_gate_params gp;
  asymspec_default_gate_params(&gp);
  if (gate_params) gp = *gate_params;
  int st = check_params(&gp);
  if (st) return st;
  const bool stoch = gp.mode == ASYMSPEC_MODE_STOCHASTIC;
  if (!logits_full || !logits_comp || !logits_ver || !draft_tokens || !out_accept_len ||
      !out_next_token)
    return ASYMSPEC_ERR_INVALID_ARG;
  if (stoch && (!draft_probs || !uniforms)) return ASYMSPEC_ERR_INVALID_ARG;
  if (opts && opts->block_threads != 0 && opts->block_threads != kThreads)
    return ASYMSPEC_ERR_INVALID_ARG;
  const int elt = elt_size(dtype);
  if (!aligned(logits_full, elt) || !aligned(logits_comp, elt) || !aligned(logits_ver, elt) ||
      !aligned(draft_tokens, 4) || !aligned(out_accept_len, 4) || !aligned(out_next_token, 4) ||
      (draft_probs && !aligned(draft_probs, 4)) || (uniforms && !aligned(uniforms, 4)) ||
      (out_row_stats && !aligned(out_row_stats, 4)) ||
      (out_row_tokens && !aligned(out_row_tokens, 4)) ||
      (out_fused_logprobs && !aligned(out_fused_logprobs, 4)) ||
      (out_error_word && !aligned(out_error_word, 4)))
    return ASYMSPEC_ERR_MISALIGNED;
  if (!workspace || workspace_bytes < asymspec_workspace_bytes(B, K, V) ||
      !aligned(workspace, 16))
    return ASYMSPEC_ERR_WORKSPACE;
  const bool vec_ok = (static_cast<long long>(V) * elt) % 16 == 0 && aligned(logits_full, 16) &&
                      aligned(logits_comp, 16) && aligned(logits_ver, 16);
  Plan pl;
  st = make_plan(B, K, V, dtype, opts, vec_ok, &pl);
  if (st) return st;

  KParams P;
  P.a = logits_full;
  P.b = logits_comp;
  P.t = logits_ver;
  P.tokens = draft_tokens;
  P.dprobs = draft_probs;
  P.unif = uniforms;
  P.B = B;
  P.K = K;
  P.V = V;
  P.C = pl.C;
  P.W = pl.W;
  P.sh_off = pl.sh_off;
  P.gamma = gp.gamma;
  P.beta = gp.beta;
  P.lambda = gp.lambda;
  P.ln_gamma = logf(gp.gamma);
  P.divergence = gp.divergence;
  P.fuse_bonus = gp.fuse_bonus ? 1 : 0;
  P.need_lse_s = (stoch || out_fused_logprobs || out_row_stats) ? 1 : 0;
  P.need_pass2 = (stoch || out_fused_logprobs || gp.divergence == ASYMSPEC_DIV_JSD ||
                  gp.divergence == ASYMSPEC_DIV_KL)
                     ? 1
                     : 0;
  P.out_len = out_accept_len;
  P.out_next = out_next_token;
  P.row_stats = out_row_stats;
  P.row_tokens = out_row_tokens;
  P.logprobs = out_fused_logprobs;
  P.err_word = out_error_word;
  P.recs = static_cast<int4*>(workspace);
  P.tickets = reinterpret_cast<unsigned int*>(static_cast<char*>(workspace) +
                                              ws_records_bytes(B, K));

  int device = 0;
  cudaError_t e = cudaGetDevice(&device);
  if (e != cudaSuccess) return cuda_fail(e);
  KernelFn fn = pick_kernel(dtype, vec_ok, stoch);
  e = prepare_kernel(fn, device);
  if (e != cudaSuccess) return cuda_fail(e);

  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(pl.ctas));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = pl.smem;
  cfg.stream = static_cast<cudaStream_t>(stream);
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, fn, P);
  if (e != cudaSuccess) return cuda_fail(e);
  return ASYMSPEC_OK;
}

int asymspec_fuse_verify(const void* logits_full, const void* logits_comp,
                         const void* logits_ver, const int32_t* draft_tokens,
                         const float* draft_probs, const float* uniforms, int B, int K,
                         int V, int dtype, const asymspec_gate_params* gate_params,
                         int32_t* out_accept_len, int32_t* out_next_token, void* stream) {
  if (B < 1 || K < 1 || V < 2) return ASYMSPEC_ERR_INVALID_ARG;
  const size_t bytes = asymspec_workspace_bytes(B, K, V);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void* ws = nullptr;
  cudaError_t e = cudaMallocAsync(&ws, bytes, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaMemsetAsync(ws, 0, bytes, s);
  if (e != cudaSuccess) {
    cudaFreeAsync(ws, s);
    return cuda_fail(e);
  }
  const int st = asymspec_fuse_verify_ex(logits_full, logits_comp, logits_ver, draft_tokens,
                                         draft_probs, uniforms, B, K, V, dtype, gate_params,
                                         out_accept_len, out_next_token, ws, bytes, nullptr,
                                         nullptr, nullptr, nullptr, nullptr, stream);
  e = cudaFreeAsync(ws, s);
  if (st != ASYMSPEC_OK) return st;
  if (e != cudaSuccess) return cuda_fail(e);
  return ASYMSPEC_OK;
}

const char* asymspec_status_string(int status) {
  switch (status) {
    case ASYMSPEC_OK: return "ok";
    case ASYMSPEC_ERR_INVALID_ARG: return "invalid argument";
    case ASYMSPEC_ERR_UNSUPPORTED: return "unsupported dtype, mode or divergence";
    case ASYMSPEC_ERR_MISALIGNED: return "pointer not aligned to its element size";
    case ASYMSPEC_ERR_WORKSPACE: return "workspace missing or too small";
    case ASYMSPEC_ERR_CUDA: return "CUDA error (see asymspec_last_cuda_error)";
    case ASYMSPEC_ERR_TOO_LARGE: return "problem too large for the on-chip row slices";
    default: return "unknown status";
  }
}

int asymspec_last_cuda_error(void) { return g_last_cuda_error; }

int asymspec_version(void) { return 100; }

}  // extern "C"
