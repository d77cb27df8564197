// Fast fuse-and-verify kernel for 16-byte aligned rows.
//
// One cluster of C CTAs per row triple (one launch of the cluster per row;
// the hardware hands out rows as clusters finish).  CTA r owns vocabulary
// entries [r W, (r+1) W) of the row and brings its slice of a, b and t into
// shared memory with 1-D bulk copies (cp.async.bulk), split into kChunks
// chunks that each complete on their own mbarrier, so pass 1 starts on the
// first chunk while the rest are still arriving.  The slice is then worked
// on chip only: each logit row is read from HBM once.
//
// Per row the work depends on what the mode needs:
//   greedy, draft rows   pass 1: LSE(a), LSE(b), LSE(t), argmax s
//                        pass 2: JSD (or KL) terms                 (Eqs. 2-4)
//   greedy, bonus row    pass 1: argmax t only (a, b not even copied), or
//                        argmax s with fuse_bonus                  (Algorithm 1)
//   stochastic, drafts   pass 1: LSE(a), LSE(b), LSE(s)
//                        pass 2: JSD terms, residual and fused masses
//   stochastic, bonus    pass 1: LSE(s); pass 2: fused masses
// Debug outputs (row statistics, fused log-probs) switch every row to the
// full program.  Two fp32 values travel per add/sub/mul/fma instruction
// (f32x2); exponentials and logarithms use ex2.approx / lg2.approx.
//
// Reductions: per stream, the maximum first (warp shuffles), then each lane
// rescales its own sum once and the sums are added; warp -> CTA in shared
// memory.  Each CTA then pushes its record into every peer's shared memory
// (DSMEM stores) before a cluster barrier, so after the barrier every CTA
// combines local copies, identically, and holds bit-identical row values;
// nothing is read remotely after a barrier, so CTAs may leave as soon as
// they are done.  Two barriers per row (one when no pass 2 is needed); the
// stochastic draw reaches rank 0 through a remote mbarrier arrive.  The draft
// token's three logits come from the shared memory of the CTA whose slice
// holds it.
//
// Every wait is bounded: a chunk that does not land within 200 ms marks the
// row with ASYMSPEC_DATA_TIMEOUT; the CTA still reaches every cluster
// barrier, so no CTA of the cluster is left waiting, and before it exits it
// waits (bounded again) for any copy still in flight.
#pragma once

#include "device_common.cuh"

namespace asymspec_impl {

constexpr int kTThreads = 256;
constexpr int kTWarps = kTThreads / 32;
constexpr int kMaxRounds = 10;  // 16-byte vectors per thread per slice
constexpr int kChunks = 4;      // bulk-copy chunks per slice
constexpr unsigned long long kCopyTimeoutNs = 200ull * 1000ull * 1000ull;

enum : unsigned { F_LA = 1, F_LB = 2, F_LT = 4, F_LS = 8, F_AS = 16, F_AT = 32 };
enum : unsigned { G_JSD = 1, G_KL = 2, G_RES = 4, G_QF = 8 };

struct __align__(16) X1 {  // pass-1 result (per thread, per warp, per CTA, per row)
  float m[4];
  float s[4];
  float vs;
  int is;
  float vt;
  int it;
  unsigned bad;
  float da, db, dt;  // a, b, t at the draft token (set by the CTA that holds it)
};

struct __align__(16) X2 {  // pass-2 sums
  float j, msum, kl, R, Q;
  float pad[3];
};

// Fixed part of the shared state; the C pass-1 and C pass-2 records pushed
// by the cluster follow it (recv1(), recv2()).
struct __align__(16) SharedTma {
  unsigned long long bar[kChunks];   // one mbarrier per chunk
  unsigned long long sample_bar;     // rank 0: the draw has arrived
  union {                            // per-warp scratch, one use at a time
    X1 w1[kTWarps];
    X2 w2[kTWarps];
    float wr[kMaxRounds][kTWarps];
  };
  float lse[4];
  int is, it;
  unsigned bad;
  float da, db, dt;
  float D, mass_total, tau_local;
  int owner, use_r;
  int sample;  // rank 0: written by the CTA that owns the draw
  int found, jstar;
  float tau_j;
  float scan[kTWarps];
  unsigned broken;
  __device__ X1* recv1() { return reinterpret_cast<X1*>(this + 1); }
  __device__ X2* recv2(int C) { return reinterpret_cast<X2*>(recv1() + C); }
};

// The pushed records are copied with 16-byte stores.
static_assert(sizeof(X1) % 16 == 0 && alignof(X1) == 16, "X1 must be 16-byte aligned");
static_assert(sizeof(X2) % 16 == 0 && alignof(X2) == 16, "X2 must be 16-byte aligned");
static_assert(sizeof(SharedTma) % 16 == 0, "records after SharedTma must stay 16-byte aligned");

// Shared bytes after the slices for a cluster of C CTAs (the stochastic
// kernel adds rounds * kTThreads floats of per-vector masses).
__host__ __device__ constexpr int shared_tma_bytes(int C) {
  return static_cast<int>(sizeof(SharedTma) + C * (sizeof(X1) + sizeof(X2)));
}
__host__ __device__ constexpr int mass_bytes(int rounds) {
  return rounds * kTThreads * static_cast<int>(sizeof(float));
}

__device__ __forceinline__ X1 x1_neutral() {
  X1 r;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    r.m[q] = -INFINITY;
    r.s[q] = 0.f;
  }
  r.vs = -INFINITY;
  r.is = INT_MAX;
  r.vt = -INFINITY;
  r.it = INT_MAX;
  r.bad = 0;
  r.da = r.db = r.dt = 0.f;
  return r;
}

__device__ __forceinline__ X2 x2_zero() {
  X2 r;
  r.j = r.msum = r.kl = r.R = r.Q = 0.f;
  r.pad[0] = r.pad[1] = r.pad[2] = 0.f;
  return r;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, v, off);
    const int i2 = __shfl_xor_sync(0xffffffffu, i, off);
    if (v2 > v || (v2 == v && i2 < i)) {
      v = v2;
      i = i2;
    }
  }
}

// Warp-wide combine of the streams a program computes: the maximum first,
// then every lane rescales its own sum to it and the sums are added.  Every
// lane ends with the same (bit-identical) result.
template <unsigned F>
__device__ __forceinline__ void warp_reduce_x1(X1& e) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
    if (F & bit) {
      const float M = warp_max(e.m[q]);
      const float s = (e.m[q] == M) ? e.s[q] : e.s[q] * ex2((e.m[q] - M) * kLog2e);
      e.m[q] = M;
      e.s[q] = warp_sum(s);
    }
  }
  if (F & F_AS) warp_argmax(e.vs, e.is);
  if (F & F_AT) warp_argmax(e.vt, e.it);
  e.bad = __reduce_or_sync(0xffffffffu, e.bad);
}

// Cluster barrier.  Only the warp that pushed records needs release
// ordering; the others arrive relaxed.  Everyone waits with acquire.
__device__ __forceinline__ void cluster_barrier(bool released) {
  if (released)
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  else
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The record of this CTA goes into slot `rank` of every CTA of the cluster
// (lane r of warp 0 writes to CTA r); a cluster barrier must follow.
template <typename R>
__device__ __forceinline__ void push_record(const R& rec, R* slots, int rank, int C,
                                            cg::cluster_group& cluster) {
  const int lane = threadIdx.x & 31;
  if (lane < C) {
    R* dst = cluster.map_shared_rank(slots, lane) + rank;
    const float4* src = reinterpret_cast<const float4*>(&rec);
    float4* d = reinterpret_cast<float4*>(dst);
#pragma unroll
    for (int w = 0; w < static_cast<int>(sizeof(R) / 16); ++w) d[w] = src[w];
  }
}

template <unsigned G>
__device__ __forceinline__ void warp_reduce_x2(X2& x) {
  if (G & G_JSD) {
    x.j = warp_sum(x.j);
    x.msum = warp_sum(x.msum);
  }
  if (G & G_KL) x.kl = warp_sum(x.kl);
  if (G & G_RES) x.R = warp_sum(x.R);
  if (G & (G_RES | G_QF)) x.Q = warp_sum(x.Q);
}

// Maximum of the 2*NP values of a vector (NaN ignored / NaN propagated).
template <int NP>
__device__ __forceinline__ float vmax_pairs(const f2 (&x)[NP]) {
  float v[2 * NP];
#pragma unroll
  for (int h = 0; h < NP; ++h) upk(x[h], v[2 * h], v[2 * h + 1]);
  if constexpr (NP == 4) {
    const float m1 = max3(v[0], v[1], v[2]);
    const float m2 = max3(v[3], v[4], v[5]);
    return fmaxf(max3(m1, m2, v[6]), v[7]);
  } else {
    return fmaxf(max3(v[0], v[1], v[2]), v[3]);
  }
}
template <int NP>
__device__ __forceinline__ float vmax_pairs_nan(const f2 (&x)[NP]) {
  float m = lo_of(x[0]);
  m = max_nan(m, hi_of(x[0]));
#pragma unroll
  for (int h = 1; h < NP; ++h) m = max_nan(max_nan(m, lo_of(x[h])), hi_of(x[h]));
  return m;
}

// Argmax tracking per vector, branch-free: the best vector maximum so far
// and the index of its vector (a strict improvement wins, so the earliest
// vector keeps a tie); a non-finite maximum is flagged.  The element inside
// the best vector is resolved once at the end of the pass (arg_resolve).
__device__ __forceinline__ void arg_track(float& v, int& vec, float c, int i, unsigned& bad,
                                          unsigned bit) {
  if (!(c <= 3.402823466e38f)) bad |= bit;
  const bool better = c > v;
  v = better ? c : v;
  vec = better ? i : vec;
}

// Lowest index inside vector `vec` whose value equals v (INT_MAX if none).
template <int NP>
__device__ __forceinline__ int arg_in_vector(const f2 (&x)[NP], float v, int base) {
  int idx = INT_MAX;
#pragma unroll
  for (int h = NP - 1; h >= 0; --h) {
    float lo, hi;
    upk(x[h], lo, hi);
    if (hi == v) idx = base + 2 * h + 1;
    if (lo == v) idx = base + 2 * h;
  }
  return idx;
}

// Residual max(0, q - p) and fused q masses of one vector (stochastic mode);
// pass 2 and the inverse-CDF walk share this, so they see identical values.
template <int NP>
__device__ __forceinline__ void vec_masses(const f2 (&xa)[NP], const f2 (&xb)[NP],
                                           const f2 (&xt)[NP], f2 beta2, f2 L2, f2 nA2, f2 nS2,
                                           f2 (&p)[NP], f2 (&qf)[NP], f2 (&r)[NP]) {
#pragma unroll
  for (int h = 0; h < NP; ++h) {
    p[h] = ex2_2(fma2(xa[h], L2, nA2));
    const f2 s = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
    qf[h] = ex2_2(fma2(s, L2, nS2));
    r[h] = relu2(sub2(qf[h], p[h]));
  }
}

template <int NP>
__device__ __forceinline__ float vsum(const f2 (&x)[NP]) {
  if constexpr (NP == 4) return hsum2(add2(add2(x[0], x[1]), add2(x[2], x[3])));
  else return hsum2(add2(x[0], x[1]));
}

// ---------------------------------------------------------------- pass 1

// Running (max m, packed sum of 2^((x - m) log2 e)) over two vectors of
// pairs (one rescale check per 2 VE entries); returns their maximum.
template <int NP>
__device__ __forceinline__ float online_pairs2(float& m, f2& acc, const f2 (&x)[NP],
                                               const f2 (&y)[NP], f2 L2) {
  const float cm = fmaxf(vmax_pairs(x), vmax_pairs(y));
  if (cm > m) {
    const float f = ex2((m - cm) * kLog2e);
    acc = mul2(acc, pk(f, f));
    m = cm;
  }
  const float nm = -m * kLog2e;
  const f2 nm2 = pk(nm, nm);
  f2 e[NP];
#pragma unroll
  for (int h = 0; h < NP; ++h)
    e[h] = add2(ex2_2(fma2(x[h], L2, nm2)), ex2_2(fma2(y[h], L2, nm2)));
  if constexpr (NP == 4) {
    acc = add2(acc, add2(add2(e[0], e[1]), add2(e[2], e[3])));
  } else {
    acc = add2(acc, add2(e[0], e[1]));
  }
  return cm;
}

template <typename T, int NP>
__device__ __forceinline__ void load_or_fill(const T* p, bool ok, f2 (&x)[NP]) {
  if (ok) {
    load_pairs(p, x);
  } else {
#pragma unroll
    for (int h = 0; h < NP; ++h) x[h] = pk(-1e30f, -1e30f);  // contributes nothing
  }
}

// Vector i of the slice lives in round i / NT; chunk c holds rounds
// [c rc, (c+1) rc).  Every thread waits for a chunk before its first round.
// Rounds are taken two at a time.
template <typename T, unsigned F>
__device__ __forceinline__ void pass1(const T* ra, const T* rb, const T* rt, int nv, int rounds,
                                      int rc, int lo, float beta, SharedTma* sh, X1& e) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needA = (F & (F_LA | F_LS | F_AS)) != 0;
  constexpr bool needB = (F & (F_LB | F_LS | F_AS)) != 0;
  constexpr bool needT = (F & (F_LT | F_LS | F_AS | F_AT)) != 0;
  constexpr bool needS = (F & (F_LS | F_AS)) != 0;
  constexpr int STEP = 2 * kTThreads * VE;  // elements per two rounds
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  f2 acc[4] = {0ull, 0ull, 0ull, 0ull};
  int vec_s = -1, vec_t = -1;  // vectors holding the best s and t so far
  const int tid = static_cast<int>(threadIdx.x);
  for (int c = 0, r0 = 0; c < kChunks && r0 < rounds; ++c, r0 += rc) {
    if (!sh->broken && !mbar_wait_bounded(&sh->bar[c], 0, kCopyTimeoutNs))
      atomicOr(&sh->broken, kBadTimeout);
    const int r1 = min(rounds, r0 + rc);
    int i0 = r0 * kTThreads + tid;          // vector index of this thread's first vector
    int e0 = i0 * VE;                       // its element offset in the slice
    for (int kr = r0; kr < r1; kr += 2, i0 += 2 * kTThreads, e0 += STEP) {
      if (i0 >= nv) break;
      const bool has1 = (kr + 1 < r1) && (i0 + kTThreads < nv);
      const int e1 = e0 + kTThreads * VE;
      f2 xa[NP], xb[NP], xt[NP], xs[NP], ya[NP], yb[NP], yt[NP], ys[NP];
      if (needA) {
        load_pairs(ra + e0, xa);
        load_or_fill(ra + e1, has1, ya);
      }
      if (needB) {
        load_pairs(rb + e0, xb);
        load_or_fill(rb + e1, has1, yb);
      }
      if (needT) {
        load_pairs(rt + e0, xt);
        load_or_fill(rt + e1, has1, yt);
      }
      if (needS) {
#pragma unroll
        for (int h = 0; h < NP; ++h) {
          xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
          ys[h] = fma2(beta2, sub2(ya[h], yb[h]), yt[h]);
        }
      }
      if (F & F_LA) online_pairs2(e.m[0], acc[0], xa, ya, L2);
      if (F & F_LB) online_pairs2(e.m[1], acc[1], xb, yb, L2);
      float ct0 = 0.f, ct1 = 0.f, cs0 = 0.f, cs1 = 0.f;
      if (F & F_LT) {
        online_pairs2(e.m[2], acc[2], xt, yt, L2);
        if (F & F_AT) {
          ct0 = vmax_pairs(xt);
          ct1 = vmax_pairs(yt);
        }
      } else if (F & F_AT) {
        ct0 = vmax_pairs_nan(xt);
        ct1 = vmax_pairs_nan(yt);
      }
      if (F & F_LS) {
        online_pairs2(e.m[3], acc[3], xs, ys, L2);
        if (F & F_AS) {
          cs0 = vmax_pairs(xs);
          cs1 = vmax_pairs(ys);
        }
      } else if (F & F_AS) {
        cs0 = vmax_pairs_nan(xs);
        cs1 = vmax_pairs_nan(ys);
      }
      if (F & F_AS) {
        arg_track(e.vs, vec_s, cs0, i0, e.bad, kBadS);
        if (has1) arg_track(e.vs, vec_s, cs1, i0 + kTThreads, e.bad, kBadS);
      }
      if (F & F_AT) {
        arg_track(e.vt, vec_t, ct0, i0, e.bad, kBadT);
        if (has1) arg_track(e.vt, vec_t, ct1, i0 + kTThreads, e.bad, kBadT);
      }
    }
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) e.s[q] = hsum2(acc[q]);
  // the element of the best vector (re-read once from shared memory)
  if ((F & F_AS) && vec_s >= 0) {
    f2 xa[NP], xb[NP], xt[NP], xs[NP];
    load_pairs(ra + vec_s * VE, xa);
    load_pairs(rb + vec_s * VE, xb);
    load_pairs(rt + vec_s * VE, xt);
#pragma unroll
    for (int h = 0; h < NP; ++h) xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
    e.is = arg_in_vector(xs, e.vs, lo + vec_s * VE);
  }
  if ((F & F_AT) && vec_t >= 0) {
    f2 xt[NP];
    load_pairs(rt + vec_t * VE, xt);
    e.it = arg_in_vector(xt, e.vt, lo + vec_t * VE);
  }
}

// Pass 1, block combine, push to the cluster, barrier, local combine; leaves
// the row values in sh.  dtok: the row's draft token (-1 if none).
template <typename T, unsigned F>
__device__ __forceinline__ void pass1_and_combine(const T* ra, const T* rb, const T* rt, int nv,
                                                  int rounds, int rc, int lo, int n, int W,
                                                  float beta, int dtok, SharedTma* sh, int rank,
                                                  int C, cg::cluster_group& cluster) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  X1 e = x1_neutral();
  pass1<T, F>(ra, rb, rt, nv, rounds, rc, lo, beta, sh, e);
  warp_reduce_x1<F>(e);
  if (lane == 0) sh->w1[warp] = e;
  __syncthreads();
  if (warp == 0) {
    X1 w = (lane < kTWarps) ? sh->w1[lane] : x1_neutral();
    warp_reduce_x1<F>(w);
    w.bad |= sh->broken;
    if (dtok >= lo && dtok < lo + n) {  // this CTA's slice holds the draft token
      w.da = to_f32(ra[dtok - lo]);
      w.db = to_f32(rb[dtok - lo]);
      w.dt = to_f32(rt[dtok - lo]);
    }
    push_record(w, sh->recv1(), rank, C, cluster);
  }
  cluster_barrier(warp == 0);  // B1: every CTA's pass-1 record is in every CTA
  if (warp == 0) {
    X1 w = (lane < C) ? sh->recv1()[lane] : x1_neutral();
    warp_reduce_x1<F>(w);
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < 4; ++q) sh->lse[q] = w.m[q] + logf(w.s[q]);
      sh->is = w.is;
      sh->it = w.it;
      sh->bad = w.bad;
      if (dtok >= 0 && W > 0) {
        const X1& o = sh->recv1()[dtok / W < C ? dtok / W : 0];
        sh->da = o.da;
        sh->db = o.db;
        sh->dt = o.dt;
      }
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------- pass 2

// Divergence terms of one vector (Eq. 3): JSD terms p (log2 p - log2 m) and
// q (log2 q - log2 m) with m = p + q, their mass m, or KL terms.
template <int NP, bool JSD, bool KL>
__device__ __forceinline__ void div_terms(const f2 (&xa)[NP], const f2 (&xb)[NP], const f2 (&p)[NP],
                                          f2 L2, f2 nA2, f2 nB2, f2 tiny2, f2& ja, f2& jb,
                                          f2& ms2, f2& kl2) {
#pragma unroll
  for (int h = 0; h < NP; ++h) {
    const f2 la2 = fma2(xa[h], L2, nA2);
    const f2 lb2 = fma2(xb[h], L2, nB2);
    if (JSD) {
      const f2 q = ex2_2(lb2);
      const f2 m = add2(add2(p[h], q), tiny2);
      const f2 lg = lg2_2(m);
      ja = fma2(p[h], sub2(la2, lg), ja);
      jb = fma2(q, sub2(lb2, lg), jb);
      ms2 = add2(ms2, m);
    }
    if (KL) kl2 = fma2(p[h], sub2(la2, lb2), kl2);
  }
}

// Pass 2 over the slice, two vectors per step (an absent second vector is
// filled with -1e30, which contributes nothing).
template <typename T, unsigned G, bool LP>
__device__ __forceinline__ void pass2(const T* ra, const T* rb, const T* rt, int nv, int rounds,
                                      float beta, float A2, float B2, float S2, float lse_s, X2& x,
                                      float* lp, float* vmass) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool JSD = (G & G_JSD) != 0, KL = (G & G_KL) != 0, RES = (G & G_RES) != 0;
  constexpr bool QF = (G & G_QF) != 0;
  constexpr bool needT = RES || QF || LP;
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  const f2 nA2 = pk(-A2, -A2), nB2 = pk(-B2, -B2), nS2 = pk(-S2, -S2);
  const f2 tiny2 = pk(kMinNormal, kMinNormal);
  const f2 nl2 = pk(-lse_s, -lse_s);
  f2 ja = 0ull, jb = 0ull, ms2 = 0ull, kl2 = 0ull, R2 = 0ull, Q2 = 0ull;
  for (int kr = 0; kr < rounds; kr += 2) {
    const int i0 = kr * kTThreads + static_cast<int>(threadIdx.x);
    const int i1 = i0 + kTThreads;
    if (i0 >= nv) {
      if (RES || QF) {
        vmass[kr * kTThreads + threadIdx.x] = 0.f;
        if (kr + 1 < rounds) vmass[(kr + 1) * kTThreads + threadIdx.x] = 0.f;
      }
      continue;
    }
    const bool has1 = i1 < nv;
    f2 xa[NP], xb[NP], xt[NP], ya[NP], yb[NP], yt[NP];
    load_pairs(ra + i0 * VE, xa);
    load_pairs(rb + i0 * VE, xb);
    load_or_fill(ra + i1 * VE, has1, ya);
    load_or_fill(rb + i1 * VE, has1, yb);
    if (needT) {
      load_pairs(rt + i0 * VE, xt);
      load_or_fill(rt + i1 * VE, has1, yt);
    }
    f2 px[NP], py[NP];
    if (RES) {
      f2 qx[NP], qy[NP], rx[NP], ry[NP];
      vec_masses(xa, xb, xt, beta2, L2, nA2, nS2, px, qx, rx);
      vec_masses(ya, yb, yt, beta2, L2, nA2, nS2, py, qy, ry);
#pragma unroll
      for (int h = 0; h < NP; ++h) Q2 = add2(Q2, add2(qx[h], qy[h]));
      // residual mass of each vector, kept for the inverse-CDF walk
      const float r0 = vsum(rx), r1 = vsum(ry);
      R2 = add2(R2, pk(r0, r1));
      vmass[kr * kTThreads + threadIdx.x] = r0;
      if (kr + 1 < rounds) vmass[(kr + 1) * kTThreads + threadIdx.x] = r1;
    } else if (QF) {
      f2 qx[NP], qy[NP];
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        qx[h] = ex2_2(fma2(fma2(beta2, sub2(xa[h], xb[h]), xt[h]), L2, nS2));
        qy[h] = ex2_2(fma2(fma2(beta2, sub2(ya[h], yb[h]), yt[h]), L2, nS2));
      }
      // fused mass of each vector, kept for the inverse-CDF walk
      const float q0 = vsum(qx), q1 = vsum(qy);
      Q2 = add2(Q2, pk(q0, q1));
      vmass[kr * kTThreads + threadIdx.x] = q0;
      if (kr + 1 < rounds) vmass[(kr + 1) * kTThreads + threadIdx.x] = q1;
    } else if (JSD || KL) {
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        px[h] = ex2_2(fma2(xa[h], L2, nA2));
        py[h] = ex2_2(fma2(ya[h], L2, nA2));
      }
    }
    if (JSD || KL) {
      div_terms<NP, JSD, KL>(xa, xb, px, L2, nA2, nB2, tiny2, ja, jb, ms2, kl2);
      div_terms<NP, JSD, KL>(ya, yb, py, L2, nA2, nB2, tiny2, ja, jb, ms2, kl2);
    }
    if (LP) {
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        float l0, l1;
        upk(add2(fma2(beta2, sub2(xa[h], xb[h]), xt[h]), nl2), l0, l1);
        lp[i0 * VE + 2 * h] = l0;
        lp[i0 * VE + 2 * h + 1] = l1;
        if (has1) {
          upk(add2(fma2(beta2, sub2(ya[h], yb[h]), yt[h]), nl2), l0, l1);
          lp[i1 * VE + 2 * h] = l0;
          lp[i1 * VE + 2 * h + 1] = l1;
        }
      }
    }
  }
  x.j = hsum2(add2(ja, jb));
  x.msum = hsum2(ms2);
  x.kl = hsum2(kl2);
  x.R = hsum2(R2);
  x.Q = hsum2(Q2);
}

// Pass 2, block combine, push to the cluster, barrier, local combine:
// divergence, inverse-CDF mass and the CTA that owns the draw.
template <typename T, unsigned G, bool LP, bool STOCH>
__device__ __forceinline__ void pass2_and_combine(const T* ra, const T* rb, const T* rt, int nv,
                                                  int rounds, float beta, float* lp,
                                                  SharedTma* sh, int rank, int C, bool r_allowed,
                                                  float u_last, float* vmass,
                                                  cg::cluster_group& cluster) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float lse_a = sh->lse[0], lse_b = sh->lse[1], lse_s = sh->lse[3];
  X2 x = x2_zero();
  pass2<T, G, LP>(ra, rb, rt, nv, rounds, beta, lse_a * kLog2e, lse_b * kLog2e, lse_s * kLog2e,
                  lse_s, x, lp, vmass);
  warp_reduce_x2<G>(x);
  if (lane == 0) sh->w2[warp] = x;
  __syncthreads();
  if (warp == 0) {
    X2 w = (lane < kTWarps) ? sh->w2[lane] : x2_zero();
    warp_reduce_x2<G>(w);
    push_record(w, sh->recv2(C), rank, C, cluster);
  }
  cluster_barrier(warp == 0);  // B2: every CTA's pass-2 record is in every CTA
  if (warp == 0) {
    const X2 w = (lane < C) ? sh->recv2(C)[lane] : x2_zero();
    X2 tot = w;
    warp_reduce_x2<G>(tot);
    float D = 0.f;
    if (G & G_JSD) D = 0.5f * kLn2 * (tot.j + tot.msum);
    else if (G & G_KL) D = kLn2 * tot.kl;
    if (STOCH) {
      // inclusive prefix of the inverse-CDF mass over ranks, in rank order
      float incl_R = w.R, incl_Q = w.Q;
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
      const bool r_ok = r_allowed && (R_all > 0.f);
      const float incl = r_ok ? incl_R : incl_Q;
      const float mass = r_ok ? w.R : w.Q;
      const float total = r_ok ? R_all : Q_all;
      const float tau = u_last * total;
      const unsigned over = __ballot_sync(0xffffffffu, lane < C && incl > tau);
      const unsigned pos = __ballot_sync(0xffffffffu, lane < C && mass > 0.f);
      int owner = -1;
      if (over) owner = __ffs(over) - 1;
      else if (pos) owner = 31 - __clz(pos);
      const float incl_o = __shfl_sync(0xffffffffu, incl, owner < 0 ? 0 : owner);
      const float mass_o = __shfl_sync(0xffffffffu, mass, owner < 0 ? 0 : owner);
      if (lane == 0) {
        sh->mass_total = total;
        sh->use_r = r_ok ? 1 : 0;
        sh->owner = owner;
        sh->tau_local = fmaxf(tau - (incl_o - mass_o), 0.f);
      }
    }
    if (lane == 0) sh->D = D;
  }
  __syncthreads();
}

// ---------------------------------------------------------------- inverse-CDF walk

// Residual (use_r) or fused mass of vector i of the slice, summed.
template <typename T>
__device__ __forceinline__ float vec_mass(const T* ra, const T* rb, const T* rt, int i, bool use_r,
                                          f2 beta2, f2 L2, f2 nA2, f2 nS2) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  f2 xa[NP], xb[NP], xt[NP], p[NP], qf[NP], r[NP];
  load_pairs(ra + i * VE, xa);
  load_pairs(rb + i * VE, xb);
  load_pairs(rt + i * VE, xt);
  vec_masses(xa, xb, xt, beta2, L2, nA2, nS2, p, qf, r);
  return use_r ? vsum(r) : vsum(qf);
}

// In the CTA that owns the target: the smallest slice index whose cumulative
// mass (index order: round, thread, element) exceeds tau_local.  The masses
// are recomputed here exactly as pass 2 computed them.  Returns the index
// within the row, or -1.
template <typename T>
__device__ int walk(SharedTma* sh, const T* ra, const T* rb, const T* rt, int nv, int rounds,
                    int lo, float beta, const float* vmass, bool stored_r) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool use_r = sh->use_r != 0;
  const float tau = sh->tau_local;
  const float A2 = sh->lse[0] * kLog2e, S2 = sh->lse[3] * kLog2e;
  const f2 beta2 = pk(beta, beta), L2 = pk(kLog2e, kLog2e);
  const f2 nA2 = pk(-A2, -A2), nS2 = pk(-S2, -S2);
  // pass 2 kept the residual masses of draft rows and the fused masses of
  // the bonus row; the other kind (a draft row whose residual is zero) is
  // recomputed exactly as pass 2 computes it
  const bool stored = (use_r == stored_r);
  int last_pos = -1;  // this thread's last vector with positive mass
  for (int j = 0; j < rounds; ++j) {
    const int i = j * kTThreads + tid;
    float v = 0.f;
    if (i < nv)
      v = stored ? vmass[j * kTThreads + tid] : vec_mass(ra, rb, rt, i, use_r, beta2, L2, nA2, nS2);
    if (v > 0.f) last_pos = i;
    const float ws = warp_sum(v);
    if (lane == 0) sh->wr[j][warp] = ws;
  }
  __syncthreads();
  if (tid == 0) {
    float cum = 0.f, tj = 0.f;
    int js = -1;
    for (int j = 0; j < rounds; ++j) {
      float tot = 0.f;
      for (int w = 0; w < kTWarps; ++w) tot += sh->wr[j][w];
      if (cum + tot > tau) {
        js = j;
        tj = fmaxf(tau - cum, 0.f);
        break;
      }
      cum += tot;
    }
    sh->jstar = js;
    sh->tau_j = tj;
    sh->found = -1;
  }
  __syncthreads();
  const int js = sh->jstar;
  if (js >= 0) {
    const int i = js * kTThreads + tid;
    float x = 0.f;
    if (i < nv)
      x = stored ? vmass[js * kTThreads + tid] : vec_mass(ra, rb, rt, i, use_r, beta2, L2, nA2, nS2);
    float incl = x;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    if (lane == 31) sh->scan[warp] = incl;
    __syncthreads();
    float woff = 0.f;
    for (int w = 0; w < warp; ++w) woff += sh->scan[w];
    incl += woff;
    const float excl = incl - x;
    const float tj = sh->tau_j;
    if (x > 0.f && excl <= tj && tj < incl) {
      f2 xa[NP], xb[NP], xt[NP], p[NP], qf[NP], r[NP];
      load_pairs(ra + i * VE, xa);
      load_pairs(rb + i * VE, xb);
      load_pairs(rt + i * VE, xt);
      vec_masses(xa, xb, xt, beta2, L2, nA2, nS2, p, qf, r);
      float cum = excl;
      int pick = -1, last = -1;
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        float v0, v1;
        upk(use_r ? r[h] : qf[h], v0, v1);
        if (v0 > 0.f) last = 2 * h;
        cum += v0;
        if (pick < 0 && cum > tj) pick = 2 * h;
        if (v1 > 0.f) last = 2 * h + 1;
        cum += v1;
        if (pick < 0 && cum > tj) pick = 2 * h + 1;
      }
      if (pick < 0) pick = last;
      if (pick >= 0) sh->found = lo + i * VE + pick;
    }
  }
  __syncthreads();
  const int found0 = sh->found;
  __syncthreads();
  if (found0 < 0) {
    // the target fell into the rounding gap at the end: last positive element
    if (last_pos >= 0) atomicMax(&sh->found, last_pos);
    __syncthreads();
    const int kmax = sh->found;
    __syncthreads();
    if (tid == 0) sh->found = -1;
    __syncthreads();
    if (kmax >= 0 && last_pos == kmax) {
      f2 xa[NP], xb[NP], xt[NP], p[NP], qf[NP], r[NP];
      load_pairs(ra + kmax * VE, xa);
      load_pairs(rb + kmax * VE, xb);
      load_pairs(rt + kmax * VE, xt);
      vec_masses(xa, xb, xt, beta2, L2, nA2, nS2, p, qf, r);
      int last = -1;
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        float v0, v1;
        upk(use_r ? r[h] : qf[h], v0, v1);
        if (v0 > 0.f) last = 2 * h;
        if (v1 > 0.f) last = 2 * h + 1;
      }
      if (last >= 0) sh->found = lo + kmax * VE + last;
    }
    __syncthreads();
  }
  return sh->found;
}

// ---------------------------------------------------------------- the kernel

template <typename T, bool STOCH>
__global__ void __launch_bounds__(kTThreads, 2) fuse_verify_tma(const KParams P) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  extern __shared__ __align__(128) unsigned char smem_tma[];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int tid = threadIdx.x;
  const int C = P.C;
  const long long row = blockIdx.x / C;
  const int K1 = P.K + 1;
  const int bi = static_cast<int>(row / K1);
  const int k = static_cast<int>(row % K1);
  const bool bonus = (k == P.K);
  const int V = P.V, W = P.W;
  const int lo = rank * W;
  const int n = max(0, min(W, V - lo));
  const int nv = n / VE;
  const int rounds = (nv + kTThreads - 1) / kTThreads;
  // rounds per chunk, even so that pass 1's pairs of rounds never straddle a chunk
  const int rc = max(2, ((rounds + kChunks - 1) / kChunks + 1) & ~1);
  T* sa = reinterpret_cast<T*>(smem_tma);
  T* sb = sa + W;
  T* st = sb + W;
  SharedTma* sh = reinterpret_cast<SharedTma*>(smem_tma + P.sh_off);
  // stochastic: per-thread, per-round sampling masses after the records
  float* vmass = reinterpret_cast<float*>(reinterpret_cast<unsigned char*>(sh) +
                                          shared_tma_bytes(C));
  const float beta = P.beta;
  const bool leader = (rank == 0 && tid == 0);
  const bool only_t = !STOCH && !P.full && bonus && !P.fuse_bonus;

  if (tid == 0) {
#pragma unroll
    for (int c = 0; c < kChunks; ++c) mbar_init(&sh->bar[c], 1);
    mbar_init(&sh->sample_bar, 1);
    sh->broken = 0;
    sh->sample = -1;
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) {
    const size_t off = static_cast<size_t>(row) * V + lo;
    const T* ga = static_cast<const T*>(P.a) + off;
    const T* gb = static_cast<const T*>(P.b) + off;
    const T* gt = static_cast<const T*>(P.t) + off;
#pragma unroll
    for (int c = 0; c < kChunks; ++c) {
      const int v0 = min(nv, c * rc * kTThreads);
      const int v1 = min(nv, (c + 1) * rc * kTThreads);
      const unsigned bytes = static_cast<unsigned>(v1 - v0) * 16u;
      mbar_arrive_expect_tx(&sh->bar[c], bytes * (only_t ? 1u : 3u));
      if (bytes) {
        const int e0 = v0 * VE;
        if (!only_t) {
          bulk_load(sa + e0, ga + e0, bytes, &sh->bar[c]);
          bulk_load(sb + e0, gb + e0, bytes, &sh->bar[c]);
        }
        bulk_load(st + e0, gt + e0, bytes, &sh->bar[c]);
      }
    }
  }
  // the scalars of this row, loaded while the slice is in flight
  const int dtok = bonus ? -1 : P.tokens[static_cast<size_t>(bi) * P.K + k];
  const float u_last = STOCH ? P.unif[static_cast<size_t>(bi) * K1 + P.K] : 0.f;

  // ---- pass 1 (program chosen per row; uniform over the cluster)
  if (P.full) {
    pass1_and_combine<T, F_LA | F_LB | F_LT | F_LS | F_AS | F_AT>(
        sa, sb, st, nv, rounds, rc, lo, n, W, beta, dtok, sh, rank, C, cluster);
  } else if (!STOCH) {
    if (!bonus)
      pass1_and_combine<T, F_LA | F_LB | F_LT | F_AS>(sa, sb, st, nv, rounds, rc, lo, n, W, beta,
                                                      dtok, sh, rank, C, cluster);
    else if (P.fuse_bonus)
      pass1_and_combine<T, F_AS>(sa, sb, st, nv, rounds, rc, lo, n, W, beta, dtok, sh, rank, C,
                                 cluster);
    else
      pass1_and_combine<T, F_AT>(sa, sb, st, nv, rounds, rc, lo, n, W, beta, dtok, sh, rank, C,
                                 cluster);
  } else if (!bonus) {
    if (P.want_tokens)
      pass1_and_combine<T, F_LA | F_LB | F_LS | F_AS>(sa, sb, st, nv, rounds, rc, lo, n, W, beta,
                                                      dtok, sh, rank, C, cluster);
    else
      pass1_and_combine<T, F_LA | F_LB | F_LS>(sa, sb, st, nv, rounds, rc, lo, n, W, beta, dtok,
                                               sh, rank, C, cluster);
  } else {
    if (P.want_tokens)
      pass1_and_combine<T, F_LS | F_AS>(sa, sb, st, nv, rounds, rc, lo, n, W, beta, dtok, sh,
                                        rank, C, cluster);
    else
      pass1_and_combine<T, F_LS>(sa, sb, st, nv, rounds, rc, lo, n, W, beta, dtok, sh, rank, C,
                                 cluster);
  }

  // ---- pass 2
  const bool jsd = P.divergence == ASYMSPEC_DIV_JSD;
  const bool klg = P.divergence == ASYMSPEC_DIV_KL;
  const bool run2 = STOCH || P.full || (!bonus && (jsd || klg));
  if (run2) {
    float* lp = P.logprobs ? P.logprobs + static_cast<size_t>(row) * V + lo : nullptr;
    const bool r_allowed = STOCH && !bonus;
    constexpr unsigned RQ = STOCH ? G_RES : 0u;
    if (STOCH && bonus && !P.full) {
      pass2_and_combine<T, G_QF, false, STOCH>(sa, sb, st, nv, rounds, beta, nullptr, sh, rank,
                                               C, false, u_last, vmass, cluster);
    } else if (lp) {
      if (jsd)
        pass2_and_combine<T, G_JSD | RQ, true, STOCH>(sa, sb, st, nv, rounds, beta, lp, sh, rank, C,
                                              r_allowed, u_last, vmass, cluster);
      else if (klg)
        pass2_and_combine<T, G_KL | RQ, true, STOCH>(sa, sb, st, nv, rounds, beta, lp, sh, rank, C,
                                              r_allowed, u_last, vmass, cluster);
      else
        pass2_and_combine<T, RQ, true, STOCH>(sa, sb, st, nv, rounds, beta, lp, sh, rank, C,
                                              r_allowed, u_last, vmass, cluster);
    } else {
      if (jsd)
        pass2_and_combine<T, G_JSD | RQ, false, STOCH>(sa, sb, st, nv, rounds, beta, nullptr, sh, rank, C,
                                              r_allowed, u_last, vmass, cluster);
      else if (klg)
        pass2_and_combine<T, G_KL | RQ, false, STOCH>(sa, sb, st, nv, rounds, beta, nullptr, sh, rank, C,
                                              r_allowed, u_last, vmass, cluster);
      else
        pass2_and_combine<T, RQ, false, STOCH>(sa, sb, st, nv, rounds, beta, nullptr, sh, rank, C,
                                              r_allowed, u_last, vmass, cluster);
    }
  } else if (tid == 0) {
    sh->D = 0.f;
  }

  // ---- stochastic: inverse-CDF draw in the owning CTA, handed to rank 0
  if constexpr (STOCH) {
    if (rank == sh->owner) {
      const int pick = walk<T>(sh, sa, sb, st, nv, rounds, lo, beta, vmass, !bonus || P.full);
      if (tid == 0) {
        *cluster.map_shared_rank(&sh->sample, 0) = pick;
        mbar_arrive_remote(&sh->sample_bar, 0);
      }
    }
  }

  // ---- epilogue (rank 0, thread 0)
  if (leader) {
    if (STOCH && sh->owner >= 0 &&
        !mbar_wait_cluster_bounded(&sh->sample_bar, 0, kCopyTimeoutNs))
      sh->bad |= kBadTimeout;
    const float lse_a = sh->lse[0], lse_b = sh->lse[1], lse_s = sh->lse[3];
    const bool has_ab = P.full || !bonus;
    const bool has_t = P.full || (!STOCH && !bonus);
    const bool has_s = P.full || STOCH;
    RowResult r;
    r.lse_a = has_ab ? lse_a : NAN;
    r.lse_b = has_ab ? lse_b : NAN;
    r.lse_t = has_t ? sh->lse[2] : NAN;
    r.lse_s = has_s ? lse_s : NAN;
    r.D = sh->D;
    r.is = sh->is;
    r.it = sh->it;
    r.sample = STOCH ? sh->sample : -1;
    r.mass = STOCH ? sh->mass_total : NAN;
    r.bad = sh->bad;
    r.have_lse_t = has_t;
    finish_row<STOCH>(P, row, bi, k, r, dtok, sh->da, sh->db, sh->dt);
  }
  // a copy that timed out may still land: wait for it (bounded) before exit
  if (tid == 0 && sh->broken) {
#pragma unroll
    for (int c = 0; c < kChunks; ++c) mbar_wait_bounded(&sh->bar[c], 0, kCopyTimeoutNs);
  }
}

}  // namespace asymspec_impl
