// Staged fuse-and-verify kernel for 16-byte aligned rows (every program
// but the production stochastic JSD step, which fuse_verify_row in
// kernel_row.cuh runs), and the decision kernel both row kernels feed.
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
// Normalisers: each thread sums 2^((x - ref) log2 e) against one fixed
// reference per stream and warp (the warp's largest of its threads' first
// two entries), so an entry costs one FMA, one ex2 and one add; the warps'
// references meet only in the reductions.  A thread whose sum reaches 2^100
// (an entry more than ~69 nats above its reference, or non-finite data)
// makes the CTA redo its slice with a running maximum (pass1_online).
//
// Reductions: warp maxima with redux.sync, sums with shuffles; warp -> CTA in
// shared memory.  Each CTA pushes its pass-1 record into every peer's shared
// memory (DSMEM stores) before one cluster barrier, so after the barrier
// every CTA combines local copies, identically.  After pass 2 each CTA
// stores its row statistics (rank 0), its pass-2 record and its inverse-CDF
// group masses in the workspace and exits; decide_rows (below), a second
// launch with one CTA per batch element, decides every row from those
// records (the divergence, the walk to the drawn element, the acceptance
// test) and runs Algorithm 1's scan.
//
// Every wait is bounded: a chunk that does not land within 200 ms marks the
// row with ASYMSPEC_DATA_TIMEOUT; the CTA still reaches every cluster
// barrier, so no CTA of the cluster is left waiting, and before it exits
// thread 0 waits (bounded again) for any copy still in flight.
#pragma once

#include <type_traits>

#include "device_common.cuh"

namespace asymspec_impl {

constexpr int kTThreads = 256;
constexpr int kTWarps = kTThreads / 32;
constexpr int kMaxRounds = 10;  // 16-byte vectors per thread per slice
constexpr int kWalkRounds = 16;  // steps of 32 vectors in a group the walk takes
constexpr int kChunks = 4;      // bulk-copy chunks per slice
constexpr unsigned long long kCopyTimeoutNs = 200ull * 1000ull * 1000ull;
constexpr float kSumLimit = 1.2676506e30f;  // 2^100: pass1_fast's overflow guard

enum : unsigned { F_LA = 1, F_LB = 2, F_LT = 4, F_LS = 8, F_AS = 16, F_AT = 32 };
enum : unsigned { G_JSD = 1, G_KL = 2, G_RES = 4, G_QF = 8 };

// Pass-1 result (per thread, per warp, per CTA, per row).  Stream q's
// normaliser is ref[q] + ln s[q]: s[q] sums 2^((x - ref[q]) log2 e).
struct __align__(16) X1 {
  float ref[4];
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

// Fixed part of the shared state; the C pass-1 records pushed by the
// cluster follow it (recv1()).
struct __align__(16) SharedTma {
  unsigned long long bar[kChunks];  // one mbarrier per chunk
  union {                           // per-warp records, one pass at a time
    X1 w1[kTWarps];
    X2 w2[kTWarps];
  };
  float lse[4];       // the row's normalisers (pass 2 reads them)
  unsigned broken;    // a chunk copy timed out
  float qown;         // production draft rows: this slice's fused mass, from pass 1
  unsigned long long wait_ns;  // limit of each chunk wait (KParams::copy_wait_ns)
  unsigned pad[kChunks];
  // the C pushed records
  __device__ X1* recv1() { return reinterpret_cast<X1*>(this + 1); }
};

// The pushed records are copied with 16-byte stores.
static_assert(sizeof(X1) % 16 == 0 && alignof(X1) == 16, "X1 must be 16-byte aligned");
static_assert(sizeof(X2) % 16 == 0 && alignof(X2) == 16, "X2 must be 16-byte aligned");
static_assert(sizeof(SharedTma) % 16 == 0, "records after SharedTma must stay 16-byte aligned");

// Inverse-CDF groups: group g of a slice is the 32 vectors of warp (g % 8)
// in round g / 8, i.e. vectors [32 g, 32 g + 32) in index order.
constexpr int kGroupsMax = kMaxRounds * kTWarps;

// Shared bytes after the slices for a cluster of C CTAs.
__host__ __device__ constexpr int shared_tma_bytes(int C) {
  return static_cast<int>(sizeof(SharedTma) + C * sizeof(X1));
}

__device__ __forceinline__ X1 x1_neutral() {
  X1 r;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    r.ref[q] = -INFINITY;
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

// Warp maximum (NaN ignored unless every lane holds NaN).
__device__ __forceinline__ float warp_max(float v) {
  float r;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
  return r;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// Larger value wins, the lowest index among equal values; NaN never wins.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
  const float m = warp_max(v);
  const int cand = (v == m) ? i : INT_MAX;
  i = __reduce_min_sync(0xffffffffu, cand);
  v = m;
}

// Warp-wide combine of the streams a program computes: the largest
// reference, every lane's sum rescaled to it, the sums added.  Every lane
// ends with the same (bit-identical) result.  A NaN sum stays NaN.
template <unsigned F>
__device__ __forceinline__ void warp_reduce_x1(X1& e) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
    if (F & bit) {
      const float M = warp_max(e.ref[q]);
      const float s = (e.s[q] == 0.f || e.ref[q] == M) ? e.s[q]
                                                       : e.s[q] * ex2((e.ref[q] - M) * kLog2e);
      e.ref[q] = M;
      e.s[q] = warp_sum(s);
    }
  }
  if (F & F_AS) warp_argmax(e.vs, e.is);
  if (F & F_AT) warp_argmax(e.vt, e.it);
  e.bad = __reduce_or_sync(0xffffffffu, e.bad);
}

// Sums of four values over a warp in one transposed butterfly (9 shuffles
// instead of 20); every lane ends with the four totals.
__device__ __forceinline__ void warp_sum4(float& v0, float& v1, float& v2, float& v3) {
  const int lane = threadIdx.x & 31;
  const bool up16 = (lane & 16) != 0, up8 = (lane & 8) != 0;
  // lanes 0-15 carry v0, v1 on; lanes 16-31 carry v2, v3
  const float a = (up16 ? v2 : v0) + __shfl_xor_sync(0xffffffffu, up16 ? v0 : v2, 16);
  const float b = (up16 ? v3 : v1) + __shfl_xor_sync(0xffffffffu, up16 ? v1 : v3, 16);
  // lanes with bit 3 clear carry a (v0 or v2) on, the others b (v1 or v3)
  float c = (up8 ? b : a) + __shfl_xor_sync(0xffffffffu, up8 ? a : b, 8);
#pragma unroll
  for (int off = 4; off > 0; off >>= 1) c += __shfl_xor_sync(0xffffffffu, c, off);
  // lane 0: v0, lane 8: v1, lane 16: v2, lane 24: v3
  v0 = __shfl_sync(0xffffffffu, c, 0);
  v1 = __shfl_sync(0xffffffffu, c, 8);
  v2 = __shfl_sync(0xffffffffu, c, 16);
  v3 = __shfl_sync(0xffffffffu, c, 24);
}

// As warp_reduce_x1 for records whose references are already equal across
// the warp (pass1_fast takes the warp maximum of the first vectors): the
// sums are added without rescaling.
template <unsigned F>
__device__ __forceinline__ void warp_reduce_x1_uniform(X1& e) {
  constexpr int nsum = ((F & F_LA) != 0) + ((F & F_LB) != 0) + ((F & F_LT) != 0) + ((F & F_LS) != 0);
  if constexpr (nsum >= 2) {
    warp_sum4(e.s[0], e.s[1], e.s[2], e.s[3]);
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
      if (F & bit) e.s[q] = warp_sum(e.s[q]);
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
// (lane r of the calling warp writes to CTA r); a cluster barrier must follow.
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
  constexpr int nsum = ((G & G_JSD) ? 2 : 0) + ((G & G_KL) ? 1 : 0) + ((G & G_RES) ? 2 : 0) +
                       ((!(G & G_RES) && (G & G_QF)) ? 1 : 0);
  if constexpr (nsum >= 2 && !((G & G_JSD) && (G & G_KL))) {
    // the (at most four) sums of the gate in one butterfly
    float v0 = (G & G_JSD) ? x.j : x.kl, v1 = x.msum, v2 = x.R, v3 = x.Q;
    warp_sum4(v0, v1, v2, v3);
    if (G & G_JSD) {
      x.j = v0;
      x.msum = v1;
    }
    if (G & G_KL) x.kl = v0;
    if (G & G_RES) x.R = v2;
    if (G & (G_RES | G_QF)) x.Q = v3;
  } else {
    if (G & G_JSD) {
      x.j = warp_sum(x.j);
      x.msum = warp_sum(x.msum);
    }
    if (G & G_KL) x.kl = warp_sum(x.kl);
    if (G & G_RES) x.R = warp_sum(x.R);
    if (G & (G_RES | G_QF)) x.Q = warp_sum(x.Q);
  }
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

// The first two entries of a 16-byte vector in shared memory, widened.
__device__ __forceinline__ f2 first_pair(const __nv_bfloat16* p) {
  const unsigned w = *reinterpret_cast<const unsigned*>(p);
  return pk(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}
__device__ __forceinline__ f2 first_pair(const float* p) {
  return *reinterpret_cast<const f2*>(p);
}

// The fused score s = t + beta delta of a pair (Eq. 2) for delta source DS:
// a - b (Eq. 1, ASYMSPEC_DELTA_AB), a (raw-augmented) or t - b (SCD-style).
template <int DS>
__device__ __forceinline__ f2 fuse2(f2 beta2, f2 a, f2 b, f2 t) {
  if constexpr (DS == ASYMSPEC_DELTA_A) return fma2(beta2, a, t);
  else if constexpr (DS == ASYMSPEC_DELTA_TB) return fma2(beta2, sub2(t, b), t);
  else return fma2(beta2, sub2(a, b), t);
}

// Residual max(0, q - p) and fused q masses of one vector (stochastic mode);
// pass 2 and the inverse-CDF walk share this, so they see identical values.
template <int NP, int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ void vec_masses(const f2 (&xa)[NP], const f2 (&xb)[NP],
                                           const f2 (&xt)[NP], f2 beta2, f2 L2, f2 nA2, f2 nS2,
                                           f2 (&p)[NP], f2 (&qf)[NP], f2 (&r)[NP],
                                           f2 (&la2)[NP]) {
  // delta = a - b: the fused score in log2 units as t log2 e + (beta log2 e)(a - b),
  // the form the production kernel (kernel_row.cuh) uses, so that a walk over
  // either kernel's group masses sees identical vector masses
  const f2 bL2 = mul2(beta2, L2);
#pragma unroll
  for (int h = 0; h < NP; ++h) {
    la2[h] = fma2(xa[h], L2, nA2);  // log2 softmax(a), which the divergence terms reuse
    p[h] = ex2_2(la2[h]);
    if constexpr (DS == ASYMSPEC_DELTA_AB) {
      qf[h] = ex2_2(fma2(xt[h], L2, fma2(bL2, sub2(xa[h], xb[h]), nS2)));
    } else {
      const f2 s = fuse2<DS>(beta2, xa[h], xb[h], xt[h]);
      qf[h] = ex2_2(fma2(s, L2, nS2));
    }
    r[h] = relu2(sub2(qf[h], p[h]));
  }
}

template <int NP, int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ void vec_masses(const f2 (&xa)[NP], const f2 (&xb)[NP],
                                           const f2 (&xt)[NP], f2 beta2, f2 L2, f2 nA2, f2 nS2,
                                           f2 (&p)[NP], f2 (&qf)[NP], f2 (&r)[NP]) {
  f2 la2[NP];
  vec_masses<NP, DS>(xa, xb, xt, beta2, L2, nA2, nS2, p, qf, r, la2);
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

// Pass 1 with a running maximum per stream (one rescale check per two
// vectors): the fallback for slices where pass1_fast's fixed reference
// overflows.  Vector i of the slice lives in round i / NT; chunk c holds
// rounds [c rc, (c+1) rc).  Rounds are taken two at a time.
// WAIT: the slice is in shared memory behind the chunk barriers of sh (false:
// it is in global memory and sh is not used).
template <typename T, unsigned F, bool WAIT = true, int DS = ASYMSPEC_DELTA_AB>
__device__ __noinline__ void pass1_online(const T* ra, const T* rb, const T* rt, int nv, int rounds,
                                      int rc, int lo, float beta, SharedTma* sh, X1& e,
                                      unsigned ph = 0) {
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
    if (WAIT && !sh->broken && !mbar_wait_bounded(&sh->bar[c], ph, sh->wait_ns))
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
          xs[h] = fuse2<DS>(beta2, xa[h], xb[h], xt[h]);
          ys[h] = fuse2<DS>(beta2, ya[h], yb[h], yt[h]);
        }
      }
      if (F & F_LA) online_pairs2(e.ref[0], acc[0], xa, ya, L2);
      if (F & F_LB) online_pairs2(e.ref[1], acc[1], xb, yb, L2);
      float ct0 = 0.f, ct1 = 0.f, cs0 = 0.f, cs1 = 0.f;
      if (F & F_LT) {
        online_pairs2(e.ref[2], acc[2], xt, yt, L2);
        if (F & F_AT) {
          ct0 = vmax_pairs(xt);
          ct1 = vmax_pairs(yt);
        }
      } else if (F & F_AT) {
        ct0 = vmax_pairs_nan(xt);
        ct1 = vmax_pairs_nan(yt);
      }
      if (F & F_LS) {
        online_pairs2(e.ref[3], acc[3], xs, ys, L2);
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
    for (int h = 0; h < NP; ++h) xs[h] = fuse2<DS>(beta2, xa[h], xb[h], xt[h]);
    e.is = arg_in_vector(xs, e.vs, lo + vec_s * VE);
  }
  if ((F & F_AT) && vec_t >= 0) {
    f2 xt[NP];
    load_pairs(rt + vec_t * VE, xt);
    e.it = arg_in_vector(xt, e.vt, lo + vec_t * VE);
  }
}

// Adds two vectors of pairs to a packed sum of 2^((x - ref) log2 e), with
// nm2 = -ref log2 e in both halves.
template <int NP>
__device__ __forceinline__ void fixed_pairs2(f2& acc, const f2 (&x)[NP], const f2 (&y)[NP], f2 L2,
                                             f2 nm2) {
  f2 e[NP];
#pragma unroll
  for (int h = 0; h < NP; ++h)
    e[h] = add2(ex2_2(fma2(x[h], L2, nm2)), ex2_2(fma2(y[h], L2, nm2)));
  if constexpr (NP == 4) {
    acc = add2(acc, add2(add2(e[0], e[1]), add2(e[2], e[3])));
  } else {
    acc = add2(acc, add2(e[0], e[1]));
  }
}

// Pass 1 against fixed references: each warp takes the largest of its
// threads' first-vector maxima (vector tid, in chunk 0) as the reference of
// each normaliser stream.  Returns true when one of this thread's sums reached 2^100 or is not
// finite (the caller then redoes the slice with pass1_online).  Argmax
// streams are tracked per vector as in pass1_online.
template <typename T, unsigned F, int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ bool pass1_fast(const T* ra, const T* rb, const T* rt, int nv,
                                           int rounds, int rc, int lo, float beta, SharedTma* sh,
                                           X1& e, unsigned ph = 0) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needA = (F & (F_LA | F_LS | F_AS)) != 0;
  constexpr bool needB = (F & (F_LB | F_LS | F_AS)) != 0;
  constexpr bool needT = (F & (F_LT | F_LS | F_AS | F_AT)) != 0;
  constexpr bool needS = (F & (F_LS | F_AS)) != 0;
  constexpr int STEP = 2 * kTThreads * VE;  // elements per two rounds
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  const int tid = static_cast<int>(threadIdx.x);
  // chunk 0 holds every thread's first vector
  if (!sh->broken && !mbar_wait_bounded(&sh->bar[0], ph, sh->wait_ns))
    atomicOr(&sh->broken, kBadTimeout);
  float ref[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  if (tid < nv) {
    // the first two entries of the thread's first vector: any entries do as
    // references (a sum that reaches 2^100 sends the CTA to pass1_online)
    f2 xa = 0ull, xb = 0ull, xt = 0ull;
    if (needA) xa = first_pair(ra + tid * VE);
    if (needB) xb = first_pair(rb + tid * VE);
    if (needT) xt = first_pair(rt + tid * VE);
    if (F & F_LA) ref[0] = fmaxf(lo_of(xa), hi_of(xa));
    if (F & F_LB) ref[1] = fmaxf(lo_of(xb), hi_of(xb));
    if (F & F_LT) ref[2] = fmaxf(lo_of(xt), hi_of(xt));
    if (F & F_LS) {
      const f2 xs = fuse2<DS>(beta2, xa, xb, xt);
      ref[3] = fmaxf(lo_of(xs), hi_of(xs));
    }
  }
  // one reference per warp: the largest of its threads' first-pair maxima
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
    if (F & bit) ref[q] = warp_max(ref[q]);
  }
  f2 nm[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float v = -ref[q] * kLog2e;
    nm[q] = pk(v, v);
  }
  f2 acc[4] = {0ull, 0ull, 0ull, 0ull};
  int vec_s = -1, vec_t = -1;  // vectors holding the best s and t so far
  for (int c = 0, r0 = 0; c < kChunks && r0 < rounds; ++c, r0 += rc) {
    if (c > 0 && !sh->broken && !mbar_wait_bounded(&sh->bar[c], ph, sh->wait_ns))
      atomicOr(&sh->broken, kBadTimeout);
    const int r1 = min(rounds, r0 + rc);
    int i0 = r0 * kTThreads + tid;          // vector index of this thread's first vector
    int e0 = i0 * VE;                       // its element offset in the slice
    for (int kr = r0; kr < r1; kr += 2, i0 += 2 * kTThreads, e0 += STEP) {
      if (i0 >= nv) break;
      // TWO: the thread has both vectors of the step (all but the slice's
      // last step); the other form fills the missing one (one copy each)
      auto step = [&](auto two) {
      constexpr bool TWO = decltype(two)::value;
      const bool has1 = TWO;
      const int e1 = e0 + kTThreads * VE;
      f2 xa[NP], xb[NP], xt[NP], xs[NP], ya[NP], yb[NP], yt[NP], ys[NP];
      if (needA) {
        load_pairs(ra + e0, xa);
        if (TWO) load_pairs(ra + e1, ya); else load_or_fill(ra + e1, false, ya);
      }
      if (needB) {
        load_pairs(rb + e0, xb);
        if (TWO) load_pairs(rb + e1, yb); else load_or_fill(rb + e1, false, yb);
      }
      if (needT) {
        load_pairs(rt + e0, xt);
        if (TWO) load_pairs(rt + e1, yt); else load_or_fill(rt + e1, false, yt);
      }
      if (needS) {
#pragma unroll
        for (int h = 0; h < NP; ++h) {
          xs[h] = fuse2<DS>(beta2, xa[h], xb[h], xt[h]);
          ys[h] = fuse2<DS>(beta2, ya[h], yb[h], yt[h]);
        }
      }
      if (F & F_LA) fixed_pairs2(acc[0], xa, ya, L2, nm[0]);
      if (F & F_LB) fixed_pairs2(acc[1], xb, yb, L2, nm[1]);
      if (F & F_LT) fixed_pairs2(acc[2], xt, yt, L2, nm[2]);
      if (F & F_LS) fixed_pairs2(acc[3], xs, ys, L2, nm[3]);
      if (F & F_AS) {
        const float cs0 = (F & F_LS) ? vmax_pairs(xs) : vmax_pairs_nan(xs);
        const float cs1 = (F & F_LS) ? vmax_pairs(ys) : vmax_pairs_nan(ys);
        arg_track(e.vs, vec_s, cs0, i0, e.bad, kBadS);
        if (has1) arg_track(e.vs, vec_s, cs1, i0 + kTThreads, e.bad, kBadS);
      }
      if (F & F_AT) {
        const float ct0 = (F & F_LT) ? vmax_pairs(xt) : vmax_pairs_nan(xt);
        const float ct1 = (F & F_LT) ? vmax_pairs(yt) : vmax_pairs_nan(yt);
        arg_track(e.vt, vec_t, ct0, i0, e.bad, kBadT);
        if (has1) arg_track(e.vt, vec_t, ct1, i0 + kTThreads, e.bad, kBadT);
      }
      };
      if ((kr + 1 < r1) && (i0 + kTThreads < nv)) step(std::true_type{});
      else step(std::false_type{});
    }
  }
  bool ovf = false;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
    e.ref[q] = ref[q];
    e.s[q] = hsum2(acc[q]);
    if ((F & bit) && !(e.s[q] < kSumLimit)) ovf = true;
  }
  // the element of the best vector (re-read once from shared memory)
  if ((F & F_AS) && vec_s >= 0) {
    f2 xa[NP], xb[NP], xt[NP], xs[NP];
    load_pairs(ra + vec_s * VE, xa);
    load_pairs(rb + vec_s * VE, xb);
    load_pairs(rt + vec_s * VE, xt);
#pragma unroll
    for (int h = 0; h < NP; ++h) xs[h] = fuse2<DS>(beta2, xa[h], xb[h], xt[h]);
    e.is = arg_in_vector(xs, e.vs, lo + vec_s * VE);
  }
  if ((F & F_AT) && vec_t >= 0) {
    f2 xt[NP];
    load_pairs(rt + vec_t * VE, xt);
    e.it = arg_in_vector(xt, e.vt, lo + vec_t * VE);
  }
  return ovf;
}

// Pass 1 and the CTA combine, pushed to every CTA of the cluster, up to and
// including cluster barrier B1.  dtok: the row's draft token (-1 if none),
// known to warp 0.
template <typename T, unsigned F, int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ void pass1_and_push(const T* ra, const T* rb, const T* rt, int nv,
                                               int rounds, int rc, int lo, int n, float beta,
                                               int dtok, SharedTma* sh, int rank, int C,
                                               cg::cluster_group& cluster) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  X1 e = x1_neutral();
  const bool ovf = pass1_fast<T, F, DS>(ra, rb, rt, nv, rounds, rc, lo, beta, sh, e);
  warp_reduce_x1_uniform<F>(e);  // the warp's references are equal
  if (lane == 0) sh->w1[warp] = e;
  if (__syncthreads_or(ovf)) {
    // an entry far above its thread's reference (or non-finite data): redo
    // the slice with a running maximum
    e = x1_neutral();
    pass1_online<T, F, true, DS>(ra, rb, rt, nv, rounds, rc, lo, beta, sh, e);
    warp_reduce_x1<F>(e);
    if (lane == 0) sh->w1[warp] = e;
    __syncthreads();
  }
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
}

// Thread 0: the bulk copies of a row's slice into the CTA's buffers, in
// kChunks chunks, each completing on its own mbarrier.  only_t: copy t alone
// (a greedy bonus row without fused bonus needs nothing else).
template <typename T>
__device__ __forceinline__ void issue_chunk(const KParams& P, SharedTma* sh, long long row,
                                            int lo, int nv, int rc, T* sa, T* sb, T* st,
                                            bool only_t, int c) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const size_t off = static_cast<size_t>(row) * P.V + lo;
  const int v0 = min(nv, c * rc * kTThreads);
  const int v1 = min(nv, (c + 1) * rc * kTThreads);
  const unsigned bytes = static_cast<unsigned>(v1 - v0) * 16u;
  mbar_arrive_expect_tx(&sh->bar[c], bytes * (only_t ? 1u : 3u));
  if (bytes) {
    const int e0 = v0 * VE;
    if (!only_t) {
      bulk_load(sa + e0, static_cast<const T*>(P.a) + off + e0, bytes, &sh->bar[c]);
      bulk_load(sb + e0, static_cast<const T*>(P.b) + off + e0, bytes, &sh->bar[c]);
    }
    bulk_load(st + e0, static_cast<const T*>(P.t) + off + e0, bytes, &sh->bar[c]);
  }
}
template <typename T>
__device__ __forceinline__ void issue_slice(const KParams& P, SharedTma* sh, long long row,
                                            int lo, int nv, int rc, T* sa, T* sb, T* st,
                                            bool only_t) {
#pragma unroll
  for (int c = 0; c < kChunks; ++c) issue_chunk<T>(P, sh, row, lo, nv, rc, sa, sb, st, only_t, c);
}

// After B1, in one warp: the row values from the C pushed records (every
// lane ends with them).  lse[q] = ln of stream q's normaliser.
template <unsigned F>
__device__ __forceinline__ X1 combine_pass1(SharedTma* sh, int C, float (&lse)[4]) {
  const int lane = threadIdx.x & 31;
  X1 w = (lane < C) ? sh->recv1()[lane] : x1_neutral();
  warp_reduce_x1<F>(w);
#pragma unroll
  for (int q = 0; q < 4; ++q) lse[q] = w.ref[q] + logf(w.s[q]);
  return w;
}

// The draft token's a, b, t (from the record of the CTA whose slice holds it).
__device__ __forceinline__ void draft_logits(SharedTma* sh, int dtok, int W, int C, float& ad,
                                             float& bd, float& td) {
  ad = bd = td = 0.f;
  if (dtok >= 0 && W > 0) {
    const X1& o = sh->recv1()[dtok / W < C ? dtok / W : 0];
    ad = o.da;
    bd = o.db;
    td = o.dt;
  }
}

// ---------------------------------------------------------------- pass 2

// Divergence terms of one vector (Eq. 3): JSD terms p (log2 p - log2 m) and
// q (log2 q - log2 m) with m = p + q, their mass m, or KL terms; la: log2 p.
template <int NP, bool JSD, bool KL>
__device__ __forceinline__ void div_terms(const f2 (&la)[NP], const f2 (&xb)[NP], const f2 (&p)[NP],
                                          f2 L2, f2 nB2, f2 tiny2, f2& ja, f2& jb,
                                          f2& ms2, f2& kl2) {
#pragma unroll
  for (int h = 0; h < NP; ++h) {
    const f2 la2 = la[h];
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

// As above from the logits a (log2 p = a log2 e - nA2).
template <int NP, bool JSD, bool KL>
__device__ __forceinline__ void div_terms(const f2 (&xa)[NP], const f2 (&xb)[NP], const f2 (&p)[NP],
                                          f2 L2, f2 nA2, f2 nB2, f2 tiny2, f2& ja, f2& jb,
                                          f2& ms2, f2& kl2) {
  f2 la[NP];
#pragma unroll
  for (int h = 0; h < NP; ++h) la[h] = fma2(xa[h], L2, nA2);
  div_terms<NP, JSD, KL>(la, xb, p, L2, nB2, tiny2, ja, jb, ms2, kl2);
}

// Pass-2 constants and running sums of one thread.
struct P2Const {
  f2 beta2, L2, nA2, nB2, nS2, tiny2, nl2;
};
struct P2Acc {
  f2 ja, jb, ms2, kl2, R2, Q2;
};

__device__ __forceinline__ P2Const p2_const(float beta, float A2, float B2, float S2,
                                            float lse_s) {
  P2Const k;
  k.beta2 = pk(beta, beta);
  k.L2 = pk(kLog2e, kLog2e);
  k.nA2 = pk(-A2, -A2);
  k.nB2 = pk(-B2, -B2);
  k.nS2 = pk(-S2, -S2);
  k.tiny2 = pk(kMinNormal, kMinNormal);
  k.nl2 = pk(-lse_s, -lse_s);
  return k;
}

// Pass 2 on two vectors x, y of a thread (y absent unless has1: filled with
// -1e30, which contributes nothing); g0, g1 receive their inverse-CDF masses
// (residual, or fused for G_QF).  LP: fused log-probs go to lpx, lpy.
template <int NP, unsigned G, bool LP, int DS = ASYMSPEC_DELTA_AB, bool QSUM = true>
__device__ __forceinline__ void p2_pair(const f2 (&xa)[NP], const f2 (&xb)[NP], const f2 (&xt)[NP],
                                        const f2 (&ya)[NP], const f2 (&yb)[NP], const f2 (&yt)[NP],
                                        bool has1, const P2Const& k, P2Acc& acc, float& g0,
                                        float& g1, float* lpx, float* lpy) {
  constexpr bool JSD = (G & G_JSD) != 0, KL = (G & G_KL) != 0, RES = (G & G_RES) != 0;
  constexpr bool QF = (G & G_QF) != 0;
  f2 px[NP], py[NP], lax[NP], lay[NP];
  if (RES) {
    f2 qx[NP], qy[NP], rx[NP], ry[NP];
    vec_masses<NP, DS>(xa, xb, xt, k.beta2, k.L2, k.nA2, k.nS2, px, qx, rx, lax);
    vec_masses<NP, DS>(ya, yb, yt, k.beta2, k.L2, k.nA2, k.nS2, py, qy, ry, lay);
    // the fused mass, used only when the whole residual is zero (QSUM false:
    // the caller takes the slice's fused mass from its pass-1 sum instead)
    if constexpr (QSUM) {
#pragma unroll
      for (int h = 0; h < NP; ++h) acc.Q2 = add2(acc.Q2, add2(qx[h], qy[h]));
    }
    // residual mass of each vector, summed per group for the inverse-CDF walk
    g0 = vsum(rx);
    g1 = vsum(ry);
    acc.R2 = add2(acc.R2, pk(g0, g1));
  } else if (QF) {
    f2 qx[NP], qy[NP];
#pragma unroll
    for (int h = 0; h < NP; ++h) {
      qx[h] = ex2_2(fma2(fuse2<DS>(k.beta2, xa[h], xb[h], xt[h]), k.L2, k.nS2));
      qy[h] = ex2_2(fma2(fuse2<DS>(k.beta2, ya[h], yb[h], yt[h]), k.L2, k.nS2));
    }
    // fused mass of each vector, summed per group for the inverse-CDF walk
    g0 = vsum(qx);
    g1 = vsum(qy);
    acc.Q2 = add2(acc.Q2, pk(g0, g1));
  } else if (JSD || KL) {
#pragma unroll
    for (int h = 0; h < NP; ++h) {
      lax[h] = fma2(xa[h], k.L2, k.nA2);
      lay[h] = fma2(ya[h], k.L2, k.nA2);
      px[h] = ex2_2(lax[h]);
      py[h] = ex2_2(lay[h]);
    }
  }
  if (JSD || KL) {
    div_terms<NP, JSD, KL>(lax, xb, px, k.L2, k.nB2, k.tiny2, acc.ja, acc.jb, acc.ms2, acc.kl2);
    div_terms<NP, JSD, KL>(lay, yb, py, k.L2, k.nB2, k.tiny2, acc.ja, acc.jb, acc.ms2, acc.kl2);
  }
  if (LP) {
#pragma unroll
    for (int h = 0; h < NP; ++h) {
      float l0, l1;
      upk(add2(fuse2<DS>(k.beta2, xa[h], xb[h], xt[h]), k.nl2), l0, l1);
      lpx[2 * h] = l0;
      lpx[2 * h + 1] = l1;
      if (has1) {
        upk(add2(fuse2<DS>(k.beta2, ya[h], yb[h], yt[h]), k.nl2), l0, l1);
        lpy[2 * h] = l0;
        lpy[2 * h + 1] = l1;
      }
    }
  }
}

// The inverse-CDF group masses of rounds kr and kr + 1 of one warp (every
// lane takes part, with or without a vector): one butterfly, lanes 0-15
// carrying round kr and lanes 16-31 round kr + 1.
__device__ __forceinline__ void p2_groups(float g0, float g1, float* grp, int kr, int rounds) {
  const int lane = static_cast<int>(threadIdx.x & 31), warp = static_cast<int>(threadIdx.x >> 5);
  const bool upper = lane >= 16;
  float g = (upper ? g1 : g0) + __shfl_xor_sync(0xffffffffu, upper ? g0 : g1, 16);
#pragma unroll
  for (int off = 8; off > 0; off >>= 1) g += __shfl_xor_sync(0xffffffffu, g, off);
  if (lane == 0) grp[kr * kTWarps + warp] = g;
  if (lane == 16 && kr + 1 < rounds) grp[(kr + 1) * kTWarps + warp] = g;
}

// As p2_groups for four rounds kr .. kr + 3 (v0 .. v3) in one transposed
// butterfly: lanes 0, 8, 16 and 24 end with the four group masses.  NW: warps
// per CTA (group r NW + w is warp w's 32 vectors of round r).
template <int NW = kTWarps>
__device__ __forceinline__ void p2_groups4(float v0, float v1, float v2, float v3, float* grp,
                                           int kr, int rounds) {
  const int lane = static_cast<int>(threadIdx.x & 31), warp = static_cast<int>(threadIdx.x >> 5);
  const bool up16 = (lane & 16) != 0, up8 = (lane & 8) != 0;
  const float a = (up16 ? v2 : v0) + __shfl_xor_sync(0xffffffffu, up16 ? v0 : v2, 16);
  const float b = (up16 ? v3 : v1) + __shfl_xor_sync(0xffffffffu, up16 ? v1 : v3, 16);
  float c = (up8 ? b : a) + __shfl_xor_sync(0xffffffffu, up8 ? a : b, 8);
#pragma unroll
  for (int off = 4; off > 0; off >>= 1) c += __shfl_xor_sync(0xffffffffu, c, off);
  const int r = kr + (lane >> 3);
  if ((lane & 7) == 0 && r < rounds) grp[r * NW + warp] = c;
}

__device__ __forceinline__ void p2_finish(const P2Acc& acc, X2& x) {
  x.j = hsum2(add2(acc.ja, acc.jb));
  x.msum = hsum2(acc.ms2);
  x.kl = hsum2(acc.kl2);
  x.R = hsum2(acc.R2);
  x.Q = hsum2(acc.Q2);
}

// Pass 2 over the slice, two vectors per step.
template <typename T, unsigned G, bool LP, int DS = ASYMSPEC_DELTA_AB, bool QSUM = true>
__device__ __forceinline__ void pass2(const T* ra, const T* rb, const T* rt, int nv, int rounds,
                                      float beta, float A2, float B2, float S2, float lse_s, X2& x,
                                      float* lp, float* grp) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needT = (G & (G_RES | G_QF)) != 0 || LP;
  const P2Const k = p2_const(beta, A2, B2, S2, lse_s);
  P2Acc acc = {0ull, 0ull, 0ull, 0ull, 0ull, 0ull};
  float gp0 = 0.f, gp1 = 0.f;  // the previous step's masses, reduced with this step's
  bool pending = false;
  for (int kr = 0; kr < rounds; kr += 2) {
    const int i0 = kr * kTThreads + static_cast<int>(threadIdx.x);
    const int i1 = i0 + kTThreads;
    float g0 = 0.f, g1 = 0.f;  // this thread's vector masses in rounds kr and kr + 1
    if (i0 < nv) {
      // TWO: both vectors present (all but the slice's last step)
      auto step = [&](auto two) {
        constexpr bool TWO = decltype(two)::value;
        f2 xa[NP], xb[NP], xt[NP], ya[NP], yb[NP], yt[NP];
        load_pairs(ra + i0 * VE, xa);
        load_pairs(rb + i0 * VE, xb);
        if (TWO) {
          load_pairs(ra + i1 * VE, ya);
          load_pairs(rb + i1 * VE, yb);
        } else {
          load_or_fill(ra + i1 * VE, false, ya);
          load_or_fill(rb + i1 * VE, false, yb);
        }
        if (needT) {
          load_pairs(rt + i0 * VE, xt);
          if (TWO) load_pairs(rt + i1 * VE, yt); else load_or_fill(rt + i1 * VE, false, yt);
        }
        p2_pair<NP, G, LP, DS, QSUM>(xa, xb, xt, ya, yb, yt, TWO, k, acc, g0, g1,
                               LP ? lp + i0 * VE : nullptr, LP ? lp + i1 * VE : nullptr);
      };
      if (i1 < nv) step(std::true_type{});
      else step(std::false_type{});
    }
    if (G & (G_RES | G_QF)) {
      // group masses leave the warp four rounds at a time
      if (pending) p2_groups4(gp0, gp1, g0, g1, grp, kr - 2, rounds);
      gp0 = g0;
      gp1 = g1;
      pending = !pending;
    }
  }
  if ((G & (G_RES | G_QF)) && pending) p2_groups(gp0, gp1, grp, ((rounds - 1) & ~1), rounds);
  p2_finish(acc, x);
}

// Pass 2 and the CTA combine; warp 0 stores the CTA's pass-2 record in the
// workspace (groups: this CTA's group masses there, stored by pass 2).
template <typename T, unsigned G, bool LP, int DS = ASYMSPEC_DELTA_AB, bool QSUM = true>
__device__ __forceinline__ void pass2_and_store(const T* ra, const T* rb, const T* rt, int nv,
                                                int rounds, float beta, float* lp, SharedTma* sh,
                                                float* rec, float* groups) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float lse_a = sh->lse[0], lse_b = sh->lse[1], lse_s = sh->lse[3];
  X2 x = x2_zero();
  pass2<T, G, LP, DS, QSUM>(ra, rb, rt, nv, rounds, beta, lse_a * kLog2e, lse_b * kLog2e,
                            lse_s * kLog2e, lse_s, x, lp, groups);
  warp_reduce_x2<G>(x);
  if (lane == 0) sh->w2[warp] = x;
  __syncthreads();
  if (warp == 0) {
    X2 w = (lane < kTWarps) ? sh->w2[lane] : x2_zero();
    warp_reduce_x2<G>(w);
    if (!QSUM && (G & G_RES)) w.Q = sh->qown;
    if (sh->broken) w.pad[0] = __uint_as_float(kBadTimeout);
    if (lane < static_cast<int>(sizeof(X2) / 16))
      reinterpret_cast<float4*>(rec)[lane] = reinterpret_cast<const float4*>(&w)[lane];
  }
}

// The divergence of Eq. 3 from the summed pass-2 records (nats).
template <unsigned G>
__device__ __forceinline__ float divergence_of(const X2& tot) {
  if (G & G_JSD) return 0.5f * kLn2 * (tot.j + tot.msum);
  if (G & G_KL) return kLn2 * tot.kl;
  return 0.f;
}

// ---------------------------------------------------------------- inverse-CDF walk

// Masses of vector v of a slice held in global memory, as pass 2 computes them.
template <typename T, int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ void slice_vector_masses(const T* ga, const T* gb, const T* gt, int v,
                                                    f2 beta2, f2 L2, f2 nA2, f2 nS2,
                                                    f2 (&p)[8 / sizeof(T)],
                                                    f2 (&qf)[8 / sizeof(T)],
                                                    f2 (&r)[8 / sizeof(T)]) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  f2 xa[NP], xb[NP], xt[NP];
  load_pairs(ga + v * VE, xa);
  load_pairs(gb + v * VE, xb);
  load_pairs(gt + v * VE, xt);
  vec_masses<NP, DS>(xa, xb, xt, beta2, L2, nA2, nS2, p, qf, r);
}

// The inverse-CDF draw inside one slice, by one warp: the smallest slice
// index (index order) whose cumulative residual (use_r) or fused mass
// exceeds tau, or the last index with positive mass when rounding leaves tau
// at or beyond the slice's total.  The slice (ga, gb, gt: global memory,
// entries from lo) is cut into groups of 32 vectors; gm holds their masses
// when `stored` (else they are recomputed: the rare fallback to the fused
// masses of a draft row whose residual is zero).  Lane l takes groups
// [l P, l P + P) (P = ceil(ngroups / 32) <= kWalkGroupsPerLane), then the lane
// holding the target recomputes its group's vectors, one per lane, and the
// element.  Returns the index within the row, or -1 when the slice holds no
// mass.
constexpr int kWalkGroupsPerLane = 8;  // slices of up to 256 groups (32 rounds)

template <typename T, bool GM_GLOBAL, int DS = ASYMSPEC_DELTA_AB>
__device__ __noinline__ int group_walk(const T* ga, const T* gb, const T* gt, int nvec, int lo,
                                       int ngroups, float beta, const float* gm, bool stored,
                                       bool use_r, float A2, float S2, float tau) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr int GP = kWalkGroupsPerLane;
  const int lane = threadIdx.x & 31;
  const int gpl = (ngroups + 31) / 32;
  const f2 beta2 = pk(beta, beta), L2 = pk(kLog2e, kLog2e);
  const f2 nA2 = pk(-A2, -A2), nS2 = pk(-S2, -S2);
  float gl[GP];
#pragma unroll
  for (int h = 0; h < GP; ++h) {
    const int g = gpl * lane + h;
    float m = 0.f;
    if (h < gpl && g < ngroups) {
      if (stored) {
        m = GM_GLOBAL ? __ldcg(gm + g) : gm[g];
      } else {
        for (int u = 0; u < 32; ++u) {
          const int v = 32 * g + u;
          if (v < nvec) {
            f2 p[NP], qf[NP], r[NP];
            slice_vector_masses<T, DS>(ga, gb, gt, v, beta2, L2, nA2, nS2, p, qf, r);
            m += vsum(use_r ? r : qf);
          }
        }
      }
    }
    gl[h] = m;
  }
  float pl = 0.f;
#pragma unroll
  for (int h = 0; h < GP; ++h) pl += gl[h];
  float incl = pl;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float v = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += v;
  }
  const float excl = incl - pl;
  bool take_last = false;
  const unsigned hit = __ballot_sync(0xffffffffu, pl > 0.f && excl <= tau && tau < incl);
  int lc;
  if (hit) {
    lc = __ffs(hit) - 1;
  } else {
    const unsigned pos = __ballot_sync(0xffffffffu, pl > 0.f);
    if (!pos) return -1;
    lc = 31 - __clz(pos);
    take_last = true;
  }
  // the group, within lane lc
  int gsel = -1;
  float trem = 0.f;
  if (lane == lc) {
    float cum = excl;
    int glast = -1;
#pragma unroll
    for (int h = 0; h < GP; ++h) {
      if (gl[h] > 0.f) glast = gpl * lane + h;
      if (h < gpl && !take_last && gsel < 0) {
        if (cum + gl[h] > tau) {
          gsel = gpl * lane + h;
          trem = fmaxf(tau - cum, 0.f);
        } else {
          cum += gl[h];
        }
      }
    }
    if (gsel < 0) {
      gsel = glast;
      take_last = true;
    }
  }
  gsel = __shfl_sync(0xffffffffu, gsel, lc);
  trem = __shfl_sync(0xffffffffu, trem, lc);
  take_last = __shfl_sync(0xffffffffu, take_last ? 1 : 0, lc) != 0;
  // the vector: lane u recomputes vector 32 gsel + u
  const int v = 32 * gsel + lane;
  f2 p[NP], qf[NP], r[NP];
  float mv = 0.f;
  if (v < nvec) {
    slice_vector_masses<T, DS>(ga, gb, gt, v, beta2, L2, nA2, nS2, p, qf, r);
    mv = vsum(use_r ? r : qf);
  }
  float vin = mv;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float w = __shfl_up_sync(0xffffffffu, vin, off);
    if (lane >= off) vin += w;
  }
  const float vex = vin - mv;
  const unsigned vh =
      __ballot_sync(0xffffffffu, !take_last && mv > 0.f && vex <= trem && trem < vin);
  int vc;
  if (vh) {
    vc = __ffs(vh) - 1;
  } else {
    const unsigned pos = __ballot_sync(0xffffffffu, mv > 0.f);
    if (!pos) return -1;
    vc = 31 - __clz(pos);
    take_last = true;
  }
  int found = -1;
  if (lane == vc) {
    const float te = fmaxf(trem - vex, 0.f);
    float cum = 0.f;
    int pick = -1, last = -1;
#pragma unroll
    for (int h = 0; h < NP; ++h) {
      float v0, v1;
      upk(use_r ? r[h] : qf[h], v0, v1);
      if (v0 > 0.f) last = 2 * h;
      cum += v0;
      if (!take_last && pick < 0 && cum > te) pick = 2 * h;
      if (v1 > 0.f) last = 2 * h + 1;
      cum += v1;
      if (!take_last && pick < 0 && cum > te) pick = 2 * h + 1;
    }
    if (pick < 0) pick = last;
    if (pick >= 0) found = lo + v * VE + pick;
  }
  return __shfl_sync(0xffffffffu, found, vc);
}

// The block of warp w in fuse_verify_row (kernel_row.cuh): vectors
// [w bw, min(nv, (w + 1) bw)) of the slice, bw = ceil(nv / NW); the warp's
// lane l takes vector w bw + 32 r + l in step r.
__host__ __device__ __forceinline__ int row_block_vectors(int nv, int nw) {
  return (nv + nw - 1) / nw;
}

// The inverse-CDF draw inside vectors [b0, b1) of a slice (one group of
// fuse_verify_row: a warp's block), by one warp: the smallest index whose
// cumulative residual (use_r) or fused mass exceeds trem, or with take_last
// (rounding left the target at or beyond the group's mass) the last index
// with positive mass.  The group's vectors of the three rows are first
// copied into the warp's staging area `stg` (16-byte cp.async, all in
// flight at once: one round trip; 3 x 32 ceil((b1 - b0) / 32) vectors), then
// their masses are scanned 32 vectors at a time in index order; the masses
// are formed exactly as the row kernel's pass 2 forms them.  Returns the
// index within the row, or -1 if the group holds no mass.
template <typename T>
__device__ __noinline__ int walk_vectors(const T* ga, const T* gb, const T* gt, int b0, int b1,
                                         int lo, float beta, bool use_r, float A2, float S2,
                                         float trem, bool take_last, uint4* stg) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  const int lane = threadIdx.x & 31;
  const f2 beta2 = pk(beta, beta), L2 = pk(kLog2e, kLog2e);
  const f2 nA2 = pk(-A2, -A2), nS2 = pk(-S2, -S2);
  // staging: vector j of the group (vector b0 + j of the slice) of stream
  // a, b, t at stg[j], stg[cap + j], stg[2 cap + j]
  const int nvb = max(0, b1 - b0), cap = (nvb + 31) & ~31;
  T* sa = reinterpret_cast<T*>(stg);
  T* sb = reinterpret_cast<T*>(stg + cap);
  T* st = reinterpret_cast<T*>(stg + 2 * cap);
  for (int j = lane; j < nvb; j += 32) {
    cp_async16(sa + j * VE, ga + (b0 + j) * VE);
    cp_async16(sb + j * VE, gb + (b0 + j) * VE);
    cp_async16(st + j * VE, gt + (b0 + j) * VE);
  }
  cp_async_wait_all();
  __syncwarp();
  float mvs[kWalkRounds];
#pragma unroll
  for (int s = 0; s < kWalkRounds; ++s) {
    const int j = 32 * s + lane;
    mvs[s] = 0.f;
    if (j < nvb) {
      f2 p[NP], qf[NP], r[NP];
      slice_vector_masses<T>(sa, sb, st, j, beta2, L2, nA2, nS2, p, qf, r);
      mvs[s] = vsum(use_r ? r : qf);
    }
  }
  float run = 0.f;
  int vsel = -1, vlast = -1;
  float tin = 0.f;  // the target's offset inside the selected vector
#pragma unroll
  for (int s = 0; s < kWalkRounds; ++s) {
    const int base = b0 + 32 * s;
    if (base >= b1 || vsel >= 0) break;
    const float mv = mvs[s];
    float vin = mv;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float w = __shfl_up_sync(0xffffffffu, vin, off);
      if (lane >= off) vin += w;
    }
    const float vex = vin - mv;
    const unsigned pos = __ballot_sync(0xffffffffu, mv > 0.f);
    if (pos) vlast = base + 31 - __clz(pos);
    const unsigned vh = __ballot_sync(0xffffffffu, !take_last && mv > 0.f && run + vex <= trem &&
                                                       trem < run + vin);
    if (vh) {
      const int vc = __ffs(vh) - 1;
      vsel = base + vc;
      tin = fmaxf(trem - run - __shfl_sync(0xffffffffu, vex, vc), 0.f);
    }
    run += __shfl_sync(0xffffffffu, vin, 31);
  }
  if (vsel < 0) {  // rounding left the target beyond the group: its last positive vector
    if (vlast < 0) return -1;
    vsel = vlast;
    take_last = true;
  }
  int found = -1;
  if (lane == 0) {
    f2 p[NP], qf[NP], r[NP];
    slice_vector_masses<T>(sa, sb, st, vsel - b0, beta2, L2, nA2, nS2, p, qf, r);
    float cum = 0.f;
    int pick = -1, last = -1;
#pragma unroll
    for (int h = 0; h < NP; ++h) {
      float m0, m1;
      upk(use_r ? r[h] : qf[h], m0, m1);
      if (m0 > 0.f) last = 2 * h;
      cum += m0;
      if (!take_last && pick < 0 && cum > tin) pick = 2 * h;
      if (m1 > 0.f) last = 2 * h + 1;
      cum += m1;
      if (!take_last && pick < 0 && cum > tin) pick = 2 * h + 1;
    }
    if (pick < 0) pick = last;
    if (pick >= 0) found = lo + vsel * VE + pick;
  }
  return __shfl_sync(0xffffffffu, found, 0);
}

// ---------------------------------------------------------------- the kernel

// Per-row values the row programs share.
struct RowCtx {
  const void* sa;
  const void* sb;
  const void* st;
  int nv, rounds, rc, lo, n, W, rank, C, k, bi;
  long long row;
  bool bonus;
  int dtok;           // warp 0 only: the row's draft token (-1 on the bonus row)
  SharedTma* sh;
};

// Rank 0: what pass 1 leaves for the row's decision.
__device__ __forceinline__ void store_row_stat(const KParams& P, long long row,
                                               const float (&lse)[4], int is, int it,
                                               unsigned bad, int dtok, float ad, float bd,
                                               float td) {
  RowStat st;
#pragma unroll
  for (int q = 0; q < 4; ++q) st.lse[q] = lse[q];
  st.is = is;
  st.it = it;
  st.bad = bad;
  st.dtok = dtok;
  st.da = ad;
  st.db = bd;
  st.dt = td;
  st.pad = 0.f;
  static_cast<RowStat*>(P.row_stat)[row] = st;
}

// One row with pass-1 program F and pass-2 program G (R2: pass 2 runs; LP:
// it writes the fused log-probs).
template <typename T, bool STOCH, unsigned F, unsigned G, bool LP, bool R2,
          int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ void run_row(const KParams& P, const RowCtx& c,
                                        cg::cluster_group& cluster) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const T* ra = static_cast<const T*>(c.sa);
  const T* rb = static_cast<const T*>(c.sb);
  const T* rt = static_cast<const T*>(c.st);
  SharedTma* sh = c.sh;
  const float beta = P.beta;
  // the residual rows of the production programs take their fused mass (used
  // only when the whole residual is zero) from pass 1; the full program (the
  // only one with F_AT and pass 2) sums it in pass 2, for every row alike
  constexpr bool QSUM = !((G & G_RES) && !(F & F_AT) && (F & F_LS));
  pass1_and_push<T, F, DS>(ra, rb, rt, c.nv, c.rounds, c.rc, c.lo, c.n, beta, c.dtok, sh, c.rank,
                           c.C, cluster);
  if constexpr (!R2) {
    // no pass 2: rank 0 leaves the row's pass-1 results for the decision kernel
    if (c.rank == 0 && warp == 0) {
      float lse[4];
      const X1 w = combine_pass1<F>(sh, c.C, lse);
      float ad, bd, td;
      draft_logits(sh, c.dtok, c.W, c.C, ad, bd, td);
      if (lane == 0) store_row_stat(P, c.row, lse, w.is, w.it, w.bad, c.dtok, ad, bd, td);
    }
    return;
  } else {
    if (warp == 0) {
      float lse[4];
      const X1 w = combine_pass1<F>(sh, c.C, lse);
      if (lane == 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) sh->lse[q] = lse[q];
        if (!QSUM) {
          // this slice's fused mass sum exp(s - LSE(s)), from its own pass-1 record
          const X1& own = sh->recv1()[c.rank];
          sh->qown = own.s[3] * ex2((own.ref[3] - lse[3]) * kLog2e);
        }
        if (c.rank == 0) {
          float ad, bd, td;
          draft_logits(sh, c.dtok, c.W, c.C, ad, bd, td);
          store_row_stat(P, c.row, lse, w.is, w.it, w.bad, c.dtok, ad, bd, td);
        }
      }
    }
    __syncthreads();
    float* lp = LP ? P.logprobs + static_cast<size_t>(c.row) * P.V + c.lo : nullptr;
    const size_t slot = static_cast<size_t>(c.row) * c.C + c.rank;
    pass2_and_store<T, G, LP, DS, QSUM>(ra, rb, rt, c.nv, c.rounds, beta, lp, sh,
                                        P.pass2_rec + slot * 8,
                                        P.group_mass + slot * P.group_stride);
  }
}

template <typename T, bool STOCH, unsigned F, unsigned RQ, int DS = ASYMSPEC_DELTA_AB>
__device__ __forceinline__ void run_full(const KParams& P, const RowCtx& c,
                                         cg::cluster_group& cluster) {
  const bool jsd = P.divergence == ASYMSPEC_DIV_JSD;
  const bool klg = P.divergence == ASYMSPEC_DIV_KL;
  if (P.logprobs) {
    if (jsd) run_row<T, STOCH, F, G_JSD | RQ, true, true, DS>(P, c, cluster);
    else if (klg) run_row<T, STOCH, F, G_KL | RQ, true, true, DS>(P, c, cluster);
    else run_row<T, STOCH, F, RQ, true, true, DS>(P, c, cluster);
  } else {
    if (jsd) run_row<T, STOCH, F, G_JSD | RQ, false, true, DS>(P, c, cluster);
    else if (klg) run_row<T, STOCH, F, G_KL | RQ, false, true, DS>(P, c, cluster);
    else run_row<T, STOCH, F, RQ, false, true, DS>(P, c, cluster);
  }
}

// Program set 0: every row program, chosen at run time, for delta source DS.
template <typename T, bool STOCH, int DS>
__device__ __forceinline__ void run_any(const KParams& P, const RowCtx& c, bool bonus,
                                        cg::cluster_group& cluster) {
  if (P.full) {
    run_full<T, STOCH, F_LA | F_LB | F_LT | F_LS | F_AS | F_AT, STOCH ? G_RES : 0u, DS>(P, c, cluster);
  } else if (!STOCH) {
    const bool jsd = P.divergence == ASYMSPEC_DIV_JSD;
    const bool klg = P.divergence == ASYMSPEC_DIV_KL;
    constexpr unsigned FD = F_LA | F_LB | F_LT | F_AS;
    if (bonus) {
      if (P.fuse_bonus) run_row<T, STOCH, F_AS, 0, false, false, DS>(P, c, cluster);
      else run_row<T, STOCH, F_AT, 0, false, false, DS>(P, c, cluster);
    } else if (jsd) {
      run_row<T, STOCH, FD, G_JSD, false, true, DS>(P, c, cluster);
    } else if (klg) {
      run_row<T, STOCH, FD, G_KL, false, true, DS>(P, c, cluster);
    } else {
      run_row<T, STOCH, FD, 0, false, false, DS>(P, c, cluster);
    }
  } else if (!bonus) {
    const bool jsd = P.divergence == ASYMSPEC_DIV_JSD;
    const bool klg = P.divergence == ASYMSPEC_DIV_KL;
    if (P.want_tokens) {
      constexpr unsigned FS = F_LA | F_LB | F_LS | F_AS;
      if (jsd) run_row<T, STOCH, FS, G_JSD | G_RES, false, true, DS>(P, c, cluster);
      else if (klg) run_row<T, STOCH, FS, G_KL | G_RES, false, true, DS>(P, c, cluster);
      else run_row<T, STOCH, FS, G_RES, false, true, DS>(P, c, cluster);
    } else {
      constexpr unsigned FS = F_LA | F_LB | F_LS;
      if (jsd) run_row<T, STOCH, FS, G_JSD | G_RES, false, true, DS>(P, c, cluster);
      else if (klg) run_row<T, STOCH, FS, G_KL | G_RES, false, true, DS>(P, c, cluster);
      else run_row<T, STOCH, FS, G_RES, false, true, DS>(P, c, cluster);
    }
  } else {
    if (P.want_tokens) run_row<T, STOCH, F_LS | F_AS, G_QF, false, true, DS>(P, c, cluster);
    else run_row<T, STOCH, F_LS, G_QF, false, true, DS>(P, c, cluster);
  }

}

// Program sets.  SEL 0 chooses among every row program at run time (debug
// outputs, per-row tokens, any gate, any delta source).  SEL > 0 compiles
// only the two
// programs of one production configuration (draft rows, bonus row), which
// keeps the instruction footprint of the two CTAs an SM runs small:
//   stochastic  SEL = 1 + d
//   greedy      SEL = 1 + d + 3 fuse_bonus
// with d = 0 for the JSD gate, 1 for KL, 2 for none or lambda.
constexpr int kTmaProgramSets = 7;

__host__ __device__ constexpr int tma_program_set(bool stoch, int divergence, bool fuse_bonus,
                                                  bool full, bool want_tokens, int delta_src) {
  return (full || (stoch && want_tokens) || delta_src != ASYMSPEC_DELTA_AB)
             ? 0
             : 1 + (divergence == ASYMSPEC_DIV_JSD ? 0 : divergence == ASYMSPEC_DIV_KL ? 1 : 2) +
                   ((!stoch && fuse_bonus) ? 3 : 0);
}

// One cluster of C CTAs per row (grid = rows x C); CTA r of the cluster
// takes entries [r W, (r+1) W) of the row.
template <typename T, bool STOCH, int SEL>
__global__ void __launch_bounds__(kTThreads, 2) fuse_verify_tma(const KParams P) {
  // the decision kernel (a programmatic dependent) may be scheduled once
  // every CTA of this grid has started; it waits for this grid's completion
  // before it reads anything the grid writes
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  extern __shared__ __align__(128) unsigned char smem_tma[];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int tid = threadIdx.x;
  const int C = P.C;
  // 32-bit row arithmetic: the host keeps rows x C below 2^31
  const unsigned row32 = blockIdx.x / static_cast<unsigned>(C);
  const unsigned K1 = static_cast<unsigned>(P.K) + 1u;
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
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
  const int bi = static_cast<int>(row32 / K1);
  const int k = static_cast<int>(row32 - static_cast<unsigned>(bi) * K1);
  const bool bonus = (k == P.K);

  if (tid == 0) {
#pragma unroll
    for (int q = 0; q < kChunks; ++q) mbar_init(&sh->bar[q], 1);
    sh->broken = 0;
    sh->wait_ns = P.copy_wait_ns;
    fence_mbar_init();
    // a greedy bonus row without fused bonus needs t alone (Algorithm 1 emits argmax t)
    const bool only_t = !STOCH && !P.full && bonus && !P.fuse_bonus;
    issue_slice<T>(P, sh, row32, lo, nv, rc, sa, sb, st, only_t);
  }
  RowCtx c;
  c.sa = sa;
  c.sb = sb;
  c.st = st;
  c.nv = nv;
  c.rounds = rounds;
  c.rc = rc;
  c.lo = lo;
  c.n = n;
  c.W = W;
  c.rank = rank;
  c.C = C;
  c.sh = sh;
  c.k = k;
  c.bi = bi;
  c.row = row32;
  c.bonus = bonus;
  // warp 0 keeps the row's draft token, loaded while the slice is in flight
  c.dtok = -1;
  if ((tid >> 5) == 0 && !bonus) c.dtok = P.tokens[static_cast<size_t>(bi) * P.K + k];
  __syncthreads();  // the chunk barriers are initialised

  if constexpr (SEL > 0 && STOCH) {
    constexpr int d = SEL - 1;
    constexpr unsigned GD = d == 0 ? G_JSD : d == 1 ? G_KL : 0u;
    if (!bonus)
      run_row<T, STOCH, F_LA | F_LB | F_LS, GD | G_RES, false, true, ASYMSPEC_DELTA_AB>(P, c,
                                                                                     cluster);
    else
      run_row<T, STOCH, F_LS, G_QF, false, true, ASYMSPEC_DELTA_AB>(P, c, cluster);
  } else if constexpr (SEL > 0) {
    constexpr int d = (SEL - 1) % 3;
    constexpr bool fused_bonus = SEL > 3;
    constexpr unsigned FD = F_LA | F_LB | F_LT | F_AS;
    if (bonus) {
      if (fused_bonus) run_row<T, STOCH, F_AS, 0, false, false, ASYMSPEC_DELTA_AB>(P, c, cluster);
      else run_row<T, STOCH, F_AT, 0, false, false, ASYMSPEC_DELTA_AB>(P, c, cluster);
    } else if (d == 0) {
      run_row<T, STOCH, FD, G_JSD, false, true, ASYMSPEC_DELTA_AB>(P, c, cluster);
    } else if (d == 1) {
      run_row<T, STOCH, FD, G_KL, false, true, ASYMSPEC_DELTA_AB>(P, c, cluster);
    } else {
      run_row<T, STOCH, FD, 0, false, false, ASYMSPEC_DELTA_AB>(P, c, cluster);
    }
  } else if (P.delta_src == ASYMSPEC_DELTA_A) {
    run_any<T, STOCH, ASYMSPEC_DELTA_A>(P, c, bonus, cluster);
  } else if (P.delta_src == ASYMSPEC_DELTA_TB) {
    run_any<T, STOCH, ASYMSPEC_DELTA_TB>(P, c, bonus, cluster);
  } else {
    run_any<T, STOCH, ASYMSPEC_DELTA_AB>(P, c, bonus, cluster);
  }

  // a copy that timed out may still land: wait for it (bounded, always with
  // the normal limit) before exit
  if (tid == 0 && sh->broken) {
#pragma unroll
    for (int q = 0; q < kChunks; ++q) mbar_wait_bounded(&sh->bar[q], 0u, kCopyTimeoutNs);
  }
}

// ---------------------------------------------------------------- row decisions

constexpr int kDecideThreads = 512;  // at most 16 warps; each takes rows k, k + 16, ...
constexpr int kDecideSmemRows = 64;  // rows of an element whose records the scan reads from shared memory

// ---- rows of fuse_verify_row (kernel_row.cuh): one pass-2 record per warp
// block, each block one inverse-CDF group

constexpr int kRowMaxWarps = 8;  // warps per CTA of fuse_verify_row; records per CTA

// What the decision of row (bi, k) needs from the kernel's inputs (not from
// the row kernel): the draft token, its three logits, the row's scalars.
// Loaded before griddepcontrol.wait, so that the loads overlap the row
// kernel's last CTAs.
struct RowInputs {
  int dtok;
  float ad, bd, td;
  RowScalars sc;
};

template <typename T>
__device__ __forceinline__ RowInputs load_row_inputs(const KParams& P, int bi, int k) {
  RowInputs d;
  d.dtok = -1;
  d.ad = d.bd = d.td = 0.f;
  d.sc = load_row_scalars(P, bi, k);
  if (k < P.K) {
    d.dtok = P.tokens[static_cast<size_t>(bi) * P.K + k];
    if (d.dtok >= 0 && d.dtok < P.V) {
      const size_t o = (static_cast<size_t>(bi) * (P.K + 1) + k) * P.V + d.dtok;
      d.ad = to_f32(static_cast<const T*>(P.a)[o]);
      d.bd = to_f32(static_cast<const T*>(P.b)[o]);
      d.td = to_f32(static_cast<const T*>(P.t)[o]);
    }
  }
  return d;
}

// The row's results from its C x NW warp records (one warp): the divergence
// of Eq. 3 and the inverse-CDF draw at u_K (the residual's groups, or the
// fused masses when the whole residual is zero and on the bonus row).  Lane
// l takes groups 4l .. 4l + 3 (group g = warp g % NW of rank g / NW, in index
// order), the lane holding the target picks the group, walk_vectors the
// element.
template <typename T>
__device__ __forceinline__ RowResult block_row_result(const KParams& P, int k, long long row,
                                                      const RowScalars& sc, uint4* stg) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const int lane = threadIdx.x & 31;
  const int C = P.C, NW = P.tma_threads / 32, ng = C * NW;
  const bool bonus = (k == P.K);
  // (read from L2: another CTA wrote it during this launch)
  RowStat st;
  {
    const float4* src = reinterpret_cast<const float4*>(static_cast<const RowStat*>(P.row_stat) + row);
    float4* dst = reinterpret_cast<float4*>(&st);
    dst[0] = __ldcg(src);
    dst[1] = __ldcg(src + 1);
    dst[2] = __ldcg(src + 2);
  }
  float j = 0.f, Rm[4], Qm[4];
  bool late = false;
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    const int g = 4 * lane + h;
    Rm[h] = Qm[h] = 0.f;
    if (g < ng) {
      const int r = g / NW, w = g - r * NW;
      const float4* rec = reinterpret_cast<const float4*>(
          P.pass2_rec + ((static_cast<size_t>(row) * C + r) * kRowMaxWarps + w) * 8);
      const float4 x0 = __ldcg(rec), x1 = __ldcg(rec + 1);
      j += x0.x;
      Rm[h] = x0.w;
      Qm[h] = x1.x;
      late = late || __float_as_uint(x1.y) != 0u;
    }
  }
  RowResult rr;
  rr.lse_a = bonus ? NAN : st.lse[0];
  rr.lse_b = bonus ? NAN : st.lse[1];
  rr.lse_t = NAN;
  rr.lse_s = st.lse[3];
  rr.D = bonus ? 0.f : 0.5f * kLn2 * warp_sum(j);  // j sums 2 JSD in bits
  rr.is = rr.it = INT_MAX;
  rr.bad = st.bad | (__any_sync(0xffffffffu, late) ? kBadTimeout : 0u);
  rr.have_lse_t = false;
  const float Rl = (Rm[0] + Rm[1]) + (Rm[2] + Rm[3]), Ql = (Qm[0] + Qm[1]) + (Qm[2] + Qm[3]);
  const float R_all = warp_sum(Rl), Q_all = warp_sum(Ql);
  const bool r_ok = !bonus && R_all > 0.f;
  const float ml = r_ok ? Rl : Ql, total = r_ok ? R_all : Q_all;
  rr.mass = total;
  const float tau = sc.u_last * total;
  float incl = ml;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float v = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += v;
  }
  const float excl = incl - ml;
  bool take_last = false;
  const unsigned hit = __ballot_sync(0xffffffffu, ml > 0.f && excl <= tau && tau < incl);
  int lc;
  if (hit) {
    lc = __ffs(hit) - 1;
  } else {
    const unsigned pos = __ballot_sync(0xffffffffu, ml > 0.f);
    if (!pos) {
      rr.sample = -1;
      return rr;
    }
    lc = 31 - __clz(pos);
    take_last = true;
  }
  // the group, inside lane lc's four
  int gsel = -1, glast = -1;
  float trem = 0.f;
  if (lane == lc) {
    float cum = excl;
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      const float m = r_ok ? Rm[h] : Qm[h];
      if (m > 0.f) glast = 4 * lane + h;
      if (!take_last && gsel < 0) {
        if (m > 0.f && cum + m > tau) {
          gsel = 4 * lane + h;
          trem = fmaxf(tau - cum, 0.f);
        } else {
          cum += m;
        }
      }
    }
    if (gsel < 0) {
      gsel = glast;
      take_last = true;
    }
  }
  gsel = __shfl_sync(0xffffffffu, gsel, lc);
  trem = __shfl_sync(0xffffffffu, trem, lc);
  take_last = __shfl_sync(0xffffffffu, take_last ? 1 : 0, lc) != 0;
  const int r = gsel / NW, w = gsel - r * NW;
  const int lo_r = r * P.W;
  const int nv_r = max(0, min(P.W, P.V - lo_r)) / VE;
  const int bw = row_block_vectors(nv_r, NW);
  const int b0 = min(nv_r, w * bw), b1 = min(nv_r, b0 + bw);
  const size_t off = static_cast<size_t>(row) * P.V + lo_r;
  rr.sample = walk_vectors<T>(static_cast<const T*>(P.a) + off, static_cast<const T*>(P.b) + off,
                              static_cast<const T*>(P.t) + off, b0, b1, lo_r, P.beta, r_ok,
                              st.lse[0] * kLog2e, st.lse[3] * kLog2e, trem, take_last, stg);
  return rr;
}

// The decisions of one batch element's K+1 rows (one CTA per element, one
// warp per row) from what fuse_verify_tma left in the workspace, then
// Algorithm 1's scan over them in shared memory.  Per row: the divergence
// (Eq. 3) from the C pass-2 records; in stochastic mode the CTA whose slice
// holds the inverse-CDF target (prefix over ranks) and the draw inside it
// (group_walk, reading that slice back from L2); the acceptance test and
// the emitted candidate (row_record, kept in the workspace's records).
template <typename T, bool STOCH>
__global__ void __launch_bounds__(kDecideThreads) decide_rows(const KParams P) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const int bi = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int K = P.K, K1 = K + 1, C = P.C;
  const bool jsd = P.divergence == ASYMSPEC_DIV_JSD;
  const bool klg = P.divergence == ASYMSPEC_DIV_KL;
  __shared__ int4 srec[kDecideSmemRows];  // the element's records (K + 1 <= kDecideSmemRows)
  // rows of fuse_verify_row: each warp's staging area for its walks
  extern __shared__ uint4 walk_stage[];
  uint4* stg = walk_stage + static_cast<size_t>(warp) * (P.walk_stage / 16);
  // the kernel inputs of this warp's first row, loaded before the wait
  RowInputs pre{-1, 0.f, 0.f, 0.f, RowScalars{0.f, 0.f, 0.f}};
  if (STOCH && P.row_blocks && warp < K1) pre = load_row_inputs<T>(P, bi, warp);
  // launched as a programmatic dependent of the row kernel: its CTAs may
  // start early; nothing of the workspace is read before that kernel is done
  asm volatile("griddepcontrol.wait;" ::: "memory");
  for (int k = warp; k < K1; k += nw) {
    const long long row = static_cast<long long>(bi) * K1 + k;
    if constexpr (STOCH) {
      if (P.row_blocks) {  // a row of fuse_verify_row
        const RowInputs din = (k == warp) ? pre : load_row_inputs<T>(P, bi, k);
        const RowResult rr = block_row_result<T>(P, k, row, din.sc, stg);
        if (lane == 0) {
          const int4 rec = row_record<true>(P, row, k, rr, din.dtok, din.ad, din.bd, din.td, din.sc);
          P.recs[row] = rec;
          if (k < kDecideSmemRows) srec[k] = rec;
        }
        continue;
      }
    }
    const bool bonus = (k == K);
    const bool pass2 = STOCH || P.full || (!bonus && (jsd || klg));
    RowStat st = static_cast<const RowStat*>(P.row_stat)[row];
    X2 w = x2_zero();
    if (pass2 && lane < C) w = reinterpret_cast<const X2*>(P.pass2_rec)[row * C + lane];
    const unsigned late = __ballot_sync(0xffffffffu, pass2 && lane < C &&
                                                         __float_as_uint(w.pad[0]) != 0u);
    if (late) st.bad |= kBadTimeout;
    const float j = warp_sum(w.j), msum = warp_sum(w.msum), kl = warp_sum(w.kl);
    float D = 0.f;
    if (pass2 && jsd) D = 0.5f * kLn2 * (j + msum);
    else if (pass2 && klg) D = kLn2 * kl;
    int sample = -1;
    float mass_total = NAN;
    const RowScalars sc = STOCH ? load_row_scalars(P, bi, k) : RowScalars{0.f, 0.f, 0.f};
    if constexpr (STOCH) {
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
      const bool r_ok = !bonus && (R_all > 0.f);
      const float incl = r_ok ? incl_R : incl_Q;
      const float mass = r_ok ? w.R : w.Q;
      const float total = r_ok ? R_all : Q_all;
      mass_total = total;
      const float tau = sc.u_last * total;
      const unsigned over = __ballot_sync(0xffffffffu, lane < C && incl > tau);
      const unsigned pos = __ballot_sync(0xffffffffu, lane < C && mass > 0.f);
      int owner = -1;
      if (over) owner = __ffs(over) - 1;
      else if (pos) owner = 31 - __clz(pos);
      if (owner >= 0) {
        const float incl_o = __shfl_sync(0xffffffffu, incl, owner);
        const float mass_o = __shfl_sync(0xffffffffu, mass, owner);
        const float tau_local = fmaxf(tau - (incl_o - mass_o), 0.f);
        const int lo_o = owner * P.W;
        const int nv_o = max(0, min(P.W, P.V - lo_o)) / VE;
        const int ng_o = ((nv_o + P.tma_threads - 1) / P.tma_threads) * (P.tma_threads / 32);
        const size_t off = static_cast<size_t>(row) * P.V + lo_o;
        // the group masses are residual ones for draft rows and fused ones for
        // the bonus row; the other kind (a draft row whose residual is zero)
        // is recomputed exactly as pass 2 computes it
        const bool stored_r = !bonus || P.full;
        const T* ga = static_cast<const T*>(P.a) + off;
        const T* gb = static_cast<const T*>(P.b) + off;
        const T* gt = static_cast<const T*>(P.t) + off;
        const float* gm = P.group_mass + (row * C + owner) * P.group_stride;
        const float A2 = st.lse[0] * kLog2e, S2 = st.lse[3] * kLog2e;
        const bool stored = r_ok == stored_r;
        if (P.delta_src == ASYMSPEC_DELTA_A)
          sample = group_walk<T, true, ASYMSPEC_DELTA_A>(ga, gb, gt, nv_o, lo_o, ng_o, P.beta, gm,
                                                         stored, r_ok, A2, S2, tau_local);
        else if (P.delta_src == ASYMSPEC_DELTA_TB)
          sample = group_walk<T, true, ASYMSPEC_DELTA_TB>(ga, gb, gt, nv_o, lo_o, ng_o, P.beta, gm,
                                                          stored, r_ok, A2, S2, tau_local);
        else
          sample = group_walk<T, true>(ga, gb, gt, nv_o, lo_o, ng_o, P.beta, gm, stored, r_ok, A2,
                                       S2, tau_local);
      }
    }
    const bool has_ab = P.full || !bonus;
    const bool has_t = P.full || (!STOCH && !bonus);
    RowResult r;
    r.lse_a = has_ab ? st.lse[0] : NAN;
    r.lse_b = has_ab ? st.lse[1] : NAN;
    r.lse_t = has_t ? st.lse[2] : NAN;
    r.lse_s = (P.full || STOCH) ? st.lse[3] : NAN;
    r.D = D;
    r.is = st.is;
    r.it = st.it;
    r.sample = sample;
    r.mass = mass_total;
    r.bad = st.bad;
    r.have_lse_t = has_t;
    if (lane == 0) {
      const int4 rec = row_record<STOCH>(P, row, k, r, st.dtok, st.da, st.db, st.dt, sc);
      P.recs[row] = rec;
      if (k < kDecideSmemRows) srec[k] = rec;
    }
  }
  __syncthreads();  // the element's records are visible to the block
  const int4* recs = P.recs + static_cast<size_t>(bi) * K1;
  const bool in_smem = K1 <= kDecideSmemRows;
  if (warp != 0) return;
  // Algorithm 1: the first rejected draft, or K if none; any data error voids the element
  bool any_err = false;
  int len = -1, next = -1;
  for (int base = 0; base < K1; base += 32) {
    const int j = base + lane;
    int4 v = make_int4(1, -1, 0, 0);
    if (j < K1) v = in_smem ? srec[j] : __ldcg(&recs[j]);
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
  }
}

}  // namespace asymspec_impl
