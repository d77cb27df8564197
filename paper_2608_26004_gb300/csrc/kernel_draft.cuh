// The augmented drafter's draw (Section 3.2, item 1; the drafting step of
// Algorithm 1): per position, greedy d = argmax a (lowest index on ties) or,
// sampling, the inverse CDF of softmax(a) at the position's uniform, plus
// the drafter's probability of its draw, softmax(a)[d].
//
// One cluster of C CTAs (1 <= C <= 8) per row: CTA c owns the vectors
// [c W, (c + 1) W) of the row (VE elements each; the last slice may be
// shorter or empty).  In a slice, vector v0 + r kDThreads + t is handled by
// thread t in round r, kDUnroll rounds' loads issued before any is used (in
// sampling, the next kDUnroll rounds' too).
// Each CTA reads its slice once from HBM and pushes a summary (reference,
// mass relative to it, finiteness sum, argmax index) into every CTA of the
// cluster; after one cluster barrier every CTA combines the C summaries
// locally and identically, so no shared memory is read remotely.
//   greedy    per thread a running maximum, the lowest vector that holds it
//             and the sum of 2^((x - m) log2 e), rescaled when the maximum
//             moves.  Rank 0 writes d (the lowest index holding the row
//             maximum) and softmax(a)[d] = 1 / S.
//   sampling  one pass: every warp takes as its reference R_w the maximum of
//             its first round's vectors and stores the mass 2^((x - R_w)
//             log2 e) of each group of 32 consecutive vectors (one warp in one
//             round) in shared memory.  If any group's mass reaches 2^100 (an
//             entry ~69 nats above its warp's reference) the CTA redoes the
//             slice against the slice maximum.  Combining: the row reference
//             R is the largest R_w; the CTA whose slice holds the target u S
//             (S in units of 2^R) walks its groups, the 32 vectors of the
//             group (recomputed against R) and the elements of the vector.
//             If rounding leaves the target at or past a boundary with no
//             owner, the last entry of positive mass is taken.
// Non-finite data: every element also enters f = sum x 2^-40, finite
// exactly when all elements are (2^-40 keeps 2^20 fp32 maxima finite).  A
// row with a non-finite logit, or a uniform outside [0, 1), gets token -1
// and probability NaN.
#pragma once

#include "device_common.cuh"

namespace asymspec_impl {

constexpr int kDThreads = 256;
constexpr int kDWarps = kDThreads / 32;
constexpr int kDUnroll = 4;
constexpr int kDMaxCluster = 8;
constexpr float kDFinScale = 9.094947017729282e-13f;  // 2^-40
constexpr float kDGuard = 1.2676506002282294e30f;     // 2^100

struct DParams {
  const void* logits;  // [rows, V], row stride V
  const float* unif;   // [rows] (sampling)
  int32_t* tokens;     // [rows]
  float* probs;        // [rows]
  int rows, V, nv;     // nv = V / VE vectors per row
  int W;               // vectors per CTA slice
};

// A CTA's summary of its slice.
struct __align__(16) DSlice {
  float ref;  // greedy: the slice maximum; sampling: the largest warp reference
  float sum;  // sum of 2^((x - ref) log2 e) over the slice
  float fin;  // sum of x 2^-40 over the slice
  int idx;    // greedy: lowest element index holding the maximum (INT_MAX if none)
};

struct DShared {
  DSlice slot[kDMaxCluster];  // slot c: CTA c's summary (pushed by CTA c)
  float red[2 * kDWarps];
  int redi[kDWarps];
  float wref[kDWarps];    // sampling: the warps' references
  float wscale[kDWarps];  // sampling: 2^((R_w - R) log2 e)
};

__device__ __forceinline__ float dwarp_max(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

__device__ __forceinline__ float dwarp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ float dwarp_incl_scan(float v, int lane) {
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, v, off);
    if (lane >= off) v += y;
  }
  return v;
}

// A vector of VE consecutive logits as loaded: 8 packed bf16, 4 fp32, or one
// element of either type (widened on load).
template <typename T, int VE>
struct DRaw;
template <>
struct DRaw<__nv_bfloat16, 8> {
  uint4 q;
};
template <>
struct DRaw<float, 4> {
  float4 q;
};
template <typename T>
struct DRaw<T, 1> {
  float x;
};

__device__ __forceinline__ void dld(const __nv_bfloat16* row, int v, DRaw<__nv_bfloat16, 8>& r) {
  r.q = __ldg(reinterpret_cast<const uint4*>(row) + v);
}
__device__ __forceinline__ void dld(const float* row, int v, DRaw<float, 4>& r) {
  r.q = __ldg(reinterpret_cast<const float4*>(row) + v);
}
__device__ __forceinline__ void dld(const float* row, int v, DRaw<float, 1>& r) { r.x = __ldg(row + v); }
__device__ __forceinline__ void dld(const __nv_bfloat16* row, int v, DRaw<__nv_bfloat16, 1>& r) {
  r.x = __uint_as_float(static_cast<unsigned>(__ldg(reinterpret_cast<const unsigned short*>(row) + v))
                        << 16);
}

// The vector widened to fp32.
__device__ __forceinline__ void dwiden(const DRaw<__nv_bfloat16, 8>& r, float (&x)[8]) {
  const unsigned w[4] = {r.q.x, r.q.y, r.q.z, r.q.w};
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    x[2 * h] = __uint_as_float(w[h] << 16);
    x[2 * h + 1] = __uint_as_float(w[h] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void dwiden(const DRaw<float, 4>& r, float (&x)[4]) {
  x[0] = r.q.x;
  x[1] = r.q.y;
  x[2] = r.q.z;
  x[3] = r.q.w;
}
template <typename T>
__device__ __forceinline__ void dwiden(const DRaw<T, 1>& r, float (&x)[1]) {
  x[0] = r.x;
}

// The finiteness sum f = sum x 2^-40: packed bf16 pairs for bf16 vectors
// (non-finite values propagate through bf16 arithmetic as through fp32), fp32
// pairs for fp32 vectors.
template <typename T, int VE>
struct DFin;
template <>
struct DFin<__nv_bfloat16, 8> {
  unsigned acc = 0u;  // two bf16 partial sums
  __device__ __forceinline__ void add(const DRaw<__nv_bfloat16, 8>& r) {
    const unsigned scale = 0x2B802B80u;  // 2^-40 in both halves
    const unsigned w[4] = {r.q.x, r.q.y, r.q.z, r.q.w};
#pragma unroll
    for (int h = 0; h < 4; ++h) asm("fma.rn.bf16x2 %0, %1, %2, %0;" : "+r"(acc) : "r"(w[h]), "r"(scale));
  }
  __device__ __forceinline__ float value() const {
    return __uint_as_float(acc << 16) + __uint_as_float(acc & 0xFFFF0000u);
  }
};
template <>
struct DFin<float, 4> {
  f2 acc = 0ull;
  __device__ __forceinline__ void add(const DRaw<float, 4>& r) {
    const f2 scale = pk(kDFinScale, kDFinScale);
    acc = fma2(pk(r.q.x, r.q.y), scale, acc);
    acc = fma2(pk(r.q.z, r.q.w), scale, acc);
  }
  __device__ __forceinline__ float value() const { return hsum2(acc); }
};
template <typename T>
struct DFin<T, 1> {
  float acc = 0.f;
  __device__ __forceinline__ void add(const DRaw<T, 1>& r) { acc = fmaf(r.x, kDFinScale, acc); }
  __device__ __forceinline__ float value() const { return acc; }
};

template <int VE>
__device__ __forceinline__ float dvmax(const float (&x)[VE]) {
  float m = x[0];
#pragma unroll
  for (int e = 1; e < VE; ++e) m = fmaxf(m, x[e]);
  return m;
}

// Sum of 2^(x log2 e + nm2) over a vector (nm2 = -ref log2 e), in fp32 pairs.
template <int VE>
__device__ __forceinline__ float dmass(const float (&x)[VE], float nm2) {
  if constexpr (VE == 1) {
    return ex2(fmaf(x[0], kLog2e, nm2));
  } else {
    const f2 l2 = pk(kLog2e, kLog2e), n2 = pk(nm2, nm2);
    f2 acc = ex2_2(fma2(pk(x[0], x[1]), l2, n2));
#pragma unroll
    for (int h = 1; h < VE / 2; ++h) acc = add2(acc, ex2_2(fma2(pk(x[2 * h], x[2 * h + 1]), l2, n2)));
    return hsum2(acc);
  }
}

// Warp sums of four per-lane values at once: lane l returns the sum over the
// warp of value q(l) = 2 (bit 4 of l) + (bit 3 of l), so lanes 0, 8, 16 and 24
// hold the sums of m0, m1, m2 and m3 (six shuffles instead of twenty).
__device__ __forceinline__ float dwarp_sum4(float m0, float m1, float m2, float m3, int lane) {
  const bool h16 = (lane & 16) != 0, h8 = (lane & 8) != 0;
  float a = h16 ? m2 : m0, b = h16 ? m3 : m1;
  a += __shfl_xor_sync(0xffffffffu, h16 ? m0 : m2, 16);
  b += __shfl_xor_sync(0xffffffffu, h16 ? m1 : m3, 16);
  float c = h8 ? b : a;
  c += __shfl_xor_sync(0xffffffffu, h8 ? a : b, 8);
  c += __shfl_xor_sync(0xffffffffu, c, 4);
  c += __shfl_xor_sync(0xffffffffu, c, 2);
  c += __shfl_xor_sync(0xffffffffu, c, 1);
  return c;
}

__device__ __forceinline__ bool dfinite(float f) { return fabsf(f) <= 3.402823466e38f; }

// 2^((ref - R) log2 e) times a mass; an empty mass stays 0 whatever ref is.
__device__ __forceinline__ float drescale(float mass, float ref, float R) {
  return mass > 0.f ? mass * ex2((ref - R) * kLog2e) : 0.f;
}

// ---------------------------------------------------------------- greedy slice

template <typename T, int VE>
__device__ __forceinline__ DSlice slice_greedy(const T* a, int v0, int v1, DShared& sh) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n = v1 - v0, full = n / kDThreads, rounds = (n + kDThreads - 1) / kDThreads;
  float m = -INFINITY, s = 0.f;
  DFin<T, VE> fin;
  int bvec = INT_MAX;
  auto take = [&](const DRaw<T, VE>& raw, int v) {
    float x[VE];
    dwiden(raw, x);
    const float vm = dvmax(x);
    if (vm > m) {  // strict: the lowest vector of this thread keeps the maximum
      s *= ex2((m - vm) * kLog2e);
      m = vm;
      bvec = v;
    }
    s += dmass(x, -m * kLog2e);
    fin.add(raw);
  };
  int r = 0;
  for (; r + kDUnroll <= full; r += kDUnroll) {
    DRaw<T, VE> raw[kDUnroll];
#pragma unroll
    for (int u = 0; u < kDUnroll; ++u) dld(a, v0 + (r + u) * kDThreads + tid, raw[u]);
#pragma unroll
    for (int u = 0; u < kDUnroll; ++u) take(raw[u], v0 + (r + u) * kDThreads + tid);
  }
  for (; r < rounds; ++r) {
    const int v = v0 + r * kDThreads + tid;
    if (v < v1) {
      DRaw<T, VE> raw;
      dld(a, v, raw);
      take(raw, v);
    }
  }
  // the CTA maximum, the lowest vector holding it, the sum rescaled to it
  const float w = dwarp_max(m);
  if (lane == 0) sh.red[warp] = w;
  __syncthreads();
  const float M = dwarp_max(lane < kDWarps ? sh.red[lane] : -INFINITY);
  const int vsel = __reduce_min_sync(0xffffffffu, m == M ? bvec : INT_MAX);
  const float ws = dwarp_sum(drescale(s, m, M));
  const float wf = dwarp_sum(fin.value());
  __syncthreads();
  if (lane == 0) {
    sh.redi[warp] = vsel;
    sh.red[warp] = ws;
    sh.red[kDWarps + warp] = wf;
  }
  __syncthreads();
  DSlice out;
  out.ref = M;
  out.sum = dwarp_sum(lane < kDWarps ? sh.red[lane] : 0.f);
  out.fin = dwarp_sum(lane < kDWarps ? sh.red[kDWarps + lane] : 0.f);
  const int vi = __reduce_min_sync(0xffffffffu, lane < kDWarps ? sh.redi[lane] : INT_MAX);
  int idx = INT_MAX;
  if (warp == 0 && lane == 0 && vi < v1) {
    DRaw<T, VE> raw;
    dld(a, vi, raw);
    float x[VE];
    dwiden(raw, x);
#pragma unroll
    for (int e = VE - 1; e >= 0; --e)
      if (x[e] == M) idx = vi * VE + e;
  }
  out.idx = __shfl_sync(0xffffffffu, idx, 0);
  return out;  // valid in warp 0
}

// -------------------------------------------------------------- sampling slice

// Loads of rounds [r, r + kDUnroll) of the slice (vectors past v1 skipped).
template <typename T, int VE>
__device__ __forceinline__ void dld_batch(const T* a, int v0, int v1, int r,
                                          DRaw<T, VE> (&raw)[kDUnroll]) {
#pragma unroll
  for (int u = 0; u < kDUnroll; ++u) {
    const int v = v0 + (r + u) * kDThreads + threadIdx.x;
    if (v < v1) dld(a, v, raw[u]);
  }
}

// Group masses of the slice against the warp reference `ref`: gm[r kDWarps +
// warp] = the mass of vectors v0 + r kDThreads + warp 32 + [0, 32), summed
// kDUnroll rounds at a time.  `cur` holds the first batch's loads (rounds
// 0 .. kDUnroll - 1); each next batch is loaded before the current one is
// used, so a slice of two batches costs one memory round trip.  Adds the
// thread's share to tot (and, when FIN, its finiteness sum to fin); returns
// true if a group's mass reached kDGuard (or is not a number).
template <typename T, int VE, bool FIN>
__device__ __forceinline__ bool slice_masses(const T* a, int v0, int v1, float ref, float* gm,
                                             float& tot, DFin<T, VE>& fin,
                                             DRaw<T, VE> (&cur)[kDUnroll]) {
  static_assert(kDUnroll == 4, "dwarp_sum4 sums four rounds");
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rounds = (v1 - v0 + kDThreads - 1) / kDThreads;
  const float nm2 = -ref * kLog2e;
  bool over = false;
  for (int r = 0; r < rounds; r += kDUnroll) {
    DRaw<T, VE> nxt[kDUnroll];
    if (r + kDUnroll < rounds) dld_batch<T, VE>(a, v0, v1, r + kDUnroll, nxt);
    float mv[kDUnroll];
#pragma unroll
    for (int u = 0; u < kDUnroll; ++u) {
      mv[u] = 0.f;
      if (v0 + (r + u) * kDThreads + tid < v1) {  // implies r + u < rounds
        float x[VE];
        dwiden(cur[u], x);
        mv[u] = dmass(x, nm2);
        if (FIN) fin.add(cur[u]);
      }
      tot += mv[u];
    }
    const float g = dwarp_sum4(mv[0], mv[1], mv[2], mv[3], lane);
    over |= !(g < kDGuard);
    const int q = lane >> 3;  // lanes 0, 8, 16, 24 hold rounds r .. r + 3
    if ((lane & 7) == 0 && r + q < rounds) gm[(r + q) * kDWarps + warp] = g;
#pragma unroll
    for (int u = 0; u < kDUnroll; ++u) cur[u] = nxt[u];
  }
  return over;
}

template <typename T, int VE>
__device__ __forceinline__ DSlice slice_sample(const T* a, int v0, int v1, float* gm, DShared& sh) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // the first batch of rounds; the warp reference: the maximum of the
  // warp's first-round vectors (-inf if none)
  DRaw<T, VE> first[kDUnroll];
  dld_batch<T, VE>(a, v0, v1, 0, first);
  float ref;
  {
    float r0 = -INFINITY;
    if (v0 + tid < v1) {
      float x[VE];
      dwiden(first[0], x);
      r0 = dvmax(x);
    }
    ref = dwarp_max(r0);
  }
  float tot = 0.f;
  DFin<T, VE> fin;
  const bool over = slice_masses<T, VE, true>(a, v0, v1, ref, gm, tot, fin, first);
  if (__syncthreads_or(over)) {
    // an entry far above its warp's reference: the exact slice maximum, then
    // every group again against it
    float m = -INFINITY;
    const int rounds = (v1 - v0 + kDThreads - 1) / kDThreads;
    for (int r = 0; r < rounds; ++r) {
      const int v = v0 + r * kDThreads + tid;
      if (v < v1) {
        DRaw<T, VE> raw;
        dld(a, v, raw);
        float x[VE];
        dwiden(raw, x);
        m = fmaxf(m, dvmax(x));
      }
    }
    const float w = dwarp_max(m);
    if (lane == 0) sh.red[warp] = w;
    __syncthreads();
    ref = dwarp_max(lane < kDWarps ? sh.red[lane] : -INFINITY);
    tot = 0.f;
    DFin<T, VE> unused;
    dld_batch<T, VE>(a, v0, v1, 0, first);
    slice_masses<T, VE, false>(a, v0, v1, ref, gm, tot, unused, first);
    __syncthreads();  // every warp has read sh.red
  }
  const float wt = dwarp_sum(tot), wf = dwarp_sum(fin.value());
  if (lane == 0) {
    sh.wref[warp] = ref;
    sh.red[warp] = wt;
    sh.red[kDWarps + warp] = wf;
  }
  __syncthreads();  // the group masses and the warp totals are in place
  DSlice out;
  const float rw = lane < kDWarps ? sh.wref[lane] : -INFINITY;
  out.ref = dwarp_max(rw);
  out.sum = dwarp_sum(lane < kDWarps ? drescale(sh.red[lane], rw, out.ref) : 0.f);
  out.fin = dwarp_sum(lane < kDWarps ? sh.red[kDWarps + lane] : 0.f);
  out.idx = 0;
  return out;
}

// The owner CTA's walk: the group, the vector and the element holding the
// target tau (in units of 2^R) inside the slice; `last` takes the last entry
// of positive mass instead.  Warp 0 only; lane `vc` writes the row's outputs.
template <typename T, int VE>
__device__ __forceinline__ void slice_walk(const DParams& P, const T* a, int v0, int v1,
                                           const float* gm, const DShared& sh, float R, float S,
                                           float tau, bool last, int row) {
  const int lane = threadIdx.x & 31;
  const int ng = (v1 - v0 + kDThreads - 1) / kDThreads * kDWarps, gpl = (ng + 31) / 32;
  // lane l owns groups [l gpl, (l + 1) gpl)
  float pl = 0.f;
  for (int h = 0; h < gpl; ++h) {
    const int g = lane * gpl + h;
    if (g < ng) pl += gm[g] * sh.wscale[g & (kDWarps - 1)];
  }
  const float incl = dwarp_incl_scan(pl, lane), excl = incl - pl;
  const unsigned hit = __ballot_sync(0xffffffffu, !last && pl > 0.f && excl <= tau && tau < incl);
  const unsigned posl = __ballot_sync(0xffffffffu, pl > 0.f);
  if (!hit) last = true;
  const int lc = hit ? __ffs(hit) - 1 : (posl ? 31 - __clz(posl) : 0);
  int gsel = -1;
  float trem = 0.f;
  if (lane == lc) {
    float cum = excl;
    int glast = -1;
    for (int h = 0; h < gpl; ++h) {
      const int g = lane * gpl + h;
      if (g >= ng) break;
      const float gv = gm[g] * sh.wscale[g & (kDWarps - 1)];
      if (gv > 0.f) glast = g;
      if (!last && gsel < 0) {
        if (cum + gv > tau) {
          gsel = g;
          trem = tau - cum;
        } else {
          cum += gv;
        }
      }
    }
    if (gsel < 0) {
      gsel = glast;
      last = true;
    }
  }
  gsel = __shfl_sync(0xffffffffu, gsel, lc);
  trem = fmaxf(__shfl_sync(0xffffffffu, trem, lc), 0.f);
  last = __shfl_sync(0xffffffffu, last ? 1 : 0, lc) != 0;
  // the vector: lane l recomputes vector v0 + 32 gsel + l against R
  const float nm2 = -R * kLog2e;
  const int v = v0 + 32 * max(gsel, 0) + lane;
  float x[VE];
  float mv = 0.f;
  if (gsel >= 0 && v < v1) {
    DRaw<T, VE> raw;
    dld(a, v, raw);
    dwiden(raw, x);
    mv = dmass(x, nm2);
  }
  const float vin = dwarp_incl_scan(mv, lane), vex = vin - mv;
  const unsigned vh = __ballot_sync(0xffffffffu, !last && mv > 0.f && vex <= trem && trem < vin);
  const unsigned posv = __ballot_sync(0xffffffffu, mv > 0.f);
  if (!vh) last = true;
  const int vc = vh ? __ffs(vh) - 1 : (posv ? 31 - __clz(posv) : 0);
  if (lane != vc) return;
  // the element
  int tok = -1;
  float pr = NAN;
  if (gsel >= 0 && v < v1) {
    const float te = fmaxf(trem - vex, 0.f);
    float cum = 0.f, qpick = 0.f, qlast = 0.f;
    int pick = -1, lastp = -1;
#pragma unroll
    for (int e = 0; e < VE; ++e) {
      const float q = ex2(fmaf(x[e], kLog2e, nm2));
      if (q > 0.f) {
        lastp = e;
        qlast = q;
      }
      cum += q;
      if (!last && pick < 0 && cum > te) {
        pick = e;
        qpick = q;
      }
    }
    if (pick < 0) {
      pick = lastp;
      qpick = qlast;
    }
    if (pick >= 0) {
      tok = v * VE + pick;
      pr = qpick / S;
    }
  }
  P.tokens[row] = tok;
  P.probs[row] = pr;
}

// ------------------------------------------------------------------- the kernel

// Grid: rows x C CTAs in clusters of C.  Shared memory (sampling): one float
// of group mass per warp and round of a slice.
template <typename T, int VE, bool STOCH>
__global__ void __launch_bounds__(kDThreads) draft_kernel(const __grid_constant__ DParams P) {
  extern __shared__ float gm[];
  __shared__ DShared sh;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = static_cast<int>(cluster.num_blocks());
  const int rank = static_cast<int>(cluster.block_rank());
  const int row = static_cast<int>(blockIdx.x) / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const T* a = static_cast<const T*>(P.logits) + static_cast<size_t>(row) * P.V;
  const int v0 = min(rank * P.W, P.nv), v1 = min(v0 + P.W, P.nv);

  const DSlice mine = STOCH ? slice_sample<T, VE>(a, v0, v1, gm, sh) : slice_greedy<T, VE>(a, v0, v1, sh);
  if (warp == 0 && lane < C) *cluster.map_shared_rank(&sh.slot[rank], lane) = mine;
  cluster.sync();  // every CTA's summary is in every CTA; nothing remote after this
  if (warp != 0) return;

  const DSlice s = lane < C ? sh.slot[lane] : DSlice{-INFINITY, 0.f, 0.f, INT_MAX};
  const float R = dwarp_max(s.ref);
  const float mass = lane < C ? drescale(s.sum, s.ref, R) : 0.f;
  const float S = dwarp_sum(mass);
  const float F = dwarp_sum(s.fin);
  if constexpr (!STOCH) {
    const int idx = __reduce_min_sync(0xffffffffu, s.ref == R ? s.idx : INT_MAX);
    if (rank == 0 && lane == 0) {
      const bool ok = dfinite(F) && dfinite(R) && idx != INT_MAX;
      P.tokens[row] = ok ? idx : -1;
      P.probs[row] = ok ? 1.f / S : NAN;  // the maximum's own mass is 2^0
    }
  } else {
    const float u = P.unif[row];
    if (!(dfinite(F) && dfinite(R) && u >= 0.f && u < 1.f)) {
      if (rank == 0 && lane == 0) {
        P.tokens[row] = -1;
        P.probs[row] = NAN;
      }
      return;
    }
    // the slice holding the target (the last with positive mass if none does)
    const float tau = u * S;
    const float incl = dwarp_incl_scan(mass, lane), excl = incl - mass;
    const unsigned hit = __ballot_sync(0xffffffffu, mass > 0.f && excl <= tau && tau < incl);
    const unsigned pos = __ballot_sync(0xffffffffu, mass > 0.f);
    const int owner = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
    if (owner != rank) return;
    const float tloc = fmaxf(tau - __shfl_sync(0xffffffffu, excl, owner), 0.f);
    if (lane < kDWarps) sh.wscale[lane] = drescale(1.f, sh.wref[lane], R);
    __syncwarp();
    slice_walk<T, VE>(P, a, v0, v1, gm, sh, R, S, tloc, hit == 0u, row);
  }
}

}  // namespace asymspec_impl
