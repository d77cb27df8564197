// Production kernel of the stochastic step (JSD gate, delta = a - b, no
// debug outputs): the program bench workloads and serving run.
//
// Same decomposition as fuse_verify_tma (kernel_tma.cuh), whose records it
// leaves for the same decision kernel: one cluster of C CTAs per row triple
// (a_k, b_k, t_k), CTA r taking entries [r W, (r+1) W) of the three rows;
// pass 1 (the normalisers of Eqs. 1-3) over the slice; every warp pushes its
// pass-1 record into every CTA of the cluster (distributed shared memory,
// st.async completing on the receiver's mbarrier); pass 2 (the divergence of
// Eq. 3 and the masses of the fused and residual distributions) over the
// slice again.
//
// What differs from fuse_verify_tma is where the slice lives between the
// passes and the shape of the work:
//   * no slice is held in shared memory.  Each warp owns a contiguous block
//     of the slice and reads it twice through a small ring in shared memory
//     (kRing steps of 32 consecutive 16-byte vectors per stream, filled with
//     cp.async): pass 1 from HBM, pass 2 from the L2, where pass 1 just
//     brought it.  The rows in flight at once (one per resident cluster:
//     97 clusters of 6 CTAs on GB300 for V = 128256 bf16, 75 MB; the host
//     picks C so that they stay within its L2 budget) sit inside the 129 MB
//     L2, so each logit row comes from HBM about once.  With 48 KB of rings
//     and the cluster's pass-1 records in shared memory, four 256-thread CTAs
//     fit on an SM (the register file is the limit), against three when the
//     slice is staged whole; the ring keeps four steps of every warp in
//     flight without holding registers, and pass 2's first steps are issued
//     while the records are exchanged;
//   * no CTA or cluster barrier between the passes but the one __syncthreads
//     after warp 0 has combined the records: a warp pushes its record as soon
//     as its block is done, and the exchange completes on each receiver's
//     mbarrier when the last record of the cluster lands;
//   * the block of a warp is one inverse-CDF group: its mass is the warp's
//     residual (or fused) sum, which the warp reduces anyway, so pass 2 needs
//     no per-step group reductions (the decision kernel walks the group's
//     vectors);
//   * one 16-byte vector per stream per step, unpacked pair by pair from the
//     raw words (bf16 -> fp32 is a shift or a mask), two fp32 lanes per
//     add/sub/mul/fma instruction;
//   * the divergence of Eq. 3 in one product per pair.  With p = softmax(a),
//     q = softmax(b) in log2 units, e = q/p = 2^d (d = log2 q - log2 p) and
//     w = 1 + e, each entry contributes to 2 JSD (in bits)
//         p log2(2p/(p+q)) + q log2(2q/(p+q)) = p [w (1 - log2 w) + e d],
//     a sum of small non-negative terms with no cancellation at the end;
//   * the residual max(0, q_f - p) and fused score (t + beta (a - b)) log2 e
//     are formed exactly as the decision kernel's inverse-CDF walk forms
//     them (res_pair), so the group masses and the walk agree bit for bit.
//
// Waits: one cluster barrier at the start (every CTA's mbarrier is
// initialised before the first push), CTA barriers, its own cp.async groups,
// and the record exchange's mbarrier, bounded by %globaltimer: a wait that
// gives up reports ASYMSPEC_DATA_TIMEOUT for the row, and is waited for once
// more (bounded) before the CTA exits, so that a late push finds it alive.
#pragma once

#include "kernel_tma.cuh"

namespace asymspec_impl {

// A 16-byte vector of the slice, as raw words; pair(h) widens entries
// 2h, 2h + 1 to fp32.
template <typename T>
struct RawVec;
template <>
struct RawVec<__nv_bfloat16> {
  static constexpr int NP = 4;
  uint4 v;
  __device__ __forceinline__ f2 pair(int h) const {
    const unsigned w = h == 0 ? v.x : h == 1 ? v.y : h == 2 ? v.z : v.w;
    return pk(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
  }
};
template <>
struct RawVec<float> {
  static constexpr int NP = 2;
  float4 v;
  __device__ __forceinline__ f2 pair(int h) const { return h == 0 ? pk(v.x, v.y) : pk(v.z, v.w); }
};
// A vector from global memory (read-only for the kernel's lifetime).
template <typename T>
__device__ __forceinline__ RawVec<T> raw_ldg(const T* p) {
  RawVec<T> r;
  r.v = __ldg(reinterpret_cast<const decltype(r.v)*>(p));
  return r;
}

// Constants of a row's pass 2 (log2 units): L2 = log2 e, bL2 = beta log2 e,
// nA2 = -LSE(a) log2 e, nS2 = -LSE(s) log2 e, cAB2 = (LSE(a) - LSE(b)) log2 e.
struct ResConst {
  f2 L2, nL2, bL2, nA2, nS2, cAB2, one2;
};

__device__ __forceinline__ ResConst res_const(float beta, float A2, float B2, float S2) {
  ResConst k;
  k.L2 = pk(kLog2e, kLog2e);
  k.nL2 = pk(-kLog2e, -kLog2e);
  const float bl = beta * kLog2e;
  k.bL2 = pk(bl, bl);
  k.nA2 = pk(-A2, -A2);
  k.nS2 = pk(-S2, -S2);
  const float c = A2 - B2;
  k.cAB2 = pk(c, c);
  k.one2 = pk(1.f, 1.f);
  return k;
}

// The masses of one pair of entries: p = softmax(a), the fused q_f =
// softmax(t + beta (a - b)) and the residual r = max(0, q_f - p); amb = a - b.
// The row kernel's pass 2 and the decision kernel's walk both use this.
__device__ __forceinline__ void res_pair(f2 a2, f2 b2, f2 t2, const ResConst& k, f2& amb, f2& p,
                                         f2& qf, f2& r) {
  amb = sub2(a2, b2);
  p = ex2_2(fma2(a2, k.L2, k.nA2));
  qf = ex2_2(fma2(t2, k.L2, fma2(k.bL2, amb, k.nS2)));
  r = relu2(sub2(qf, p));
}

// The JSD term of a pair (see the header): p [w (1 - log2 w) + e d] with
// d = log2 q - log2 p = -(a - b) log2 e + (LSE(a) - LSE(b)) log2 e.
__device__ __forceinline__ f2 jsd_pair(f2 amb, f2 p, const ResConst& k, f2 jacc) {
  const f2 d = fma2(amb, k.nL2, k.cAB2);
  const f2 e = ex2_2(d);
  const f2 w = add2(e, k.one2);
  const f2 x = sub2(k.one2, lg2_2(w));
  return fma2(p, fma2(w, x, mul2(e, d)), jacc);
}

// ---------------------------------------------------------------- layout

constexpr int kRowThreads = 256;  // threads per CTA of the row kernel
constexpr int kRowMinBlocks = 4;  // CTAs per SM (64 registers a thread)
static_assert(kRowThreads / 32 <= kRowMaxWarps, "one pass-2 record slot per warp");

// A warp's pass-1 record: the references (nats) and sums of
// 2^((x - ref) log2 e) of a, b and the fused score, and its data-error bits.
struct __align__(16) W1 {
  float ref[3], s[3];
  unsigned bad;
  float pad;
};

// Shared state of the row kernel; the pass-1 records of every warp of the
// cluster follow it (recv(): C x kRowThreads / 32 records, the record of
// warp w of CTA r at r kRowThreads / 32 + w).
struct __align__(16) RowShared {
  float lse[4];             // the row's normalisers (a, b, -, s)
  unsigned long long xbar;  // completes when the cluster's records have landed
  unsigned long long pad2;
  __device__ W1* recv() { return reinterpret_cast<W1*>(this + 1); }
};
static_assert(sizeof(W1) == 32, "one warp record is two 16-byte words");
static_assert(sizeof(RowShared) % 16 == 0, "records after RowShared stay 16-byte aligned");

__host__ __device__ constexpr int row_shared_bytes(int C) {
  return static_cast<int>(sizeof(RowShared) + C * (kRowThreads / 32) * sizeof(W1));
}

// ---------------------------------------------------------------- the rings

// Each warp reads its block through a ring of kRing steps in shared memory:
// lane l copies its vector of the three streams for a step into the step's
// slot with 16-byte cp.async (one commit group per step) and later reads
// back only what it copied itself, so no barrier is needed; kRing steps of
// every warp are in flight without holding registers.
constexpr int kRing = 4;
constexpr int kRingBytes = (kRowThreads / 32) * kRing * 3 * 32 * 16;  // per CTA (48 KB)

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Lane's vector i of the three streams into ring slot `slot` (one commit
// group per step, committed by the caller).
template <typename T>
__device__ __forceinline__ void ring_issue(uint4* ring, int slot, const T* ga, const T* gb,
                                           const T* gt, int i) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  uint4* d = ring + slot * 96 + (threadIdx.x & 31);
  cp_async16(d, ga + i * VE);
  cp_async16(d + 32, gb + i * VE);
  cp_async16(d + 64, gt + i * VE);
}
template <typename T>
__device__ __forceinline__ void ring_read(const uint4* ring, int slot, RawVec<T>& va,
                                          RawVec<T>& vb, RawVec<T>& vt) {
  using V = decltype(va.v);
  const V* d = reinterpret_cast<const V*>(ring + slot * 96 + (threadIdx.x & 31));
  va.v = d[0];
  vb.v = d[32];
  vt.v = d[64];
}
// Before step r (r >= 1) reads its slot: step r + kRing - 1 into the slot
// step r - 1 used (slot `slot`, a constant once the loops are unrolled).  That slot's values were consumed by instructions this thread has
// already issued, so the copy cannot overwrite unread data.  pa, pb, pt: the
// lane's vector of step 0 of each stream.
template <typename T>
__device__ __forceinline__ void ring_refill(uint4* ring, int slot, const T* pa, const T* pb,
                                            const T* pt, int i0, int v1, int r) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const int q = r + kRing - 1;
  if (i0 + 32 * q < v1) {
    uint4* d = ring + slot * 96 + (threadIdx.x & 31);
    const size_t o = static_cast<size_t>(q) * 32 * VE;
    cp_async16(d, pa + o);
    cp_async16(d + 32, pb + o);
    cp_async16(d + 64, pt + o);
  }
  cp_async_commit();
}
// The first kRing steps of a pass into the ring (one group each, empty past R).
template <typename T>
__device__ __forceinline__ void ring_prologue(uint4* ring, const T* ga, const T* gb, const T* gt,
                                              int v0, int v1, int R) {
  const int i0 = v0 + static_cast<int>(threadIdx.x & 31);
#pragma unroll
  for (int q = 0; q < kRing; ++q) {
    const int i = i0 + 32 * q;
    if (q < R && i < v1) ring_issue<T>(ring, q, ga, gb, gt, i);
    cp_async_commit();
  }
}

// ---------------------------------------------------------------- pass 1

// Pass 1 over the warp's block [v0, v1) of the slice (ga, gb, gt: the
// slice's first entries in global memory; R steps), its vectors read through
// the warp's ring (the caller issued the prologue), with one fixed reference
// per warp and stream: the largest of the first pairs of the lanes' first
// vectors.  DRAFT: the normalisers of a, b and the fused score s; the bonus
// row needs s only.  Returns true when a lane's sum reached 2^100 or is not
// finite (the CTA then redoes its slice with a running maximum).  Every lane
// ends with the warp's record.
template <typename T, bool DRAFT>
__device__ __forceinline__ bool row_pass1(uint4* ring, const T* ga, const T* gb, const T* gt,
                                           int v0, int v1, int R, float beta, W1& e) {
  constexpr int NP = RawVec<T>::NP;
  const int lane = static_cast<int>(threadIdx.x & 31);
  const f2 L2 = pk(kLog2e, kLog2e);
  const float bl = beta * kLog2e;
  const f2 bL2 = pk(bl, bl);
  const int i0 = v0 + lane;
  float ra0 = -INFINITY, rb0 = -INFINITY, rs0 = -INFINITY;
  cp_async_wait<kRing - 1>();  // step 0 (this lane's own copies)
  RawVec<T> va, vb, vt;
  if (i0 < v1) {
    ring_read<T>(ring, 0, va, vb, vt);
    const f2 a2 = va.pair(0), b2 = vb.pair(0), t2 = vt.pair(0);
    const f2 s2 = fma2(pk(beta, beta), sub2(a2, b2), t2);
    ra0 = fmaxf(lo_of(a2), hi_of(a2));
    rb0 = fmaxf(lo_of(b2), hi_of(b2));
    rs0 = fmaxf(lo_of(s2), hi_of(s2));
  }
  if (DRAFT) {
    ra0 = warp_max(ra0);
    rb0 = warp_max(rb0);
  }
  rs0 = warp_max(rs0);
  const float nA = -ra0 * kLog2e, nB = -rb0 * kLog2e, nS = -rs0 * kLog2e;
  const f2 nA2 = pk(nA, nA), nB2 = pk(nB, nB), nS2 = pk(nS, nS);
  f2 acc_a = 0ull, acc_b = 0ull, acc_s = 0ull;
  constexpr int VE = 2 * NP;
  const T* pa = ga + static_cast<size_t>(i0) * VE;
  const T* pb = gb + static_cast<size_t>(i0) * VE;
  const T* pt = gt + static_cast<size_t>(i0) * VE;
  // unrolled by the ring's depth, so that every slot is a constant
  for (int r0 = 0; r0 < R; r0 += kRing) {
#pragma unroll
    for (int u = 0; u < kRing; ++u) {
      const int r = r0 + u;
      if (r >= R) break;
      if (r > 0) {
        ring_refill<T>(ring, (u + kRing - 1) % kRing, pa, pb, pt, i0, v1, r);
        cp_async_wait<kRing - 1>();
      }
      if (i0 + 32 * r < v1) {
        if (r > 0) ring_read<T>(ring, u, va, vb, vt);
#pragma unroll
        for (int h = 0; h < NP; ++h) {
          const f2 a2 = va.pair(h), b2 = vb.pair(h), t2 = vt.pair(h);
          if (DRAFT) {
            acc_a = add2(acc_a, ex2_2(fma2(a2, L2, nA2)));
            acc_b = add2(acc_b, ex2_2(fma2(b2, L2, nB2)));
          }
          acc_s = add2(acc_s, ex2_2(fma2(t2, L2, fma2(bL2, sub2(a2, b2), nS2))));
        }
      }
    }
  }
  float sa = DRAFT ? hsum2(acc_a) : 0.f, sb = DRAFT ? hsum2(acc_b) : 0.f, ss = hsum2(acc_s);
  const bool ovf = !(ss < kSumLimit) || (DRAFT && (!(sa < kSumLimit) || !(sb < kSumLimit)));
  float z = 0.f;
  warp_sum4(sa, sb, ss, z);
  e.ref[0] = ra0;
  e.ref[1] = rb0;
  e.ref[2] = rs0;
  e.s[0] = sa;
  e.s[1] = sb;
  e.s[2] = ss;
  e.bad = 0u;
  e.pad = 0.f;
  return ovf;
}

// Fallback of row_pass1 (a sum reached 2^100, or non-finite data): each lane
// keeps a running maximum per stream over its vectors of the warp's block,
// rescaling its sum when the maximum rises; the lanes then merge.
template <typename T, bool DRAFT>
__device__ __forceinline__ void row_pass1_online(const T* ga, const T* gb, const T* gt, int v0,
                                                 int v1, float beta, W1& e) {
  constexpr int NP = RawVec<T>::NP;
  constexpr int VE = 2 * NP;
  const int lane = static_cast<int>(threadIdx.x & 31);
  float m[3] = {-INFINITY, -INFINITY, -INFINITY};  // running maxima of a, b, s (nats)
  float s[3] = {0.f, 0.f, 0.f};                    // sums of 2^((x - m) log2 e)
  for (int i = v0 + lane; i < v1; i += 32) {
    const RawVec<T> va = raw_ldg(ga + i * VE), vb = raw_ldg(gb + i * VE);
    const RawVec<T> vt = raw_ldg(gt + i * VE);
#pragma unroll
    for (int h = 0; h < NP; ++h) {
      const f2 a2 = va.pair(h), b2 = vb.pair(h), t2 = vt.pair(h);
      const f2 s2 = fma2(pk(beta, beta), sub2(a2, b2), t2);
      float x[3][2];
      upk(a2, x[0][0], x[0][1]);
      upk(b2, x[1][0], x[1][1]);
      upk(s2, x[2][0], x[2][1]);
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        if (!DRAFT && q < 2) continue;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const float v = x[q][j];
          if (v > m[q]) {
            s[q] = s[q] * ex2((m[q] - v) * kLog2e);
            m[q] = v;
          }
          s[q] += ex2((v - m[q]) * kLog2e);
        }
      }
    }
  }
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    const float M = warp_max(m[q]);
    const float sc = (s[q] == 0.f || m[q] == M) ? s[q] : s[q] * ex2((m[q] - M) * kLog2e);
    e.ref[q] = M;
    e.s[q] = warp_sum(sc);
  }
  if (!DRAFT) {
    e.ref[0] = e.ref[1] = -INFINITY;
    e.s[0] = e.s[1] = 0.f;
  }
}

// ---------------------------------------------------------------- pass 2

// Pass 2 over the warp's block (from the L2, where pass 1 left it), through
// the warp's ring (the caller issued the prologue): DRAFT, the JSD terms
// (see the header) and the residual masses; the bonus row, the fused
// masses.  Returns through jsum / msum the warp's sums (every lane ends with
// them): msum is the mass of the warp's inverse-CDF group.
template <typename T, bool DRAFT>
__device__ __forceinline__ void row_pass2(uint4* ring, const T* ga, const T* gb, const T* gt,
                                           int v0, int v1, int R, const ResConst& k, float& jsum,
                                           float& msum) {
  constexpr int NP = RawVec<T>::NP;
  const int lane = static_cast<int>(threadIdx.x & 31);
  f2 jacc = 0ull, macc = 0ull;
  const int i0 = v0 + lane;
  constexpr int VE = 2 * NP;
  const T* pa = ga + static_cast<size_t>(i0) * VE;
  const T* pb = gb + static_cast<size_t>(i0) * VE;
  const T* pt = gt + static_cast<size_t>(i0) * VE;
  for (int r0 = 0; r0 < R; r0 += kRing) {
#pragma unroll
    for (int u = 0; u < kRing; ++u) {
      const int r = r0 + u;
      if (r >= R) break;
      if (r > 0) ring_refill<T>(ring, (u + kRing - 1) % kRing, pa, pb, pt, i0, v1, r);
      cp_async_wait<kRing - 1>();
      if (i0 + 32 * r < v1) {
        RawVec<T> va, vb, vt;
        ring_read<T>(ring, u, va, vb, vt);
#pragma unroll
        for (int h = 0; h < NP; ++h) {
          f2 amb, p, qf, rr;
          res_pair(va.pair(h), vb.pair(h), vt.pair(h), k, amb, p, qf, rr);
          if (DRAFT) {
            macc = add2(macc, rr);
            jacc = jsd_pair(amb, p, k, jacc);
          } else {
            macc = add2(macc, qf);
          }
        }
      }
    }
  }
  float j = hsum2(jacc), m = hsum2(macc), z0 = 0.f, z1 = 0.f;
  warp_sum4(j, m, z0, z1);
  jsum = j;
  msum = m;
}

// ---------------------------------------------------------------- the kernel

// 16 bytes into CTA `rank`'s copy of the shared variable at `local`,
// completing 16 bytes of the transaction count of that CTA's copy of `bar`.
__device__ __forceinline__ void st_async16(const void* local, unsigned rank,
                                           unsigned long long* bar, float4 v) {
  unsigned ra, rb;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rb) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(ra),
      "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rb)
      : "memory");
}
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}
// The row's pass-1 result from the n warp records of its cluster, by one
// warp: lane l merges records l, l + 32, ... (each stream's sums restated
// against the largest of their references), then the lanes' results are
// combined as warp_reduce_x1 combines them.  Every lane ends with the same
// (bit-identical) result, and so does every CTA, whose records are the same.
__device__ __forceinline__ void combine_records(const W1* rec, int n, float (&ref)[3],
                                                float (&sum)[3]) {
  const int lane = static_cast<int>(threadIdx.x & 31);
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    ref[q] = -INFINITY;
    sum[q] = 0.f;
  }
  for (int i = lane; i < n; i += 32) {
    const W1 r = rec[i];
#pragma unroll
    for (int q = 0; q < 3; ++q) {
      const float M = fmaxf(ref[q], r.ref[q]);
      const float a = (sum[q] == 0.f || ref[q] == M) ? sum[q] : sum[q] * ex2((ref[q] - M) * kLog2e);
      const float b = (r.s[q] == 0.f || r.ref[q] == M) ? r.s[q] : r.s[q] * ex2((r.ref[q] - M) * kLog2e);
      ref[q] = M;
      sum[q] = a + b;
    }
  }
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    const float M = warp_max(ref[q]);
    const float v = (sum[q] == 0.f || ref[q] == M) ? sum[q] : sum[q] * ex2((ref[q] - M) * kLog2e);
    ref[q] = M;
    sum[q] = warp_sum(v);
  }
}

// The cluster's index in the grid: (row k of batch element bi) = (x, y).
__device__ __forceinline__ unsigned cluster_id_x() {
  unsigned r;
  asm("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ unsigned cluster_id_y() {
  unsigned r;
  asm("mov.u32 %0, %%clusterid.y;" : "=r"(r));
  return r;
}

// Grid: (C (K+1), B) CTAs of kRowThreads threads in clusters of (C, 1, 1);
// cluster (k, bi) takes row k of batch element bi.  What it leaves for the
// decision kernel: rank 0's row statistics (the normalisers, data-error
// bits) and one pass-2 record per warp of every CTA (KParams::pass2_rec,
// kRowMaxWarps records per CTA): the warp's JSD sum, the residual and fused
// masses of its block (its inverse-CDF group).  Dynamic shared memory: the
// fixed state and pushed records (row_shared_bytes(C)), then the warps'
// rings (kRingBytes) at KParams::sh_off.  Pass 2's first kRing steps are
// issued before the records are exchanged: they do not depend on the
// normalisers.
template <typename T>
__global__ void __launch_bounds__(kRowThreads, kRowMinBlocks) fuse_verify_row(const KParams P) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  constexpr int NW = kRowThreads / 32;
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  extern __shared__ __align__(128) unsigned char smem_row[];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int tid = static_cast<int>(threadIdx.x);
  const int lane = tid & 31, warp = tid >> 5;
  const int C = P.C;
  const int k = static_cast<int>(cluster_id_x());
  const int bi = static_cast<int>(cluster_id_y());
  const unsigned row32 = static_cast<unsigned>(bi) * static_cast<unsigned>(P.K + 1) +
                         static_cast<unsigned>(k);
  const int W = P.W;
  const int lo = rank * W;
  const int n = max(0, min(W, P.V - lo));
  const int nv = n / VE;
  const int bw = row_block_vectors(nv, NW);
  const int v0 = min(nv, warp * bw), v1 = min(nv, v0 + bw);
  const int R = (v1 - v0 + 31) / 32;
  const size_t off = static_cast<size_t>(row32) * P.V + lo;
  const T* ga = static_cast<const T*>(P.a) + off;
  const T* gb = static_cast<const T*>(P.b) + off;
  const T* gt = static_cast<const T*>(P.t) + off;
  RowShared* sh = reinterpret_cast<RowShared*>(smem_row);
  uint4* ring = reinterpret_cast<uint4*>(smem_row + P.sh_off) + warp * (kRing * 96);
  const bool draft = k < P.K;
  const int nrec = C * NW;  // pass-1 records the cluster exchanges
  if (tid == 0) {
    mbar_init(&sh->xbar, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(&sh->xbar, static_cast<unsigned>(nrec * sizeof(W1)));
  }
  cluster_arrive_relaxed();
  ring_prologue<T>(ring, ga, gb, gt, v0, v1, R);
  // every CTA's barrier is initialised before any push (the CTAs of a
  // cluster start together; this wait overlaps the first loads)
  cluster_wait();

  // ---- pass 1: the row normalisers, combined over the cluster
  W1 e;
  bool ovf = draft ? row_pass1<T, true>(ring, ga, gb, gt, v0, v1, R, P.beta, e)
                   : row_pass1<T, false>(ring, ga, gb, gt, v0, v1, R, P.beta, e);
  cp_async_wait<0>();  // the pass's trailing (empty) groups; the ring is free
  // pass 2's first steps do not depend on the normalisers
  ring_prologue<T>(ring, ga, gb, gt, v0, v1, R);
  if (__any_sync(0xffffffffu, ovf)) {
    // an entry far above the warp's reference (or non-finite data): redo the
    // block with running maxima
    if (draft) row_pass1_online<T, true>(ga, gb, gt, v0, v1, P.beta, e);
    else row_pass1_online<T, false>(ga, gb, gt, v0, v1, P.beta, e);
  }
  e.bad = 0u;
  e.pad = 0.f;
  if (lane < C) {
    // this warp's record into slot rank NW + warp of every CTA (lane j to CTA j)
    const float4* slot = reinterpret_cast<const float4*>(sh->recv() + rank * NW + warp);
    st_async16(slot, static_cast<unsigned>(lane), &sh->xbar,
               make_float4(e.ref[0], e.ref[1], e.ref[2], e.s[0]));
    st_async16(slot + 1, static_cast<unsigned>(lane), &sh->xbar,
               make_float4(e.s[1], e.s[2], 0.f, 0.f));
  }
  bool got = true;
  if (warp == 0) {
    // every warp's record of the cluster is in this CTA once the barrier completes
    got = mbar_wait_cluster_bounded(&sh->xbar, 0, kCopyTimeoutNs);
    float ref[3], sum[3];
    combine_records(sh->recv(), nrec, ref, sum);
    if (lane == 0) {
      float lse[4];
      lse[0] = draft ? ref[0] + logf(sum[0]) : NAN;
      lse[1] = draft ? ref[1] + logf(sum[1]) : NAN;
      lse[2] = NAN;
      lse[3] = ref[2] + logf(sum[2]);
#pragma unroll
      for (int q = 0; q < 4; ++q) sh->lse[q] = lse[q];
      // the draft token's logits are read by the decision kernel itself
      if (rank == 0)
        store_row_stat(P, row32, lse, INT_MAX, INT_MAX, got ? 0u : kBadTimeout, -1, 0.f, 0.f, 0.f);
    }
  }
  __syncthreads();

  // ---- pass 2: divergence terms and inverse-CDF masses
  const float A2 = sh->lse[0] * kLog2e, B2 = sh->lse[1] * kLog2e, S2 = sh->lse[3] * kLog2e;
  const ResConst kc = res_const(P.beta, A2, B2, S2);
  float jsum, msum;
  if (draft) row_pass2<T, true>(ring, ga, gb, gt, v0, v1, R, kc, jsum, msum);
  else row_pass2<T, false>(ring, ga, gb, gt, v0, v1, R, kc, jsum, msum);
  cp_async_wait<0>();
  if (lane == 0) {
    // this warp's record: its block is one inverse-CDF group of the row.  A
    // draft row's fused mass (the draw's fallback when the row's whole
    // residual is zero) comes from the warp's pass-1 sum.
    const float qf = draft ? e.s[2] * ex2(e.ref[2] * kLog2e - S2) : msum;
    float4* rec = reinterpret_cast<float4*>(
        P.pass2_rec + ((static_cast<size_t>(row32) * C + rank) * kRowMaxWarps + warp) * 8);
    rec[0] = make_float4(jsum, 0.f, 0.f, draft ? msum : 0.f);
    rec[1] = make_float4(qf, 0.f, 0.f, 0.f);
  }
  // no CTA exits while a push to it may be in flight: once the barrier has
  // completed every push has landed; after a wait that gave up, warp 0 waits
  // once more (bounded) before the CTA may exit
  if (warp == 0 && !got) mbar_wait_cluster_bounded(&sh->xbar, 0, kCopyTimeoutNs);
}

}  // namespace asymspec_impl
