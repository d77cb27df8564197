// Persistent cluster kernel for 16-byte aligned rows (the default).
//
// A grid of as many clusters of C CTAs as the device holds at once; cluster
// q takes rows q, q + NCL, q + 2 NCL, ... (NCL clusters), and CTA r of the
// cluster owns entries [r W, (r+1) W) of each of them, as in the one-shot
// cluster kernel (kernel_tma.cuh), whose per-entry arithmetic this kernel
// shares.  What differs is where the slice lives:
//
// both passes stream the slice through a ring of kRStages shared-memory
// stages, one round (256 vectors of each of a, b, t) per stage, filled by
// 1-D bulk copies that thread 0 keeps issuing ahead of the consumers, across
// pass and row boundaries: for each row the ring carries the slice's rounds
// for pass 1 (from HBM), then the same rounds again for pass 2, which finds
// them in L2 one slice later (L2 policy evict_first on the second copy).
// A row without pass 2 still takes its ring positions, with no copies.
//
// Between the passes each CTA pushes its pass-1 record to every CTA of the
// cluster (DSMEM stores plus a remote mbarrier arrive) and waits for the
// others', while the ring keeps loading.  Each CTA keeps kRSlots record
// slots, so a peer that is ahead never overwrites a record not yet read.  No cluster-wide barrier is
// taken per row; each row's decision is left to decide_rows, from the same
// workspace records the one-shot kernel writes.
//
// Only the production programs run here, optionally with the per-row token
// output; calls that ask for row statistics or fused log-probs go to
// fuse_verify_tma.
//
// Every wait is bounded (kCopyTimeoutNs); a wait that gives up marks the row
// ASYMSPEC_DATA_TIMEOUT, and before the CTA exits thread 0 waits (bounded
// again) for any copy still in flight.
#pragma once

#include "kernel_tma.cuh"

namespace asymspec_impl {

constexpr int kRStages = 8;                             // ring stages (rounds in flight)
constexpr int kRThreads = kTThreads + 32;               // 8 consumer warps + 1 producer warp
constexpr int kRMaxRounds = 32;                         // rounds per slice (group walk: 256 groups)
constexpr int kRSlots = 4;                              // pass-1 record slots per peer
constexpr int kRStreamBytes = kTThreads * 16;           // one round of one stream
constexpr int kRStageBytes = 3 * kRStreamBytes;         // one round of a, b and t
constexpr int kRRingBytes = kRStages * kRStageBytes;

// Shared state after the ring; kRSlots x C pass-1 records follow it.
struct __align__(16) SharedRing {
  unsigned long long full[kRStages];   // a stage's copies landed (1 arrive + bytes)
  unsigned long long empty[kRStages];  // every consumer warp is done with a stage
  unsigned long long rowbar[kRSlots];  // C remote arrivals per row
  X1 w1[2][kTWarps];                   // per-warp pass-1 records, by row parity
  X2 w2[kTWarps];
  float lse[4];                        // the row's normalisers, for pass 2
  unsigned broken;                     // a copy or a peer timed out
  unsigned pad[3];
  __device__ X1* recv(int slot, int C) { return reinterpret_cast<X1*>(this + 1) + slot * C; }
};
static_assert(sizeof(SharedRing) % 16 == 0, "records after SharedRing stay 16-byte aligned");

__host__ __device__ constexpr int ring_smem_bytes(int C) {
  return kRRingBytes + static_cast<int>(sizeof(SharedRing)) + kRSlots * C * static_cast<int>(sizeof(X1));
}

// Per-CTA constants and the ring position (identical in every thread; the
// issue position `issued` is kept by thread 0 only).
struct RingCtx {
  SharedRing* sh;
  unsigned char* ring;
  int C, rank, q, ncl, nrows;  // cluster q of ncl takes nrows rows
  int W, lo, n, nv, rounds;    // this CTA's slice
  unsigned seq;                // next ring sequence number to consume
  unsigned issued;             // next to issue (thread 0)
  unsigned total;              // nrows * 2 * rounds
  unsigned long long pol1;     // L2 policy of the pass-1 copies
  unsigned long long pol2;     // L2 policy of the pass-2 copies
};

__device__ __forceinline__ long long ring_row(const RingCtx& c, int i) {
  return static_cast<long long>(c.q) + static_cast<long long>(i) * c.ncl;
}

// Greedy bonus rows without the fused bonus need t only (Algorithm 1 emits argmax t).
template <bool STOCH>
__device__ __forceinline__ bool ring_only_t(const KParams& P, long long row) {
  return !STOCH && !P.fuse_bonus && static_cast<int>(row % (P.K + 1)) == P.K;
}

// Rows with a pass 2: every stochastic row; greedy draft rows with a JSD or KL gate.
template <bool STOCH>
__device__ __forceinline__ bool ring_has_pass2(const KParams& P, long long row) {
  if (STOCH) return true;
  return static_cast<int>(row % (P.K + 1)) != P.K &&
         (P.divergence == ASYMSPEC_DIV_JSD || P.divergence == ASYMSPEC_DIV_KL);
}

// What thread 0 needs to issue copies (passed by value).
struct RingIssue {
  SharedRing* sh;
  unsigned char* ring;
  int q, ncl, rounds, nv, lo;
  unsigned total;
  unsigned long long pol1, pol2;
};

__device__ __forceinline__ RingIssue ring_issue_of(const RingCtx& c) {
  return RingIssue{c.sh, c.ring, c.q, c.ncl, c.rounds, c.nv, c.lo, c.total, c.pol1, c.pol2};
}

// Thread 0: the copies of ring sequence number n into stage n % kRStages.
// Local row i takes sequence numbers [2 i R, 2 i R + R) for pass 1 and the
// next R for pass 2 (R = rounds); round kr of a pass is vectors
// [256 kr, 256 kr + 256) of the slice.
template <typename T, bool STOCH>
__device__ __forceinline__ void ring_issue(const KParams& P, const RingIssue& c, unsigned n) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const int s = static_cast<int>(n % kRStages);
  const unsigned R = static_cast<unsigned>(c.rounds);
  const int i = static_cast<int>(n / (2u * R));
  const unsigned w = n - static_cast<unsigned>(i) * 2u * R;
  const bool second = w >= R;
  const int kr = static_cast<int>(second ? w - R : w);
  const long long row = static_cast<long long>(c.q) + static_cast<long long>(i) * c.ncl;
  unsigned long long* bar = &c.sh->full[s];
  if (second && !ring_has_pass2<STOCH>(P, row)) {
    mbar_arrive(bar);  // an empty position: nothing to copy
    return;
  }
  const unsigned long long pol = second ? c.pol2 : c.pol1;
  const bool only_t = ring_only_t<STOCH>(P, row);
  const int v0 = kr * kTThreads;
  const int v1 = min(c.nv, v0 + kTThreads);
  const unsigned bytes = static_cast<unsigned>(v1 - v0) * 16u;
  unsigned char* st = c.ring + s * kRStageBytes;
  mbar_arrive_expect_tx(bar, bytes * (only_t ? 1u : 3u));
  const size_t off = static_cast<size_t>(row) * P.V + c.lo + static_cast<size_t>(v0) * VE;
  if (!only_t) {
    bulk_load_hint(st, static_cast<const T*>(P.a) + off, bytes, bar, pol);
    bulk_load_hint(st + kRStreamBytes, static_cast<const T*>(P.b) + off, bytes, bar, pol);
  }
  bulk_load_hint(st + 2 * kRStreamBytes, static_cast<const T*>(P.t) + off, bytes, bar, pol);
}

// Thread 0: issues every sequence number from `issued` on whose stage is
// free, without waiting; with `block`, waits (bounded) for the stages up to
// sequence number `upto`.  Returns the next sequence number to issue.
template <typename T, bool STOCH>
__device__ __noinline__ unsigned ring_top_up_impl(const KParams& P, RingIssue c, unsigned issued,
                                                  unsigned upto, bool block) {
  while (issued < c.total) {
    if (c.sh->broken) break;  // after a timeout nothing more is issued
    const unsigned n = issued;
    if (n >= static_cast<unsigned>(kRStages)) {
      // the stage's previous use, sequence n - kRStages, must be released
      unsigned long long* e = &c.sh->empty[n % kRStages];
      const unsigned par = ((n / kRStages) + 1u) & 1u;
      if (!mbar_test_wait(e, par)) {
        if (!block || n > upto) break;
        if (!mbar_wait_bounded(e, par, kCopyTimeoutNs)) {
          atomicOr(&c.sh->broken, kBadTimeout);
          break;
        }
      }
    }
    ring_issue<T, STOCH>(P, c, n);
    issued = n + 1;
  }
  return issued;
}

// The producer warp's lane 0: every sequence number in order, each once its
// stage's previous use has been released (bounded waits).
template <typename T, bool STOCH>
__device__ __forceinline__ void ring_produce(const KParams& P, RingCtx& c) {
  c.issued = ring_top_up_impl<T, STOCH>(P, ring_issue_of(c), 0u, c.total, true);
}

// Waits (bounded) for the stage of sequence number n; false on a timeout.
__device__ __forceinline__ bool ring_wait(RingCtx& c, unsigned n) {
  if (c.sh->broken) return false;
  if (mbar_wait_bounded(&c.sh->full[n % kRStages], (n / kRStages) & 1u, kCopyTimeoutNs)) return true;
  atomicOr(&c.sh->broken, kBadTimeout);
  return false;
}

// Every consumer warp releases the stage of sequence number n once.
__device__ __forceinline__ void ring_release(RingCtx& c, unsigned n) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&c.sh->empty[n % kRStages]);
}

// Barrier over the 256 consumer threads (named barrier 1; the producer warp
// never takes part), and its OR-reduction form.
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kTThreads) : "memory");
}
__device__ __forceinline__ bool consumer_sync_or(bool v) {
  unsigned r;
  asm volatile(
      "{ .reg .pred p, q; setp.ne.u32 p, %1, 0; bar.red.or.pred q, 1, %2, p; selp.u32 %0, 1, 0, q; }"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(kTThreads)
      : "memory");
  return r != 0;
}

// Vector `slot` (0 .. 255) of stream q (0 a, 1 b, 2 t) in the stage of n.
template <typename T>
__device__ __forceinline__ const T* ring_vec(const RingCtx& c, unsigned n, int q, int slot) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  return reinterpret_cast<const T*>(c.ring + (n % kRStages) * kRStageBytes + q * kRStreamBytes) +
         slot * VE;
}

// ---------------------------------------------------------------- pass 1

// Pass 1 of one row from the ring, against fixed references (the maximum
// of each thread's first vector, as in pass1_fast), two rounds per step.
// Returns true when one of this thread's sums reached 2^100 or is not
// finite.  ga, gb, gt: the slice in global memory, for the argmax elements.
template <typename T, bool STOCH, unsigned F>
__device__ __forceinline__ bool ring_pass1(const KParams& P, RingCtx& c, const T* ga,
                                           const T* gb, const T* gt, X1& e) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needA = (F & (F_LA | F_LS | F_AS)) != 0;
  constexpr bool needB = (F & (F_LB | F_LS | F_AS)) != 0;
  constexpr bool needT = (F & (F_LT | F_LS | F_AS | F_AT)) != 0;
  constexpr bool needS = (F & (F_LS | F_AS)) != 0;
  const int tid = static_cast<int>(threadIdx.x);
  const float beta = P.beta;
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  const unsigned s0 = c.seq;
  c.seq = s0 + static_cast<unsigned>(c.rounds);
  if (c.rounds == 0) {
#pragma unroll
    for (int q = 0; q < 4; ++q) e.s[q] = 0.f;
    return false;
  }
  ring_wait(c, s0);
  float ref[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  if (tid < c.nv) {
    f2 xa[NP], xb[NP], xt[NP], xs[NP];
    if (needA) load_pairs(ring_vec<T>(c, s0, 0, tid), xa);
    if (needB) load_pairs(ring_vec<T>(c, s0, 1, tid), xb);
    if (needT) load_pairs(ring_vec<T>(c, s0, 2, tid), xt);
    if (F & F_LA) ref[0] = vmax_pairs(xa);
    if (F & F_LB) ref[1] = vmax_pairs(xb);
    if (F & F_LT) ref[2] = vmax_pairs(xt);
    if (F & F_LS) {
#pragma unroll
      for (int h = 0; h < NP; ++h) xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
      ref[3] = vmax_pairs(xs);
    }
  }
  f2 nm[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float v = -ref[q] * kLog2e;
    nm[q] = pk(v, v);
  }
  f2 acc[4] = {0ull, 0ull, 0ull, 0ull};
  int vec_s = -1, vec_t = -1;
  for (int kr = 0; kr < c.rounds; kr += 2) {
    const unsigned n0 = s0 + static_cast<unsigned>(kr);
    const bool two = kr + 1 < c.rounds;
    if (kr > 0) ring_wait(c, n0);
    if (two) ring_wait(c, n0 + 1);
    const int i0 = kr * kTThreads + tid;
    const bool has0 = i0 < c.nv;
    const bool has1 = two && i0 + kTThreads < c.nv;
    f2 xa[NP], xb[NP], xt[NP], xs[NP], ya[NP], yb[NP], yt[NP], ys[NP];
    if (needA) {
      load_or_fill(ring_vec<T>(c, n0, 0, tid), has0, xa);
      load_or_fill(ring_vec<T>(c, n0 + 1, 0, tid), has1, ya);
    }
    if (needB) {
      load_or_fill(ring_vec<T>(c, n0, 1, tid), has0, xb);
      load_or_fill(ring_vec<T>(c, n0 + 1, 1, tid), has1, yb);
    }
    if (needT) {
      load_or_fill(ring_vec<T>(c, n0, 2, tid), has0, xt);
      load_or_fill(ring_vec<T>(c, n0 + 1, 2, tid), has1, yt);
    }
    if (needS) {
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
        ys[h] = fma2(beta2, sub2(ya[h], yb[h]), yt[h]);
      }
    }
    if (F & F_LA) fixed_pairs2(acc[0], xa, ya, L2, nm[0]);
    if (F & F_LB) fixed_pairs2(acc[1], xb, yb, L2, nm[1]);
    if (F & F_LT) fixed_pairs2(acc[2], xt, yt, L2, nm[2]);
    if (F & F_LS) fixed_pairs2(acc[3], xs, ys, L2, nm[3]);
    if (F & F_AS) {
      const float cs0 = (F & F_LS) ? vmax_pairs(xs) : vmax_pairs_nan(xs);
      const float cs1 = (F & F_LS) ? vmax_pairs(ys) : vmax_pairs_nan(ys);
      if (has0) arg_track(e.vs, vec_s, cs0, i0, e.bad, kBadS);
      if (has1) arg_track(e.vs, vec_s, cs1, i0 + kTThreads, e.bad, kBadS);
    }
    if (F & F_AT) {
      const float ct0 = (F & F_LT) ? vmax_pairs(xt) : vmax_pairs_nan(xt);
      const float ct1 = (F & F_LT) ? vmax_pairs(yt) : vmax_pairs_nan(yt);
      if (has0) arg_track(e.vt, vec_t, ct0, i0, e.bad, kBadT);
      if (has1) arg_track(e.vt, vec_t, ct1, i0 + kTThreads, e.bad, kBadT);
    }
    ring_release(c, n0);
    if (two) ring_release(c, n0 + 1);
  }
  bool ovf = false;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
    e.ref[q] = ref[q];
    e.s[q] = hsum2(acc[q]);
    if ((F & bit) && !(e.s[q] < kSumLimit)) ovf = true;
  }
  // the element of the best vector, re-read from global memory (L2)
  if ((F & F_AS) && vec_s >= 0) {
    f2 xa[NP], xb[NP], xt[NP], xs[NP];
    load_pairs(ga + vec_s * VE, xa);
    load_pairs(gb + vec_s * VE, xb);
    load_pairs(gt + vec_s * VE, xt);
#pragma unroll
    for (int h = 0; h < NP; ++h) xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
    e.is = arg_in_vector(xs, e.vs, c.lo + vec_s * VE);
  }
  if ((F & F_AT) && vec_t >= 0) {
    f2 xt[NP];
    load_pairs(gt + vec_t * VE, xt);
    e.it = arg_in_vector(xt, e.vt, c.lo + vec_t * VE);
  }
  return ovf;
}

// ---------------------------------------------------------------- pass 2

// Pass 2 of one row from the ring (the second R sequence numbers of the row),
// two rounds per step; as pass2 in kernel_tma.cuh, with the slice's rounds in
// ring stages instead of a resident slice.
template <typename T, bool STOCH, unsigned G>
__device__ __forceinline__ void ring_pass2(const KParams& P, RingCtx& c, float A2, float B2,
                                           float S2, float lse_s, X2& x, float* grp) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needT = (G & (G_RES | G_QF)) != 0;
  const int tid = static_cast<int>(threadIdx.x);
  const unsigned s0 = c.seq;
  c.seq = s0 + static_cast<unsigned>(c.rounds);
  const P2Const k = p2_const(P.beta, A2, B2, S2, lse_s);
  P2Acc acc = {0ull, 0ull, 0ull, 0ull, 0ull, 0ull};
  for (int kr = 0; kr < c.rounds; kr += 2) {
    const unsigned n0 = s0 + static_cast<unsigned>(kr);
    const bool two = kr + 1 < c.rounds;
    ring_wait(c, n0);
    if (two) ring_wait(c, n0 + 1);
    const int i0 = kr * kTThreads + tid;
    const bool has1 = two && i0 + kTThreads < c.nv;
    float g0 = 0.f, g1 = 0.f;
    if (i0 < c.nv) {
      f2 xa[NP], xb[NP], xt[NP], ya[NP], yb[NP], yt[NP];
      load_pairs(ring_vec<T>(c, n0, 0, tid), xa);
      load_pairs(ring_vec<T>(c, n0, 1, tid), xb);
      load_or_fill(ring_vec<T>(c, n0 + 1, 0, tid), has1, ya);
      load_or_fill(ring_vec<T>(c, n0 + 1, 1, tid), has1, yb);
      if (needT) {
        load_pairs(ring_vec<T>(c, n0, 2, tid), xt);
        load_or_fill(ring_vec<T>(c, n0 + 1, 2, tid), has1, yt);
      }
      p2_pair<NP, G, false>(xa, xb, xt, ya, yb, yt, has1, k, acc, g0, g1, nullptr, nullptr);
    }
    if (G & (G_RES | G_QF)) p2_groups(g0, g1, grp, kr, c.rounds);
    ring_release(c, n0);
    if (two) ring_release(c, n0 + 1);
  }
  p2_finish(acc, x);
}

// The ring positions of a row without pass 2 (no copies behind them).
template <typename T, bool STOCH>
__device__ __forceinline__ void ring_skip(const KParams& P, RingCtx& c) {
  const unsigned s0 = c.seq;
  c.seq = s0 + static_cast<unsigned>(c.rounds);
  for (int kr = 0; kr < c.rounds; ++kr) {
    const unsigned n = s0 + static_cast<unsigned>(kr);
    ring_wait(c, n);
    ring_release(c, n);
  }
}

// The CTA's pass-1 record of row i goes into slot i % kRSlots of every CTA
// of the cluster (lane r of warp 0 stores into CTA r and arrives, with
// cluster-scope release, on that CTA's row barrier).
template <typename T, bool STOCH, unsigned F>
__device__ __forceinline__ void ring_row_pass1(const KParams& P, RingCtx& c, int i,
                                               cg::cluster_group& cluster) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  (void)VE;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const long long row = ring_row(c, i);
  const size_t off = static_cast<size_t>(row) * P.V + c.lo;
  const T* ga = static_cast<const T*>(P.a) + off;
  const T* gb = static_cast<const T*>(P.b) + off;
  const T* gt = static_cast<const T*>(P.t) + off;
  SharedRing* sh = c.sh;
  X1 e = x1_neutral();
  const bool ovf = ring_pass1<T, STOCH, F>(P, c, ga, gb, gt, e);
  warp_reduce_x1<F>(e);
  X1* w1 = sh->w1[i & 1];
  if (lane == 0) w1[warp] = e;
  if (consumer_sync_or(ovf)) {
    // an entry far above its thread's reference (or non-finite data): redo
    // the slice, from global memory, with a running maximum
    e = x1_neutral();
    pass1_online<T, F, false>(ga, gb, gt, c.nv, c.rounds, (c.rounds + 1) & ~1, c.lo, P.beta,
                              nullptr, e);
    warp_reduce_x1<F>(e);
    if (lane == 0) w1[warp] = e;
    consumer_sync();
  }
  if (warp == 0) {
    X1 w = (lane < kTWarps) ? w1[lane] : x1_neutral();
    warp_reduce_x1<F>(w);
    w.bad |= sh->broken;
    const int K1 = P.K + 1;
    const int k = static_cast<int>(row % K1);
    if (k < P.K) {
      const int dtok = P.tokens[static_cast<size_t>(row / K1) * P.K + k];
      if (dtok >= c.lo && dtok < c.lo + c.n) {  // this CTA's slice holds the draft token
        w.da = to_f32(ga[dtok - c.lo]);
        w.db = to_f32(gb[dtok - c.lo]);
        w.dt = to_f32(gt[dtok - c.lo]);
      }
    }
    const int slot = i % kRSlots;
    if (lane < c.C) {
      X1* dst = cluster.map_shared_rank(sh->recv(slot, c.C), lane) + c.rank;
      const float4* src = reinterpret_cast<const float4*>(&w);
      float4* d = reinterpret_cast<float4*>(dst);
#pragma unroll
      for (int q = 0; q < static_cast<int>(sizeof(X1) / 16); ++q) d[q] = src[q];
      mbar_arrive_remote(&sh->rowbar[slot], static_cast<unsigned>(lane));
    }
  }
}

// Row i once every CTA's pass-1 record is in: its normalisers (rank 0
// leaves the row's pass-1 results for decide_rows) and, with R2, pass 2 from
// the ring and this CTA's pass-2 record and group masses (else the row's
// empty pass-2 positions are passed over).
template <typename T, bool STOCH, unsigned F, unsigned G, bool R2>
__device__ __forceinline__ void ring_row_finish(const KParams& P, RingCtx& c, int i) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const long long row = ring_row(c, i);
  SharedRing* sh = c.sh;
  if (warp == 0) {
    const int slot = i % kRSlots;
    const bool ok =
        mbar_wait_cluster_bounded(&sh->rowbar[slot], (i / kRSlots) & 1, kCopyTimeoutNs);
    const X1* recv = sh->recv(slot, c.C);
    X1 w = (lane < c.C) ? recv[lane] : x1_neutral();
    warp_reduce_x1<F>(w);
    float lse[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) lse[q] = w.ref[q] + logf(w.s[q]);
    if (!ok) w.bad |= kBadTimeout;
    if (lane == 0) {
      if (R2) {
#pragma unroll
        for (int q = 0; q < 4; ++q) sh->lse[q] = lse[q];
      }
      if (c.rank == 0) {
        const int K1 = P.K + 1;
        const int k = static_cast<int>(row % K1);
        int dtok = -1;
        float ad = 0.f, bd = 0.f, td = 0.f;
        if (k < P.K) {
          dtok = P.tokens[static_cast<size_t>(row / K1) * P.K + k];
          if (dtok >= 0 && c.W > 0) {
            const X1& o = recv[dtok / c.W < c.C ? dtok / c.W : 0];
            ad = o.da;
            bd = o.db;
            td = o.dt;
          }
        }
        store_row_stat(P, row, lse, w.is, w.it, w.bad | (ok ? 0u : kBadTimeout), dtok, ad, bd,
                       td);
      }
    }
  }
  if constexpr (R2) {
    consumer_sync();
    const size_t slot = static_cast<size_t>(row) * c.C + c.rank;
    const float lse_a = sh->lse[0], lse_b = sh->lse[1], lse_s = sh->lse[3];
    X2 x = x2_zero();
    ring_pass2<T, STOCH, G>(P, c, lse_a * kLog2e, lse_b * kLog2e, lse_s * kLog2e, lse_s, x,
                            P.group_mass + slot * P.group_stride);
    warp_reduce_x2<G>(x);
    if (lane == 0) sh->w2[warp] = x;
    consumer_sync();
    if (warp == 0) {
      X2 w = (lane < kTWarps) ? sh->w2[lane] : x2_zero();
      warp_reduce_x2<G>(w);
      if (sh->broken) w.pad[0] = __uint_as_float(kBadTimeout);
      if (lane < static_cast<int>(sizeof(X2) / 16))
        reinterpret_cast<float4*>(P.pass2_rec + slot * 8)[lane] =
            reinterpret_cast<const float4*>(&w)[lane];
    }
  } else {
    ring_skip<T, STOCH>(P, c);
  }
}

// The programs of the production modes (see the table in kernel_tma.cuh).
template <typename T, bool STOCH>
__device__ __forceinline__ void ring_dispatch_pass1(const KParams& P, RingCtx& c, int i,
                                                    cg::cluster_group& cluster) {
  const bool bonus = static_cast<int>(ring_row(c, i) % (P.K + 1)) == P.K;
  if constexpr (!STOCH) {
    if (bonus) {
      if (P.fuse_bonus) ring_row_pass1<T, STOCH, F_AS>(P, c, i, cluster);
      else ring_row_pass1<T, STOCH, F_AT>(P, c, i, cluster);
    } else {
      ring_row_pass1<T, STOCH, F_LA | F_LB | F_LT | F_AS>(P, c, i, cluster);
    }
  } else if (P.want_tokens) {  // argmax s as well, for the per-row token output
    if (bonus) ring_row_pass1<T, STOCH, F_LS | F_AS>(P, c, i, cluster);
    else ring_row_pass1<T, STOCH, F_LA | F_LB | F_LS | F_AS>(P, c, i, cluster);
  } else {
    if (bonus) ring_row_pass1<T, STOCH, F_LS>(P, c, i, cluster);
    else ring_row_pass1<T, STOCH, F_LA | F_LB | F_LS>(P, c, i, cluster);
  }
}

template <typename T, bool STOCH>
__device__ __forceinline__ void ring_dispatch_finish(const KParams& P, RingCtx& c, int i) {
  const bool bonus = static_cast<int>(ring_row(c, i) % (P.K + 1)) == P.K;
  const bool jsd = P.divergence == ASYMSPEC_DIV_JSD;
  const bool klg = P.divergence == ASYMSPEC_DIV_KL;
  if constexpr (!STOCH) {
    constexpr unsigned FD = F_LA | F_LB | F_LT | F_AS;
    if (bonus) {
      if (P.fuse_bonus) ring_row_finish<T, STOCH, F_AS, 0, false>(P, c, i);
      else ring_row_finish<T, STOCH, F_AT, 0, false>(P, c, i);
    } else if (jsd) {
      ring_row_finish<T, STOCH, FD, G_JSD, true>(P, c, i);
    } else if (klg) {
      ring_row_finish<T, STOCH, FD, G_KL, true>(P, c, i);
    } else {
      ring_row_finish<T, STOCH, FD, 0, false>(P, c, i);
    }
  } else if (P.want_tokens) {
    constexpr unsigned FS = F_LA | F_LB | F_LS | F_AS;
    if (bonus) ring_row_finish<T, STOCH, F_LS | F_AS, G_QF, true>(P, c, i);
    else if (jsd) ring_row_finish<T, STOCH, FS, G_JSD | G_RES, true>(P, c, i);
    else if (klg) ring_row_finish<T, STOCH, FS, G_KL | G_RES, true>(P, c, i);
    else ring_row_finish<T, STOCH, FS, G_RES, true>(P, c, i);
  } else {
    constexpr unsigned FS = F_LA | F_LB | F_LS;
    if (bonus) ring_row_finish<T, STOCH, F_LS, G_QF, true>(P, c, i);
    else if (jsd) ring_row_finish<T, STOCH, FS, G_JSD | G_RES, true>(P, c, i);
    else if (klg) ring_row_finish<T, STOCH, FS, G_KL | G_RES, true>(P, c, i);
    else ring_row_finish<T, STOCH, FS, G_RES, true>(P, c, i);
  }
}

// ---------------------------------------------------------------- the kernel

template <typename T, bool STOCH>
__global__ void __launch_bounds__(kRThreads, 2) fuse_verify_ring(const __grid_constant__ KParams P) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  extern __shared__ __align__(128) unsigned char smem_ring[];
  cg::cluster_group cluster = cg::this_cluster();
  RingCtx c;
  c.ring = smem_ring;
  c.sh = reinterpret_cast<SharedRing*>(smem_ring + kRRingBytes);
  c.C = P.C;
  c.rank = static_cast<int>(cluster.block_rank());
  c.ncl = static_cast<int>(gridDim.x) / c.C;
  c.q = static_cast<int>(blockIdx.x) / c.C;
  c.nrows = (P.rows > c.q) ? static_cast<int>((P.rows - c.q + c.ncl - 1) / c.ncl) : 0;
  c.W = P.W;
  c.lo = c.rank * c.W;
  c.n = max(0, min(c.W, P.V - c.lo));
  c.nv = c.n / VE;
  c.rounds = (c.nv + kTThreads - 1) / kTThreads;
  c.seq = 0;
  c.issued = 0;
  c.total = static_cast<unsigned>(c.nrows) * 2u * static_cast<unsigned>(c.rounds);
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(c.pol1));
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(c.pol2));
  SharedRing* sh = c.sh;
  if (threadIdx.x == 0) {
#pragma unroll
    for (int s = 0; s < kRStages; ++s) {
      mbar_init(&sh->full[s], 1);
      mbar_init(&sh->empty[s], kTWarps);
    }
#pragma unroll
    for (int s = 0; s < kRSlots; ++s) mbar_init(&sh->rowbar[s], static_cast<unsigned>(c.C));
    sh->broken = 0;
    fence_mbar_init();
  }
  __syncwarp();
  cluster.sync();  // every CTA's barriers are initialised before any remote arrive
  if (threadIdx.x >= kTThreads) {
    // the producer warp: lane 0 keeps the ring full
    if (threadIdx.x == kTThreads) ring_produce<T, STOCH>(P, c);
    __syncwarp();
  } else {
    for (int i = 0; i < c.nrows; ++i) {
      ring_dispatch_pass1<T, STOCH>(P, c, i, cluster);
      ring_dispatch_finish<T, STOCH>(P, c, i);
    }
  }
  // after a timeout, copies still in flight land before the CTA exits
  if (threadIdx.x == kTThreads && sh->broken) {
    for (unsigned n = c.issued > static_cast<unsigned>(kRStages) ? c.issued - kRStages : 0u;
         n < c.issued; ++n)
      mbar_wait_bounded(&sh->full[n % kRStages], (n / kRStages) & 1u, kCopyTimeoutNs);
  }
  __syncwarp();
  cluster.sync();  // no CTA leaves while a peer may still push into it
}

}  // namespace asymspec_impl
