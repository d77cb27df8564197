// Streaming fuse-and-verify kernel: the two passes over a row read it twice,
// once from HBM and once from L2, instead of holding it in shared memory.
//
// Work items.  Row r of the B(K+1) verify rows is cut into NT tiles of TS
// vocabulary entries (8 vectors of 16 bytes per thread and tile).  A tile has
// a pass-1 item (partial normalisers and argmaxes) and a pass-2 item
// (divergence terms and inverse-CDF masses, which need the row's
// normalisers).  Items are laid out in steps: step s holds the pass-1 items
// of row s and the pass-2 items of row s - D, so a row's second read comes D
// rows after its first, while the row is still in L2 (pass-1 loads carry an
// evict_last policy, pass-2 loads evict_first).  D spans more than one wave
// of the grid, so pass-2 items seldom wait.
//
// Persistent grid.  Exactly as many CTAs as are resident together (a
// cooperative launch, so the hardware refuses otherwise); CTA c takes items
// c, c+G, c+2G, ...  A pass-2 item waits only for pass-1 items of lower
// index, which resident CTAs are working on or have finished, so every wait
// ends; each wait is bounded all the same (200 ms, then the row is marked
// ASYMSPEC_DATA_TIMEOUT).
//
// Per item: every warp reduces its threads' partials, a __syncthreads, then
// one warp (rotating with the item count) combines the eight warp records,
// stores the tile record and takes the row's ticket; the warp that completes
// a row's pass 1 publishes its normalisers (tagged 64-bit words that pass-2
// items poll), the warp that completes its pass 2 draws from the inverse CDF
// and decides the row (Algorithm 1's scan through the element's ticket).
// All per-row counters, flags and tags return to zero when the row is done.
#pragma once

#include "kernel_tma.cuh"

namespace asymspec_impl {

constexpr int kSThreads = 256;
constexpr int kSWarps = kSThreads / 32;
constexpr int kSRounds = 8;                     // vectors per thread and tile
constexpr int kSGroups = kSRounds * kSWarps;    // 32-vector groups per tile
constexpr unsigned long long kWaitNs = 200ull * 1000ull * 1000ull;

enum : int {
  PG_GREEDY_DRAFT_JSD, PG_GREEDY_DRAFT_KL, PG_GREEDY_DRAFT_NONE,
  PG_GREEDY_BONUS_T, PG_GREEDY_BONUS_S,
  PG_STOCH_DRAFT_JSD, PG_STOCH_DRAFT_KL, PG_STOCH_DRAFT_NONE,
  PG_STOCH_DRAFT_JSD_TOK, PG_STOCH_DRAFT_KL_TOK, PG_STOCH_DRAFT_NONE_TOK,
  PG_STOCH_BONUS, PG_STOCH_BONUS_TOK,
  PG_FULL_JSD, PG_FULL_KL, PG_FULL_NONE, PG_FULL_JSD_LP, PG_FULL_KL_LP, PG_FULL_NONE_LP
};

// Workspace of the streaming kernel (device pointers into one allocation).
struct StreamWs {
  int4* recs;                   // [B(K+1)] row records (Algorithm 1's scan)
  unsigned* tickets;            // [B]
  unsigned* p1cnt;              // [B(K+1)] pass-1 tiles done
  unsigned* p2cnt;              // [B(K+1)] pass-2 tiles done
  unsigned* ready;              // [B(K+1)] RowStat published (release)
  unsigned long long* tags;     // [B(K+1)][4] (value, 1) words: lse_a, lse_b, lse_s in log2 units, lse_s
  RowStat* stat;                // [B(K+1)]
  X1* p1rec;                    // [B(K+1)][NT]
  X2* p2rec;                    // [B(K+1)][NT]
  float* groups;                // [B(K+1)][NT][kSGroups] inverse-CDF mass of each 32-vector group
};

struct SParams {
  KParams P;                    // the arguments (P.recs / P.tickets alias ws)
  StreamWs ws;
  int NT, TS, D;                // tiles per row, entries per tile, look-ahead in rows
  long long NI;                 // items
  int program[2];               // row program of draft rows / of the bonus row
};

__device__ __forceinline__ unsigned long long policy_evict_last() {
  unsigned long long p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ unsigned long long policy_evict_first() {
  unsigned long long p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// 16 bytes of read-only input straight to registers, with an L2 policy.
__device__ __forceinline__ uint4 ldg16(const void* p, unsigned long long pol) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ void pairs_of(uint4 v, const float*, f2 (&x)[2]) {
  x[0] = pk(__uint_as_float(v.x), __uint_as_float(v.y));
  x[1] = pk(__uint_as_float(v.z), __uint_as_float(v.w));
}
__device__ __forceinline__ void pairs_of(uint4 v, const __nv_bfloat16*, f2 (&x)[4]) {
  const unsigned w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int h = 0; h < 4; ++h)
    x[h] = pk(__uint_as_float(w[h] << 16), __uint_as_float(w[h] & 0xFFFF0000u));
}
template <typename T, int NP>
__device__ __forceinline__ void gload_pairs(const T* p, unsigned long long pol, f2 (&x)[NP]) {
  pairs_of(ldg16(p, pol), p, x);
}
template <typename T, int NP>
__device__ __forceinline__ void gload_or_fill(const T* p, bool ok, unsigned long long pol,
                                              f2 (&x)[NP]) {
  if (ok) {
    gload_pairs(p, pol, x);
  } else {
#pragma unroll
    for (int h = 0; h < NP; ++h) x[h] = pk(-1e30f, -1e30f);  // contributes nothing
  }
}

__device__ __forceinline__ unsigned long long ld_relaxed64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_relaxed64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release32(unsigned* p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned long long tag_word(float v) {
  return (1ull << 32) | static_cast<unsigned long long>(__float_as_uint(v));
}

// The ring: kSStages stages of one round each (a vector of a, b and t per
// thread, 4 KB per stream), filled by 1-D bulk copies that thread 0 issues
// up to kSStages - 1 chunks ahead of consumption, across item boundaries.
constexpr int kSStages = 8;
constexpr int kStreamBytes = kSThreads * 16;
constexpr int kStageBytes = 3 * kStreamBytes;
constexpr int kRingBytes = kSStages * kStageBytes;

// Producer state (thread 0 alone reads and writes it).
struct ItemInfo {
  long long row;
  int tile, prog, nvec, nch;  // tile vectors, chunks (rounds of kSThreads vectors)
  unsigned streams;           // bit 0: a, bit 1: b, bit 2: t copied into the ring
  bool p2;
};
struct Ring {
  long long pi;       // item of the next chunk to issue
  long long issued;   // chunks issued so far
  int pc;             // that chunk's index within its item
  int pvalid;
  ItemInfo pit;
};

struct SharedStream {
  unsigned long long full[kSStages];   // a stage's copies have landed (count 1 + bytes)
  unsigned long long empty[kSStages];  // every warp is done with a stage (count kSWarps)
  X1 w1[2][kSWarps];                   // per-warp records, by item parity
  X2 w2[2][kSWarps];
  Ring prod;
  unsigned broken;                     // a chunk wait ran out of time
};

// ---------------------------------------------------------------- row program

__device__ __forceinline__ int row_program(const SParams& S, int k) {
  return S.program[k == S.P.K ? 1 : 0];
}

// Whether rows of this program have a pass 2.
__host__ __device__ constexpr bool program_has_pass2(int prog) {
  return !(prog == PG_GREEDY_DRAFT_NONE || prog == PG_GREEDY_BONUS_T || prog == PG_GREEDY_BONUS_S);
}

// One work item as the producer and the consumers see it.

template <typename T>
__device__ __forceinline__ bool item_info(const SParams& S, long long i, ItemInfo& it) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const long long per_step = 2ll * S.NT;
  const long long s = i / per_step;
  const int slot = static_cast<int>(i - s * per_step);
  it.p2 = slot >= S.NT;
  it.row = it.p2 ? s - S.D : s;
  if (it.row < 0 || it.row >= S.P.rows) return false;
  const int k = static_cast<int>(it.row % (S.P.K + 1));
  it.prog = row_program(S, k);
  if (it.p2 && !program_has_pass2(it.prog)) return false;
  it.tile = it.p2 ? slot - S.NT : slot;
  const int t0 = it.tile * S.TS;
  it.nvec = (min(S.P.V, t0 + S.TS) - t0) / VE;
  it.nch = (it.nvec + kSThreads - 1) / kSThreads;
  const bool greedy_div = it.prog == PG_GREEDY_DRAFT_JSD || it.prog == PG_GREEDY_DRAFT_KL;
  if (!it.p2) it.streams = it.prog == PG_GREEDY_BONUS_T ? 4u : 7u;
  else it.streams = greedy_div ? 3u : 7u;
  return true;
}

template <typename T>
__device__ __forceinline__ void ring_seek(const SParams& S, Ring& R) {
  while (R.pi < S.NI && !item_info<T>(S, R.pi, R.pit)) R.pi += gridDim.x;
  R.pvalid = R.pi < S.NI ? 1 : 0;
  R.pc = 0;
}

// Thread 0: issue every chunk before consumption index q_cons + kSStages.
// A stage is reused once all warps have released its previous chunk.
template <typename T>
__device__ __noinline__ void ring_top_up(const SParams& S, SharedStream* sh, unsigned char* buf,
                                         long long q_cons) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  Ring& R = sh->prod;
  while (R.pvalid && R.issued < q_cons + kSStages) {
    const long long q = R.issued;
    const int st = static_cast<int>(q % kSStages);
    if (q >= kSStages &&
        !mbar_wait_bounded(&sh->empty[st], static_cast<unsigned>((q / kSStages - 1) & 1), kWaitNs))
      sh->broken = 1u;
    const int v0 = R.pc * kSThreads;
    const int nv = min(kSThreads, R.pit.nvec - v0);
    const unsigned bytes = static_cast<unsigned>(nv) * 16u;
    const unsigned ns = __popc(R.pit.streams);
    mbar_arrive_expect_tx(&sh->full[st], bytes * ns);
    const size_t off = static_cast<size_t>(R.pit.row) * S.P.V + R.pit.tile * S.TS + v0 * VE;
    const unsigned long long pol = R.pit.p2 ? policy_evict_first() : policy_evict_last();
    unsigned char* dst = buf + st * kStageBytes;
    if (R.pit.streams & 1u)
      bulk_load_hint(dst, static_cast<const T*>(S.P.a) + off, bytes, &sh->full[st], pol);
    if (R.pit.streams & 2u)
      bulk_load_hint(dst + kStreamBytes, static_cast<const T*>(S.P.b) + off, bytes, &sh->full[st],
                     pol);
    if (R.pit.streams & 4u)
      bulk_load_hint(dst + 2 * kStreamBytes, static_cast<const T*>(S.P.t) + off, bytes,
                     &sh->full[st], pol);
    ++R.issued;
    if (++R.pc == R.pit.nch) {
      R.pi += gridDim.x;
      ring_seek<T>(S, R);
    }
  }
}

// Consumer side of chunk q: wait for it (bounded) and return its stage.
__device__ __forceinline__ unsigned char* ring_acquire(SharedStream* sh, unsigned char* buf,
                                                       long long q) {
  const int st = static_cast<int>(q % kSStages);
  if (!mbar_wait_bounded(&sh->full[st], static_cast<unsigned>((q / kSStages) & 1), kWaitNs))
    sh->broken = 1u;
  return buf + st * kStageBytes;
}

// Every lane of the warp is done reading chunk q.
__device__ __forceinline__ void ring_release(SharedStream* sh, long long q) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&sh->empty[q % kSStages]);
}

// ---------------------------------------------------------------- pass-1 item

// Per-thread pass 1 over one tile from global memory (evict_last: the tile
// is read again by its pass-2 item), against fixed references as in
// pass1_fast; argmaxes are resolved in registers when they improve.
// Returns true on overflow (the caller then redoes the tile online).
template <typename T, unsigned F, bool ONLINE>
__device__ __forceinline__ bool tile_pass1(const T* ra, const T* rb, const T* rt, int nvec,
                                           int t0, float beta, unsigned long long pol, X1& e) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needA = (F & (F_LA | F_LS | F_AS)) != 0;
  constexpr bool needB = (F & (F_LB | F_LS | F_AS)) != 0;
  constexpr bool needT = (F & (F_LT | F_LS | F_AS | F_AT)) != 0;
  constexpr bool needS = (F & (F_LS | F_AS)) != 0;
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  const int tid = static_cast<int>(threadIdx.x);
  float ref[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  f2 acc[4] = {0ull, 0ull, 0ull, 0ull};
  f2 nm[4];
  bool first = true;
#pragma unroll 1
  for (int j = 0; j < kSRounds; j += 2) {
    const int i0 = j * kSThreads + tid, i1 = i0 + kSThreads;
    if (i0 >= nvec) break;
    const bool has1 = i1 < nvec;
    f2 xa[NP], xb[NP], xt[NP], xs[NP], ya[NP], yb[NP], yt[NP], ys[NP];
    if (needA) {
      gload_pairs(ra + i0 * VE, pol, xa);
      gload_or_fill(ra + i1 * VE, has1, pol, ya);
    }
    if (needB) {
      gload_pairs(rb + i0 * VE, pol, xb);
      gload_or_fill(rb + i1 * VE, has1, pol, yb);
    }
    if (needT) {
      gload_pairs(rt + i0 * VE, pol, xt);
      gload_or_fill(rt + i1 * VE, has1, pol, yt);
    }
    if (needS) {
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
        ys[h] = fma2(beta2, sub2(ya[h], yb[h]), yt[h]);
      }
    }
    if constexpr (ONLINE) {
      if (F & F_LA) online_pairs2(ref[0], acc[0], xa, ya, L2);
      if (F & F_LB) online_pairs2(ref[1], acc[1], xb, yb, L2);
      if (F & F_LT) online_pairs2(ref[2], acc[2], xt, yt, L2);
      if (F & F_LS) online_pairs2(ref[3], acc[3], xs, ys, L2);
    } else {
      if (first) {  // this thread's first vector sets its references
        if (F & F_LA) ref[0] = vmax_pairs(xa);
        if (F & F_LB) ref[1] = vmax_pairs(xb);
        if (F & F_LT) ref[2] = vmax_pairs(xt);
        if (F & F_LS) ref[3] = vmax_pairs(xs);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float v = -ref[q] * kLog2e;
          nm[q] = pk(v, v);
        }
        first = false;
      }
      if (F & F_LA) fixed_pairs2(acc[0], xa, ya, L2, nm[0]);
      if (F & F_LB) fixed_pairs2(acc[1], xb, yb, L2, nm[1]);
      if (F & F_LT) fixed_pairs2(acc[2], xt, yt, L2, nm[2]);
      if (F & F_LS) fixed_pairs2(acc[3], xs, ys, L2, nm[3]);
    }
    if (F & F_AS) {
      const float cs0 = (F & F_LS) ? vmax_pairs(xs) : vmax_pairs_nan(xs);
      const float cs1 = (F & F_LS) ? vmax_pairs(ys) : vmax_pairs_nan(ys);
      if (!(cs0 <= 3.402823466e38f)) e.bad |= kBadS;
      if (cs0 > e.vs) {
        e.vs = cs0;
        e.is = arg_in_vector(xs, cs0, t0 + i0 * VE);
      }
      if (has1) {
        if (!(cs1 <= 3.402823466e38f)) e.bad |= kBadS;
        if (cs1 > e.vs) {
          e.vs = cs1;
          e.is = arg_in_vector(ys, cs1, t0 + i1 * VE);
        }
      }
    }
    if (F & F_AT) {
      const float ct0 = (F & F_LT) ? vmax_pairs(xt) : vmax_pairs_nan(xt);
      const float ct1 = (F & F_LT) ? vmax_pairs(yt) : vmax_pairs_nan(yt);
      if (!(ct0 <= 3.402823466e38f)) e.bad |= kBadT;
      if (ct0 > e.vt) {
        e.vt = ct0;
        e.it = arg_in_vector(xt, ct0, t0 + i0 * VE);
      }
      if (has1) {
        if (!(ct1 <= 3.402823466e38f)) e.bad |= kBadT;
        if (ct1 > e.vt) {
          e.vt = ct1;
          e.it = arg_in_vector(yt, ct1, t0 + i1 * VE);
        }
      }
    }
  }
  bool ovf = false;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const unsigned bit = q == 0 ? F_LA : q == 1 ? F_LB : q == 2 ? F_LT : F_LS;
    e.ref[q] = ref[q];
    e.s[q] = hsum2(acc[q]);
    if (!ONLINE && (F & bit) && !(e.s[q] < kSumLimit)) ovf = true;
  }
  return ovf;
}

// Vector `tid` of a ring stage (stream s = 0 a, 1 b, 2 t), or the fill value.
template <typename T, int NP>
__device__ __forceinline__ void stage_pairs(const unsigned char* stage, int s, bool ok,
                                            f2 (&x)[NP]) {
  if (ok) {
    load_pairs(reinterpret_cast<const T*>(stage + s * kStreamBytes) +
                   threadIdx.x * (16 / static_cast<int>(sizeof(T))),
               x);
  } else {
#pragma unroll
    for (int h = 0; h < NP; ++h) x[h] = pk(-1e30f, -1e30f);  // contributes nothing
  }
}

// Pass 1 over one tile from the ring (chunks q, q+1, ... of this CTA), two
// chunks per step; as tile_pass1 with fixed references.  Thread 0 keeps the
// ring topped up.  Returns true on overflow.
template <typename T, unsigned F>
__device__ __forceinline__ bool ring_pass1(const SParams& S, SharedStream* sh,
                                           unsigned char* buf, long long q, int nvec, int nch,
                                           int t0, float beta, X1& e) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool needA = (F & (F_LA | F_LS | F_AS)) != 0;
  constexpr bool needB = (F & (F_LB | F_LS | F_AS)) != 0;
  constexpr bool needT = (F & (F_LT | F_LS | F_AS | F_AT)) != 0;
  constexpr bool needS = (F & (F_LS | F_AS)) != 0;
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  const int tid = static_cast<int>(threadIdx.x);
  float ref[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  f2 acc[4] = {0ull, 0ull, 0ull, 0ull};
  f2 nm[4];
  for (int c = 0; c < nch; c += 2, q += 2) {
    const bool two = c + 1 < nch;
    if (tid == 0) ring_top_up<T>(S, sh, buf, q);
    const unsigned char* s0 = ring_acquire(sh, buf, q);
    const unsigned char* s1 = two ? ring_acquire(sh, buf, q + 1) : s0;
    const int i0 = c * kSThreads + tid, i1 = i0 + kSThreads;
    const bool has0 = i0 < nvec, has1 = two && i1 < nvec;
    f2 xa[NP], xb[NP], xt[NP], xs[NP], ya[NP], yb[NP], yt[NP], ys[NP];
    if (needA) {
      stage_pairs<T>(s0, 0, has0, xa);
      stage_pairs<T>(s1, 0, has1, ya);
    }
    if (needB) {
      stage_pairs<T>(s0, 1, has0, xb);
      stage_pairs<T>(s1, 1, has1, yb);
    }
    if (needT) {
      stage_pairs<T>(s0, 2, has0, xt);
      stage_pairs<T>(s1, 2, has1, yt);
    }
    ring_release(sh, q);
    if (two) ring_release(sh, q + 1);
    if (needS) {
#pragma unroll
      for (int h = 0; h < NP; ++h) {
        xs[h] = fma2(beta2, sub2(xa[h], xb[h]), xt[h]);
        ys[h] = fma2(beta2, sub2(ya[h], yb[h]), yt[h]);
      }
    }
    if (c == 0) {  // this thread's first vector sets its references
      if (has0) {
        if (F & F_LA) ref[0] = vmax_pairs(xa);
        if (F & F_LB) ref[1] = vmax_pairs(xb);
        if (F & F_LT) ref[2] = vmax_pairs(xt);
        if (F & F_LS) ref[3] = vmax_pairs(xs);
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float v = -ref[k] * kLog2e;
        nm[k] = pk(v, v);
      }
    }
    if (has0) {
      if (F & F_LA) fixed_pairs2(acc[0], xa, ya, L2, nm[0]);
      if (F & F_LB) fixed_pairs2(acc[1], xb, yb, L2, nm[1]);
      if (F & F_LT) fixed_pairs2(acc[2], xt, yt, L2, nm[2]);
      if (F & F_LS) fixed_pairs2(acc[3], xs, ys, L2, nm[3]);
      if (F & F_AS) {
        const float cs0 = (F & F_LS) ? vmax_pairs(xs) : vmax_pairs_nan(xs);
        if (!(cs0 <= 3.402823466e38f)) e.bad |= kBadS;
        if (cs0 > e.vs) {
          e.vs = cs0;
          e.is = arg_in_vector(xs, cs0, t0 + i0 * VE);
        }
        if (has1) {
          const float cs1 = (F & F_LS) ? vmax_pairs(ys) : vmax_pairs_nan(ys);
          if (!(cs1 <= 3.402823466e38f)) e.bad |= kBadS;
          if (cs1 > e.vs) {
            e.vs = cs1;
            e.is = arg_in_vector(ys, cs1, t0 + i1 * VE);
          }
        }
      }
      if (F & F_AT) {
        const float ct0 = (F & F_LT) ? vmax_pairs(xt) : vmax_pairs_nan(xt);
        if (!(ct0 <= 3.402823466e38f)) e.bad |= kBadT;
        if (ct0 > e.vt) {
          e.vt = ct0;
          e.it = arg_in_vector(xt, ct0, t0 + i0 * VE);
        }
        if (has1) {
          const float ct1 = (F & F_LT) ? vmax_pairs(yt) : vmax_pairs_nan(yt);
          if (!(ct1 <= 3.402823466e38f)) e.bad |= kBadT;
          if (ct1 > e.vt) {
            e.vt = ct1;
            e.it = arg_in_vector(yt, ct1, t0 + i1 * VE);
          }
        }
      }
    }
  }
  bool ovf = false;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const unsigned bit = k == 0 ? F_LA : k == 1 ? F_LB : k == 2 ? F_LT : F_LS;
    e.ref[k] = ref[k];
    e.s[k] = hsum2(acc[k]);
    if ((F & bit) && !(e.s[k] < kSumLimit)) ovf = true;
  }
  return ovf;
}

// The tile again with a running maximum (the rare fallback of pass 1).
template <typename T, unsigned F>
__device__ __noinline__ void redo_pass1(const T* ra, const T* rb, const T* rt, int nvec, int t0,
                                        float beta, unsigned long long pol, X1* slot) {
  X1 e = x1_neutral();
  tile_pass1<T, F, true>(ra, rb, rt, nvec, t0, beta, pol, e);
  warp_reduce_x1<F>(e);
  if ((threadIdx.x & 31) == 0) *slot = e;
}

// ---------------------------------------------------------------- pass-2 item

// Pass 2 over one tile from the ring, two chunks per step.  Group g of the
// tile is vectors [32 g, 32 g + 32), the 32 lanes of warp (g % 8) in round
// g / 8; lane 0 stores its residual (or, for the bonus row, fused) mass.
template <typename T, unsigned G, bool LP>
__device__ __forceinline__ void ring_pass2(const SParams& S, SharedStream* sh,
                                           unsigned char* buf, long long q, int nvec, int nch,
                                           float beta, float A2, float B2, float S2, float lse_s,
                                           X2& x, float* lp, float* groups) {
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int NP = VE / 2;
  constexpr bool JSD = (G & G_JSD) != 0, KL = (G & G_KL) != 0, RES = (G & G_RES) != 0;
  constexpr bool QF = (G & G_QF) != 0;
  constexpr bool needT = RES || QF || LP;
  const int tid = static_cast<int>(threadIdx.x), lane = tid & 31, warp = tid >> 5;
  const f2 beta2 = pk(beta, beta);
  const f2 L2 = pk(kLog2e, kLog2e);
  const f2 nA2 = pk(-A2, -A2), nB2 = pk(-B2, -B2), nS2 = pk(-S2, -S2);
  const f2 tiny2 = pk(kMinNormal, kMinNormal);
  const f2 nl2 = pk(-lse_s, -lse_s);
  f2 ja = 0ull, jb = 0ull, ms2 = 0ull, kl2 = 0ull, R2 = 0ull, Q2 = 0ull;
  for (int c = 0; c < nch; c += 2, q += 2) {
    const bool two = c + 1 < nch;
    if (tid == 0) ring_top_up<T>(S, sh, buf, q);
    const unsigned char* s0 = ring_acquire(sh, buf, q);
    const unsigned char* s1 = two ? ring_acquire(sh, buf, q + 1) : s0;
    const int i0 = c * kSThreads + tid, i1 = i0 + kSThreads;
    const bool has0 = i0 < nvec, has1 = two && i1 < nvec;
    f2 xa[NP], xb[NP], xt[NP], ya[NP], yb[NP], yt[NP];
    stage_pairs<T>(s0, 0, has0, xa);
    stage_pairs<T>(s0, 1, has0, xb);
    stage_pairs<T>(s1, 0, has1, ya);
    stage_pairs<T>(s1, 1, has1, yb);
    if (needT) {
      stage_pairs<T>(s0, 2, has0, xt);
      stage_pairs<T>(s1, 2, has1, yt);
    }
    ring_release(sh, q);
    if (two) ring_release(sh, q + 1);
    float g0 = 0.f, g1 = 0.f;  // this thread's vector masses (groups of rounds c, c+1)
    if (__any_sync(0xffffffffu, has0)) {
      f2 px[NP], py[NP];
      if (RES) {
        f2 qx[NP], qy[NP], rx[NP], ry[NP];
        vec_masses(xa, xb, xt, beta2, L2, nA2, nS2, px, qx, rx);
        vec_masses(ya, yb, yt, beta2, L2, nA2, nS2, py, qy, ry);
#pragma unroll
        for (int h = 0; h < NP; ++h) Q2 = add2(Q2, add2(qx[h], qy[h]));
        g0 = vsum(rx);
        g1 = vsum(ry);
        R2 = add2(R2, pk(g0, g1));
      } else if (QF) {
        f2 qx[NP], qy[NP];
#pragma unroll
        for (int h = 0; h < NP; ++h) {
          qx[h] = ex2_2(fma2(fma2(beta2, sub2(xa[h], xb[h]), xt[h]), L2, nS2));
          qy[h] = ex2_2(fma2(fma2(beta2, sub2(ya[h], yb[h]), yt[h]), L2, nS2));
        }
        g0 = vsum(qx);
        g1 = vsum(qy);
        Q2 = add2(Q2, pk(g0, g1));
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
          if (has0) {
            upk(add2(fma2(beta2, sub2(xa[h], xb[h]), xt[h]), nl2), l0, l1);
            lp[i0 * VE + 2 * h] = l0;
            lp[i0 * VE + 2 * h + 1] = l1;
          }
          if (has1) {
            upk(add2(fma2(beta2, sub2(ya[h], yb[h]), yt[h]), nl2), l0, l1);
            lp[i1 * VE + 2 * h] = l0;
            lp[i1 * VE + 2 * h + 1] = l1;
          }
        }
      }
    }
    if (RES || QF) {
      const float m0 = warp_sum(g0), m1 = warp_sum(g1);
      if (lane == 0) {
        groups[c * kSWarps + warp] = m0;
        if (two) groups[(c + 1) * kSWarps + warp] = m1;
      }
    }
  }
  if (RES || QF) {  // groups of rounds the tile does not reach hold no mass
    for (int c = nch + (nch & 1); c < kSRounds; ++c)
      if (lane == 0) groups[c * kSWarps + warp] = 0.f;
    if ((nch & 1) && lane == 0) groups[nch * kSWarps + warp] = 0.f;
  }
  x.j = hsum2(add2(ja, jb));
  x.msum = hsum2(ms2);
  x.kl = hsum2(kl2);
  x.R = hsum2(R2);
  x.Q = hsum2(Q2);
}

// ---------------------------------------------------------------- inverse-CDF draw

// ---------------------------------------------------------------- row completion

// After the last pass-1 tile of a row (one warp, records acquired): the row's
// normalisers, argmaxes and draft logits.  Publishes them for pass 2, or,
// when the row has no pass 2, decides it.
template <typename T, bool STOCH, unsigned F, bool R2>
__device__ __noinline__ void row_after_pass1(const SParams& S, long long row, int bi, int k) {
  const KParams& P = S.P;
  const int lane = threadIdx.x & 31;
  const X1* rec = S.ws.p1rec + row * S.NT;
  X1 w = x1_neutral();
  // the records were written by other CTAs: read them from L2
  if (lane < S.NT) {
    const float4* src = reinterpret_cast<const float4*>(rec + lane);
    float4* dst = reinterpret_cast<float4*>(&w);
#pragma unroll
    for (int q = 0; q < static_cast<int>(sizeof(X1) / 16); ++q) dst[q] = __ldcg(src + q);
  }
  const bool bonus = (k == P.K);
  const int dtok = bonus ? -1 : __ldg(P.tokens + static_cast<size_t>(bi) * P.K + k);
  float ad = 0.f, bd = 0.f, td = 0.f;
  if (dtok >= 0 && dtok < P.V) {
    const size_t o = static_cast<size_t>(row) * P.V + dtok;
    ad = to_f32(static_cast<const T*>(P.a)[o]);
    bd = to_f32(static_cast<const T*>(P.b)[o]);
    td = to_f32(static_cast<const T*>(P.t)[o]);
  }
  warp_reduce_x1<F>(w);
  float lse[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) lse[q] = w.ref[q] + logf(w.s[q]);
  if constexpr (!R2) {
    const bool has_ab = P.full || !bonus;
    const bool has_t = P.full || (!STOCH && !bonus);
    RowResult r;
    r.lse_a = has_ab ? lse[0] : NAN;
    r.lse_b = has_ab ? lse[1] : NAN;
    r.lse_t = has_t ? lse[2] : NAN;
    r.lse_s = (P.full || STOCH) ? lse[3] : NAN;
    r.D = 0.f;
    r.is = w.is;
    r.it = w.it;
    r.sample = -1;
    r.mass = NAN;
    r.bad = w.bad;
    r.have_lse_t = has_t;
    const RowScalars sc = STOCH ? load_row_scalars(P, bi, k) : RowScalars{0.f, 0.f, 0.f};
    finish_row_warp<STOCH>(P, row, bi, k, r, dtok, ad, bd, td, sc);
    if (lane == 0) S.ws.p1cnt[row] = 0u;
  } else {
    if (lane == 0) {
      RowStat st;
#pragma unroll
      for (int q = 0; q < 4; ++q) st.lse[q] = lse[q];
      st.is = w.is;
      st.it = w.it;
      st.bad = w.bad;
      st.dtok = dtok;
      st.da = ad;
      st.db = bd;
      st.dt = td;
      st.pad = 0.f;
      S.ws.stat[row] = st;
      unsigned long long* tg = S.ws.tags + row * 4;
      st_relaxed64(tg + 0, tag_word(lse[0] * kLog2e));
      st_relaxed64(tg + 1, tag_word(lse[1] * kLog2e));
      st_relaxed64(tg + 2, tag_word(lse[3] * kLog2e));
      st_relaxed64(tg + 3, tag_word(lse[3]));
      S.ws.p1cnt[row] = 0u;
      st_release32(S.ws.ready + row, 1u);
    }
  }
}

// After the last pass-2 tile of a row (one warp, records acquired): the
// divergence, the inverse-CDF draw (stochastic), and the row decision.
template <typename T, bool STOCH, unsigned G>
__device__ __noinline__ void row_after_pass2(const SParams& S, long long row, int bi, int k) {
  const KParams& P = S.P;
  const int lane = threadIdx.x & 31;
  const bool bonus = (k == P.K);
  // the RowStat of pass 1 (released through `ready`)
  unsigned rdy = 0;
  if (lane == 0) {
    const unsigned long long t0 = global_ns();
    while ((rdy = ld_acquire32(S.ws.ready + row)) == 0u) {
      if (global_ns() - t0 > kWaitNs) break;
      __nanosleep(128);
    }
  }
  rdy = __shfl_sync(0xffffffffu, rdy, 0);
  __syncwarp();
  RowStat st;
  {
    const float4* src = reinterpret_cast<const float4*>(S.ws.stat + row);
    float4* dst = reinterpret_cast<float4*>(&st);
#pragma unroll
    for (int q = 0; q < static_cast<int>(sizeof(RowStat) / 16); ++q) dst[q] = __ldcg(src + q);
  }
  if (!rdy) st.bad |= kBadTimeout;
  X2 w = x2_zero();
  if (lane < S.NT) {
    const float4* src = reinterpret_cast<const float4*>(S.ws.p2rec + row * S.NT + lane);
    float4* dst = reinterpret_cast<float4*>(&w);
#pragma unroll
    for (int q = 0; q < static_cast<int>(sizeof(X2) / 16); ++q) dst[q] = __ldcg(src + q);
  }
  const RowScalars sc = STOCH ? load_row_scalars(P, bi, k) : RowScalars{0.f, 0.f, 0.f};
  if (__any_sync(0xffffffffu, __float_as_uint(w.pad[0]) != 0u)) st.bad |= kBadTimeout;
  X2 tot = w;
  warp_reduce_x2<G>(tot);
  const float D = divergence_of<G>(tot);
  int sample = -1;
  float mass_total = NAN;
  if constexpr (STOCH) {
    // inclusive prefix of the inverse-CDF mass over tiles, in tile order
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
    const unsigned over = __ballot_sync(0xffffffffu, lane < S.NT && incl > tau);
    const unsigned pos = __ballot_sync(0xffffffffu, lane < S.NT && mass > 0.f);
    int owner = -1;
    if (over) owner = __ffs(over) - 1;
    else if (pos) owner = 31 - __clz(pos);
    if (owner >= 0) {
      const float incl_o = __shfl_sync(0xffffffffu, incl, owner);
      const float mass_o = __shfl_sync(0xffffffffu, mass, owner);
      const float tau_local = fmaxf(tau - (incl_o - mass_o), 0.f);
      const int t0 = owner * S.TS;
      const int nvec = (min(P.V, t0 + S.TS) - t0) / (16 / static_cast<int>(sizeof(T)));
      const size_t off = static_cast<size_t>(row) * P.V + t0;
      // group masses were stored for the residual of draft rows and the
      // fused masses of the bonus row; a draft row with zero residual
      // recomputes its fused masses
      const bool stored = (r_ok == (!bonus || P.full));
      sample = group_walk<T, true>(static_cast<const T*>(P.a) + off,
                                   static_cast<const T*>(P.b) + off,
                                   static_cast<const T*>(P.t) + off, nvec, t0, kSGroups, P.beta,
                                   S.ws.groups + (row * S.NT + owner) * kSGroups, stored, r_ok,
                                   st.lse[0] * kLog2e, st.lse[3] * kLog2e, tau_local);
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
  finish_row_warp<STOCH>(P, row, bi, k, r, st.dtok, st.da, st.db, st.dt, sc);
  if (lane == 0) {
    unsigned long long* tg = S.ws.tags + row * 4;
#pragma unroll
    for (int q = 0; q < 4; ++q) st_relaxed64(tg + q, 0ull);
    S.ws.ready[row] = 0u;
    S.ws.p2cnt[row] = 0u;
  }
}

// ---------------------------------------------------------------- items

template <typename T, bool STOCH, unsigned F, bool R2>
__device__ __noinline__ void item_pass1(const SParams& S, SharedStream* sh, unsigned char* buf,
                                        long long q, long long row, int tile, int par,
                                        int tail_warp) {
  const KParams& P = S.P;
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int K1 = P.K + 1;
  const int bi = static_cast<int>(row / K1), k = static_cast<int>(row % K1);
  const int t0 = tile * S.TS;
  const int nvec = (min(P.V, t0 + S.TS) - t0) / VE;
  const size_t off = static_cast<size_t>(row) * P.V + t0;
  const T* ra = static_cast<const T*>(P.a) + off;
  const T* rb = static_cast<const T*>(P.b) + off;
  const T* rt = static_cast<const T*>(P.t) + off;
  const unsigned long long pol = policy_evict_last();
  X1 e = x1_neutral();
  const bool ovf = ring_pass1<T, F>(S, sh, buf, q, nvec, (nvec + kSThreads - 1) / kSThreads, t0,
                                    P.beta, e);
  warp_reduce_x1<F>(e);
  if (lane == 0) sh->w1[par][warp] = e;
  if (__syncthreads_or(ovf)) {
    // an entry far above its thread's reference (or non-finite data)
    redo_pass1<T, F>(ra, rb, rt, nvec, t0, P.beta, pol, &sh->w1[par][warp]);
    __syncthreads();
  }
  if (warp != tail_warp) return;
  X1 w = (lane < kSWarps) ? sh->w1[par][lane] : x1_neutral();
  warp_reduce_x1<F>(w);
  if (sh->broken) w.bad |= kBadTimeout;
  unsigned ticket = 0;
  if (lane == 0) {
    X1* dst = S.ws.p1rec + row * S.NT + tile;
    *dst = w;
    ticket = atom_add_acq_rel(S.ws.p1cnt + row, 1u);
  }
  ticket = __shfl_sync(0xffffffffu, ticket, 0);
  if (ticket + 1 != static_cast<unsigned>(S.NT)) return;
  __syncwarp();
  row_after_pass1<T, STOCH, F, R2>(S, row, bi, k);
}

template <typename T, bool STOCH, unsigned G, bool LP>
__device__ __noinline__ void item_pass2(const SParams& S, SharedStream* sh, unsigned char* buf,
                                        long long q, long long row, int tile, int par,
                                        int tail_warp) {
  const KParams& P = S.P;
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int K1 = P.K + 1;
  const int bi = static_cast<int>(row / K1), k = static_cast<int>(row % K1);
  const int t0 = tile * S.TS;
  const int nvec = (min(P.V, t0 + S.TS) - t0) / VE;
  // the row's normalisers, published by its pass 1 as tagged words
  float v[4] = {0.f, 0.f, 0.f, 0.f};
  bool late = false;
  if (lane < 4) {
    const unsigned long long* tg = S.ws.tags + row * 4 + lane;
    unsigned long long wd = ld_relaxed64(tg);
    if ((wd >> 32) == 0ull) {
      const unsigned long long w0 = global_ns();
      while (((wd = ld_relaxed64(tg)) >> 32) == 0ull) {
        if (global_ns() - w0 > kWaitNs) {
          late = true;
          break;
        }
        __nanosleep(256);
      }
    }
    v[0] = __uint_as_float(static_cast<unsigned>(wd));
  }
  const float A2 = __shfl_sync(0xffffffffu, v[0], 0);
  const float B2 = __shfl_sync(0xffffffffu, v[0], 1);
  const float S2 = __shfl_sync(0xffffffffu, v[0], 2);
  const float lse_s = __shfl_sync(0xffffffffu, v[0], 3);
  late = __any_sync(0xffffffffu, late);
  X2 x = x2_zero();
  float* lp = LP ? P.logprobs + static_cast<size_t>(row) * P.V + t0 : nullptr;
  float* groups = S.ws.groups + (row * S.NT + tile) * kSGroups;
  ring_pass2<T, G, LP>(S, sh, buf, q, nvec, (nvec + kSThreads - 1) / kSThreads, P.beta, A2, B2,
                       S2, lse_s, x, lp, groups);
  if (late) x.j = x.msum = x.kl = x.R = x.Q = NAN;  // pass 1 never published: a data error
  warp_reduce_x2<G>(x);
  if (lane == 0) sh->w2[par][warp] = x;
  __syncthreads();
  if (warp != tail_warp) return;
  X2 w = (lane < kSWarps) ? sh->w2[par][lane] : x2_zero();
  warp_reduce_x2<G>(w);
  w.pad[0] = __uint_as_float(sh->broken ? kBadTimeout : 0u);  // this tile's copies timed out
  unsigned ticket = 0;
  if (lane == 0) {
    S.ws.p2rec[row * S.NT + tile] = w;
    ticket = atom_add_acq_rel(S.ws.p2cnt + row, 1u);
  }
  ticket = __shfl_sync(0xffffffffu, ticket, 0);
  if (ticket + 1 != static_cast<unsigned>(S.NT)) return;
  __syncwarp();
  row_after_pass2<T, STOCH, G>(S, row, bi, k);
}

template <typename T, bool STOCH>
__device__ __forceinline__ void run_item(const SParams& S, SharedStream* sh, unsigned char* buf,
                                         long long q, int prog, bool p2, long long row, int tile,
                                         int par, int tw) {
  constexpr unsigned FG = F_LA | F_LB | F_LT | F_AS;
  constexpr unsigned FF = F_LA | F_LB | F_LT | F_LS | F_AS | F_AT;
  constexpr unsigned RQ = STOCH ? G_RES : 0u;
#define P1(F, R2) item_pass1<T, STOCH, F, R2>(S, sh, buf, q, row, tile, par, tw)
#define P2(G, LP) item_pass2<T, STOCH, G, LP>(S, sh, buf, q, row, tile, par, tw)
  if (!STOCH) {
    switch (prog) {
      case PG_GREEDY_DRAFT_JSD: if (p2) P2(G_JSD, false); else P1(FG, true); return;
      case PG_GREEDY_DRAFT_KL: if (p2) P2(G_KL, false); else P1(FG, true); return;
      case PG_GREEDY_DRAFT_NONE: if (!p2) P1(FG, false); return;
      case PG_GREEDY_BONUS_T: if (!p2) P1(F_AT, false); return;
      case PG_GREEDY_BONUS_S: if (!p2) P1(F_AS, false); return;
      default: break;
    }
  } else {
    switch (prog) {
      case PG_STOCH_DRAFT_JSD: if (p2) P2(G_JSD | G_RES, false); else P1(F_LA | F_LB | F_LS, true); return;
      case PG_STOCH_DRAFT_KL: if (p2) P2(G_KL | G_RES, false); else P1(F_LA | F_LB | F_LS, true); return;
      case PG_STOCH_DRAFT_NONE: if (p2) P2(G_RES, false); else P1(F_LA | F_LB | F_LS, true); return;
      case PG_STOCH_DRAFT_JSD_TOK: if (p2) P2(G_JSD | G_RES, false); else P1(F_LA | F_LB | F_LS | F_AS, true); return;
      case PG_STOCH_DRAFT_KL_TOK: if (p2) P2(G_KL | G_RES, false); else P1(F_LA | F_LB | F_LS | F_AS, true); return;
      case PG_STOCH_DRAFT_NONE_TOK: if (p2) P2(G_RES, false); else P1(F_LA | F_LB | F_LS | F_AS, true); return;
      case PG_STOCH_BONUS: if (p2) P2(G_QF, false); else P1(F_LS, true); return;
      case PG_STOCH_BONUS_TOK: if (p2) P2(G_QF, false); else P1(F_LS | F_AS, true); return;
      default: break;
    }
  }
  switch (prog) {
    case PG_FULL_JSD: if (p2) P2(G_JSD | RQ, false); else P1(FF, true); return;
    case PG_FULL_KL: if (p2) P2(G_KL | RQ, false); else P1(FF, true); return;
    case PG_FULL_NONE: if (p2) P2(RQ, false); else P1(FF, true); return;
    case PG_FULL_JSD_LP: if (p2) P2(G_JSD | RQ, true); else P1(FF, true); return;
    case PG_FULL_KL_LP: if (p2) P2(G_KL | RQ, true); else P1(FF, true); return;
    case PG_FULL_NONE_LP: if (p2) P2(RQ, true); else P1(FF, true); return;
    default: return;
  }
#undef P1
#undef P2
}

template <typename T, bool STOCH>
__global__ void __launch_bounds__(kSThreads, 2) fuse_verify_stream(const SParams S) {
  __shared__ SharedStream sh;
  extern __shared__ __align__(128) unsigned char ring_buf[];
  const int tid = threadIdx.x;
  if (tid == 0) {
#pragma unroll
    for (int s = 0; s < kSStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], kSWarps);
    }
    sh.broken = 0u;
    fence_mbar_init();
    sh.prod.pi = blockIdx.x;
    sh.prod.issued = 0;
    ring_seek<T>(S, sh.prod);
    ring_top_up<T>(S, &sh, ring_buf, 0);
  }
  __syncthreads();
  long long q = 0;  // chunks this CTA has consumed
  int n = 0;        // items this CTA has taken
  for (long long i = blockIdx.x; i < S.NI; i += gridDim.x) {
    ItemInfo it;
    if (!item_info<T>(S, i, it)) continue;
    run_item<T, STOCH>(S, &sh, ring_buf, q, it.prog, it.p2, it.row, it.tile, n & 1, n % kSWarps);
    q += it.nch;
    ++n;
  }
  // a copy that timed out may still land: wait for the last stages (bounded)
  if (tid == 0 && sh.broken) {
    for (long long c = q > kSStages ? q - kSStages : 0; c < q; ++c)
      mbar_wait_bounded(&sh.full[c % kSStages], static_cast<unsigned>((c / kSStages) & 1), kWaitNs);
  }
}

}  // namespace asymspec_impl
