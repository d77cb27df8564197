// Cross-family vocabularies (Section 4, "Cross-family portability", and the
// appendix of the same name): the drafter and the verifier tokenise
// differently and share S string-identical tokens, the pairs
// (map_d[j], map_v[j]).  The step is run on the rows restricted to the
// pairs: a'_j = a[map_d[j]], b'_j = b[map_d[j]] (drafter vocabulary, so
// delta = a' - b' is computed there and carried to pair j) and
// t'_j = t[map_v[j]] (verifier vocabulary); the emitted pair index j is
// committed as the verifier token map_v[j].
//
//   xvocab_inv_fill, xvocab_inv_build
//                  the map check: inverse maps inv_d[V_d], inv_v[V_v] (the
//                  pair of each token, -1 if unpaired) built with atomicCAS,
//                  and a map-error word that an entry outside its vocabulary
//                  or a token claimed by two pairs sets.
//   xvocab_gather  restricts every row of a and b (and, for rows that are
//                  not 16-byte aligned, t) to the pairs, in pair order, into
//                  dense [rows, S] arrays the fuse-and-verify kernels then
//                  read as rows of a vocabulary of S entries.
//   xvocab_gather_inv
//                  the same for t, each restricted row built in shared
//                  memory through the inverse map and written out whole.
//   xvocab_emit    turns the emitted pair index of each batch element into
//                  its verifier token (every element is a data error if the
//                  map-error word is set).
//
// HBM-bound, no contraction: per row the gather reads the 3 S paired
// entries through the maps and writes them densely.  A warp reading global
// memory through a random map asks for one sector per entry, which bounds
// such a gather by the L1's sector rate, not by HBM; so the verifier side,
// whose map is the random one in the paper's pairing, is built in shared
// memory instead, where scattered writes cost a few bank cycles a warp.
#pragma once

#include "device_common.cuh"

namespace asymspec_impl {

constexpr int kXThreads = 256;
constexpr int kXJ = 4;     // pair indices per thread
constexpr int kXRows = 8;  // rows per CTA

struct XGatherParams {
  const void* a;
  const void* b;
  const void* t;
  const int32_t* map_d;
  const int32_t* map_v;
  void* ga;
  void* gb;
  void* gt;
  uint32_t* err_word;
  long long rows;
  int V_d, V_v, S;
  const int* inv_v;      // xvocab_gather_inv: the pair of each verifier token, -1 if none
  const unsigned* map_err;  // xvocab_gather_inv: the map check's error word
};

constexpr int kXInvThreads = 512;

template <typename T>
__device__ __forceinline__ T x_nan();
template <>
__device__ __forceinline__ float x_nan<float>() {
  return __int_as_float(0x7fc00000);
}
template <>
__device__ __forceinline__ __nv_bfloat16 x_nan<__nv_bfloat16>() {
  return __ushort_as_bfloat16(static_cast<unsigned short>(0x7FC0));
}

// The drafter-side restriction (and, with WITH_T, the verifier's too)
// through global memory, kXJ pair indices per thread for kXRows rows: a
// warp's loads through the increasing map_d touch a few sectors; loads
// through a random map_v ask for one sector per entry.  Every map entry is
// checked against its vocabulary (ASYMSPEC_DATA_BAD_MAP).
template <typename T, bool WITH_T>
__global__ void __launch_bounds__(kXThreads) xvocab_gather(XGatherParams P) {
  // xvocab_gather_inv (launched as a programmatic dependent when t is built
  // in shared memory) reads nothing this kernel writes: let it start
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const T* __restrict__ a = static_cast<const T*>(P.a);
  const T* __restrict__ b = static_cast<const T*>(P.b);
  const T* __restrict__ t = static_cast<const T*>(P.t);
  T* __restrict__ ga = static_cast<T*>(P.ga);
  T* __restrict__ gb = static_cast<T*>(P.gb);
  T* __restrict__ gt = static_cast<T*>(P.gt);
  const int S = P.S;
  const int j0 = blockIdx.x * (kXThreads * kXJ) + static_cast<int>(threadIdx.x);
  int md[kXJ], mv[kXJ];
  bool in[kXJ], okd[kXJ], okv[kXJ];
  bool bad = false;
#pragma unroll
  for (int i = 0; i < kXJ; ++i) {
    const int j = j0 + i * kXThreads;
    in[i] = j < S;
    md[i] = in[i] ? __ldg(P.map_d + j) : 0;
    mv[i] = in[i] ? __ldg(P.map_v + j) : 0;
    okd[i] = static_cast<unsigned>(md[i]) < static_cast<unsigned>(P.V_d);
    okv[i] = static_cast<unsigned>(mv[i]) < static_cast<unsigned>(P.V_v);
    bad |= in[i] && !(okd[i] && okv[i]);
  }
  if (bad && P.err_word) atomicOr(P.err_word, ASYMSPEC_DATA_BAD_MAP);
  const long long r0 = static_cast<long long>(blockIdx.y) * kXRows;
  const long long r1 = r0 + kXRows < P.rows ? r0 + kXRows : P.rows;
  const T nan = x_nan<T>();
  for (long long r = r0; r < r1; ++r) {
    const T* ra = a + r * P.V_d;
    const T* rb = b + r * P.V_d;
    const T* rt = t + r * P.V_v;
    T va[kXJ], vb[kXJ], vt[kXJ];
#pragma unroll
    for (int i = 0; i < kXJ; ++i) {
      va[i] = okd[i] ? ra[md[i]] : nan;
      vb[i] = okd[i] ? rb[md[i]] : nan;
      if (WITH_T) vt[i] = okv[i] ? rt[mv[i]] : nan;
    }
    const long long o = r * S;
#pragma unroll
    for (int i = 0; i < kXJ; ++i) {
      if (in[i]) {
        const int j = j0 + i * kXThreads;
        ga[o + j] = va[i];
        gb[o + j] = vb[i];
        if (WITH_T) gt[o + j] = vt[i];
      }
    }
  }
}

// Entry e of a 16-byte vector of T (e a compile-time index after unrolling).
template <typename T>
__device__ __forceinline__ T x_elem(const uint4& v, int e);
template <>
__device__ __forceinline__ float x_elem<float>(const uint4& v, int e) {
  return __uint_as_float(e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w);
}
template <>
__device__ __forceinline__ __nv_bfloat16 x_elem<__nv_bfloat16>(const uint4& v, int e) {
  const int k = e >> 1;
  const unsigned w = k == 0 ? v.x : k == 1 ? v.y : k == 2 ? v.z : v.w;
  return __ushort_as_bfloat16(static_cast<unsigned short>((e & 1) ? (w >> 16) : (w & 0xFFFFu)));
}

// The verifier-side restriction t'_j = t[map_v[j]], one CTA per row (or per
// contiguous part of the pairs when a restricted row exceeds a CTA's shared
// memory), for a map_v in any order: the restricted row is built in shared
// memory by reading the verifier row and its inverse map inv_v (the pair of
// each token, -1 if unpaired; built by the map check) in index order,
// 16-byte loads, and placing each paired entry at its pair index; the row
// is then written out densely.  Every DRAM sector of t is read once and
// every sector of t' written whole.  When the map check found an error
// (which the inverse map cannot express), the row is read through map_v
// instead, an entry outside the vocabulary reading NaN.
template <typename T>
__global__ void __launch_bounds__(kXInvThreads, 1) xvocab_gather_inv(XGatherParams P) {
  extern __shared__ __align__(16) unsigned char xrow[];
  T* out = reinterpret_cast<T*>(xrow);
  constexpr int VE = 16 / static_cast<int>(sizeof(T));
  constexpr int U = 4;
  // CTA (r, h) builds pairs [j0, j0 + S) of row r: gridDim.y parts of
  // P.S / gridDim.y pairs (rounded up to whole 16-byte vectors)
  const long long r = blockIdx.x;
  const int part = ((P.S + gridDim.y - 1) / gridDim.y + VE - 1) / VE * VE;
  const int j0 = static_cast<int>(blockIdx.y) * part;
  const T* src = static_cast<const T*>(P.t) + r * P.V_v;
  T* dst = static_cast<T*>(P.gt) + r * P.S + j0;
  const int S = max(0, min(part, P.S - j0)), V = P.V_v;
  const int tid = static_cast<int>(threadIdx.x), nt = static_cast<int>(blockDim.x);
  const T nan = x_nan<T>();
  if (*P.map_err) {
    // the map check failed (a token out of range or in two pairs, which the
    // inverse map cannot express): read each pair's entry through map_v
    for (int i = tid; i < S; i += nt) {
      const int u = __ldg(P.map_v + j0 + i);
      dst[i] = static_cast<unsigned>(u) < static_cast<unsigned>(V) ? src[u] : nan;
    }
    return;
  }
  // a map that passed the check pairs every j with a distinct token in
  // range: every entry of the row is written below
  // (the host takes this kernel for 16-byte aligned rows of t only)
  const int nvec = V / VE;
  for (int i0 = tid; i0 < nvec; i0 += U * nt) {
    uint4 v[U];
    int4 jv[U][VE / 4];
#pragma unroll
    for (int q = 0; q < U; ++q) {
      const int i = i0 + q * nt;
      if (i < nvec) {
        v[q] = __ldg(reinterpret_cast<const uint4*>(src) + i);
#pragma unroll
        for (int h = 0; h < VE / 4; ++h)
          jv[q][h] = __ldg(reinterpret_cast<const int4*>(P.inv_v) + i * (VE / 4) + h);
      }
    }
#pragma unroll
    for (int q = 0; q < U; ++q) {
      const int i = i0 + q * nt;
      if (i < nvec) {
#pragma unroll
        for (int h = 0; h < VE / 4; ++h) {
          // (unsigned compares: unpaired tokens, -1, fall outside too)
          const int4 j4 = jv[q][h];
          if (static_cast<unsigned>(j4.x - j0) < static_cast<unsigned>(S)) out[j4.x - j0] = x_elem<T>(v[q], 4 * h);
          if (static_cast<unsigned>(j4.y - j0) < static_cast<unsigned>(S)) out[j4.y - j0] = x_elem<T>(v[q], 4 * h + 1);
          if (static_cast<unsigned>(j4.z - j0) < static_cast<unsigned>(S)) out[j4.z - j0] = x_elem<T>(v[q], 4 * h + 2);
          if (static_cast<unsigned>(j4.w - j0) < static_cast<unsigned>(S)) out[j4.w - j0] = x_elem<T>(v[q], 4 * h + 3);
        }
      }
    }
  }
  for (int u = nvec * VE + tid; u < V; u += nt) {
    const int j = P.inv_v[u];
    if (static_cast<unsigned>(j - j0) < static_cast<unsigned>(S)) out[j - j0] = src[u];
  }
  __syncthreads();
  const bool vec_out = (reinterpret_cast<uintptr_t>(dst) & 15u) == 0;
  const int nout = vec_out ? S / VE : 0;
  for (int i = tid; i < nout; i += nt) reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(out)[i];
  for (int i = nout * VE + tid; i < S; i += nt) dst[i] = out[i];
}

// inv[v] = -1 for every token of both vocabularies; the map-error word is
// cleared.  (I = int; a template so that the header can be included twice.)
template <typename I>
__global__ void __launch_bounds__(256) xvocab_inv_fill(I* __restrict__ inv_d, int V_d,
                                                       I* __restrict__ inv_v, int V_v,
                                                       unsigned* __restrict__ map_err) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < V_d) inv_d[i] = -1;
  if (i < V_v) inv_v[i] = -1;
  if (i == 0) *map_err = 0u;
}

// inv_d[map_d[j]] = j and inv_v[map_v[j]] = j; an entry outside its
// vocabulary, or a token that a second pair claims, sets the error word.
template <typename I>
__global__ void __launch_bounds__(256) xvocab_inv_build(const I* __restrict__ map_d,
                                                        const I* __restrict__ map_v, int S,
                                                        I* __restrict__ inv_d, int V_d,
                                                        I* __restrict__ inv_v, int V_v,
                                                        unsigned* __restrict__ map_err,
                                                        uint32_t* __restrict__ err_word) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= S) return;
  const I md = map_d[j], mv = map_v[j];
  bool bad = false;
  if (static_cast<unsigned>(md) < static_cast<unsigned>(V_d))
    bad |= atomicCAS(inv_d + md, I(-1), I(j)) != I(-1);
  else
    bad = true;
  if (static_cast<unsigned>(mv) < static_cast<unsigned>(V_v))
    bad |= atomicCAS(inv_v + mv, I(-1), I(j)) != I(-1);
  else
    bad = true;
  if (bad) {
    atomicOr(map_err, 1u);
    if (err_word) atomicOr(err_word, ASYMSPEC_DATA_BAD_MAP);
  }
}

// out_next[b] = map_v[next_index[b]] (-1 stays -1: a data error); with the
// map-error word set, every element is a data error (its pair index too).
template <typename I>
__global__ void __launch_bounds__(256) xvocab_emit(I* __restrict__ next_index,
                                                   const I* __restrict__ map_v, int S, int B,
                                                   const unsigned* __restrict__ map_err,
                                                   I* __restrict__ out_len,
                                                   I* __restrict__ out_next) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B) return;
  const I j = next_index[i];
  if (*map_err) {
    out_len[i] = -1;
    out_next[i] = -1;
    next_index[i] = -1;
    return;
  }
  out_next[i] = (j >= 0 && j < S) ? map_v[j] : -1;
}

}  // namespace asymspec_impl
