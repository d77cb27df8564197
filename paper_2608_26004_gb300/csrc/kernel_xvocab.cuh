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
//   xvocab_gather  restricts every row of a, b and t to the pairs, in pair
//                  order, into dense [rows, S] arrays the fuse-and-verify
//                  kernels then read as rows of a vocabulary of S entries.
//   xvocab_emit    turns the emitted pair index of each batch element into
//                  its verifier token (every element is a data error if the
//                  map-error word is set).
//
// HBM-bound, no contraction: per row the gather reads the 3 S paired
// entries through the maps and writes them densely.  A warp reading through
// a random map asks L2 for a sector per entry (a sequential read of the
// source row scattered through the inverse map into a shared-memory copy of
// the restricted row was measured no faster: the int32 inverse map doubles
// the bytes each source row brings from L2).
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
};

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

template <typename T>
__global__ void __launch_bounds__(kXThreads) xvocab_gather(XGatherParams P) {
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
      vt[i] = okv[i] ? rt[mv[i]] : nan;
    }
    const long long o = r * S;
#pragma unroll
    for (int i = 0; i < kXJ; ++i) {
      if (in[i]) {
        const int j = j0 + i * kXThreads;
        ga[o + j] = va[i];
        gb[o + j] = vb[i];
        gt[o + j] = vt[i];
      }
    }
  }
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
