// AsymSpec per-step fuse-and-verify on GB300 (sm_103a): host side of the C ABI
// declared in include/asymspec.h, and the launch of its kernels.
//
//   fuse_verify_tma      (kernel_tma.cuh) one cluster per row, each CTA's
//                        slice brought in by chunked 1-D bulk copies, per-row
//                        programs; the default for 16-byte aligned rows.  Its
//                        rows are decided, and Algorithm 1's scan run, by
//                        decide_rows, a second launch.
//   fuse_verify_row      (kernel_row.cuh) the same decomposition with no
//                        slice in shared memory (pass 1 from HBM, pass 2 from
//                        the L2, four CTAs per SM) and the lean per-entry
//                        arithmetic: the production program of the
//                        stochastic JSD step (no debug outputs, delta = a - b).
//   fuse_verify_generic  (kernel_generic.cuh) one cluster per row, any
//                        element-aligned input; folds the scan into the same
//                        launch through a per-element ticket in the workspace.
//
// Each reads every logit row from HBM once.
#include <algorithm>
#include <mutex>

#include "device_common.cuh"
#include "kernel_generic.cuh"
#include "kernel_tma.cuh"
#include "kernel_row.cuh"
#include "kernel_draft.cuh"
#include "kernel_xvocab.cuh"
#include "kernels.h"

namespace {

using namespace asymspec_impl;

thread_local int g_last_cuda_error = 0;

int cuda_fail(cudaError_t e) {
  g_last_cuda_error = static_cast<int>(e);
  return ASYMSPEC_ERR_CUDA;
}

constexpr int kTmaPreferredSmem = 113 * 1024;  // two CTAs per SM

struct Plan {
  int kernel;  // ASYMSPEC_KERNEL_*
  int C, W, VE, sh_off, smem;
  int group_stride;  // TMA kernels: floats per row and CTA of group masses
  long long rows;
  long long ctas;  // grid size
  bool vector_path;
  bool row;          // the production row kernel (fuse_verify_row) runs
  int nt;            // threads per CTA (kRowThreads or kTThreads)
  int grid_y;        // the row kernel's grid is (C (K+1), B): grid_y = B (1 otherwise)
};

// Shared memory one SM offers its CTAs, and what each CTA costs beyond its
// own allocation.
constexpr int kSmemPerSm = 228 * 1024;
constexpr int kSmemPerCta = 1024;

const void* row_kernel(int dtype) {
  return dtype == ASYMSPEC_FP32 ? row_kernel_f32() : row_kernel_bf16();
}


int elt_size(int dtype) { return dtype == ASYMSPEC_FP32 ? 4 : 2; }

long long round_up_ll(long long x, long long a) { return (x + a - 1) / a * a; }

// Cluster sizes tried, in order of preference (8 packs GB300's GPCs best).
constexpr int kClusterOrder[] = {1, 2, 4, 8, 10, 12, 16};

// Generic kernel: first C whose slice fits the preferred size, else C=16.
bool plan_generic(int V, int elt, int VE, int forced_C, Plan* pl) {
  const int shared_bytes = static_cast<int>(sizeof(SharedGeneric));
  auto fill = [&](int C) {
    const long long per = (static_cast<long long>(V) + C - 1) / C;
    const long long W = round_up_ll(per, VE);
    const long long sh_off = round_up_ll(3 * W * elt, 16);
    pl->C = C;
    pl->W = static_cast<int>(W);
    pl->sh_off = static_cast<int>(sh_off);
    pl->smem = static_cast<int>(sh_off + shared_bytes);
    return sh_off + shared_bytes <= kMaxSmem;
  };
  if (forced_C > 0) return fill(forced_C);
  for (int C : kClusterOrder)
    if (fill(C) && pl->sh_off <= kPreferredSliceBytes) return true;
  return fill(16);
}

// TMA kernel: first C whose slice (and shared state) fits two CTAs per SM,
// else the first that fits one; a slice holds at most kMaxRounds vectors
// per thread.
bool plan_tma(int V, int elt, int forced_C, Plan* pl) {
  const int VE = 16 / elt;
  auto fill = [&](int C) {
    const long long per = (static_cast<long long>(V) + C - 1) / C;
    const long long W = round_up_ll(per, VE);
    const int shared_bytes = shared_tma_bytes(C);
    const long long sh_off = round_up_ll(3 * W * elt, 128);
    pl->C = C;
    pl->W = static_cast<int>(W);
    pl->sh_off = static_cast<int>(sh_off);
    pl->smem = static_cast<int>(sh_off + shared_bytes);
    pl->group_stride = kGroupsMax;
    return sh_off + shared_bytes <= kMaxSmem &&
           W / VE <= static_cast<long long>(kMaxRounds) * kTThreads;
  };
  if (forced_C > 0) return fill(forced_C);
  for (int C : kClusterOrder)
    if (fill(C) && pl->smem <= kTmaPreferredSmem) return true;
  for (int C : kClusterOrder)
    if (fill(C)) return true;
  return false;
}

// The production row kernel.  Pass 2 re-reads each row from the L2, so the
// rows in flight (one per resident cluster) must stay well inside it, while
// fewer CTAs per row give each warp a longer block over which the fixed
// costs of a CTA (its launch, the first loads, the exchange of the pass-1
// records) are spread.  With at least one wave of clusters of 8 (rows x 8 >=
// 4 CTAs x SMs): the smallest C of kRowClusters whose resident clusters
// hold at most kRowL2Budget of rows.  Measured on GB300 (kernel time, rows
// in flight):
//   B=64, K=7, V=128256 bf16:  C=5 103.4 us (90 MB), C=6 97.3 us (75 MB), C=8 102.4 us (57 MB)
//   B=32, K=8, V=151936 bf16:  C=6 70.7 us (88 MB), C=7 71.7 us (74 MB), C=8 75.8 us (67 MB)
//   B=128, K=4, V=151936 fp32: C=12 207.9 us (84 MB), C=16 247.8 us (60 MB)
// Smaller batches take C = 8.  A warp's block takes at most kWalkRounds
// steps (the decision kernel's walk loads a whole block at once).  Only the
// pass-1 records live in shared memory.  forced_C: the caller's
// asymspec_launch_opts.
constexpr int kRowClusters[] = {4, 5, 6, 7, 8, 10, 12, 16};
constexpr double kRowL2Budget = 86.0e6;

struct DeviceShape {
  int device, sms;
  bool ok;
};
DeviceShape device_shape() {
  DeviceShape d{0, 152, false};  // GB300 when no device answers
  int n = 0;
  if (cudaGetDevice(&d.device) == cudaSuccess &&
      cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, d.device) == cudaSuccess && n > 0) {
    d.sms = n;
    d.ok = true;
  }
  cudaGetLastError();
  return d;
}

const void* row_kernel(int dtype);
cudaError_t prepare_kernel(const void* fn, int device);
cudaError_t active_clusters(const void* fn, const Plan& pl, int device, int* out);

bool plan_row(int V, int dtype, int forced_C, long long rows, Plan* pl) {
  const int elt = elt_size(dtype);
  const int VE = 16 / elt;
  auto width = [&](int C) {
    const long long per = (static_cast<long long>(V) + C - 1) / C;
    return round_up_ll(per, VE);
  };
  auto fits = [&](int C) {
    return width(C) / VE <= static_cast<long long>(kWalkRounds) * kRowThreads;
  };
  int C = 0;
  if (forced_C) {
    if (fits(forced_C)) C = forced_C;
  } else {
    const DeviceShape dev = device_shape();
    const long long slots = static_cast<long long>(dev.sms) * kRowMinBlocks;
    const double row_bytes = 3.0 * V * elt;
    if (rows * 8 < slots) {
      if (fits(8)) C = 8;
    } else {
      const void* fn = row_kernel(dtype);
      const bool query = dev.ok && prepare_kernel(fn, dev.device) == cudaSuccess;
      for (int c : kRowClusters) {
        if (!fits(c)) continue;
        // the clusters the device holds at once (an estimate without a device)
        long long resident = slots / c;
        Plan q = *pl;
        q.C = c;
        q.smem = row_shared_bytes(c) + kRingBytes;
        q.nt = kRowThreads;
        q.kernel = ASYMSPEC_KERNEL_TMA;
        q.grid_y = 1;
        int n = 0;
        if (query && active_clusters(fn, q, dev.device, &n) == cudaSuccess && n > 0) resident = n;
        cudaGetLastError();
        if (static_cast<double>(std::min(rows, resident)) * row_bytes <= kRowL2Budget) {
          C = c;
          break;
        }
      }
    }
    if (!C) {  // nothing within the budget (or no full wave): the largest cluster that fits
      for (int c : kRowClusters)
        if (fits(c)) C = c;
    }
  }
  if (!C) return false;
  pl->C = C;
  pl->W = static_cast<int>(width(C));
  pl->sh_off = row_shared_bytes(C);  // the warps' rings follow the fixed state
  pl->smem = row_shared_bytes(C) + kRingBytes;
  pl->group_stride = kGroupsMax;
  pl->nt = kRowThreads;
  return true;
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

size_t ws_records_bytes(int B, int K) {
  return round_up(static_cast<size_t>(B) * (K + 1) * sizeof(int4), 256);
}

size_t cluster_ws_bytes(int B, int K) {
  return ws_records_bytes(B, K) + round_up(static_cast<size_t>(B) * sizeof(unsigned), 256);
}

// Workspace of the cluster TMA kernel for clusters of C CTAs: the records
// and tickets first (same offsets), then what each row leaves for the
// decision kernel: the row's pass-1 results, one pass-2 record per CTA and
// each CTA's inverse-CDF group masses.
struct TmaLayout {
  size_t stat, p2rec, groups, total;
};

// group_stride: floats of group masses per row and CTA.
TmaLayout tma_layout(int B, int K, int C, int group_stride = kGroupsMax) {
  TmaLayout L;
  const size_t R = static_cast<size_t>(B) * (K + 1);
  size_t off = cluster_ws_bytes(B, K);
  L.stat = off;
  off += round_up(R * sizeof(RowStat), 256);
  L.p2rec = off;
  // one record per CTA (fuse_verify_tma) or per warp (fuse_verify_row)
  off += round_up(R * C * kRowMaxWarps * sizeof(X2), 256);
  L.groups = off;
  off += round_up(R * C * static_cast<size_t>(group_stride) * sizeof(float), 256);
  L.total = off;
  return L;
}

// prod_row: the call is the production stochastic JSD step (no debug
// outputs, no per-row tokens, delta = a - b), which fuse_verify_row runs.
int make_plan(int B, int K, int V, int dtype, const asymspec_launch_opts* opts, bool vec_ok,
              size_t ws_bytes, bool prod_row, Plan* pl) {
  const int elt = elt_size(dtype);
  const int forced_C = (opts && opts->cluster_size > 0) ? opts->cluster_size : 0;
  const int forced_kernel = opts ? opts->kernel : 0;
  if (forced_C < 0 || forced_C > 16) return ASYMSPEC_ERR_INVALID_ARG;
  if (forced_kernel != 0 && forced_kernel != ASYMSPEC_KERNEL_GENERIC &&
      forced_kernel != ASYMSPEC_KERNEL_TMA)
    return ASYMSPEC_ERR_INVALID_ARG;
  pl->rows = static_cast<long long>(B) * (K + 1);
  pl->vector_path = vec_ok;
  pl->row = false;
  pl->nt = kTThreads;
  pl->grid_y = 1;
  if (ws_bytes < cluster_ws_bytes(B, K)) return ASYMSPEC_ERR_WORKSPACE;
  bool ok = false;
  // (its grid is (C (K+1), B): B up to 65535)
  if (forced_kernel != ASYMSPEC_KERNEL_GENERIC && vec_ok && prod_row && B <= 65535 &&
      plan_row(V, dtype, forced_C, static_cast<long long>(B) * (K + 1), pl)) {
    if (ws_bytes >= tma_layout(B, K, pl->C).total) {
      pl->kernel = ASYMSPEC_KERNEL_TMA;
      pl->VE = 16 / elt;
      pl->row = true;
      pl->grid_y = B;
      ok = true;
    } else if (forced_kernel == ASYMSPEC_KERNEL_TMA) {
      return ASYMSPEC_ERR_WORKSPACE;
    }
  }
  if (ok) {
    // the production row kernel
  } else if (forced_kernel != ASYMSPEC_KERNEL_GENERIC && vec_ok && plan_tma(V, elt, forced_C, pl)) {
    // the TMA kernel leaves each row's results in the workspace; the generic
    // kernel, which needs only the records and tickets, runs when it is short
    if (ws_bytes >= tma_layout(B, K, pl->C).total) {
      pl->kernel = ASYMSPEC_KERNEL_TMA;
      pl->VE = 16 / elt;
      ok = true;
    } else if (forced_kernel == ASYMSPEC_KERNEL_TMA) {
      return ASYMSPEC_ERR_WORKSPACE;
    }
  } else if (forced_kernel == ASYMSPEC_KERNEL_TMA) {
    return vec_ok ? ASYMSPEC_ERR_TOO_LARGE : ASYMSPEC_ERR_UNSUPPORTED;
  }
  if (!ok) {
    pl->kernel = ASYMSPEC_KERNEL_GENERIC;
    pl->VE = vec_ok ? 16 / elt : 1;
    if (!plan_generic(V, elt, pl->VE, forced_C, pl)) return ASYMSPEC_ERR_TOO_LARGE;
  }
  pl->ctas = pl->rows * pl->C;
  if (pl->ctas > INT_MAX) return ASYMSPEC_ERR_TOO_LARGE;
  return ASYMSPEC_OK;
}

using KernelFn = const void*;  // a __global__ function taking KParams (or SParams)

// sel: the TMA kernel's program set (tma_program_set; 0 = run-time dispatch)
KernelFn pick_kernel(const Plan& pl, int dtype, bool stoch, int sel = 0) {
  if (pl.row) return row_kernel(dtype);
  if (pl.kernel == ASYMSPEC_KERNEL_TMA)
    return dtype == ASYMSPEC_FP32 ? tma_kernel_f32(stoch, sel) : tma_kernel_bf16(stoch, sel);
  return generic_kernel(dtype, pl.vector_path, stoch);
}

KernelFn pick_decide(int dtype, bool stoch) {
  return dtype == ASYMSPEC_FP32 ? decide_kernel_f32(stoch) : decide_kernel_bf16(stoch);
}

// Per (kernel, device): attributes set once; cluster occupancy cached per
// (cluster size, shared memory size).
std::mutex g_mu;
struct AttrEntry {
  const void* fn;
  int device;
};
AttrEntry g_attr_done[64];
int g_attr_count = 0;
struct OccEntry {
  const void* fn;
  int device, C, smem, clusters;
};
OccEntry g_occ[128];
int g_occ_count = 0;

cudaError_t prepare_kernel(KernelFn fn, int device) {
  std::lock_guard<std::mutex> lock(g_mu);
  const void* f = fn;
  for (int i = 0; i < g_attr_count; ++i)
    if (g_attr_done[i].fn == f && g_attr_done[i].device == device) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  if (g_attr_count < 64) g_attr_done[g_attr_count++] = {f, device};
  return cudaSuccess;
}

// A kernel without clusters whose dynamic shared memory may reach max_bytes
// (the decision kernel's walk staging: what its static records leave of the
// per-CTA limit; the gather's restricted row of t).
cudaError_t prepare_plain_kernel(KernelFn fn, int device, int max_bytes) {
  std::lock_guard<std::mutex> lock(g_mu);
  const void* f = fn;
  for (int i = 0; i < g_attr_count; ++i)
    if (g_attr_done[i].fn == f && g_attr_done[i].device == device) return cudaSuccess;
  const cudaError_t e =
      cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, max_bytes);
  if (e != cudaSuccess) return e;
  if (g_attr_count < 64) g_attr_done[g_attr_count++] = {f, device};
  return cudaSuccess;
}

cudaLaunchConfig_t launch_config(const Plan& pl, long long ctas, cudaStream_t stream,
                                 cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = pl.grid_y > 1 ? dim3(static_cast<unsigned>(ctas / pl.grid_y),
                                     static_cast<unsigned>(pl.grid_y))
                              : dim3(static_cast<unsigned>(ctas));
  cfg.blockDim = dim3(pl.kernel == ASYMSPEC_KERNEL_GENERIC ? kThreads : pl.nt);
  cfg.dynamicSmemBytes = pl.smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

// Clusters of this shape the device holds at once (0 if it cannot).
cudaError_t active_clusters(KernelFn fn, const Plan& pl, int device, int* out) {
  const void* f = fn;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    for (int i = 0; i < g_occ_count; ++i)
      if (g_occ[i].fn == f && g_occ[i].device == device && g_occ[i].C == pl.C &&
          g_occ[i].smem == pl.smem) {
        *out = g_occ[i].clusters;
        return cudaSuccess;
      }
  }
  cudaLaunchAttribute attr[1];
  Plan one = pl;  // a grid of one cluster
  one.grid_y = 1;
  cudaLaunchConfig_t cfg = launch_config(one, pl.C, nullptr, attr);
  int n = 0;
  const cudaError_t e = cudaOccupancyMaxActiveClusters(&n, fn, &cfg);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_occ_count < 128) g_occ[g_occ_count++] = {f, device, pl.C, pl.smem, n};
  *out = n;
  return cudaSuccess;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_params(const asymspec_gate_params* gp) {
  if (!(gp->gamma > 0.f && gp->gamma <= 1.f)) return ASYMSPEC_ERR_INVALID_ARG;
  if (!(std::isfinite(gp->beta) && gp->beta >= 0.f)) return ASYMSPEC_ERR_INVALID_ARG;
  if (gp->mode != ASYMSPEC_MODE_GREEDY && gp->mode != ASYMSPEC_MODE_STOCHASTIC)
    return ASYMSPEC_ERR_UNSUPPORTED;
  if (gp->divergence < ASYMSPEC_DIV_JSD || gp->divergence > ASYMSPEC_DIV_LAMBDA)
    return ASYMSPEC_ERR_UNSUPPORTED;
  if (gp->divergence == ASYMSPEC_DIV_LAMBDA && !std::isfinite(gp->lambda))
    return ASYMSPEC_ERR_INVALID_ARG;
  // flags: bits 0-1 the delta source, every other bit reserved
  if ((gp->flags & ~ASYMSPEC_FLAG_DELTA_MASK) != 0) return ASYMSPEC_ERR_INVALID_ARG;
  const int ds = gp->flags & ASYMSPEC_FLAG_DELTA_MASK;
  if (ds != ASYMSPEC_DELTA_AB && ds != ASYMSPEC_DELTA_A && ds != ASYMSPEC_DELTA_TB)
    return ASYMSPEC_ERR_INVALID_ARG;
  return ASYMSPEC_OK;
}

int check_opts(const asymspec_launch_opts* opts) {
  // every kernel runs 256-thread CTAs
  if (opts && opts->block_threads != 0 && opts->block_threads != 256)
    return ASYMSPEC_ERR_INVALID_ARG;
  if (opts && (opts->test_flags & ~ASYMSPEC_TEST_COPY_GIVE_UP) != 0) return ASYMSPEC_ERR_INVALID_ARG;
  if (opts && ((opts->timing_begin == nullptr) != (opts->timing_end == nullptr)))
    return ASYMSPEC_ERR_INVALID_ARG;
  return ASYMSPEC_OK;
}

// The caller's timing events around the fused row kernel (asymspec_launch_opts).
cudaError_t record_timing(const asymspec_launch_opts* opts, bool begin, cudaStream_t s) {
  if (!opts || !opts->timing_begin) return cudaSuccess;
  return cudaEventRecord(static_cast<cudaEvent_t>(begin ? opts->timing_begin : opts->timing_end), s);
}

// Scratch of asymspec_fuse_verify_static, used as asymspec_fuse_verify_ex
// uses any workspace.  The generic kernel needs records for
// ASYMSPEC_STATIC_MAX_ROWS rows and tickets for the largest batch that can
// have that many rows (K >= 1, so B <= ASYMSPEC_STATIC_MAX_ROWS / 2): 144 KiB.
// 4 MiB also holds the cluster kernels' per-row results (48 + 576 C bytes a
// row for clusters of C: about 890 rows at C = 8, 1190 at C = 6); larger
// batches take the generic kernel.
constexpr size_t kStaticScratchBytes = ASYMSPEC_STATIC_SCRATCH_BYTES;
static_assert(kStaticScratchBytes >= static_cast<size_t>(ASYMSPEC_STATIC_MAX_ROWS) * sizeof(int4) +
                                         static_cast<size_t>(ASYMSPEC_STATIC_MAX_ROWS / 2) *
                                             sizeof(unsigned),
              "the static scratch holds the generic kernel's records and tickets");
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Device address of g_static_scratch in the current device's context, looked
// up on every call: a cached address would outlive a context that
// cudaDeviceReset tore down (the module, and the array, are loaded again in
// the next context).  Once the module is loaded the lookup is a host-side
// table read; the first lookup in a context may load the module.
constexpr int kMaxDevices = 64;

int static_scratch(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
  if (e != cudaSuccess) return cuda_fail(e);
  *out = p;
  return ASYMSPEC_OK;
}

// asymspec_fuse_verify_host: the scratch layout (each part 256-byte aligned)
// and the chunking of the batch.
struct HostLayout {
  int P, Bc;  // chunks, batch elements per chunk (the last may have fewer)
  size_t a, b, t, tok, prob, unif, len, next, ws, ws_each, total;
};

HostLayout host_layout(int B, int K, int V, int dtype) {
  HostLayout L;
  L.Bc = (B + ASYMSPEC_HOST_CHUNKS - 1) / ASYMSPEC_HOST_CHUNKS;
  L.P = (B + L.Bc - 1) / L.Bc;
  const size_t R = static_cast<size_t>(B) * (K + 1);
  const size_t row = static_cast<size_t>(V) * elt_size(dtype);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += round_up(bytes, 256);
    return o;
  };
  L.a = take(R * row);
  L.b = take(R * row);
  L.t = take(R * row);
  L.tok = take(static_cast<size_t>(B) * K * sizeof(int32_t));
  L.prob = take(static_cast<size_t>(B) * K * sizeof(float));
  L.unif = take(R * sizeof(float));
  L.len = take(static_cast<size_t>(B) * sizeof(int32_t));
  L.next = take(static_cast<size_t>(B) * sizeof(int32_t));
  L.ws_each = round_up(asymspec_workspace_bytes(L.Bc, K, V), 256);
  L.ws = take(L.ws_each * L.P);
  L.total = off;
  return L;
}

// Per device: the copy stream and its per-chunk events (created on first use).
struct HostRes {
  cudaStream_t copy;
  cudaEvent_t start;
  cudaEvent_t chunk[ASYMSPEC_HOST_CHUNKS];
  bool ready;
};
std::mutex g_host_mu;
HostRes g_host[kMaxDevices] = {};

int host_resources(HostRes** out) {
  int device = 0;
  cudaError_t e = cudaGetDevice(&device);
  if (e != cudaSuccess) return cuda_fail(e);
  if (device < 0 || device >= kMaxDevices) return ASYMSPEC_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_host_mu);
  HostRes& r = g_host[device];
  if (!r.ready) {
    e = cudaStreamCreateWithFlags(&r.copy, cudaStreamNonBlocking);
    if (e != cudaSuccess) return cuda_fail(e);
    e = cudaEventCreateWithFlags(&r.start, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(e);
    for (int c = 0; c < ASYMSPEC_HOST_CHUNKS; ++c) {
      e = cudaEventCreateWithFlags(&r.chunk[c], cudaEventDisableTiming);
      if (e != cudaSuccess) return cuda_fail(e);
    }
    r.ready = true;
  }
  *out = &r;
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
  // the TMA kernel's layout for the largest cluster
  return tma_layout(B, K, 16).total;
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
  int st = check_opts(opts);
  if (st) return st;
  asymspec_gate_params gp;
  asymspec_default_gate_params(&gp);
  if (gate_params) gp = *gate_params;
  st = check_params(&gp);
  if (st) return st;
  const bool vec_ok = (static_cast<long long>(V) * elt_size(dtype)) % 16 == 0;
  Plan pl = {};
  const bool stoch_p = gp.mode == ASYMSPEC_MODE_STOCHASTIC;
  st = make_plan(B, K, V, dtype, opts, vec_ok, asymspec_workspace_bytes(B, K, V),
                 stoch_p && gp.divergence == ASYMSPEC_DIV_JSD &&
                     (gp.flags & ASYMSPEC_FLAG_DELTA_MASK) == ASYMSPEC_DELTA_AB,
                 &pl);
  if (st) return st;
  out->cluster_size = pl.C;
  out->block_threads = pl.kernel == ASYMSPEC_KERNEL_GENERIC ? kThreads : pl.nt;
  out->slice_elems = pl.W;
  out->smem_bytes = pl.smem;
  out->ctas = pl.ctas;
  out->vector_path = vec_ok ? 1 : 0;
  out->max_active_clusters = 0;
  out->kernel = pl.kernel;
  out->launches = pl.kernel == ASYMSPEC_KERNEL_TMA ? 2 : 1;
  out->row_kernel = pl.row ? 1 : 0;
  int device = 0;
  if (cudaGetDevice(&device) == cudaSuccess) {
    const bool st_mode = gp.mode == ASYMSPEC_MODE_STOCHASTIC;
    KernelFn fn = pick_kernel(pl, dtype, st_mode,
                              tma_program_set(st_mode, gp.divergence, gp.fuse_bonus != 0, false,
                                              false, gp.flags & ASYMSPEC_FLAG_DELTA_MASK));
    int ncl = 0;
    if (fn && prepare_kernel(fn, device) == cudaSuccess &&
        active_clusters(fn, pl, device, &ncl) == cudaSuccess)
      out->max_active_clusters = ncl;
  }
  cudaGetLastError();
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
  int st = check_opts(opts);
  if (st) return st;
  asymspec_gate_params gp;
  asymspec_default_gate_params(&gp);
  if (gate_params) gp = *gate_params;
  st = check_params(&gp);
  if (st) return st;
  const bool stoch = gp.mode == ASYMSPEC_MODE_STOCHASTIC;
  if (!logits_full || !logits_comp || !logits_ver || !draft_tokens || !out_accept_len ||
      !out_next_token)
    return ASYMSPEC_ERR_INVALID_ARG;
  if (stoch && (!draft_probs || !uniforms)) return ASYMSPEC_ERR_INVALID_ARG;
  const int elt = elt_size(dtype);
  if (!aligned(logits_full, elt) || !aligned(logits_comp, elt) || !aligned(logits_ver, elt) ||
      !aligned(draft_tokens, 4) || !aligned(out_accept_len, 4) || !aligned(out_next_token, 4) ||
      (draft_probs && !aligned(draft_probs, 4)) || (uniforms && !aligned(uniforms, 4)) ||
      (out_row_stats && !aligned(out_row_stats, 4)) ||
      (out_row_tokens && !aligned(out_row_tokens, 4)) ||
      (out_fused_logprobs && !aligned(out_fused_logprobs, 4)) ||
      (out_error_word && !aligned(out_error_word, 4)))
    return ASYMSPEC_ERR_MISALIGNED;
  if (!workspace || !aligned(workspace, 16)) return ASYMSPEC_ERR_WORKSPACE;
  const bool vec_ok = (static_cast<long long>(V) * elt) % 16 == 0 && aligned(logits_full, 16) &&
                      aligned(logits_comp, 16) && aligned(logits_ver, 16);
  Plan pl = {};
  const bool prod_row = stoch && gp.divergence == ASYMSPEC_DIV_JSD && !out_row_stats &&
                        !out_fused_logprobs && !out_row_tokens &&
                        (gp.flags & ASYMSPEC_FLAG_DELTA_MASK) == ASYMSPEC_DELTA_AB;
  st = make_plan(B, K, V, dtype, opts, vec_ok, workspace_bytes, prod_row, &pl);
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
  P.delta_src = gp.flags & ASYMSPEC_FLAG_DELTA_MASK;
  P.fuse_bonus = gp.fuse_bonus ? 1 : 0;
  P.need_lse_s = (stoch || out_fused_logprobs || out_row_stats) ? 1 : 0;
  P.need_pass2 = (stoch || out_fused_logprobs || gp.divergence == ASYMSPEC_DIV_JSD ||
                  gp.divergence == ASYMSPEC_DIV_KL)
                     ? 1
                     : 0;
  P.full = (out_row_stats || out_fused_logprobs) ? 1 : 0;
  P.want_tokens = out_row_tokens ? 1 : 0;
  P.rows = pl.rows;
  P.out_len = out_accept_len;
  P.out_next = out_next_token;
  P.row_stats = out_row_stats;
  P.row_tokens = out_row_tokens;
  P.logprobs = out_fused_logprobs;
  P.err_word = out_error_word;
  P.recs = static_cast<int4*>(workspace);
  P.row_stat = nullptr;
  P.pass2_rec = nullptr;
  P.group_mass = nullptr;
  P.tma_threads = pl.nt;
  P.row_blocks = pl.row ? 1 : 0;
  // the chunk waits of the TMA kernel: bounded, or (test hook) giving up at once
  P.walk_stage = 0;
  P.copy_wait_ns =
      (opts && (opts->test_flags & ASYMSPEC_TEST_COPY_GIVE_UP)) ? 0ull : kCopyTimeoutNs;
  P.tickets = reinterpret_cast<unsigned int*>(static_cast<char*>(workspace) +
                                              ws_records_bytes(B, K));

  int device = 0;
  cudaError_t e = cudaGetDevice(&device);
  if (e != cudaSuccess) return cuda_fail(e);
  KernelFn fn = pick_kernel(pl, dtype, stoch,
                            tma_program_set(stoch, gp.divergence, gp.fuse_bonus != 0, P.full != 0,
                                            P.want_tokens != 0, P.delta_src));
  if (!fn) return ASYMSPEC_ERR_UNSUPPORTED;
  e = prepare_kernel(fn, device);
  if (e != cudaSuccess) return cuda_fail(e);
  const long long ctas = pl.ctas;  // one cluster of C CTAs per row
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = launch_config(pl, ctas, static_cast<cudaStream_t>(stream), attr);
  void* args[] = {&P};
  P.group_stride = pl.group_stride;
  if (pl.kernel == ASYMSPEC_KERNEL_TMA) {
    const TmaLayout L = tma_layout(B, K, pl.C, pl.group_stride);
    char* base = static_cast<char*>(workspace);
    P.row_stat = base + L.stat;
    P.pass2_rec = reinterpret_cast<float*>(base + L.p2rec);
    P.group_mass = reinterpret_cast<float*>(base + L.groups);
  }
  e = record_timing(opts, true, cfg.stream);
  if (e == cudaSuccess) e = cudaLaunchKernelExC(&cfg, fn, args);
  if (e == cudaSuccess) e = record_timing(opts, false, cfg.stream);
  if (e != cudaSuccess) return cuda_fail(e);
  if (pl.kernel == ASYMSPEC_KERNEL_TMA) {
    // the rows' decisions and Algorithm 1's scan: one CTA per batch element
    // as a programmatic dependent launch: its launch overlaps the row
    // kernel's last CTAs, and it waits (griddepcontrol.wait) for that kernel
    int warps = std::min(K + 1, kDecideThreads / 32);
    // rows of the production row kernel: each warp stages the vectors of the
    // inverse-CDF group it walks (at most one warp block: 3 streams x 32
    // vectors per step) in shared memory
    P.walk_stage = 0;
    if (pl.row) {
      const int nv = pl.W / pl.VE;
      const int steps = (row_block_vectors(nv, pl.nt / 32) + 31) / 32;
      P.walk_stage = 3 * steps * 32 * 16;
      warps = std::min(warps, (kMaxSmem - kDecideSmemRows * 16) / P.walk_stage);
    }
    const KernelFn dfn = pick_decide(dtype, stoch);
    e = prepare_plain_kernel(dfn, device, kMaxSmem - kDecideSmemRows * 16);
    if (e != cudaSuccess) return cuda_fail(e);
    cudaLaunchConfig_t dcfg = {};
    cudaLaunchAttribute dattr[1];
    dattr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    dattr[0].val.programmaticStreamSerializationAllowed = 1;
    dcfg.gridDim = dim3(static_cast<unsigned>(B));
    dcfg.blockDim = dim3(32 * warps);
    dcfg.dynamicSmemBytes = static_cast<size_t>(warps) * P.walk_stage;
    dcfg.stream = static_cast<cudaStream_t>(stream);
    dcfg.attrs = dattr;
    dcfg.numAttrs = 1;
    e = cudaLaunchKernelExC(&dcfg, dfn, args);
    if (e != cudaSuccess) return cuda_fail(e);
  }
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

int asymspec_fuse_verify_static(const void* logits_full, const void* logits_comp,
                                const void* logits_ver, const int32_t* draft_tokens,
                                const float* draft_probs, const float* uniforms, int B, int K,
                                int V, int dtype, const asymspec_gate_params* gate_params,
                                int32_t* out_accept_len, int32_t* out_next_token,
                                void* stream) {
  if (B < 1 || K < 1 || V < 2) return ASYMSPEC_ERR_INVALID_ARG;
  if (static_cast<long long>(B) * (K + 1) > ASYMSPEC_STATIC_MAX_ROWS)
    return ASYMSPEC_ERR_SCRATCH_LIMIT;
  void* scratch = nullptr;
  int st = static_scratch(&scratch);
  if (st) return st;
  // the tickets must start at zero; a call that did not complete may have
  // left some set, so they are cleared on the caller's stream every time
  cudaError_t e = cudaMemsetAsync(static_cast<char*>(scratch) + ws_records_bytes(B, K), 0,
                                  static_cast<size_t>(B) * sizeof(unsigned),
                                  static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e);
  return asymspec_fuse_verify_ex(logits_full, logits_comp, logits_ver, draft_tokens,
                                 draft_probs, uniforms, B, K, V, dtype, gate_params,
                                 out_accept_len, out_next_token, scratch, kStaticScratchBytes,
                                 nullptr, nullptr, nullptr, nullptr, nullptr, stream);
}

size_t asymspec_host_scratch_bytes(int B, int K, int V, int dtype) {
  if (B < 1 || K < 1 || V < 2) return 0;
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return 0;
  return host_layout(B, K, V, dtype).total;
}

int asymspec_fuse_verify_host(const void* h_logits_full, const void* h_logits_comp,
                              const void* h_logits_ver, const int32_t* h_draft_tokens,
                              const float* h_draft_probs, const float* h_uniforms, int B, int K,
                              int V, int dtype, const asymspec_gate_params* gate_params,
                              int32_t* h_out_accept_len, int32_t* h_out_next_token,
                              void* d_scratch, size_t scratch_bytes, void* stream) {
  if (B < 1 || K < 1 || V < 2) return ASYMSPEC_ERR_INVALID_ARG;
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return ASYMSPEC_ERR_UNSUPPORTED;
  asymspec_gate_params gp;
  asymspec_default_gate_params(&gp);
  if (gate_params) gp = *gate_params;
  int st = check_params(&gp);
  if (st) return st;
  const bool stoch = gp.mode == ASYMSPEC_MODE_STOCHASTIC;
  if (!h_logits_full || !h_logits_comp || !h_logits_ver || !h_draft_tokens ||
      !h_out_accept_len || !h_out_next_token)
    return ASYMSPEC_ERR_INVALID_ARG;
  if (stoch && (!h_draft_probs || !h_uniforms)) return ASYMSPEC_ERR_INVALID_ARG;
  const HostLayout L = host_layout(B, K, V, dtype);
  if (!d_scratch || !aligned(d_scratch, 256) || scratch_bytes < L.total)
    return ASYMSPEC_ERR_WORKSPACE;
  HostRes* r = nullptr;
  st = host_resources(&r);
  if (st) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(d_scratch);
  const size_t row = static_cast<size_t>(V) * elt_size(dtype);
  const int K1 = K + 1;
  // the copies start after everything already on `stream` (which may still
  // read this scratch), then run back to back on the copy stream
  cudaError_t e = cudaEventRecord(r->start, s);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(r->copy, r->start, 0);
  if (e != cudaSuccess) return cuda_fail(e);
  auto h2d = [&](size_t dst, const void* src, size_t off, size_t bytes) {
    return cudaMemcpyAsync(base + dst + off, static_cast<const char*>(src) + off, bytes,
                           cudaMemcpyHostToDevice, r->copy);
  };
  for (int c = 0; c < L.P && e == cudaSuccess; ++c) {
    const int b0 = c * L.Bc, nb = std::min(L.Bc, B - b0);
    const size_t r0 = static_cast<size_t>(b0) * K1, nr = static_cast<size_t>(nb) * K1;
    e = h2d(L.a, h_logits_full, r0 * row, nr * row);
    if (e == cudaSuccess) e = h2d(L.b, h_logits_comp, r0 * row, nr * row);
    if (e == cudaSuccess) e = h2d(L.t, h_logits_ver, r0 * row, nr * row);
    if (e == cudaSuccess)
      e = h2d(L.tok, h_draft_tokens, static_cast<size_t>(b0) * K * 4, static_cast<size_t>(nb) * K * 4);
    if (stoch && e == cudaSuccess)
      e = h2d(L.prob, h_draft_probs, static_cast<size_t>(b0) * K * 4, static_cast<size_t>(nb) * K * 4);
    if (stoch && e == cudaSuccess) e = h2d(L.unif, h_uniforms, r0 * 4, nr * 4);
    if (e == cudaSuccess) e = cudaEventRecord(r->chunk[c], r->copy);
  }
  if (e != cudaSuccess) {
    cudaStreamSynchronize(r->copy);
    return cuda_fail(e);
  }
  // each chunk's step on `stream` once its copies have landed
  for (int c = 0; c < L.P; ++c) {
    const int b0 = c * L.Bc, nb = std::min(L.Bc, B - b0);
    const size_t r0 = static_cast<size_t>(b0) * K1;
    char* ws = base + L.ws + static_cast<size_t>(c) * L.ws_each;
    e = cudaStreamWaitEvent(s, r->chunk[c], 0);
    if (e == cudaSuccess)
      e = cudaMemsetAsync(ws + ws_records_bytes(nb, K), 0, static_cast<size_t>(nb) * sizeof(unsigned), s);
    if (e != cudaSuccess) {
      cudaStreamSynchronize(r->copy);
      return cuda_fail(e);
    }
    int32_t* d_len = reinterpret_cast<int32_t*>(base + L.len) + b0;
    int32_t* d_next = reinterpret_cast<int32_t*>(base + L.next) + b0;
    st = asymspec_fuse_verify_ex(
        base + L.a + r0 * row, base + L.b + r0 * row, base + L.t + r0 * row,
        reinterpret_cast<const int32_t*>(base + L.tok) + static_cast<size_t>(b0) * K,
        stoch ? reinterpret_cast<const float*>(base + L.prob) + static_cast<size_t>(b0) * K : nullptr,
        stoch ? reinterpret_cast<const float*>(base + L.unif) + r0 : nullptr, nb, K, V, dtype, &gp,
        d_len, d_next, ws, L.ws_each, nullptr, nullptr, nullptr, nullptr, nullptr, stream);
    if (st != ASYMSPEC_OK) {
      cudaStreamSynchronize(r->copy);
      return st;
    }
    e = cudaMemcpyAsync(h_out_accept_len + b0, d_len, static_cast<size_t>(nb) * 4,
                        cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(h_out_next_token + b0, d_next, static_cast<size_t>(nb) * 4,
                          cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) {
      cudaStreamSynchronize(r->copy);
      return cuda_fail(e);
    }
  }
  return ASYMSPEC_OK;
}

int asymspec_draft_sample(const void* logits, int rows, int V, int dtype, int mode,
                          const float* uniforms, int32_t* out_tokens, float* out_probs,
                          int cluster_size, void* stream) {
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return ASYMSPEC_ERR_UNSUPPORTED;
  if (mode != ASYMSPEC_MODE_GREEDY && mode != ASYMSPEC_MODE_STOCHASTIC)
    return ASYMSPEC_ERR_UNSUPPORTED;
  if (rows < 0 || V < 2) return ASYMSPEC_ERR_INVALID_ARG;
  if (cluster_size != 0 && cluster_size != 1 && cluster_size != 2 && cluster_size != 4 &&
      cluster_size != kDMaxCluster)
    return ASYMSPEC_ERR_INVALID_ARG;
  if (V > ASYMSPEC_DRAFT_MAX_V || rows > (1 << 27)) return ASYMSPEC_ERR_TOO_LARGE;
  if (rows == 0) return ASYMSPEC_OK;
  const bool stoch = mode == ASYMSPEC_MODE_STOCHASTIC;
  if (!logits || !out_tokens || !out_probs || (stoch && !uniforms)) return ASYMSPEC_ERR_INVALID_ARG;
  const int elt = elt_size(dtype);
  if (!aligned(logits, elt) || !aligned(out_tokens, 4) || !aligned(out_probs, 4) ||
      (stoch && !aligned(uniforms, 4)))
    return ASYMSPEC_ERR_MISALIGNED;
  const bool vec = (static_cast<long long>(V) * elt) % 16 == 0 && aligned(logits, 16);
  const int VE = vec ? 16 / elt : 1;
  const int nv = V / VE;
  int C = cluster_size;
  if (C == 0) {
    int device = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return cuda_fail(e);
    C = 1;
    while (C < kDMaxCluster && static_cast<long long>(rows) * C < 4LL * sms &&
           (nv + 2 * C - 1) / (2 * C) >= 512)
      C *= 2;
  }
  DParams P;
  P.logits = logits;
  P.unif = stoch ? uniforms : nullptr;
  P.tokens = out_tokens;
  P.probs = out_probs;
  P.rows = rows;
  P.V = V;
  P.nv = nv;
  P.W = (nv + C - 1) / C;
  // sampling: one float of group mass per warp and round of a slice
  const size_t smem =
      stoch ? static_cast<size_t>((P.W + kDThreads - 1) / kDThreads) * kDWarps * sizeof(float) : 0;
  const void* fn = draft_kernel_ptr(dtype, vec, stoch);
  cudaError_t e = cudaSuccess;
  if (smem > 48 * 1024)
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return cuda_fail(e);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(static_cast<long long>(rows) * C));
  cfg.blockDim = dim3(kDThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = static_cast<cudaStream_t>(stream);
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {&P};
  e = cudaLaunchKernelExC(&cfg, fn, args);
  return e == cudaSuccess ? ASYMSPEC_OK : cuda_fail(e);
}

}  // extern "C"

// ------------------------------------------------- cross-family vocabularies

namespace {

// Scratch of asymspec_xvocab_gather, each part 256-byte aligned: inv_d[V_d],
// inv_v[V_v] (int32) and the map-error word.
struct XScratch {
  size_t inv_d, inv_v, err, total;
};

XScratch xvocab_scratch_layout(int V_d, int V_v) {
  XScratch L;
  L.inv_d = 0;
  L.inv_v = round_up(static_cast<size_t>(V_d) * sizeof(int32_t), 256);
  L.err = L.inv_v + round_up(static_cast<size_t>(V_v) * sizeof(int32_t), 256);
  L.total = L.err + 256;
  return L;
}

// Workspace of asymspec_fuse_verify_xvocab, each part 256-byte aligned: the
// restricted rows a', b', t' ([B, K+1, S] each), the emitted pair indices
// ([B] int32), the gather's scratch, then the step's own workspace for a
// vocabulary of S entries.
struct XLayout {
  size_t ga, gb, gt, idx, scratch, scratch_bytes, step, step_bytes, total;
};

XLayout xvocab_layout(int B, int K, int S, int V_d, int V_v, int dtype) {
  XLayout L;
  const size_t plane = round_up(static_cast<size_t>(B) * (K + 1) * S * elt_size(dtype), 256);
  L.ga = 0;
  L.gb = plane;
  L.gt = 2 * plane;
  L.idx = 3 * plane;
  L.scratch = L.idx + round_up(static_cast<size_t>(B) * sizeof(int32_t), 256);
  L.scratch_bytes = xvocab_scratch_layout(V_d, V_v).total;
  L.step = L.scratch + L.scratch_bytes;
  L.step_bytes = asymspec_workspace_bytes(B, K, S);
  L.total = L.step + L.step_bytes;
  return L;
}

}  // namespace

extern "C" {

size_t asymspec_xvocab_gather_scratch_bytes(int V_d, int V_v) {
  if (V_d < 1 || V_v < 1) return 0;
  return xvocab_scratch_layout(V_d, V_v).total;
}

size_t asymspec_xvocab_workspace_bytes(int B, int K, int S, int V_d, int V_v, int dtype) {
  if (B < 1 || K < 1 || S < 2 || V_d < 1 || V_v < 1) return 0;
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return 0;
  return xvocab_layout(B, K, S, V_d, V_v, dtype).total;
}

int asymspec_xvocab_gather(const void* logits_full, const void* logits_comp, int V_d,
                           const void* logits_ver, int V_v, const int32_t* map_d,
                           const int32_t* map_v, int S, int rows, int dtype, void* out_full,
                           void* out_comp, void* out_ver, uint32_t* out_error_word,
                           void* scratch, size_t scratch_bytes, void* stream) {
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return ASYMSPEC_ERR_UNSUPPORTED;
  if (rows < 0 || S < 2 || V_d < 1 || V_v < 1) return ASYMSPEC_ERR_INVALID_ARG;
  if (rows == 0) return ASYMSPEC_OK;
  if (!logits_full || !logits_comp || !logits_ver || !map_d || !map_v || !out_full ||
      !out_comp || !out_ver)
    return ASYMSPEC_ERR_INVALID_ARG;
  const int elt = elt_size(dtype);
  if (!aligned(logits_full, elt) || !aligned(logits_comp, elt) || !aligned(logits_ver, elt) ||
      !aligned(out_full, elt) || !aligned(out_comp, elt) || !aligned(out_ver, elt) ||
      !aligned(map_d, 4) || !aligned(map_v, 4) || (out_error_word && !aligned(out_error_word, 4)))
    return ASYMSPEC_ERR_MISALIGNED;
  const XScratch XL = xvocab_scratch_layout(V_d, V_v);
  if (scratch && (!aligned(scratch, 256) || scratch_bytes < XL.total)) return ASYMSPEC_ERR_WORKSPACE;
  const long long ycount = (static_cast<long long>(rows) + kXRows - 1) / kXRows;
  if (ycount > 65535) return ASYMSPEC_ERR_TOO_LARGE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSuccess;
  if (scratch) {
    // the map check: inverse maps built with atomicCAS, the map-error word
    char* base = static_cast<char*>(scratch);
    int* inv_d = reinterpret_cast<int*>(base + XL.inv_d);
    int* inv_v = reinterpret_cast<int*>(base + XL.inv_v);
    unsigned* merr = reinterpret_cast<unsigned*>(base + XL.err);
    int Vd = V_d, Vv = V_v, S_ = S;
    void* fargs[] = {&inv_d, &Vd, &inv_v, &Vv, &merr};
    const int vmax = std::max(V_d, V_v);
    e = cudaLaunchKernel(xvocab_inv_fill_ptr(), dim3((vmax + 255) / 256), dim3(256), fargs, 0, st);
    if (e != cudaSuccess) return cuda_fail(e);
    const int32_t* md = map_d;
    const int32_t* mv = map_v;
    uint32_t* ew = out_error_word;
    void* bargs[] = {&md, &mv, &S_, &inv_d, &Vd, &inv_v, &Vv, &merr, &ew};
    e = cudaLaunchKernel(xvocab_inv_build_ptr(), dim3((S + 255) / 256), dim3(256), bargs, 0, st);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  XGatherParams P;
  P.inv_v = scratch ? reinterpret_cast<const int*>(static_cast<char*>(scratch) + XL.inv_v) : nullptr;
  P.map_err =
      scratch ? reinterpret_cast<const unsigned*>(static_cast<char*>(scratch) + XL.err) : nullptr;
  P.a = logits_full;
  P.b = logits_comp;
  P.t = logits_ver;
  P.map_d = map_d;
  P.map_v = map_v;
  P.ga = out_full;
  P.gb = out_comp;
  P.gt = out_ver;
  P.err_word = out_error_word;
  P.rows = rows;
  P.V_d = V_d;
  P.V_v = V_v;
  P.S = S;
  const dim3 grid(static_cast<unsigned>((S + kXThreads * kXJ - 1) / (kXThreads * kXJ)),
                  static_cast<unsigned>(ycount));
  void* args[] = {&P};
  // t built in shared memory through the inverse map (its map may be in any
  // order) when the caller gave the scratch (where the map check builds the
  // inverse map), every row of t starts on a 16-byte boundary and a
  // restricted row fits in one CTA's shared memory; a and b (and otherwise
  // t) through global memory
  // (one CTA per row; a restricted row larger than a CTA's shared memory is
  // cut into parts, each CTA reading the whole row of t for its part)
  int parts = 1;
  while (parts < 16 && ((static_cast<size_t>(S) + parts - 1) / parts + 8) * elt >
                           static_cast<size_t>(kMaxSmem))
    ++parts;
  const size_t row_out = ((static_cast<size_t>(S) + parts - 1) / parts + 8) * elt;
  const bool inv_t = scratch && row_out <= static_cast<size_t>(kMaxSmem) &&
                     aligned(logits_ver, 16) && (static_cast<size_t>(V_v) * elt) % 16 == 0;
  e = cudaLaunchKernel(xvocab_gather_ptr(dtype, !inv_t), grid, dim3(kXThreads), args, 0, st);
  if (e != cudaSuccess) return cuda_fail(e);
  if (inv_t) {
    const KernelFn fn = xvocab_gather_inv_ptr(dtype);
    int device = 0;
    e = cudaGetDevice(&device);
    if (e == cudaSuccess) e = prepare_plain_kernel(fn, device, kMaxSmem);
    if (e == cudaSuccess) {
      // a programmatic dependent of the a/b gather, which it does not read:
      // the two gathers overlap (the map check before them is complete)
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[0].val.programmaticStreamSerializationAllowed = 1;
      cfg.gridDim = dim3(static_cast<unsigned>(rows), static_cast<unsigned>(parts));
      cfg.blockDim = dim3(kXInvThreads);
      cfg.dynamicSmemBytes = round_up(row_out, 16);
      cfg.stream = st;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      e = cudaLaunchKernelExC(&cfg, fn, args);
    }
  }
  return e == cudaSuccess ? ASYMSPEC_OK : cuda_fail(e);
}

int asymspec_fuse_verify_xvocab(const void* logits_full, const void* logits_comp, int V_d,
                                const void* logits_ver, int V_v, const int32_t* map_d,
                                const int32_t* map_v, int S, const int32_t* draft_index,
                                const float* draft_probs, const float* uniforms, int B, int K,
                                int dtype, const asymspec_gate_params* gate_params,
                                int32_t* out_accept_len, int32_t* out_next_token,
                                int32_t* out_next_index, void* workspace,
                                size_t workspace_bytes, uint32_t* out_error_word, void* stream) {
  if (B < 1 || K < 1 || S < 2 || V_d < 1 || V_v < 1) return ASYMSPEC_ERR_INVALID_ARG;
  if (dtype != ASYMSPEC_FP32 && dtype != ASYMSPEC_BF16) return ASYMSPEC_ERR_UNSUPPORTED;
  asymspec_gate_params gp;
  asymspec_default_gate_params(&gp);
  if (gate_params) gp = *gate_params;
  int st = check_params(&gp);
  if (st) return st;
  if (!draft_index || !out_accept_len || !out_next_token) return ASYMSPEC_ERR_INVALID_ARG;
  if (gp.mode == ASYMSPEC_MODE_STOCHASTIC && (!draft_probs || !uniforms))
    return ASYMSPEC_ERR_INVALID_ARG;
  if (!aligned(out_next_token, 4) || !aligned(out_accept_len, 4) ||
      (out_next_index && !aligned(out_next_index, 4)))
    return ASYMSPEC_ERR_MISALIGNED;
  const XLayout L = xvocab_layout(B, K, S, V_d, V_v, dtype);
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < L.total)
    return ASYMSPEC_ERR_WORKSPACE;
  char* base = static_cast<char*>(workspace);
  st = asymspec_xvocab_gather(logits_full, logits_comp, V_d, logits_ver, V_v, map_d, map_v, S,
                              B * (K + 1), dtype, base + L.ga, base + L.gb, base + L.gt,
                              out_error_word, base + L.scratch, L.scratch_bytes, stream);
  if (st) return st;
  int32_t* idx = out_next_index ? out_next_index : reinterpret_cast<int32_t*>(base + L.idx);
  st = asymspec_fuse_verify_ex(base + L.ga, base + L.gb, base + L.gt, draft_index, draft_probs,
                               uniforms, B, K, S, dtype, &gp, out_accept_len, idx,
                               base + L.step, L.step_bytes, nullptr, nullptr, nullptr,
                               out_error_word, nullptr, stream);
  if (st) return st;
  int32_t* next = out_next_token;
  int32_t* len = out_accept_len;
  const int32_t* mv = map_v;
  const unsigned* merr =
      reinterpret_cast<const unsigned*>(base + L.scratch + xvocab_scratch_layout(V_d, V_v).err);
  int S_ = S, B_ = B;
  void* args[] = {&idx, &mv, &S_, &B_, &merr, &len, &next};
  const cudaError_t e = cudaLaunchKernel(xvocab_emit_ptr(), dim3((B + 255) / 256), dim3(256),
                                         args, 0, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ASYMSPEC_OK : cuda_fail(e);
}

const char* asymspec_status_string(int status) {
  switch (status) {
    case ASYMSPEC_OK: return "ok";
    case ASYMSPEC_ERR_INVALID_ARG: return "invalid argument";
    case ASYMSPEC_ERR_UNSUPPORTED: return "unsupported dtype, mode, divergence or kernel";
    case ASYMSPEC_ERR_MISALIGNED: return "pointer not aligned to its element size";
    case ASYMSPEC_ERR_WORKSPACE: return "workspace missing or too small";
    case ASYMSPEC_ERR_CUDA: return "CUDA error (see asymspec_last_cuda_error)";
    case ASYMSPEC_ERR_TOO_LARGE: return "problem too large for the on-chip row slices";
    case ASYMSPEC_ERR_SCRATCH_LIMIT:
      return "B*(K+1) exceeds ASYMSPEC_STATIC_MAX_ROWS (8192), the static scratch of "
             "asymspec_fuse_verify_static; use asymspec_fuse_verify_ex with a workspace";
    default: return "unknown status";
  }
}

int asymspec_last_cuda_error(void) { return g_last_cuda_error; }

int asymspec_version(void) { return 200; }

}  // extern "C"
