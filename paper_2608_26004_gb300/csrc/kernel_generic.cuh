// Generic fuse-and-verify kernel: one cluster of C CTAs per row triple, one
// row per launch of the cluster.  Any element-aligned input works (scalar
// copies when a row is not 16-byte aligned); the streaming kernel handles
// the aligned case faster.
//
// Each CTA stages its slice of the three rows in shared memory (the single
// HBM read), then: pass 1 (online max and sum of exponentials of a, b, t and
// s = t + beta (a - b), argmaxes of s and t), a DSMEM combine of the C
// partial results, pass 2 (JSD or KL of softmax a and softmax b, residual and
// fused masses), a second combine, the inverse-CDF walk in the CTA that owns
// the target, and the shared row epilogue.
#pragma once

#include "device_common.cuh"

namespace asymspec_impl {

struct SharedGeneric {
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


// The residual / fused mass of one element (stochastic mode).  Pass 2 and the
// inverse-CDF walk both call this, so they see identical values.
__device__ __forceinline__ float sample_mass(float xa, float xb, float xt, float beta, float A2,
                                             float S2, bool use_r, int ds) {
  const float xs = fuse1(beta, xa, xb, xt, ds);
  const float qf = ex2(fmaf(xs, kLog2e, -S2));
  if (!use_r) return qf;
  const float p = ex2(fmaf(xa, kLog2e, -A2));
  return fmaxf(qf - p, 0.f);
}

template <typename T, int VE, bool STOCH>
__global__ void __launch_bounds__(kThreads, 1) fuse_verify_generic(const KParams P) {
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
  SharedGeneric* sh = reinterpret_cast<SharedGeneric*>(smem_raw + P.sh_off);

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
  if (leader) fetch_draft<T>(P, row, bi, k, dtok, ad, bd, td);
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
    for (int e = 0; e < VE; ++e) xs[e] = fuse1(beta, xa[e], xb[e], xt[e], P.delta_src);
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
          const float xs = fuse1(beta, xa[e], xb[e], xt[e], P.delta_src);
          const float qf = ex2(fmaf(xs, kLog2e, -S2));
          r2.R += fmaxf(qf - p, 0.f);
          r2.Q += qf;
        }
        if (lp) lp[i * VE + e] = fuse1(beta, xa[e], xb[e], xt[e], P.delta_src) - lse_s;
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
        const float mm = sample_mass(xa[e], xb[e], xt[e], beta, A2, S2, use_r, P.delta_src);
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
          const float mm = sample_mass(xa[e], xb[e], xt[e], beta, A2, S2, use_r, P.delta_src);
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
  RowResult r;
  r.lse_a = lse_a;
  r.lse_b = lse_b;
  r.lse_t = sh->lse[2];
  r.lse_s = (STOCH || P.need_lse_s) ? lse_s : NAN;
  r.D = sh->D;
  r.is = sh->is;
  r.it = sh->it;
  r.sample = STOCH ? sh->sample : -1;
  r.mass = STOCH ? sh->mass_total : NAN;
  r.bad = 0;
  r.have_lse_t = true;
  finish_row<STOCH>(P, row, bi, k, r, dtok, ad, bd, td);
}

}  // namespace asymspec_impl
