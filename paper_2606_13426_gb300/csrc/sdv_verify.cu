// sdv_verify.cu - verification step of speculative diffusion sampling on sm_103a.
//
// One sdv_verify call with few chains launches (on the caller's stream) a counter
// reset and ONE fused kernel, k_verify:
//   * every CTA streams one tile (chain b, step j, chunk c) of x, m^q and m^p once
//     with 16-byte loads and reduces S1 = sum (x - m^p)(m^p - m^q) and
//     S2 = sum (m^p - m^q)^2 (App. "Density ratio calculations": Z^T Delta =
//     S1/sigma^2, |Delta|^2 = S2/sigma^2), then takes a ticket on its chain;
//   * the CTA holding a chain's last ticket finishes that chain: warp 0 forms
//     ell_j and |Delta_j|, draws the coins, applies sample or block acceptance
//     (Algorithms token-/block-verification) and draws U (Algorithm u-sample);
//     then the whole CTA writes y (Algorithm decomposition-res: y = m^q +
//     sigma (U e + G - e e^T G); or reflect-res, the bonus step, or the last
//     accepted draft).
// Chains finish at staggered times, so the latency-bound per-chain work overlaps
// the streaming of other chains.  Rows longer than kFusedMaxGroups groups of four
// elements are written by two extra kernels (k_resid_dot, k_resid_write) spread
// over many CTAs.  With many chains (B >= kFusedMaxChains), and in pipelined calls,
// the same tiles are streamed by k_tiles (each partial stored with the call's tag)
// and every chain is finished by a small CTA of k_finish.
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

#include "sdv_device.cuh"
#include "sdv_host.h"

namespace sdv {

// ---------------------------------------------------------------- small helpers
template <int NT>
__device__ __forceinline__ float2 block_sum2(float a, float b, float2* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a += __shfl_xor_sync(0xffffffffu, a, o);
    b += __shfl_xor_sync(0xffffffffu, b, o);
  }
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[w] = make_float2(a, b);
  __syncthreads();
  float2 r = make_float2(0.f, 0.f);
  if (w == 0) {
    r = (lane < NT / 32) ? red[lane] : make_float2(0.f, 0.f);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      r.x += __shfl_xor_sync(0xffffffffu, r.x, o);
      r.y += __shfl_xor_sync(0xffffffffu, r.y, o);
    }
  }
  return r;  // valid in thread 0
}

__device__ __forceinline__ void unpack(const uint4& v, float (&f)[4]) {
  f[0] = __uint_as_float(v.x);
  f[1] = __uint_as_float(v.y);
  f[2] = __uint_as_float(v.z);
  f[3] = __uint_as_float(v.w);
}
__device__ __forceinline__ void unpack(const uint4& v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

// Read-once streaming load: no L1 allocation.
__device__ __forceinline__ uint4 ldg_stream(const uint4* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

template <typename T, bool VEC4>
__device__ __forceinline__ void load4(const T* p, int64_t i, int64_t d, float (&f)[4]) {
  if (VEC4 && i + 4 <= d) {
    if (sizeof(T) == 4) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(p + i));
      f[0] = v.x; f[1] = v.y; f[2] = v.z; f[3] = v.w;
    } else {
      const uint2 v = __ldg(reinterpret_cast<const uint2*>(p + i));
      f[0] = __uint_as_float(v.x << 16); f[1] = __uint_as_float(v.x & 0xffff0000u);
      f[2] = __uint_as_float(v.y << 16); f[3] = __uint_as_float(v.y & 0xffff0000u);
    }
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k) f[k] = (i + k < d) ? Elem<T>::load(p + i + k) : 0.f;
  }
}

template <typename T, bool VEC4>
__device__ __forceinline__ void store4(T* p, int64_t i, int64_t d, const float (&f)[4]) {
  if (VEC4 && i + 4 <= d) {
    if (sizeof(T) == 4) {
      *reinterpret_cast<float4*>(p + i) = make_float4(f[0], f[1], f[2], f[3]);
    } else {
      __nv_bfloat162 lo = __floats2bfloat162_rn(f[0], f[1]);
      __nv_bfloat162 hi = __floats2bfloat162_rn(f[2], f[3]);
      uint2 v;
      memcpy(&v.x, &lo, 4);
      memcpy(&v.y, &hi, 4);
      *reinterpret_cast<uint2*>(p + i) = v;
    }
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (i + k < d) Elem<T>::store(p + i + k, f[k]);
  }
}

// ---------------------------------------------------------------- tile reduction
// (S1, S2) of elements [e0, e1) of the row starting at element `base`;
// VEC: whole 16-byte vectors, VPT of them per thread and tensor per sweep.
template <typename T, bool VEC, int VPT>
__device__ __forceinline__ float2 tile_sums(const T* __restrict__ x, const T* __restrict__ mq,
                                            const T* __restrict__ mp, int64_t base, int64_t e0,
                                            int64_t e1) {
  float s1 = 0.f, s2 = 0.f;
  if (VEC) {
    constexpr int V = 16 / (int)sizeof(T);
    const int64_t v0 = (base + e0) / V;
    const int nv = (int)((e1 - e0) / V);
    const uint4* X = reinterpret_cast<const uint4*>(x) + v0;
    const uint4* Q = reinterpret_cast<const uint4*>(mq) + v0;
    const uint4* P = reinterpret_cast<const uint4*>(mp) + v0;
#pragma unroll 1
    for (int v = threadIdx.x; v < nv; v += kK1Threads * VPT) {
      uint4 bx[VPT], bq[VPT], bp[VPT];
      if (v + (VPT - 1) * kK1Threads < nv) {
        // full sweep: issue all 3 * VPT 16-byte loads before any use
#pragma unroll
        for (int u = 0; u < VPT; ++u) bx[u] = ldg_stream(X + v + u * kK1Threads);
#pragma unroll
        for (int u = 0; u < VPT; ++u) bq[u] = ldg_stream(Q + v + u * kK1Threads);
#pragma unroll
        for (int u = 0; u < VPT; ++u) bp[u] = ldg_stream(P + v + u * kK1Threads);
      } else {
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
          const int vv = v + u * kK1Threads;
          const bool ok = vv < nv;
          bx[u] = ok ? ldg_stream(X + vv) : make_uint4(0u, 0u, 0u, 0u);
          bq[u] = ok ? ldg_stream(Q + vv) : make_uint4(0u, 0u, 0u, 0u);
          bp[u] = ok ? ldg_stream(P + vv) : make_uint4(0u, 0u, 0u, 0u);
        }
      }
#pragma unroll
      for (int u = 0; u < VPT; ++u) {
        float fx[V], fq[V], fp[V];
        unpack(bx[u], fx);
        unpack(bq[u], fq);
        unpack(bp[u], fp);
#pragma unroll
        for (int k = 0; k < V; ++k) {
          const float dl = fp[k] - fq[k];  // m^p - m^q
          const float a = fx[k] - fp[k];   // yhat - m^p
          s1 = fmaf(a, dl, s1);
          s2 = fmaf(dl, dl, s2);
        }
      }
    }
  } else {
    for (int64_t e = e0 + threadIdx.x; e < e1; e += kK1Threads) {
      const float fx = Elem<T>::load(x + base + e);
      const float fq = Elem<T>::load(mq + base + e);
      const float fp = Elem<T>::load(mp + base + e);
      const float dl = fp - fq, a = fx - fp;
      s1 = fmaf(a, dl, s1);
      s2 = fmaf(dl, dl, s2);
    }
  }
  return make_float2(s1, s2);
}

// The verification seed: by value, or from device memory (sampler rounds).
__device__ __forceinline__ uint64_t seed_of(const ScanArgs& A) { return A.seed_dev ? *A.seed_dev : A.seed; }

// ---------------------------------------------------------------- chain scan (one warp)
__device__ __forceinline__ ChainState inactive_state() {
  ChainState cs;
  cs.tau = 0; cs.row = -1; cs.U = NAN; cs.la_res = 0.f; cs.sigma = NAN; cs.dnorm = NAN;
  cs.inv_norm = 0.f; cs.refl = 0.f; cs.status = 0u; cs.kind = kKindInactive;
  cs.pad[0] = cs.pad[1] = 0;
  return cs;
}

struct ScanOut {
  ChainState cs;
  UParams P;   // residual parameters of row tau - 1 (block mode, cs.kind == kKindResid)
  bool have_P;
};

__device__ __forceinline__ UParams shfl_params(const UParams& P, int src) {
  const unsigned FULL = 0xffffffffu;
  UParams R;
  R.D = __shfl_sync(FULL, P.D, src);
  R.la = __shfl_sync(FULL, P.la, src);
  R.ap = __shfl_sync(FULL, P.ap, src);
  R.am = __shfl_sync(FULL, P.am, src);
  R.lv = __shfl_sync(FULL, P.lv, src);
  R.lvn = __shfl_sync(FULL, P.lvn, src);
  R.lnd_ap = __shfl_sync(FULL, P.lnd_ap, src);
  R.g_ap = __shfl_sync(FULL, P.g_ap, src);
  R.l1mx0 = __shfl_sync(FULL, P.l1mx0, src);
  return R;
}

// Per-lane values of one chain's window, held by one warp: step j in lane j & 31 of
// segment j >> 5 (L <= 64).
struct ScanRegs {
  float ell[2], dn[2], S1[2], S2[2], sg[2];
  int g;         // window length gamma_k, clamped to [0, L]
  bool any_bad;  // a non-finite ratio, norm or sigma
  bool stale;    // a k_tiles partial without this call's tag (not yet visible)
};

// Loads chain b's ell_j and |Delta_j|: from the tile partials (S1, S2 of every tile of
// the row, read through L2) and sigma, or from given arrays.  k_tiles partials carry the
// call's tag in each 8-byte word (written whole); with check_tags, R.stale reports a
// word whose tag is not this call's.  Called by a full warp; reads only.
__device__ ScanRegs scan_load(const ScanArgs& A, int b, bool check_tags = true) {
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int L = A.L;
  ScanRegs R;
  // window length gamma_k, clamped to [0, L] (device data the host cannot check)
  R.g = A.L_eff ? max(0, min(A.L_eff[b], L)) : L;
  const int nseg = (L + 31) >> 5;
  bool bad = false, stale = false;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int j = lane + 32 * q;
    R.ell[q] = 0.f; R.dn[q] = 0.f; R.S1[q] = 0.f; R.S2[q] = 0.f; R.sg[q] = 1.f;
    if (q < nseg && j < R.g) {
      if (A.part || A.tpart) {
        // partials written by other CTAs: read through L2, summed over the row's tiles
        // in tile order
        float a1 = 0.f, a2 = 0.f;
        if (A.tpart) {
          const int64_t s0 = ((int64_t)b * L + j) * A.C;
          const ulonglong2* p = reinterpret_cast<const ulonglong2*>(A.tpart) + s0;
#pragma unroll 4
          for (int c = 0; c < A.C; ++c) {
            const ulonglong2 t = __ldcg(p + c);
            if (check_tags && ((uint32_t)(t.x >> 32) != A.tag || (uint32_t)(t.y >> 32) != A.tag)) stale = true;
            a1 += __uint_as_float((uint32_t)t.x);
            a2 += __uint_as_float((uint32_t)t.y);
          }
        } else {
          const float2* p = A.part + ((int64_t)b * L + j) * A.C;
#pragma unroll 4
          for (int c = 0; c < A.C; ++c) {
            const float2 t = __ldcg(p + c);
            a1 += t.x;
            a2 += t.y;
          }
        }
        const float s = A.sigma[(int64_t)b * A.sstride + j];
        R.S1[q] = a1; R.S2[q] = a2; R.sg[q] = s;
        const float rs = frcp_fast(s);
        R.ell[q] = -(a1 + 0.5f * a2) * (rs * rs);
        R.dn[q] = sqrtf(a2) * rs;
        if (!(s > 0.f) || !isfinite(s)) bad = true;
      } else {
        R.ell[q] = A.ell_in[(int64_t)b * L + j];
        R.dn[q] = A.dn_in[(int64_t)b * L + j];
      }
      if (!isfinite(R.ell[q]) || !isfinite(R.dn[q])) bad = true;
    }
  }
  R.any_bad = __any_sync(FULL, bad);
  R.stale = __any_sync(FULL, stale);
  return R;
}

// The per-step outputs (ell_j, |Delta_j|; zero outside the window) by the lanes of the warp
// that loaded R.
__device__ __forceinline__ void scan_write_steps(const ScanArgs& A, int b, const ScanRegs& R) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int j = lane + 32 * q;
    if (j < A.L) {
      if (A.ell_out) A.ell_out[(int64_t)b * A.L + j] = R.ell[q];
      if (A.dn_out) A.dn_out[(int64_t)b * A.L + j] = R.dn[q];
    }
  }
}

// The per-chain outputs known after the acceptance rule (accepted length, tau, log
// alpha_res), by one thread.
__device__ __forceinline__ void scan_write_chain(const ScanArgs& A, int b, const ChainState& cs) {
  if (A.ratios_only) return;
  if (A.accepted_len) A.accepted_len[b] = cs.tau > 0 ? cs.tau - 1 : 0;
  if (A.tau_out) A.tau_out[b] = cs.tau;
  if (A.la_res_out && cs.kind != kKindInactive) A.la_res_out[b] = cs.la_res;
}

// For chain b with loaded values R: coins and the acceptance rule.  In block mode every
// candidate residual row j (lane j & 31 of segment j >> 5) also gets the U-sampler setup
// at (|Delta_j|, log alpha_{j-1}) (log alpha_{-1} = 0), whose log v is the residual mass
// that h_{j-1} needs: the scan evaluates it once for both.  Called by a full warp; every
// lane returns the result.  Writes nothing.
__device__ ScanOut scan_decide(const ScanArgs& A, int b, const ScanRegs& R) {
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int L = A.L;
  const int g = R.g;
  ScanOut out;
  out.have_P = false;
  if (g <= 0 || A.ratios_only) {
    out.cs = inactive_state();
    return out;
  }
  const int nseg = (L + 31) >> 5;

  // coins: eta_j from Philox (b, j, 0, 0), word 0, compared in log space
  float leta[2];
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int j = lane + 32 * q;
    leta[q] = 0.f;
    if (q < nseg && j < g)
      leta[q] = log_uniform(philox_block(seed_of(A), (uint32_t)b, (uint32_t)j, kStreamCoin, 0u).x);
  }
  const float ellw[2] = {R.ell[0] * A.inv_omega2, R.ell[1] * A.inv_omega2};

  int tau;             // 1-based
  float la_res = 0.f;  // log alpha_{tau-1}
  if (A.mode == 0) {
    // sample verification: c_j = [eta_j < min{1, e^ell_j}]; tau = first failure
    unsigned fm[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = lane + 32 * q;
      const bool fail = (q < nseg && j < g) && !(leta[q] < fminf(0.f, ellw[q]));
      fm[q] = __ballot_sync(FULL, fail);
    }
    tau = fm[0] ? __ffs(fm[0]) : (fm[1] ? 32 + __ffs(fm[1]) : g + 1);
  } else {
    // block verification: log alpha_j = min{0, log alpha_{j-1} + ell_j}, evaluated in
    // step order by every lane on all tempered ell (gathered with independent
    // shuffles), lane j & 31 of segment j >> 5 keeping log alpha_j, so that a clamp
    // to alpha = 1 is exact exactly when the recursion reaches it
    float la[2] = {0.f, 0.f};
    float run = 0.f;
#pragma unroll 1
    for (int k = 0; k < g; ++k) {
      const float e = __shfl_sync(FULL, k < 32 ? ellw[0] : ellw[1], k & 31);
      run = fminf(0.f, run + e);
      if (k < 32) la[0] = (k == lane) ? run : la[0];
      else la[1] = (k - 32 == lane) ? run : la[1];
    }
    // log alpha_{j-1} of each candidate residual row, and its U-sampler setup
    float lap[2];
    {
      const float up0 = __shfl_up_sync(FULL, la[0], 1);
      const float last0 = __shfl_sync(FULL, la[0], 31);
      const float up1 = __shfl_up_sync(FULL, la[1], 1);
      lap[0] = (lane == 0) ? 0.f : up0;
      lap[1] = (lane == 0) ? last0 : up1;
    }
    UParams Pq[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      if (q < nseg) {  // warp-uniform
        const bool ok = (R.dn[q] > 0.f) && isfinite(R.dn[q]) && isfinite(lap[q]);
        Pq[q] = usample_setup(ok ? R.dn[q] : 1.f, ok ? fminf(lap[q], 0.f) : -1.f);
      } else {
        Pq[q] = UParams{};
      }
    }
    // h_j (0-based j) uses |Delta| and log v of step j + 1 (the paper's D_{j+1})
    const float dnx0 = __shfl_down_sync(FULL, R.dn[0], 1);
    const float dnx1 = __shfl_down_sync(FULL, R.dn[1], 1);
    const float dnf1 = __shfl_sync(FULL, R.dn[1], 0);
    const float lvx0 = __shfl_down_sync(FULL, Pq[0].lv, 1);
    const float lvx1 = __shfl_down_sync(FULL, Pq[1].lv, 1);
    const float lvf1 = __shfl_sync(FULL, Pq[1].lv, 0);
    unsigned sm[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = lane + 32 * q;
      bool succ = false;
      if (q < nseg && j < g) {
        float lh;
        if (j == g - 1) {
          lh = la[q];  // h_gamma = alpha_gamma
        } else {
          const float Dn = (q == 0) ? (lane == 31 ? dnf1 : dnx0) : dnx1;
          const float lv = (q == 0) ? (lane == 31 ? lvf1 : lvx0) : lvx1;
          lh = block_log_h(la[q], Dn, lv);
        }
        succ = leta[q] < lh;
      }
      sm[q] = __ballot_sync(FULL, succ);
    }
    int last = -1;  // 0-based index of the last success
    if (sm[1]) last = 32 + 31 - __clz(sm[1]);
    else if (sm[0]) last = 31 - __clz(sm[0]);
    tau = last + 2;
    if (tau >= 2) {
      const int k = tau - 2;
      const float v0 = __shfl_sync(FULL, la[0], k & 31);
      const float v1 = __shfl_sync(FULL, la[1], k & 31);
      la_res = (k < 32) ? v0 : v1;
    }
    if (tau <= g) {  // residual parameters of row tau - 1
      const int rr = tau - 1;
      const UParams P0 = shfl_params(Pq[0], rr & 31);
      const UParams P1 = shfl_params(Pq[1], rr & 31);
      out.P = (rr >> 5) ? P1 : P0;
      out.have_P = true;
    }
  }

  // quantities of step tau (0-based row tau-1) when a residual is drawn
  const bool resid = tau <= g;
  const int rrow = resid ? tau - 1 : 0;
  const int rq = rrow >> 5, rl = rrow & 31;
  const float Dt = rq ? __shfl_sync(FULL, R.dn[1], rl) : __shfl_sync(FULL, R.dn[0], rl);
  const float st = rq ? __shfl_sync(FULL, R.sg[1], rl) : __shfl_sync(FULL, R.sg[0], rl);
  const float S1t = rq ? __shfl_sync(FULL, R.S1[1], rl) : __shfl_sync(FULL, R.S1[0], rl);
  const float S2t = rq ? __shfl_sync(FULL, R.S2[1], rl) : __shfl_sync(FULL, R.S2[0], rl);

  uint32_t status = R.any_bad ? 2u : 0u;
  int kind;
  if (!resid) {
    kind = A.has_bonus ? kKindBonus : kKindCopy;
  } else if (!(S2t > 0.f) || !(Dt > 0.f)) {
    kind = kKindZeroDelta;
    status |= 1u;
  } else if (A.residual_kind == 1) {
    kind = kKindReflect;
  } else {
    kind = kKindResid;
  }
  ChainState& cs = out.cs;
  cs.tau = tau;
  cs.row = resid ? rrow : g - 1;
  cs.U = NAN;
  cs.la_res = la_res;
  cs.sigma = resid ? st : NAN;
  cs.dnorm = resid ? Dt : NAN;
  cs.inv_norm = (S2t > 0.f) ? rsqrtf(S2t) : 0.f;
  cs.refl = (S2t > 0.f) ? 1.0f + 2.0f * S1t / S2t : 0.f;
  cs.status = status;
  cs.kind = kind;
  cs.pad[0] = cs.pad[1] = 0;
  return out;
}

// scan_load, the per-step outputs, scan_decide and the per-chain outputs in one go (the
// kernels whose writes need not wait for an earlier grid).
__device__ ScanOut scan_warp(const ScanArgs& A, int b) {
  const ScanRegs R = scan_load(A, b);
  scan_write_steps(A, b, R);
  const ScanOut o = scan_decide(A, b, R);
  if ((threadIdx.x & 31) == 0) scan_write_chain(A, b, o.cs);
  return o;
}

// Per-chain outputs that depend on U: status bits and (U, log alpha_res, |Delta_tau|,
// sigma_tau); written by one thread (leader).
__device__ __forceinline__ void report_chain(const ScanArgs& A, int b, const ChainState& cs, bool leader) {
  if (leader && cs.kind != kKindInactive) {
    if (A.status_out) A.status_out[b] = cs.status;
    if (A.aux_out) {
      float* a = A.aux_out + 4 * (int64_t)b;
      a[0] = cs.U;
      a[1] = cs.la_res;
      a[2] = cs.dnorm;
      a[3] = cs.sigma;
    }
  }
}

// Residual 1-D draw of a finished chain by the whole CTA (CTA-uniform branch).
template <int NT>
__device__ __forceinline__ void draw_u(const ScanArgs& A, int b, ChainState& cs, const UParams* P,
                                       USampleScratch* us) {
  if (cs.kind == kKindResid && A.draw_u) {
    const uint32_t wbits = philox_block(seed_of(A), (uint32_t)b, 0u, kStreamUSample, 0u).x;
    uint32_t st = cs.status;
    const UParams Q = P ? *P : usample_setup(cs.dnorm, fminf(cs.la_res, 0.f));
    cs.U = usample_block<NT>(Q, wbits, &st, us);
    cs.status = st;
  }
}

// Grid dependencies (programmatic dependent launch).  A kernel launched with the
// programmatic-serialisation attribute may start while the previous kernel on its
// stream is still running, as soon as every CTA of that kernel has called
// griddep_launch_dependents or exited; griddep_wait blocks until the previous kernel has
// completed and its writes are visible.  Without that attribute (or with no previous
// kernel) both are no-ops.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---------------------------------------------------------------- residual row
// The thread group that writes one residual row: a whole CTA (the fused kernel's
// finishing CTA, or k_finish's).  all_sum returns the group's sum in every thread,
// reduced lane-wise within warps, then over warps in warp order.
struct CtaGroup {
  float2* red;   // [blockDim.x / 32]
  float* bcast;
  __device__ __forceinline__ int rank() const { return threadIdx.x; }
  __device__ __forceinline__ int size() const { return blockDim.x; }
  __device__ __forceinline__ float all_sum(float v) const {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5].x = v;
    __syncthreads();
    if (threadIdx.x < 32) {
      float w = (threadIdx.x < blockDim.x / 32) ? red[threadIdx.x].x : 0.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) w += __shfl_xor_sync(0xffffffffu, w, o);
      if (threadIdx.x == 0) *bcast = w;
    }
    __syncthreads();
    return *bcast;
  }
};

// The decomposition residual's coefficient U - e^T G of chain state cs (pass A: reduces
// delta^T G over the rejected row with the threads of group grp, every thread of the
// group calling it with the same cs; 0 for the other kinds).  With gcache (room for the
// row's groups, each used only by the thread that owns the group) pass A keeps G there
// for pass B (GMODE 1), or the caller has filled it already (GMODE 2: drawn by warps that
// would otherwise wait on the scan); with GMODE 0 pass B draws G again (same Philox
// counters).  Each thread handles RU groups of four elements per sweep, the loads of all
// of them issued before any use.  Reads only (and gcache with GMODE 1).
template <typename T, bool VEC4, int RU, int GMODE, typename Group>
__device__ float residual_coef(const T* __restrict__ mq, const T* __restrict__ mp, int L, int64_t d,
                               uint64_t seed, int b, const ChainState& cs, const Group& grp,
                               float4* gcache) {
  if (cs.kind != kKindResid) return 0.f;
  const int nt = grp.size();
  const int64_t ng = (d + 3) / 4;
  const int64_t rbase = ((int64_t)b * L + cs.row) * d;
  // groups past the row end load zeros (load4 guards each element)
  float sp = 0.f;
  for (int64_t g0 = grp.rank(); g0 < ng; g0 += (int64_t)nt * RU) {
    float fq[RU][4], fp[RU][4];
#pragma unroll
    for (int u = 0; u < RU; ++u) {
      load4<T, VEC4>(mq + rbase, 4 * (g0 + (int64_t)u * nt), d, fq[u]);
      load4<T, VEC4>(mp + rbase, 4 * (g0 + (int64_t)u * nt), d, fp[u]);
    }
#pragma unroll
    for (int u = 0; u < RU; ++u) {
      const int64_t gi = g0 + (int64_t)u * nt;
      const float4 G = (GMODE == 2) ? (gi < ng ? gcache[gi] : make_float4(0.f, 0.f, 0.f, 0.f))
                                    : normals4_f(seed, (uint32_t)b, (uint32_t)gi, kStreamResid, 0u);
      if (GMODE == 1 && gi < ng) gcache[gi] = G;
      sp = fmaf(fp[u][0] - fq[u][0], G.x, sp);  // tail elements load 0 and contribute 0
      sp = fmaf(fp[u][1] - fq[u][1], G.y, sp);
      sp = fmaf(fp[u][2] - fq[u][2], G.z, sp);
      sp = fmaf(fp[u][3] - fq[u][3], G.w, sp);
    }
  }
  return cs.U - grp.all_sum(sp) * cs.inv_norm;  // U - e^T G
}

// Writes y[b, :] for chain state cs with the threads of group grp (pass B): the
// decomposition residual m^q + sigma (G + e coef) with coef from residual_coef, the
// reflection x - delta (1 + 2 S1/S2), m^q + sigma G for a zero shift, the bonus step,
// or the last accepted draft.
template <typename T, bool VEC4, int RU, int GMODE, typename Group>
__device__ void residual_write(const T* __restrict__ x, const T* __restrict__ mq,
                               const T* __restrict__ mp, const T* __restrict__ mq_bonus,
                               const float* __restrict__ sigma_bonus, int L, int64_t d,
                               uint64_t seed, int b, const ChainState& cs, float coef,
                               T* __restrict__ y, const Group& grp, const float4* gcache) {
  if (cs.kind == kKindInactive) return;
  const int nt = grp.size();
  const int64_t ng = (d + 3) / 4;
  const int64_t rbase = ((int64_t)b * L + cs.row) * d;
  const int64_t ybase = (int64_t)b * d;
  // groups past the row end load zeros (load4 guards each element) and store nothing
  if (cs.kind == kKindResid) {
    for (int64_t g0 = grp.rank(); g0 < ng; g0 += (int64_t)nt * RU) {
      float fq[RU][4], fp[RU][4];
#pragma unroll
      for (int u = 0; u < RU; ++u) {
        load4<T, VEC4>(mq + rbase, 4 * (g0 + (int64_t)u * nt), d, fq[u]);
        load4<T, VEC4>(mp + rbase, 4 * (g0 + (int64_t)u * nt), d, fp[u]);
      }
#pragma unroll
      for (int u = 0; u < RU; ++u) {
        const int64_t gi = g0 + (int64_t)u * nt;
        const float4 G = GMODE ? (gi < ng ? gcache[gi] : make_float4(0.f, 0.f, 0.f, 0.f))
                                : normals4_f(seed, (uint32_t)b, (uint32_t)gi, kStreamResid, 0u);
        const float g4[4] = {G.x, G.y, G.z, G.w};
        float out[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
          out[k] = fq[u][k] + cs.sigma * fmaf((fp[u][k] - fq[u][k]) * cs.inv_norm, coef, g4[k]);
        if (gi < ng) store4<T, VEC4>(y + ybase, 4 * gi, d, out);
      }
    }
    return;
  }
  const bool bonus = cs.kind == kKindBonus;
  const bool draw = bonus || cs.kind == kKindZeroDelta;
  const float sgm = bonus ? sigma_bonus[b] : cs.sigma;
  for (int64_t g0 = grp.rank(); g0 < ng; g0 += (int64_t)nt * RU) {
    float a[RU][4], q[RU][4], p[RU][4];
#pragma unroll
    for (int u = 0; u < RU; ++u) {
      const int64_t i = 4 * (g0 + (int64_t)u * nt);
      if (cs.kind == kKindReflect) {
        load4<T, VEC4>(x + rbase, i, d, a[u]);
        load4<T, VEC4>(mq + rbase, i, d, q[u]);
        load4<T, VEC4>(mp + rbase, i, d, p[u]);
      } else if (cs.kind == kKindZeroDelta) {
        load4<T, VEC4>(mq + rbase, i, d, a[u]);
      } else if (bonus) {
        load4<T, VEC4>(mq_bonus + ybase, i, d, a[u]);
      } else {  // copy the last accepted draft
        load4<T, VEC4>(x + rbase, i, d, a[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < RU; ++u) {
      const int64_t gi = g0 + (int64_t)u * nt;
      float out[4];
      if (cs.kind == kKindReflect) {
#pragma unroll
        for (int k = 0; k < 4; ++k) out[k] = a[u][k] - (p[u][k] - q[u][k]) * cs.refl;  // x - delta (1 + 2 S1/S2)
      } else if (draw) {
        const float4 G = normals4_f(seed, (uint32_t)b, (uint32_t)gi, bonus ? kStreamBonus : kStreamResid, 0u);
        out[0] = a[u][0] + sgm * G.x; out[1] = a[u][1] + sgm * G.y;
        out[2] = a[u][2] + sgm * G.z; out[3] = a[u][3] + sgm * G.w;
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) out[k] = a[u][k];
      }
      if (gi < ng) store4<T, VEC4>(y + ybase, 4 * gi, d, out);
    }
  }
}

// Both passes (the writers that need not wait for an earlier grid in between).
template <typename T, bool VEC4, int RU, int GMODE, typename Group>
__device__ __forceinline__ void residual_row(const T* __restrict__ x, const T* __restrict__ mq,
                                             const T* __restrict__ mp, const T* __restrict__ mq_bonus,
                                             const float* __restrict__ sigma_bonus, int L, int64_t d,
                                             uint64_t seed, int b, const ChainState& cs,
                                             T* __restrict__ y, const Group& grp, float4* gcache) {
  const float coef = residual_coef<T, VEC4, RU, GMODE>(mq, mp, L, d, seed, b, cs, grp, gcache);
  residual_write<T, VEC4, RU, GMODE>(x, mq, mp, mq_bonus, sigma_bonus, L, d, seed, b, cs, coef, y, grp, gcache);
}

// The residual's G of chain b (stream kStreamResid) for groups [first, ng), every
// `step`-th group, into gcache: drawn by the finishing CTA's warps other than the
// scanning warp, before the rejected step is known (G does not depend on it).
__device__ __forceinline__ void prefill_resid_g(uint64_t seed, int b, int64_t ng, int first, int step,
                                                float4* gcache) {
  for (int64_t gi = first; gi < ng; gi += step) gcache[gi] = normals4_f(seed, (uint32_t)b, (uint32_t)gi, kStreamResid, 0u);
}

// ---------------------------------------------------------------- the fused kernel
struct VerifyArgs {
  const void* x;
  const void* mq;
  const void* mp;
  const void* mq_bonus;
  const float* sigma_bonus;
  int64_t d;
  int64_t chunk;
  void* y;
  float2* part;          // [B, L, C] fused kernel's tile partials (also read through S.part)
  uint64_t* tpart;       // the same slots as k_tiles' tagged partials (read through S.tpart)
  unsigned int* ticket;  // [B], zero at launch of the fused kernel
  ChainState* state;     // [B]; written when the residual row is left to k_resid_*
  ScanArgs S;
};

// Fetch-and-increment of chain b's ticket with acquire-release semantics at GPU scope,
// wrapping to 0 after `last` (atom.inc: old >= last ? 0 : old + 1): the CTA that draws
// `last` holds the chain's last tile, and the counter is back at 0 for the next call.
// The release publishes this CTA's partial; the holder of the last ticket acquires
// every partial released before it.
__device__ __forceinline__ unsigned int ticket_inc(unsigned int* p, unsigned int last) {
  unsigned int old;
  asm volatile("atom.acq_rel.gpu.global.inc.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(last) : "memory");
  return old;
}

// RESID: 1 = this kernel writes y (the residual's G cached in dynamic shared memory,
// (d + 3)/4 float4); 0 = it leaves the chain state for k_resid_*.  RU: groups of four
// elements per thread per residual sweep.
//
// Ordering against the previous kernel on the stream (see griddep_wait): this kernel
// writes nothing the previous one may read except its own outputs, and those only after
// griddep_wait; a finishing CTA triggers its dependents once it has read the chain's
// partials, the only workspace data that the next call overwrites.  (A call of this
// kernel clears the tickets first; pipelined calls run k_tiles + k_finish instead.)
template <typename T, bool VEC, int VPT, bool VEC4, int RESID, int RU>
__global__ void __launch_bounds__(kK1Threads, kK1MinBlocks) k_verify(VerifyArgs A) {
  __shared__ float2 red[kK1Threads / 32];
  __shared__ int last_s;
  __shared__ float bcast;
  __shared__ ChainState cs_s;
  __shared__ UParams P_s;
  __shared__ bool haveP_s;
  __shared__ USampleScratch us;
  __shared__ float ell_s[SDV_MAX_L], dn_s[SDV_MAX_L];
  extern __shared__ float4 g_s[];  // RESID: the residual's G, drawn once
  const int L = A.S.L;
  const int C = A.S.C;
  const int64_t tile = blockIdx.x;
  const int64_t r = tile / C;
  const int c = (int)(tile - r * C);
  const int b = (int)(r / L), j = (int)(r - (int64_t)b * L);
  const int g = A.S.L_eff ? max(0, min(A.S.L_eff[b], L)) : L;
  const T* x = (const T*)A.x;
  const T* mq = (const T*)A.mq;
  const T* mp = (const T*)A.mp;
  if (g == 0) {
    // inactive chain: tile (b, 0, 0) writes its outputs, nothing is streamed
    if (j == 0 && c == 0 && threadIdx.x < 32) {
      griddep_wait();
      const ChainState cs = scan_warp(A.S, b).cs;
      if (threadIdx.x == 0 && RESID == 0) A.state[b] = cs;
    }
    return;
  }
  if (j >= g) return;
  const int64_t e0 = (int64_t)c * A.chunk;
  const int64_t e1 = min(e0 + A.chunk, A.d);
  const float2 s = tile_sums<T, VEC, VPT>(x, mq, mp, r * A.d, e0, e1);
  const float2 t = block_sum2<kK1Threads>(s.x, s.y, red);
  if (threadIdx.x == 0) {
    A.part[tile] = t;
    const unsigned int last = (unsigned int)(g * C) - 1u;
    last_s = (ticket_inc(A.ticket + b, last) == last);
  }
  __syncthreads();  // thread 0's acquire reaches warp 0's partial loads through the barrier
  if (!last_s) return;
  ScanRegs R;
  if (threadIdx.x < 32) {
    R = scan_load(A.S, b);
    const int lane = threadIdx.x;
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      if (lane + 32 * q < L) {
        ell_s[lane + 32 * q] = R.ell[q];
        dn_s[lane + 32 * q] = R.dn[q];
      }
    }
  }
  __syncthreads();
  griddep_launch_dependents();  // this chain's partials are read
  if (A.S.ratios_only) {
    griddep_wait();
    if (threadIdx.x < 32) scan_write_steps(A.S, b, R);
    return;
  }
  if (threadIdx.x < 32) {
    const ScanOut so = scan_decide(A.S, b, R);
    if (threadIdx.x == 0) {
      cs_s = so.cs;
      P_s = so.P;
      haveP_s = so.have_P;
    }
  } else if (RESID) {
    prefill_resid_g(seed_of(A.S), b, (A.d + 3) / 4, threadIdx.x - 32, kK1Threads - 32, g_s);
  }
  __syncthreads();
  ChainState cs = cs_s;
  draw_u<kK1Threads>(A.S, b, cs, haveP_s ? &P_s : nullptr, &us);
  const CtaGroup grp{red, &bcast};
  float coef = 0.f;
  if (RESID) coef = residual_coef<T, VEC4, RU, 2>(mq, mp, L, A.d, seed_of(A.S), b, cs, grp, g_s);
  // every write of this call's outputs comes after the previous kernel has completed
  griddep_wait();
  for (int i = threadIdx.x; i < L; i += kK1Threads) {
    if (A.S.ell_out) A.S.ell_out[(int64_t)b * L + i] = ell_s[i];
    if (A.S.dn_out) A.S.dn_out[(int64_t)b * L + i] = dn_s[i];
  }
  if (threadIdx.x == 0) {
    scan_write_chain(A.S, b, cs);
    report_chain(A.S, b, cs, true);
    if (RESID == 0) A.state[b] = cs;
  }
  if (RESID)
    residual_write<T, VEC4, RU, 2>(x, mq, mp, (const T*)A.mq_bonus, A.sigma_bonus, L, A.d, seed_of(A.S), b, cs,
                                   coef, (T*)A.y, grp, g_s);
}

// ---------------------------------------------------------------- many-chain path
// With many chains the fused kernel's finishing CTAs (each holding a CTA slot for
// the whole latency-bound scan / U-draw / residual) take more SM time than the
// stream itself.  The many-chain path streams the same tiles without tickets
// (k_tiles: identical partials, tagged with the call) at full occupancy, then finishes every chain with
// a small CTA (k_finish: one warp's scan and U-draw, then the residual row), all
// chains at once.
// One tile's 3 VPT 16-byte vectors per thread (a tile is one full sweep: VPT vectors
// per thread and tensor), issued together with guarded loads, and its (S1, S2)
// contribution.
template <int VPT>
struct TileBuf {
  uint4 x[VPT], q[VPT], p[VPT];
};

template <typename T, int VPT>
__device__ __forceinline__ void tile_issue(const T* __restrict__ x, const T* __restrict__ mq,
                                           const T* __restrict__ mp, int64_t base, int64_t e0, int64_t e1,
                                           TileBuf<VPT>& B) {
  constexpr int V = 16 / (int)sizeof(T);
  const int64_t v0 = (base + e0) / V;
  const int nv = (int)((e1 - e0) / V);
  const uint4* X = reinterpret_cast<const uint4*>(x) + v0;
  const uint4* Q = reinterpret_cast<const uint4*>(mq) + v0;
  const uint4* P = reinterpret_cast<const uint4*>(mp) + v0;
  const uint4 z = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
  for (int u = 0; u < VPT; ++u) {
    const int vv = threadIdx.x + u * kK1Threads;
    B.x[u] = vv < nv ? ldg_stream(X + vv) : z;
  }
#pragma unroll
  for (int u = 0; u < VPT; ++u) {
    const int vv = threadIdx.x + u * kK1Threads;
    B.q[u] = vv < nv ? ldg_stream(Q + vv) : z;
  }
#pragma unroll
  for (int u = 0; u < VPT; ++u) {
    const int vv = threadIdx.x + u * kK1Threads;
    B.p[u] = vv < nv ? ldg_stream(P + vv) : z;
  }
}

template <typename T, int VPT>
__device__ __forceinline__ float2 tile_fma(const TileBuf<VPT>& B) {
  constexpr int V = 16 / (int)sizeof(T);
  float s1 = 0.f, s2 = 0.f;
#pragma unroll
  for (int u = 0; u < VPT; ++u) {
    float fx[V], fq[V], fp[V];
    unpack(B.x[u], fx);
    unpack(B.q[u], fq);
    unpack(B.p[u], fp);
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const float dl = fp[k] - fq[k];  // m^p - m^q (zero-filled vectors contribute 0)
      const float a = fx[k] - fp[k];   // yhat - m^p
      s1 = fmaf(a, dl, s1);
      s2 = fmaf(dl, dl, s2);
    }
  }
  return make_float2(s1, s2);
}

// The tag of the partial in slot `tile` of this call's set and the tag its reader
// released after reading it (acquire: the reader's loads of the slot happen before
// anything this thread does next).
__device__ __forceinline__ void slot_state(const VerifyArgs& A, int64_t tile, uint32_t& held, uint32_t& taken) {
  held = __ldcg(reinterpret_cast<const unsigned int*>(A.tpart + 2 * tile) + 1);
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(taken) : "l"(A.S.consumed + tile) : "memory");
}

// The stream of the many-chain and pipelined paths: one tile per CTA; its (S1, S2) is
// stored with the call's tag.  The FMAs of a tile and their order are those of
// tile_sums, so the partials equal the fused kernel's.  (Two or four software-pipelined tiles per CTA measured
// slower: 17.4 / 20.1 us against 16.5 us per pipelined pixel call.)
template <typename T, bool VEC, int VPT>
__global__ void __launch_bounds__(kK1Threads, tile_min_blocks(VPT)) k_tiles(VerifyArgs A) {
  __shared__ float2 red[kK1Threads / 32];
  const int L = A.S.L;
  const int C = A.S.C;
  const int64_t tile = blockIdx.x;
  const int64_t r = tile / C;
  const int c = (int)(tile - r * C);
  const int b = (int)(r / L), j = (int)(r - (int64_t)b * L);
  const int g = A.S.L_eff ? max(0, min(A.S.L_eff[b], L)) : L;
  if (j < g) {  // CTA-uniform
    const int64_t e0 = (int64_t)c * A.chunk;
    const int64_t e1 = min(e0 + A.chunk, A.d);
    // the tag now in this CTA's slot and the tag last consumed from it, loaded by thread
    // 0 once its tile loads are in flight (the acquire orders only what follows it) and
    // compared before the store
    uint32_t held = 0u, taken = 0u;
    float2 sm;
    if (VEC) {
      TileBuf<VPT> B;
      tile_issue<T, VPT>((const T*)A.x, (const T*)A.mq, (const T*)A.mp, r * A.d, e0, e1, B);
      if (threadIdx.x == 0) slot_state(A, tile, held, taken);
      sm = tile_fma<T, VPT>(B);
    } else {
      if (threadIdx.x == 0) slot_state(A, tile, held, taken);
      sm = tile_sums<T, false, 1>((const T*)A.x, (const T*)A.mq, (const T*)A.mp, r * A.d, e0, e1);
    }
    const float2 t = block_sum2<kK1Threads>(sm.x, sm.y, red);
    if (threadIdx.x == 0) {
      // the slot's partial has not been read yet by the call that wrote it (which may
      // still be finishing, since calls overlap), or this set held another layout:
      // wait for the previous kernel, whose completion implies every earlier call's
      // (in practice the slot was read long ago)
      if (A.S.fresh_set || held != taken) griddep_wait();
      // S1 and S2 each share an 8-byte word with the call's tag; each word is written
      // whole (a vector of two 8-byte elements), so k_finish can tell this call's
      // partials from those a previous call left in the slot
      const unsigned long long tg = (unsigned long long)A.S.tag << 32;
      reinterpret_cast<ulonglong2*>(A.tpart)[tile] =
          make_ulonglong2(tg | __float_as_uint(t.x), tg | __float_as_uint(t.y));
    }
  }
  if (blockIdx.x == 0) {
    // CTA 0 ties this grid's completion to the previous kernel's (so the next k_finish,
    // which writes its outputs after this grid has completed, writes after the previous
    // call's k_finish); it triggers first, its own tile done, so that k_finish can start
    __syncthreads();
    griddep_launch_dependents();
    if (threadIdx.x == 0) griddep_wait();
  }
}

// One CTA per chain: the CTA triggers its dependents at once (the next call's stream
// writes the other set of partials); warp 0 reads the chain's partials (k_finish starts
// only after every k_tiles CTA has stored its partial and exited or triggered; the tags
// confirm that each one read is this call's, else the warp waits for k_tiles to
// complete and reads them again), and after the barrier a second warp releases the
// chain's slots to the next call that writes this set; then warp 0 scans the chain and draws U
// (warp U-sampler) while the other warps draw the residual's G into shared memory
// (dynamic, (d + 3)/4 float4), and, with RESID = 1, all kFinishThreads threads write y
// (launched with 32 threads and leaving the chain state for k_resid_* when RESID = 0).
// Every output is written after griddep_wait.
template <typename T, bool VEC4, int RESID, int NT>
__global__ void __launch_bounds__(NT) k_finish(VerifyArgs A) {
  __shared__ ChainState cs_s;
  __shared__ float2 red[NT / 32];
  __shared__ float bcast;
  __shared__ float ell_s[SDV_MAX_L], dn_s[SDV_MAX_L];
  __shared__ UParams P_s;
  __shared__ bool haveP_s;
  __shared__ USampleScratch us;
  __shared__ int gw_s;             // the chain's window length (tiles written this call)
  extern __shared__ float4 g_s[];  // RESID: the residual's G, drawn once
  constexpr int RU = NT >= 256 ? kFusedResidUnroll : kFinishResidUnroll;
  const int b = blockIdx.x;
  const int L = A.S.L;
  ScanRegs R;
  // the next kernel (the next call's stream) may start now: it writes the other set of
  // partials, and a slot of this set only once this call has read it
  griddep_launch_dependents();
  if (threadIdx.x < 32) {
    R = scan_load(A.S, b);
    if (R.stale) {
      // a partial of this call is not visible yet (k_finish starts once every k_tiles
      // CTA has stored its partial and exited or triggered, so in practice they all
      // are): wait for k_tiles to complete, which makes its writes visible, and read
      // them again
      griddep_wait();
      R = scan_load(A.S, b, false);
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      if (threadIdx.x + 32 * q < L) {
        ell_s[threadIdx.x + 32 * q] = R.ell[q];
        dn_s[threadIdx.x + 32 * q] = R.dn[q];
      }
    }
    if (threadIdx.x == 0) gw_s = R.g;
  }
  __syncthreads();
  if (A.S.consumed && (int)(threadIdx.x >> 5) == (NT > 32 ? 1 : 0)) {
    // release the chain's slots (those its tiles wrote) to the next call that writes
    // this set: the barrier orders warp 0's reads of them before these stores, and that
    // call's k_tiles CTA overwrites a slot once it reads back (acquire) the tag it found
    // there.  Off warp 0's path where the CTA has a second warp.
    const int64_t s0 = (int64_t)b * L * A.S.C;
    const int n = gw_s * A.S.C;
    for (int k = threadIdx.x & 31; k < n; k += 32)
      asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(A.S.consumed + s0 + k), "r"(A.S.tag) : "memory");
  }
  if (threadIdx.x < 32) {
    const ScanOut so = scan_decide(A.S, b, R);
    ChainState cs = so.cs;
    if (NT < 256 && cs.kind == kKindResid && A.S.draw_u) {
      // a 64-thread CTA: the one-warp U-sampler while warp 1 draws the noise
      const uint32_t wbits = philox_block(seed_of(A.S), (uint32_t)b, 0u, kStreamUSample, 0u).x;
      uint32_t st = cs.status;
      const UParams Q = so.have_P ? so.P : usample_setup(cs.dnorm, fminf(cs.la_res, 0.f));
      cs.U = usample_warp(Q, wbits, &st);
      cs.status = st;
    }
    if (threadIdx.x == 0) {
      cs_s = cs;
      P_s = so.P;
      haveP_s = so.have_P;
    }
  } else if (RESID) {
    prefill_resid_g(seed_of(A.S), b, (A.d + 3) / 4, threadIdx.x - 32, NT - 32, g_s);
  }
  __syncthreads();
  ChainState cs = cs_s;
  if (NT >= 256) draw_u<NT>(A.S, b, cs, haveP_s ? &P_s : nullptr, &us);  // the CTA-wide U-sampler
  const CtaGroup grp{red, &bcast};
  float coef = 0.f;
  if (RESID)
    coef = residual_coef<T, VEC4, RU, 2>((const T*)A.mq, (const T*)A.mp, L, A.d, seed_of(A.S), b, cs, grp, g_s);
  // outputs: after k_tiles has completed, and with it the previous call (see k_tiles)
  griddep_wait();
  for (int i = threadIdx.x; i < L; i += blockDim.x) {
    if (A.S.ell_out) A.S.ell_out[(int64_t)b * L + i] = ell_s[i];
    if (A.S.dn_out) A.S.dn_out[(int64_t)b * L + i] = dn_s[i];
  }
  if (threadIdx.x == 0) {
    scan_write_chain(A.S, b, cs);
    report_chain(A.S, b, cs, true);
    if (RESID == 0) A.state[b] = cs;
  }
  if (RESID)
    residual_write<T, VEC4, RU, 2>((const T*)A.x, (const T*)A.mq, (const T*)A.mp, (const T*)A.mq_bonus,
                                   A.sigma_bonus, L, A.d, seed_of(A.S), b, cs, coef, (T*)A.y, grp, g_s);
}

// ---------------------------------------------------------------- acceptance scan only
__global__ void __launch_bounds__(kK2Threads) k_scan(ScanArgs A) {
  const int b = blockIdx.x * (kK2Threads / 32) + (threadIdx.x >> 5);
  if (b >= A.B) return;  // warp-uniform
  (void)scan_warp(A, b);
}

// ---------------------------------------------------------------- long rows: K4a / K4b
template <typename T, bool VEC4>
__global__ void __launch_bounds__(kK4Threads)
k_resid_dot(const T* __restrict__ mq, const T* __restrict__ mp, int L, int64_t d, int C4, int gpc,
            uint64_t seed_v, const uint64_t* __restrict__ seed_dev, const ChainState* __restrict__ state,
            float* __restrict__ part4) {
  __shared__ float2 red[kK4Threads / 32];
  // pipelined launches: let the next kernel launch now, then wait for the chain states
  griddep_launch_dependents();
  griddep_wait();
  const uint64_t seed = seed_dev ? *seed_dev : seed_v;
  const int b = blockIdx.x / C4, c = blockIdx.x - b * C4;
  const ChainState cs = state[b];
  if (cs.kind != kKindResid) return;
  const int64_t base = ((int64_t)b * L + cs.row) * d;
  const int64_t g0 = (int64_t)c * gpc;
  const int64_t g1 = min(g0 + gpc, (d + 3) / 4);
  float s = 0.f;
  for (int64_t gi = g0 + threadIdx.x; gi < g1; gi += kK4Threads) {
    float fq[4], fp[4];
    load4<T, VEC4>(mq + base, 4 * gi, d, fq);
    load4<T, VEC4>(mp + base, 4 * gi, d, fp);
    const float4 G = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamResid, 0u);
    s = fmaf(fp[0] - fq[0], G.x, s);
    s = fmaf(fp[1] - fq[1], G.y, s);
    s = fmaf(fp[2] - fq[2], G.z, s);
    s = fmaf(fp[3] - fq[3], G.w, s);
  }
  const float2 t = block_sum2<kK4Threads>(s, 0.f, red);
  if (threadIdx.x == 0) part4[blockIdx.x] = t.x;
}

template <typename T, bool VEC4>
__global__ void __launch_bounds__(kK4Threads)
k_resid_write(const T* __restrict__ x, const T* __restrict__ mq, const T* __restrict__ mp,
              const T* __restrict__ mq_bonus, const float* __restrict__ sigma_bonus, int L,
              int64_t d, int C4, int gpc, uint64_t seed_v, const uint64_t* __restrict__ seed_dev,
              const ChainState* __restrict__ state, const float* __restrict__ part4, T* __restrict__ y) {
  // pipelined launches: let the next call's stream launch now, then wait for the dots
  griddep_launch_dependents();
  griddep_wait();
  const uint64_t seed = seed_dev ? *seed_dev : seed_v;
  const int b = blockIdx.x / C4, c = blockIdx.x - b * C4;
  const ChainState cs = state[b];
  if (cs.kind == kKindInactive) return;
  const int64_t rbase = ((int64_t)b * L + cs.row) * d;
  const int64_t ybase = (int64_t)b * d;
  const int64_t g0 = (int64_t)c * gpc;
  const int64_t g1 = min(g0 + gpc, (d + 3) / 4);
  float coef = 0.f;  // U - e^T G for the decomposition residual
  if (cs.kind == kKindResid) {
    float T2 = 0.f;
    for (int k = 0; k < C4; ++k) T2 += part4[(int64_t)b * C4 + k];
    coef = cs.U - T2 * cs.inv_norm;
  }
  for (int64_t gi = g0 + threadIdx.x; gi < g1; gi += kK4Threads) {
    const int64_t i = 4 * gi;
    float out[4];
    if (cs.kind == kKindResid) {
      float fq[4], fp[4];
      load4<T, VEC4>(mq + rbase, i, d, fq);
      load4<T, VEC4>(mp + rbase, i, d, fp);
      const float4 G = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamResid, 0u);
      const float g4[4] = {G.x, G.y, G.z, G.w};
#pragma unroll
      for (int k = 0; k < 4; ++k)
        out[k] = fq[k] + cs.sigma * fmaf((fp[k] - fq[k]) * cs.inv_norm, coef, g4[k]);
    } else if (cs.kind == kKindReflect) {
      float fx[4], fq[4], fp[4];
      load4<T, VEC4>(x + rbase, i, d, fx);
      load4<T, VEC4>(mq + rbase, i, d, fq);
      load4<T, VEC4>(mp + rbase, i, d, fp);
#pragma unroll
      for (int k = 0; k < 4; ++k) out[k] = fx[k] - (fp[k] - fq[k]) * cs.refl;
    } else if (cs.kind == kKindZeroDelta) {
      float fq[4];
      load4<T, VEC4>(mq + rbase, i, d, fq);
      const float4 G = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamResid, 0u);
      out[0] = fq[0] + cs.sigma * G.x; out[1] = fq[1] + cs.sigma * G.y;
      out[2] = fq[2] + cs.sigma * G.z; out[3] = fq[3] + cs.sigma * G.w;
    } else if (cs.kind == kKindBonus) {
      float fb[4];
      load4<T, VEC4>(mq_bonus + ybase, i, d, fb);
      const float sb = sigma_bonus[b];
      const float4 G = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamBonus, 0u);
      out[0] = fb[0] + sb * G.x; out[1] = fb[1] + sb * G.y;
      out[2] = fb[2] + sb * G.z; out[3] = fb[3] + sb * G.w;
    } else {
      load4<T, VEC4>(x + rbase, i, d, out);
    }
    store4<T, VEC4>(y + ybase, i, d, out);
  }
}

// ---------------------------------------------------------------- stand-alone pieces
__global__ void __launch_bounds__(kK1Threads)
k_usample(const float* __restrict__ D, const float* __restrict__ la, const uint32_t* __restrict__ w,
          int n, float* __restrict__ U, uint32_t* __restrict__ st) {
  __shared__ USampleScratch us;
  const int i = blockIdx.x;  // one CTA per item
  const float Dn = D[i];
  float l = la[i];
  uint32_t status = 0u;
  float u = NAN;
  if (isnan(Dn) || isnan(l)) {
    status = 2u;
  } else if (!(Dn > 0.f) || isinf(Dn)) {
    status = 1u;
  } else {
    l = fminf(l, 0.f);
    u = usample_block<kK1Threads>(usample_setup(Dn, l), w[i], &status, &us);
  }
  if (threadIdx.x == 0) {
    U[i] = u;
    if (st) st[i] = status;
  }
}

__global__ void k_philox(const uint4* __restrict__ ctr, uint64_t seed, int n, uint4* __restrict__ out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = philox4x32_10(ctr[i], (uint32_t)seed, (uint32_t)(seed >> 32));
}

__global__ void k_special(int which, const float* __restrict__ z, int n, float* __restrict__ out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float v = z[i];
  out[i] = which == 0 ? erfcx_any(v) : (which == 1 ? log_ndtr_g(v).x : (v < -4.0f ? gprime_cf(v) : gprime_ex(v)));
}

__global__ void k_normals(uint64_t seed, int B, int64_t d, uint32_t stream, uint32_t sub, float* out) {
  const int64_t ng = (d + 3) / 4;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * ng) return;
  const int b = (int)(t / ng);
  const int64_t gi = t - (int64_t)b * ng;
  const float4 G = normals4(seed, (uint32_t)b, (uint32_t)gi, stream, sub);
  const float g[4] = {G.x, G.y, G.z, G.w};
  for (int k = 0; k < 4; ++k)
    if (4 * gi + k < d) out[(int64_t)b * d + 4 * gi + k] = g[k];
}

// ---------------------------------------------------------------- host side
static thread_local int g_last_cuda_error = 0;

void set_last_cuda_error(int err) { g_last_cuda_error = err; }

static int check_launch() {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    g_last_cuda_error = (int)e;
    return SDV_ECUDA;
  }
  return SDV_OK;
}

static bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// ---- per-thread timing ring (sdv_timing_enable / sdv_timing_read).  Records use
// cudaEventRecordExternal under stream capture, so that they become event-record
// nodes of the graph (a plain record there only expresses a dependency).
struct TimingRing {
  std::vector<cudaEvent_t> ev;  // slots x 3
  int slots = 0;
  long long next = 0;   // recorded calls
  int stride = 1;       // record one call in `stride`
  long long calls = 0;  // calls seen while enabled
};
static thread_local TimingRing g_timing;

static void timing_destroy() {
  for (cudaEvent_t e : g_timing.ev) cudaEventDestroy(e);
  g_timing.ev.clear();
  g_timing.slots = 0;
  g_timing.next = 0;
  g_timing.calls = 0;
}

static cudaEvent_t* timing_slot() {
  if (g_timing.slots == 0) return nullptr;
  if (g_timing.calls++ % g_timing.stride != 0) return nullptr;
  const int s = (int)(g_timing.next % g_timing.slots);
  ++g_timing.next;
  return &g_timing.ev[3 * (size_t)s];
}

static void timing_record(cudaEvent_t e, cudaStream_t s) {
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(s, &cap);
  if (cap == cudaStreamCaptureStatusActive) cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
  else cudaEventRecord(e, s);
}

WsLayout ws_layout(int B, int L, int64_t d, int dtype) {
  WsLayout w{};
  const int es = dtype == SDV_BF16 ? 2 : 4;
  // vectors per thread: the smallest sweep that covers a row, capped at kK1Vpt (at 2
  // for bf16 rows, whose 16-byte vectors hold 8 elements: the 40-register tiles leave
  // room on an SM for the previous pipelined call's 256-thread finishing CTA; latent
  // rows 19.5 -> 19.0 us per pipelined call), so that common row lengths run whole,
  // unguarded sweeps
  const int64_t vec_per_row = (d * es + 15) / 16;
  const int64_t vpt_cap = es == 2 ? 2 : kK1Vpt;
  w.vpt1 = (int)std::min<int64_t>(vpt_cap, std::max<int64_t>(1, (vec_per_row + kK1Threads - 1) / kK1Threads));
  w.chunk1 = (int64_t)kK1Threads * w.vpt1 * (16 / es);
  w.C1 = (int)((d + w.chunk1 - 1) / w.chunk1);
  // long-row residual chunks: about kK4TargetCtas CTAs over all chains, kK4MinChunk ..
  // kK4MaxChunk elements each (a power of two)
  int64_t chunk4 = kK4MinChunk;
  while (chunk4 < kK4MaxChunk && (int64_t)B * ((d + chunk4 - 1) / chunk4) > kK4TargetCtas) chunk4 *= 2;
  w.chunk4 = chunk4;
  w.C4 = (int)((d + chunk4 - 1) / chunk4);
  auto up = [](size_t v) { return (v + 255) & ~(size_t)255; };
  size_t off = 0;
  w.ticket_off = off;
  off = up(off + sizeof(unsigned int) * (size_t)B);
  w.part_off = off;
  const size_t slots = (size_t)B * L * w.C1;
  w.cons_off = up(2 * sizeof(uint64_t) * slots);  // within a set
  w.part_set_bytes = up(w.cons_off + sizeof(uint32_t) * slots);
  off = up(off + 2 * w.part_set_bytes);
  w.state_off = off;
  off = up(off + sizeof(ChainState) * (size_t)B);
  w.part4_off = off;
  off = up(off + sizeof(float) * (size_t)B * w.C4);
  w.total = off;
  return w;
}

static int validate_window(const void* x, const void* mq, const void* mp, const float* sigma,
                           int64_t sstride, int B, int L, int64_t d, int dtype) {
  if (!x || !mq || !mp || !sigma) return SDV_EINVAL;
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1) return SDV_EINVAL;
  if (dtype != SDV_F32 && dtype != SDV_BF16) return SDV_EINVAL;
  if (sstride < 0) return SDV_EINVAL;
  if ((double)B * L * (double)d > 9.0e18) return SDV_EINVAL;
  if (B > (1 << 30)) return SDV_EINVAL;
  const size_t es = dtype == SDV_BF16 ? 2 : 4;
  if (!aligned(x, es) || !aligned(mq, es) || !aligned(mp, es) || !aligned(sigma, 4)) return SDV_EALIGN;
  return SDV_OK;
}

// A launch through cudaLaunchKernelEx: dynamic shared memory (raising the kernel's limit
// when it passes 48 KB) and, with `overlap`, programmatic stream serialisation.
template <typename Kern, typename... Extra>
static cudaError_t launch_ex(Kern kern, unsigned grid, unsigned threads, size_t smem, bool overlap,
                             const VerifyArgs& A, cudaStream_t s, Extra... extra) {
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = overlap ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, A, extra...);
}

template <typename T, int RESID>
static cudaError_t launch_verify(const VerifyArgs& A, int B, int L, int vpt, bool overlap, cudaStream_t s) {
  constexpr int V = 16 / (int)sizeof(T);
  constexpr int RU = RESID ? kFusedResidUnroll : 1;
  const bool vec = (A.d % V == 0) && aligned(A.x, 16) && aligned(A.mq, 16) && aligned(A.mp, 16);
  const bool vec4 = (A.d % 4 == 0) && aligned(A.x, 4 * sizeof(T)) && aligned(A.mq, 4 * sizeof(T)) &&
                    aligned(A.mp, 4 * sizeof(T)) && (A.y == nullptr || aligned(A.y, 4 * sizeof(T))) &&
                    (A.mq_bonus == nullptr || aligned(A.mq_bonus, 4 * sizeof(T)));
  const unsigned tiles = (unsigned)((int64_t)B * L * A.S.C);
  const size_t smem = (RESID && !A.S.ratios_only) ? sizeof(float4) * (size_t)((A.d + 3) / 4) : 0;
#define SDV_LAUNCH(VECV, VPTV, V4) return launch_ex(k_verify<T, VECV, VPTV, V4, RESID, RU>, tiles, kK1Threads, smem, overlap, A, s)
  if (!vec) {
    if (vec4) SDV_LAUNCH(false, 1, true);
    SDV_LAUNCH(false, 1, false);
  }
  if (vec4) {
    switch (vpt) {
      case 1: SDV_LAUNCH(true, 1, true);
      case 2: SDV_LAUNCH(true, 2, true);
      case 3: SDV_LAUNCH(true, 3, true);
      default: SDV_LAUNCH(true, 4, true);
    }
  }
  switch (vpt) {
    case 1: SDV_LAUNCH(true, 1, false);
    case 2: SDV_LAUNCH(true, 2, false);
    case 3: SDV_LAUNCH(true, 3, false);
    default: SDV_LAUNCH(true, 4, false);
  }
#undef SDV_LAUNCH
}

template <typename T>
static cudaError_t launch_tiles(const VerifyArgs& A, int B, int L, int vpt, bool overlap, cudaStream_t s) {
  constexpr int V = 16 / (int)sizeof(T);
  const bool vec = (A.d % V == 0) && aligned(A.x, 16) && aligned(A.mq, 16) && aligned(A.mp, 16);
  const unsigned tiles = (unsigned)((int64_t)B * L * A.S.C);
  if (!vec) return launch_ex(k_tiles<T, false, 1>, tiles, kK1Threads, 0, overlap, A, s);
  switch (vpt) {
    case 1: return launch_ex(k_tiles<T, true, 1>, tiles, kK1Threads, 0, overlap, A, s);
    case 2: return launch_ex(k_tiles<T, true, 2>, tiles, kK1Threads, 0, overlap, A, s);
    case 3: return launch_ex(k_tiles<T, true, 3>, tiles, kK1Threads, 0, overlap, A, s);
    default: return launch_ex(k_tiles<T, true, 4>, tiles, kK1Threads, 0, overlap, A, s);
  }
}

// k_finish: 64 threads per chain, or kFinishWideThreads for rows longer than
// kFinishMaxGroups groups of four (the pipelined path), whose residual passes and noise
// a 64-thread CTA would take too long over.
template <typename T, int RESID>
static cudaError_t launch_finish(const VerifyArgs& A, int B, bool overlap, cudaStream_t s) {
  const bool vec4 = (A.d % 4 == 0) && aligned(A.x, 4 * sizeof(T)) && aligned(A.mq, 4 * sizeof(T)) &&
                    aligned(A.mp, 4 * sizeof(T)) && (A.y == nullptr || aligned(A.y, 4 * sizeof(T))) &&
                    (A.mq_bonus == nullptr || aligned(A.mq_bonus, 4 * sizeof(T)));
  const int64_t ng = (A.d + 3) / 4;
  const size_t smem = RESID ? sizeof(float4) * (size_t)ng : 0;
  if (!RESID) {
    if (vec4) return launch_ex(k_finish<T, true, 0, 32>, (unsigned)B, 32, 0, overlap, A, s);
    return launch_ex(k_finish<T, false, 0, 32>, (unsigned)B, 32, 0, overlap, A, s);
  }
  if (ng > kFinishMaxGroups) {
    if (vec4) return launch_ex(k_finish<T, true, 1, kFinishWideThreads>, (unsigned)B, kFinishWideThreads, smem, overlap, A, s);
    return launch_ex(k_finish<T, false, 1, kFinishWideThreads>, (unsigned)B, kFinishWideThreads, smem, overlap, A, s);
  }
  if (vec4) return launch_ex(k_finish<T, true, 1, kFinishThreads>, (unsigned)B, kFinishThreads, smem, overlap, A, s);
  return launch_ex(k_finish<T, false, 1, kFinishThreads>, (unsigned)B, kFinishThreads, smem, overlap, A, s);
}

// A kernel launch through cudaLaunchKernelEx, with programmatic stream serialisation when
// `overlap`.
template <typename Kern, typename... Args>
static cudaError_t launch_pdl(Kern kern, unsigned grid, unsigned threads, bool overlap, cudaStream_t s,
                              Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = overlap ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// The long-row residual kernels: one CTA per chunk of the chain's rejected row.  Plain
// calls size the chunks for about kK4TargetCtas CTAs (short kernels want many CTAs);
// pipelined calls for at most kK4PipeCtas, since these kernels wait, resident, for the
// chain states while the next call streams beside them (few and long CTAs then cost
// the stream nothing, and their time is hidden).
template <typename T>
static cudaError_t launch_k4(const void* x, const void* mq, const void* mp, const void* mqb,
                             const float* sb, int B, int L, int64_t d, uint64_t seed, const uint64_t* seed_dev,
                             const WsLayout& w, const ChainState* st, float* part4, void* y, bool overlap,
                             bool pdl, cudaStream_t s) {
  const bool vec = (d % 4 == 0) && aligned(x, 4 * sizeof(T)) && aligned(mq, 4 * sizeof(T)) &&
                   aligned(mp, 4 * sizeof(T)) && aligned(y, 4 * sizeof(T)) &&
                   (mqb == nullptr || aligned(mqb, 4 * sizeof(T)));
  int64_t chunk4 = w.chunk4;
  if (overlap)  // at least one chunk per chain
    while (chunk4 < d && (int64_t)B * ((d + chunk4 - 1) / chunk4) > kK4PipeCtas) chunk4 *= 2;
  const int C4 = (int)((d + chunk4 - 1) / chunk4);   // <= w.C4: part4 has room
  const int gpc = (int)(chunk4 / 4);
  const unsigned grid = (unsigned)((int64_t)B * C4);
  cudaError_t e;
  if (vec) {
    e = launch_pdl(k_resid_dot<T, true>, grid, kK4Threads, pdl, s, (const T*)mq, (const T*)mp, L, d, C4,
                   gpc, seed, seed_dev, st, part4);
    if (e == cudaSuccess)
      e = launch_pdl(k_resid_write<T, true>, grid, kK4Threads, pdl, s, (const T*)x, (const T*)mq,
                     (const T*)mp, (const T*)mqb, sb, L, d, C4, gpc, seed, seed_dev, st, (const float*)part4,
                     (T*)y);
  } else {
    e = launch_pdl(k_resid_dot<T, false>, grid, kK4Threads, pdl, s, (const T*)mq, (const T*)mp, L, d, C4,
                   gpc, seed, seed_dev, st, part4);
    if (e == cudaSuccess)
      e = launch_pdl(k_resid_write<T, false>, grid, kK4Threads, pdl, s, (const T*)x, (const T*)mq,
                     (const T*)mp, (const T*)mqb, sb, L, d, C4, gpc, seed, seed_dev, st, (const float*)part4,
                     (T*)y);
  }
  return e;
}

// The tag of a call's k_tiles partials: a process-wide counter, never 0 (a zeroed
// workspace holds tag 0), so consecutive calls on a workspace never share a tag (a
// captured call keeps its tag at every replay of its graph, and replays of a graph run
// one after another).
static std::atomic<uint32_t> g_partial_tag{0u};
static uint32_t next_partial_tag() {
  uint32_t t;
  do {
    t = g_partial_tag.fetch_add(1u, std::memory_order_relaxed) + 1u;
  } while (t == 0u);
  return t;
}

// The set of partials a call on `workspace` uses: the other one than the previous call
// on that workspace (remembered for the last kPartialSetSlots workspaces; a forgotten
// workspace starts again at set 0, which at worst makes a stream CTA wait for the
// previous kernel before its store).
// `fresh` when the set's last user on this workspace had another layout (or is
// unknown): the stream then waits for the previous kernel before it stores.
constexpr int kPartialSetSlots = 64;
static int next_partial_set(const void* workspace, uint64_t layout, bool* fresh) {
  struct Entry {
    const void* ws;
    int next;
    uint64_t layout[2];
  };
  static std::mutex mu;
  static Entry tab[kPartialSetSlots] = {};
  const size_t h = (reinterpret_cast<uintptr_t>(workspace) >> 8) % kPartialSetSlots;
  std::lock_guard<std::mutex> lock(mu);
  Entry& e = tab[h];
  if (e.ws != workspace) e = Entry{workspace, 0, {0u, 0u}};
  const int set = e.next;
  *fresh = e.layout[set] != layout;
  e.layout[set] = layout;
  e.next ^= 1;
  return set;
}

// Enqueue the whole step (or, with ratios_only, the log-ratio pass) for validated args.
static int enqueue_verify(const void* x_draft, const void* mu_target, const void* mu_draft,
                          const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d,
                          int dtype, uint64_t seed, const uint64_t* seed_dev, int mode, const int32_t* L_eff,
                          const void* mu_target_bonus, const float* sigma_bonus,
                          int residual_kind, float omega, int32_t* accepted_len, void* y_out,
                          float* log_ratio_out, float* delta_norm_out, uint32_t* status_out,
                          float* chain_aux_out, bool ratios_only, bool timed, bool overlap,
                          void* workspace, cudaStream_t s) {
  const WsLayout w = ws_layout(B, L, d, dtype);
  char* ws = (char*)workspace;
  VerifyArgs A{};
  A.x = x_draft; A.mq = mu_target; A.mp = mu_draft;
  A.mq_bonus = mu_target_bonus; A.sigma_bonus = sigma_bonus;
  A.d = d; A.chunk = w.chunk1; A.y = y_out;
  A.ticket = (unsigned int*)(ws + w.ticket_off);
  A.state = (ChainState*)(ws + w.state_off);
  ScanArgs& S = A.S;
  A.part = (float2*)(ws + w.part_off);
  A.tpart = (uint64_t*)(ws + w.part_off);
  S.part = A.part; S.tpart = nullptr; S.consumed = nullptr; S.tag = 0u; S.fresh_set = false;
  S.C = w.C1; S.sigma = sigma; S.sstride = sigma_stride_b;
  S.B = B; S.L = L; S.L_eff = L_eff; S.seed = seed; S.seed_dev = seed_dev; S.mode = mode;
  S.inv_omega2 = 1.0f / (omega * omega); S.residual_kind = residual_kind;
  S.has_bonus = mu_target_bonus != nullptr; S.ratios_only = ratios_only; S.draw_u = true;
  S.ell_out = log_ratio_out; S.dn_out = delta_norm_out; S.accepted_len = accepted_len;
  S.status_out = status_out; S.aux_out = chain_aux_out;

  cudaEvent_t* tev = (ratios_only || !timed) ? nullptr : timing_slot();
  if (tev) timing_record(tev[0], s);
  const int64_t ng = (d + 3) / 4;
  // Paths (rows in groups of four elements):
  //  - up to kFusedMaxGroups: the fused kernel for a plain call with fewer than
  //    kFusedMaxChains chains; otherwise k_tiles + k_finish (64 threads per chain);
  //  - up to kPipeMaxGroups: k_tiles + k_finish with 256 threads per chain, except
  //    for a plain call with many chains (k_tiles + k_finish and the long-row kernels);
  //  - longer: the fused kernel (or, with many chains or pipelined, k_tiles +
  //    k_finish) without the residual, then k_resid_dot / k_resid_write.
  // A pipelined call launches every one of its kernels to overlap its predecessor.
  overlap = overlap && !ratios_only;
  const bool wide = ng > kFinishMaxGroups && ng <= kPipeMaxGroups && (overlap || B < kManyChainMin);
  const bool many = !ratios_only && (overlap || B >= kFusedMaxChains || wide);
  const bool long_rows = !ratios_only && !wide && ng > (many ? kFinishMaxGroups : kFusedMaxGroups);
  const bool f32 = dtype == SDV_F32;
  cudaError_t e = cudaSuccess;
  if (many) {
    // k_tiles + k_finish: tagged partials in the set after the one this workspace's
    // previous call used, no counters
    // the layout key: the slot count and the set's size (never 0)
    const uint64_t layout = ((uint64_t)B * L * w.C1 << 24) ^ (uint64_t)w.part_set_bytes ^ 1u;
    bool fresh = true;
    char* set = ws + w.part_off + (size_t)next_partial_set(workspace, layout, &fresh) * w.part_set_bytes;
    S.fresh_set = fresh;
    A.tpart = (uint64_t*)set;
    S.part = nullptr;
    S.tpart = A.tpart;
    S.consumed = (uint32_t*)(set + w.cons_off);
    S.tag = next_partial_tag();
  } else if (cudaMemsetAsync(A.ticket, 0, sizeof(unsigned int) * (size_t)B, s) != cudaSuccess) {
    // the fused kernel counts the tiles of each chain from zero
    check_launch();
    return SDV_ECUDA;
  }
  if (many) {
    e = f32 ? launch_tiles<float>(A, B, L, w.vpt1, overlap, s)
            : launch_tiles<__nv_bfloat16>(A, B, L, w.vpt1, overlap, s);
  } else if (long_rows) {
    e = f32 ? launch_verify<float, 0>(A, B, L, w.vpt1, false, s)
            : launch_verify<__nv_bfloat16, 0>(A, B, L, w.vpt1, false, s);
  } else {
    e = f32 ? launch_verify<float, 1>(A, B, L, w.vpt1, overlap, s)
            : launch_verify<__nv_bfloat16, 1>(A, B, L, w.vpt1, overlap, s);
  }
  if (e != cudaSuccess) {
    g_last_cuda_error = (int)e;
    cudaGetLastError();
    return SDV_ECUDA;
  }
  int rc = check_launch();
  if (rc != SDV_OK) return rc;
  if (tev) timing_record(tev[1], s);
  // The kernels after the first of a call are always launched to overlap their
  // predecessor within the call: k_finish starts once every k_tiles CTA has stored
  // its partial (and checks their tags), and the residual kernels wait for their inputs at their start;
  // only the first kernel's overlap with the previous call needs the pipelined contract.
  if (many) {
    if (long_rows)
      e = f32 ? launch_finish<float, 0>(A, B, true, s) : launch_finish<__nv_bfloat16, 0>(A, B, true, s);
    else
      e = f32 ? launch_finish<float, 1>(A, B, true, s) : launch_finish<__nv_bfloat16, 1>(A, B, true, s);
    if (e != cudaSuccess) {
      g_last_cuda_error = (int)e;
      cudaGetLastError();
      return SDV_ECUDA;
    }
    if ((rc = check_launch()) != SDV_OK) return rc;
  }
  if (long_rows) {
    float* part4 = (float*)(ws + w.part4_off);
    e = f32 ? launch_k4<float>(x_draft, mu_target, mu_draft, mu_target_bonus, sigma_bonus, B, L, d, seed, seed_dev,
                               w, A.state, part4, y_out, overlap, true, s)
            : launch_k4<__nv_bfloat16>(x_draft, mu_target, mu_draft, mu_target_bonus, sigma_bonus, B, L, d, seed,
                                       seed_dev, w, A.state, part4, y_out, overlap, true, s);
    if (e != cudaSuccess) {
      g_last_cuda_error = (int)e;
      cudaGetLastError();
      return SDV_ECUDA;
    }
    rc = check_launch();
  }
  if (tev) timing_record(tev[2], s);
  return rc;
}

int verify_ex_impl(const void* x_draft, const void* mu_target, const void* mu_draft,
                        const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d, int dtype,
                        uint64_t seed, const uint64_t* seed_dev, int mode, const int32_t* L_eff,
                        const void* mu_target_bonus, const float* sigma_bonus, int residual_kind,
                        float omega, int32_t* accepted_len, void* y_out, float* log_ratio_out,
                        float* delta_norm_out, uint32_t* status_out, float* chain_aux_out,
                        void* workspace, size_t workspace_bytes, bool timed, void* stream, bool overlap) {
  int rc = validate_window(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype);
  if (rc != SDV_OK) return rc;
  if (mode != SDV_MODE_SAMPLE && mode != SDV_MODE_BLOCK) return SDV_EINVAL;
  if (residual_kind != SDV_RESIDUAL_DECOMPOSITION && residual_kind != SDV_RESIDUAL_REFLECTION)
    return SDV_EINVAL;
  if (residual_kind == SDV_RESIDUAL_REFLECTION && mode != SDV_MODE_SAMPLE) return SDV_EINVAL;
  if (!(omega > 0.f) || !std::isfinite(omega)) return SDV_EINVAL;
  if (!accepted_len || !y_out) return SDV_EINVAL;
  if ((mu_target_bonus == nullptr) != (sigma_bonus == nullptr)) return SDV_EINVAL;
  const size_t es = dtype == SDV_BF16 ? 2 : 4;
  if (!aligned(y_out, es) || !aligned(accepted_len, 4) ||
      (mu_target_bonus && !aligned(mu_target_bonus, es)) || (sigma_bonus && !aligned(sigma_bonus, 4)) ||
      (L_eff && !aligned(L_eff, 4)) || (log_ratio_out && !aligned(log_ratio_out, 4)) ||
      (delta_norm_out && !aligned(delta_norm_out, 4)) || (status_out && !aligned(status_out, 4)) ||
      (chain_aux_out && !aligned(chain_aux_out, 4)) || (seed_dev && !aligned(seed_dev, 8)))
    return SDV_EALIGN;
  const WsLayout w = ws_layout(B, L, d, dtype);
  if (!workspace || workspace_bytes < w.total) return SDV_ENOWORKSPACE;
  if (!aligned(workspace, 256)) return SDV_EALIGN;
  return enqueue_verify(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                        seed_dev, mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                        accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
                        chain_aux_out, false, timed, overlap, workspace, (cudaStream_t)stream);
}

}  // namespace sdv

using namespace sdv;

extern "C" {

const char* sdv_version(void) { return "specdiff-gb300 0.2 (sm_103a)"; }

const char* sdv_strerror(int code) {
  switch (code) {
    case SDV_OK: return "ok";
    case SDV_EINVAL: return "invalid argument";
    case SDV_EALIGN: return "misaligned pointer";
    case SDV_ECUDA: return "CUDA launch failure";
    case SDV_ENOWORKSPACE: return "workspace missing or too small";
    default: return "unknown error";
  }
}

int sdv_last_cuda_error(void) { return g_last_cuda_error; }

size_t sdv_workspace_bytes(int B, int L, int64_t d, int dtype) {
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1 || (dtype != SDV_F32 && dtype != SDV_BF16)) return 0;
  return ws_layout(B, L, d, dtype).total;
}

int sdv_verify_ex(const void* x_draft, const void* mu_target, const void* mu_draft,
                  const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d, int dtype,
                  uint64_t seed, int mode, const int32_t* L_eff, const void* mu_target_bonus,
                  const float* sigma_bonus, int residual_kind, float omega,
                  int32_t* accepted_len, void* y_out, float* log_ratio_out,
                  float* delta_norm_out, uint32_t* status_out, float* chain_aux_out,
                  void* workspace, size_t workspace_bytes, sdv_stream_t stream) {
  return verify_ex_impl(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                        nullptr, mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                        accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
                        chain_aux_out, workspace, workspace_bytes, true, stream, false);
}

int sdv_verify_pipelined(const void* x_draft, const void* mu_target, const void* mu_draft,
                         const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d, int dtype,
                         uint64_t seed, int mode, const int32_t* L_eff, const void* mu_target_bonus,
                         const float* sigma_bonus, int residual_kind, float omega,
                         int32_t* accepted_len, void* y_out, float* log_ratio_out,
                         float* delta_norm_out, uint32_t* status_out, float* chain_aux_out,
                         void* workspace, size_t workspace_bytes, sdv_stream_t stream) {
  return verify_ex_impl(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                        nullptr, mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                        accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
                        chain_aux_out, workspace, workspace_bytes, true, stream, true);
}

int sdv_verify(const void* x_draft, const void* mu_target, const void* mu_draft,
               const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d, int dtype,
               uint64_t seed, int mode, int32_t* accepted_len, void* y_out,
               float* log_ratio_out, float* delta_norm_out, uint32_t* status_out,
               void* workspace, size_t workspace_bytes, sdv_stream_t stream) {
  return sdv_verify_ex(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                       mode, nullptr, nullptr, nullptr, SDV_RESIDUAL_DECOMPOSITION, 1.0f,
                       accepted_len, y_out, log_ratio_out, delta_norm_out, status_out, nullptr,
                       workspace, workspace_bytes, stream);
}

int sdv_log_ratios(const void* x_draft, const void* mu_target, const void* mu_draft,
                   const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d, int dtype,
                   const int32_t* L_eff, float* log_ratio_out, float* delta_norm_out,
                   void* workspace, size_t workspace_bytes, sdv_stream_t stream) {
  int rc = validate_window(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype);
  if (rc != SDV_OK) return rc;
  if (!log_ratio_out || !delta_norm_out) return SDV_EINVAL;
  if (!aligned(log_ratio_out, 4) || !aligned(delta_norm_out, 4) || (L_eff && !aligned(L_eff, 4)))
    return SDV_EALIGN;
  const WsLayout w = ws_layout(B, L, d, dtype);
  if (!workspace || workspace_bytes < w.total) return SDV_ENOWORKSPACE;
  if (!aligned(workspace, 256)) return SDV_EALIGN;
  return enqueue_verify(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, 0,
                        nullptr, SDV_MODE_BLOCK, L_eff, nullptr, nullptr, SDV_RESIDUAL_DECOMPOSITION,
                        1.0f, nullptr, nullptr, log_ratio_out, delta_norm_out, nullptr, nullptr, true,
                        false, false, workspace, (cudaStream_t)stream);
}

int sdv_accept_scan(const float* log_ratio, const float* delta_norm, int B, int L,
                    const int32_t* L_eff, uint64_t seed, int mode, float omega, int32_t* tau_out,
                    float* log_alpha_res_out, sdv_stream_t stream) {
  if (!log_ratio || !delta_norm || !tau_out) return SDV_EINVAL;
  if (B < 1 || L < 1 || L > SDV_MAX_L || B > (1 << 30)) return SDV_EINVAL;
  if (mode != SDV_MODE_SAMPLE && mode != SDV_MODE_BLOCK) return SDV_EINVAL;
  if (!(omega > 0.f) || !std::isfinite(omega)) return SDV_EINVAL;
  if (!aligned(log_ratio, 4) || !aligned(delta_norm, 4) || !aligned(tau_out, 4) ||
      (log_alpha_res_out && !aligned(log_alpha_res_out, 4)) || (L_eff && !aligned(L_eff, 4)))
    return SDV_EALIGN;
  ScanArgs A{};
  A.ell_in = log_ratio; A.dn_in = delta_norm; A.B = B; A.L = L; A.L_eff = L_eff;
  A.seed = seed; A.mode = mode; A.inv_omega2 = 1.0f / (omega * omega);
  A.tau_out = tau_out; A.la_res_out = log_alpha_res_out; A.draw_u = false;
  k_scan<<<(B + kK2Threads / 32 - 1) / (kK2Threads / 32), kK2Threads, 0, (cudaStream_t)stream>>>(A);
  return check_launch();
}

int sdv_usample(const float* delta_norm, const float* log_alpha, const uint32_t* w_bits, int n,
                float* U_out, uint32_t* status_out, sdv_stream_t stream) {
  if (!delta_norm || !log_alpha || !w_bits || !U_out || n < 0) return SDV_EINVAL;
  if (!aligned(delta_norm, 4) || !aligned(log_alpha, 4) || !aligned(w_bits, 4) ||
      !aligned(U_out, 4) || (status_out && !aligned(status_out, 4)))
    return SDV_EALIGN;
  if (n == 0) return SDV_OK;
  k_usample<<<n, kK1Threads, 0, (cudaStream_t)stream>>>(delta_norm, log_alpha, w_bits, n, U_out, status_out);
  return check_launch();
}

int sdv_philox(const uint32_t* ctr, uint64_t seed, int n, uint32_t* out, sdv_stream_t stream) {
  if (!ctr || !out || n < 0) return SDV_EINVAL;
  if (!aligned(ctr, 16) || !aligned(out, 16)) return SDV_EALIGN;
  if (n == 0) return SDV_OK;
  k_philox<<<(n + 255) / 256, 256, 0, (cudaStream_t)stream>>>((const uint4*)ctr, seed, n, (uint4*)out);
  return check_launch();
}

int sdv_normals(uint64_t seed, int B, int64_t d, int stream_id, uint32_t sub, float* out,
                sdv_stream_t stream) {
  if (!out || B < 1 || d < 1 || stream_id < 0) return SDV_EINVAL;
  if (!aligned(out, 4)) return SDV_EALIGN;
  const int64_t n = (int64_t)B * ((d + 3) / 4);
  k_normals<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(seed, B, d, (uint32_t)stream_id, sub, out);
  return check_launch();
}

int sdv_special(int which, const float* z, int n, float* out, sdv_stream_t stream) {
  if (!z || !out || n < 0 || which < 0 || which > 2) return SDV_EINVAL;
  if (!aligned(z, 4) || !aligned(out, 4)) return SDV_EALIGN;
  if (n == 0) return SDV_OK;
  k_special<<<(n + 255) / 256, 256, 0, (cudaStream_t)stream>>>(which, z, n, out);
  return check_launch();
}

int sdv_timing_enable(int slots) {
  if (slots < 0 || slots > (1 << 20)) return SDV_EINVAL;
  timing_destroy();
  if (slots == 0) return SDV_OK;
  g_timing.ev.resize(3 * (size_t)slots);
  for (auto& e : g_timing.ev) {
    if (cudaEventCreate(&e) != cudaSuccess) {
      g_last_cuda_error = (int)cudaGetLastError();
      g_timing.ev.clear();
      return SDV_ECUDA;
    }
  }
  g_timing.slots = slots;
  return SDV_OK;
}

int sdv_timing_stride(int every) {
  if (every < 1) return SDV_EINVAL;
  g_timing.stride = every;
  g_timing.calls = 0;
  return SDV_OK;
}

int sdv_timing_read(int n_calls, float* ms3) {
  if (!ms3 || g_timing.slots == 0 || n_calls < 1 || n_calls > g_timing.slots ||
      n_calls > g_timing.next)
    return SDV_EINVAL;
  double acc[3] = {0, 0, 0};
  for (int i = 0; i < n_calls; ++i) {
    const int s = (int)((g_timing.next - 1 - i) % g_timing.slots);
    cudaEvent_t* e = &g_timing.ev[3 * (size_t)s];
    if (cudaEventSynchronize(e[2]) != cudaSuccess) {
      g_last_cuda_error = (int)cudaGetLastError();
      return SDV_ECUDA;
    }
    for (int k = 0; k < 2; ++k) {
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, e[k], e[k + 1]) != cudaSuccess) {
        g_last_cuda_error = (int)cudaGetLastError();
        return SDV_ECUDA;
      }
      acc[k] += ms;
    }
  }
  for (int k = 0; k < 3; ++k) ms3[k] = (float)acc[k];
  return SDV_OK;
}

}  // extern "C"
