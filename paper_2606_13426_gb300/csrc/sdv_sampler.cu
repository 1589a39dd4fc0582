// sdv_sampler.cu - end-to-end speculative diffusion sampler on an analytic Gaussian-
// mixture target (sm_103a): the target-mean kernel, the Free / Frozen drafter, the
// round update, the plain Euler-Maruyama chain, and the native round loop.
//
// Model (Eq. forward-process / backward-process / target-distribution):
//   VP schedule beta(t) = beta_min + (beta_max - beta_min) t, f = -beta/2, g = sqrt(beta),
//   abar_t = exp(-int_0^t beta); q_t = sum_c w_c N(sqrt(abar) mu_c, v I), v = abar s^2 + 1 - abar;
//   score s_t(x) = sum_c r_c (sqrt(abar) mu_c - x) / v, r = softmax(log w_c - |x - sqrt(abar) mu_c|^2/(2v));
//   m^q_k(y) = y + delta [beta/2 y + (1 + eps^2)/2 beta s(y)] at forward time 1 - t_k (floored),
//   sigma_k = sqrt(delta) eps sqrt(beta).
// Drafter (Eq. frozen-draft-drift and the Free drafter of Sec. "Self-Speculative Drafter"):
//   m^p = yhat + delta [beta/2 yhat + (1 + eps^2)/2 beta s_cache], yhat' = m^p + sigma G.
// Round (Alg. full-block-verification): draft gamma_k = min(L, K - k) steps, target means
// at yhat_k .. yhat_{k+gamma_k}, sdv_verify_ex, then advance k by tau (no bonus step when
// the window reaches K), keep the score at the next round's start state.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "sdv_device.cuh"
#include "sdv_host.h"

namespace sdv {

struct Sched {
  int K;
  float churn, beta_min, beta_max, t_floor, delta;
  __device__ __forceinline__ float tfwd(int k) const {
    return fmaxf((float)(K - k) / (float)K, t_floor);  // 1 - t_k, t_k = k / K
  }
  __device__ __forceinline__ float beta(float tf) const { return beta_min + (beta_max - beta_min) * tf; }
  __device__ __forceinline__ float abar(float tf) const {
    return expf(-(beta_min * tf + 0.5f * (beta_max - beta_min) * tf * tf));
  }
  __device__ __forceinline__ float sigma(int k) const {
    return sqrtf(delta) * churn * sqrtf(beta(tfwd(k)));
  }
};

struct Gmm {
  const float* means;  // [C, d]
  const float* log_w;  // [C]
  int C;
  float comp_var;
};

__host__ __device__ __forceinline__ uint64_t splitmix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Seed of round r: the (r+1)-th SplitMix64 output of a stream started at `seed`.
__host__ __device__ __forceinline__ uint64_t round_seed(uint64_t seed, int r) {
  return splitmix64(seed + (uint64_t)(r + 1) * 0x9E3779B97F4A7C15ull);
}

constexpr int kGmmThreads = 256;              // 8 warps, one state row per warp at a time
constexpr int kGmmWarps = kGmmThreads / 32;
constexpr size_t kGmmSmemCap = 96 * 1024;     // stage the means in shared memory up to this size

// One state row of a target call: state z at generative step k; outputs mq / score
// (either may be null; z may alias mq: each lane reads a group of four elements
// before it writes it, and no other lane touches that group).  add_sigma != 0 adds
// sigma * G to mq (Philox stream noise_stream of chain `chain`, sub-counter k; one
// Philox block per group of four).
struct GmmRow {
  const float* z;
  float* mq;
  float* score;
  int k;
  uint32_t chain;
  float add_sigma;
};

// m^q and the score for nr <= RB rows by one warp: every mean group read from `mu`
// (shared or global memory) serves all nr rows.  nr is warp-uniform.
// VEC: d % 4 == 0 and 16-byte aligned rows (float4 accesses); MAXC >= C components.
template <int MAXC, bool VEC, int RB>
__device__ __forceinline__ void gmm_rows_warp(const GmmRow (&R)[RB], int nr, int64_t d, const Sched& S,
                                              const Gmm& G, const float* mu, uint64_t noise_seed,
                                              uint32_t noise_stream) {
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int C = G.C;
  float sab[RB], v[RB], inv_v[RB], be[RB];
#pragma unroll
  for (int q = 0; q < RB; ++q) {
    const float tf = S.tfwd(R[q].k);
    const float ab = S.abar(tf);
    sab[q] = sqrtf(ab);
    v[q] = ab * G.comp_var + 1.0f - ab;
    inv_v[q] = 1.0f / v[q];
    be[q] = S.beta(tf);
  }
  const float cst = 0.5f * (1.0f + S.churn * S.churn);
  const int64_t ng = (d + 3) / 4;
  // groups in flight per lane: RB rows, times the unrolled sweeps
  constexpr int kU = RB >= 3 ? 1 : (RB == 2 ? 2 : 4);
  auto load_group = [&](const float* p, int64_t gi, float (&f)[4]) {
    if (VEC) {
      const float4 t = *reinterpret_cast<const float4*>(p + 4 * gi);
      f[0] = t.x; f[1] = t.y; f[2] = t.z; f[3] = t.w;
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) f[e] = (4 * gi + e < d) ? p[4 * gi + e] : 0.f;
    }
  };
  // pass 1: squared distances to the scaled centres sqrt(abar) mu_c
  float acc[RB][MAXC];
#pragma unroll
  for (int q = 0; q < RB; ++q)
#pragma unroll
    for (int c = 0; c < MAXC; ++c) acc[q][c] = 0.f;
#pragma unroll kU
  for (int64_t gi = lane; gi < ng; gi += 32) {
    float zf[RB][4];
#pragma unroll
    for (int q = 0; q < RB; ++q) {
      if (q < nr) load_group(R[q].z, gi, zf[q]);
    }
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
      if (c < C) {
        float mf[4];
        load_group(mu + (int64_t)c * d, gi, mf);
#pragma unroll
        for (int q = 0; q < RB; ++q) {
          if (q < nr) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              // the tail check is only needed without VEC (d % 4 == 0 otherwise)
              const float df = (VEC || 4 * gi + e < d) ? zf[q][e] - sab[q] * mf[e] : 0.f;
              acc[q][c] = fmaf(df, df, acc[q][c]);
            }
          }
        }
      }
    }
  }
  // responsibilities r_c = softmax(log w_c - d2_c / (2 v)), identical in every lane;
  // acc becomes r, w_sc folds the softmax normaliser and sqrt(abar)
  float w_sc[RB];
#pragma unroll
  for (int q = 0; q < RB; ++q) {
    float mx = -INFINITY;
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
      float a = acc[q][c];
      if (c < C) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(FULL, a, o);
      }
      acc[q][c] = (c < C) ? __ldg(G.log_w + c) - 0.5f * a * inv_v[q] : -INFINITY;
      mx = fmaxf(mx, acc[q][c]);
    }
    float den = 0.f;
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
      acc[q][c] = (c < C) ? expf(acc[q][c] - mx) : 0.f;
      den += acc[q][c];
    }
    w_sc[q] = sab[q] / den;
  }
  // pass 2: score and target mean
#pragma unroll kU
  for (int64_t gi = lane; gi < ng; gi += 32) {
    float zf[RB][4], wsum[RB][4];
#pragma unroll
    for (int q = 0; q < RB; ++q) {
      if (q < nr) load_group(R[q].z, gi, zf[q]);
#pragma unroll
      for (int e = 0; e < 4; ++e) wsum[q][e] = 0.f;
    }
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
      if (c < C) {
        float mf[4];
        load_group(mu + (int64_t)c * d, gi, mf);
#pragma unroll
        for (int q = 0; q < RB; ++q)
#pragma unroll
          for (int e = 0; e < 4; ++e) wsum[q][e] = fmaf(acc[q][c], mf[e], wsum[q][e]);
      }
    }
#pragma unroll
    for (int q = 0; q < RB; ++q) {
      if (q < nr) {
        float G4[4] = {0.f, 0.f, 0.f, 0.f};
        if (R[q].add_sigma != 0.f) {
          const float4 n4 = normals4(noise_seed, R[q].chain, (uint32_t)gi, noise_stream, (uint32_t)R[q].k);
          G4[0] = n4.x; G4[1] = n4.y; G4[2] = n4.z; G4[3] = n4.w;
        }
        float sc[4], m[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          sc[e] = (w_sc[q] * wsum[q][e] - zf[q][e]) * inv_v[q];
          m[e] = zf[q][e] + S.delta * (0.5f * be[q] * zf[q][e] + cst * be[q] * sc[e]) + R[q].add_sigma * G4[e];
        }
        float* score = R[q].score;
        float* mq = R[q].mq;
        if (VEC) {
          if (score) *reinterpret_cast<float4*>(score + 4 * gi) = make_float4(sc[0], sc[1], sc[2], sc[3]);
          if (mq) *reinterpret_cast<float4*>(mq + 4 * gi) = make_float4(m[0], m[1], m[2], m[3]);
        } else {
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            if (4 * gi + e < d) {
              if (score) score[4 * gi + e] = sc[e];
              if (mq) mq[4 * gi + e] = m[e];
            }
          }
        }
      }
    }
  }
}

// Stage the means in dynamic shared memory (when the launch gave it room); returns the
// pointer the warps read from.
__device__ __forceinline__ const float* stage_means(const Gmm& G, int64_t d, bool use_smem) {
  extern __shared__ float mu_s[];
  if (!use_smem) return G.means;
  const int64_t n = (int64_t)G.C * d;
  for (int64_t i = threadIdx.x; i < n; i += blockDim.x) mu_s[i] = __ldg(G.means + i);
  __syncthreads();
  return mu_s;
}

// Target means and scores for rows of a [n, d] array at steps k[row]; one warp per row;
// rows whose window mask (if given) is 0 are skipped.
template <int MAXC, bool VEC>
__global__ void __launch_bounds__(kGmmThreads)
k_gmm_rows(const float* __restrict__ states, const int32_t* __restrict__ k, const int32_t* __restrict__ mask,
           int n, int64_t d, Sched S, Gmm G, bool use_smem, float* mq, float* score) {
  const float* mu = stage_means(G, d, use_smem);
  const int warp = threadIdx.x >> 5;
  for (int row = blockIdx.x * kGmmWarps + warp; row < n; row += gridDim.x * kGmmWarps) {
    if (mask && mask[row] == 0) continue;
    const int64_t o = (int64_t)row * d;
    const GmmRow R[1] = {{states + o, mq ? mq + o : nullptr, score ? score + o : nullptr, k[row], 0u, 0.f}};
    gmm_rows_warp<MAXC, VEC, 1>(R, 1, d, S, G, mu, 0, 0);
  }
}

// Rows of a round's parallel target call per warp.
template <int MAXC> struct RoundRows { static constexpr int value = MAXC <= 8 ? 3 : 1; };

// Parallel target call of a round.  Row (b, j), j = 0 .. gamma_b, is state y[b]
// (j = 0) or x_draft[b, j-1] at step k[b] + j; its mean goes to mu_target[b, j]
// (j < gamma_b) or mu_bonus[b] (j = gamma_b, with sigma_bonus[b] = sigma_{k+gamma}),
// its score to sc_all[b, j].  The B (L+1) row slots are dealt to warps RB at a time
// (slots past gamma_b are skipped), grid-stride over persistent CTAs.
template <int MAXC, bool VEC>
__global__ void __launch_bounds__(kGmmThreads, 2)
k_round_target(const float* __restrict__ y, const float* __restrict__ x_draft,
               const int32_t* __restrict__ kk, const int32_t* __restrict__ gam, int B, int L, int64_t d,
               Sched S, Gmm G, bool use_smem, float* mu_target, float* mu_bonus, float* sigma_bonus,
               float* sc_all) {
  constexpr int RB = RoundRows<MAXC>::value;
  const float* mu = stage_means(G, d, use_smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t slots = (int64_t)B * (L + 1);
  for (int64_t r0 = ((int64_t)blockIdx.x * kGmmWarps + warp) * RB; r0 < slots;
       r0 += (int64_t)gridDim.x * kGmmWarps * RB) {
    GmmRow R[RB];
    int nr = 0;
#pragma unroll
    for (int q = 0; q < RB; ++q) {
      R[q] = GmmRow{nullptr, nullptr, nullptr, 0, 0u, 0.f};
      const int64_t slot = r0 + q;
      if (slot >= slots) continue;
      const int b = (int)(slot / (L + 1));
      const int j = (int)(slot - (int64_t)b * (L + 1));
      const int g = gam[b];
      if (j > g || g == 0) continue;
      const int kb = kk[b];
      GmmRow row;
      row.z = (j == 0) ? y + (int64_t)b * d : x_draft + ((int64_t)b * L + j - 1) * d;
      row.mq = (j < g) ? mu_target + ((int64_t)b * L + j) * d : mu_bonus + (int64_t)b * d;
      row.score = sc_all + ((int64_t)b * (L + 1) + j) * d;
      row.k = kb + j;
      row.chain = 0u;
      row.add_sigma = 0.f;
      if (j == g && lane == 0) sigma_bonus[b] = S.sigma(kb + g);
      // compact the live rows to the front (q is a compile-time index after unrolling)
#pragma unroll
      for (int t = 0; t < RB; ++t)
        if (t == nr) R[t] = row;
      ++nr;
    }
    if (nr > 0) gmm_rows_warp<MAXC, VEC, RB>(R, nr, d, S, G, mu, 0, 0);
  }
}

// Row slots of a round's target call, shared by the target-call kernels: slot
// (b, j), j = 0 .. L, is live when j <= gamma_b (and gamma_b > 0).
struct RoundRow {
  const float* z;
  float* mq;
  float* score;
  int k;
  bool live;
};

__device__ __forceinline__ RoundRow round_row(int64_t slot, int64_t slots, const float* y, const float* x_draft,
                                              const int32_t* kk, const int32_t* gam, int L, int64_t d,
                                              const Sched& S, float* mu_target, float* mu_bonus,
                                              float* sigma_bonus, float* sc_all, bool write_sigma) {
  RoundRow R{nullptr, nullptr, nullptr, 0, false};
  if (slot >= slots) return R;
  const int b = (int)(slot / (L + 1));
  const int j = (int)(slot - (int64_t)b * (L + 1));
  const int g = gam[b];
  if (j > g || g == 0) return R;
  const int kb = kk[b];
  R.z = (j == 0) ? y + (int64_t)b * d : x_draft + ((int64_t)b * L + j - 1) * d;
  R.mq = (j < g) ? mu_target + ((int64_t)b * L + j) * d : mu_bonus + (int64_t)b * d;
  R.score = sc_all + ((int64_t)b * (L + 1) + j) * d;
  R.k = kb + j;
  R.live = true;
  if (j == g && write_sigma) sigma_bonus[b] = S.sigma(kb + g);
  return R;
}

// Resident CTAs per SM k_round_target_reg is built for (its register budget).
constexpr int round_reg_blocks(int maxc) { return maxc <= 8 ? 3 : 2; }

// Parallel target call of a round for rows of up to 4 kGmmThreads elements
// (d % 4 == 0, 16-byte aligned rows): each thread owns one group of four elements
// and holds that group of every mean in registers for the whole kernel; a CTA takes
// RB = 32 / MAXC row slots at a time (grid-stride), keeps each row's group in
// registers across both passes, and reduces the RB x MAXC squared distances with one
// warp reduce-scatter (value v ends in lane v) and one pass over the warps.  Warp 0
// resolves the next batch's rows and their schedule constants into shared memory
// (three buffers: the batch being written, the one being finished and the next),
// and every thread loads the next batch's states while this batch finishes.
template <int MAXC>
__global__ void __launch_bounds__(kGmmThreads, round_reg_blocks(MAXC))
k_round_target_reg(const float* __restrict__ y, const float* __restrict__ x_draft,
                   const int32_t* __restrict__ kk, const int32_t* __restrict__ gam, int B, int L, int64_t d,
                   Sched S, Gmm G, float* mu_target, float* mu_bonus, float* sigma_bonus, float* sc_all) {
  constexpr int RB = 32 / MAXC;
  constexpr int NV = RB * MAXC;  // 32
  struct RowC {
    const float* z;
    float* mq;
    float* score;
    float sab, inv_v, be;
    int live;
  };
  __shared__ float red[kGmmWarps][NV];
  __shared__ float resp[RB][MAXC];
  __shared__ float wsc[RB];
  __shared__ RowC rows_s[3][RB];
  const unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int C = G.C;
  const int64_t ng = d / 4;
  const bool own = tid < ng;  // this thread's group exists
  const int64_t slots = (int64_t)B * (L + 1);
  const int64_t stride = (int64_t)gridDim.x * RB;
  // warp 0, lane r < RB: row slot s + r -> rows_s[buf][r]
  auto resolve = [&](int64_t s, int buf) {
    if (warp == 0 && lane < RB) {
      const RoundRow R = round_row(s + lane, slots, y, x_draft, kk, gam, L, d, S, mu_target, mu_bonus,
                                   sigma_bonus, sc_all, true);
      RowC rc;
      rc.z = R.z; rc.mq = R.mq; rc.score = R.score; rc.live = R.live ? 1 : 0;
      const float tf = S.tfwd(R.k);
      const float ab = S.abar(tf);
      rc.sab = sqrtf(ab);
      rc.inv_v = 1.0f / (ab * G.comp_var + 1.0f - ab);
      rc.be = S.beta(tf);
      rows_s[buf][lane] = rc;
    }
  };
  float4 m4[MAXC];
#pragma unroll
  for (int c = 0; c < MAXC; ++c)
    m4[c] = (own && c < C) ? __ldg(reinterpret_cast<const float4*>(G.means + (int64_t)c * d) + tid)
                           : make_float4(0.f, 0.f, 0.f, 0.f);
  const float cst = 0.5f * (1.0f + S.churn * S.churn);
  int64_t s0 = (int64_t)blockIdx.x * RB;
  int cur = 0;
  resolve(s0, cur);
  __syncthreads();
  float4 z[RB];
#pragma unroll
  for (int r = 0; r < RB; ++r)
    z[r] = (rows_s[cur][r].live && own) ? *(reinterpret_cast<const float4*>(rows_s[cur][r].z) + tid)
                                        : make_float4(0.f, 0.f, 0.f, 0.f);
  for (; s0 < slots; s0 += stride) {
    const int nxt = cur == 2 ? 0 : cur + 1;
    const RowC* R = rows_s[cur];
    // pass 1: this thread's share of |z_r - sqrt(abar_r) mu_c|^2
    float v[NV];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const float zf[4] = {z[r].x, z[r].y, z[r].z, z[r].w};
#pragma unroll
      for (int c = 0; c < MAXC; ++c) {
        const float mf[4] = {m4[c].x, m4[c].y, m4[c].z, m4[c].w};
        float a = 0.f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float df = zf[e] - R[r].sab * mf[e];
          a = fmaf(df, df, a);
        }
        v[r * MAXC + c] = a;
      }
    }
    // warp reduce-scatter: after the halving steps lane l holds the warp sum of value l
#pragma unroll
    for (int h = NV / 2; h >= 1; h >>= 1) {
      const bool up = (lane & h) != 0;
#pragma unroll
      for (int k = 0; k < h; ++k) {
        const float send = up ? v[k] : v[k + h];
        const float keep = up ? v[k + h] : v[k];
        v[k] = keep + __shfl_xor_sync(FULL, send, h);
      }
    }
    red[warp][lane] = v[0];
    resolve(s0 + stride, nxt);  // last read two batches ago, before this batch's first barrier
    __syncthreads();
    // the next batch's states, in flight while this batch finishes
    float4 zn[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r)
      zn[r] = (rows_s[nxt][r].live && own) ? *(reinterpret_cast<const float4*>(rows_s[nxt][r].z) + tid)
                                           : make_float4(0.f, 0.f, 0.f, 0.f);
    if (warp == 0) {
      // responsibilities r_c = softmax(log w_c - d2_c / (2 v)) over each row's MAXC lanes
      float t = 0.f;
#pragma unroll
      for (int w = 0; w < kGmmWarps; ++w) t += red[w][lane];
      const int r = lane / MAXC, c = lane - r * MAXC;
      float ivr = R[0].inv_v, sabr = R[0].sab;
#pragma unroll
      for (int q = 1; q < RB; ++q) {
        ivr = (r == q) ? R[q].inv_v : ivr;
        sabr = (r == q) ? R[q].sab : sabr;
      }
      const float a = (c < C) ? __ldg(G.log_w + c) - 0.5f * t * ivr : -INFINITY;
      float mx = a;
#pragma unroll
      for (int o = MAXC / 2; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(FULL, mx, o));
      const float ex = (c < C) ? expf(a - mx) : 0.f;
      float den = ex;
#pragma unroll
      for (int o = MAXC / 2; o >= 1; o >>= 1) den += __shfl_xor_sync(FULL, den, o);
      resp[r][c] = ex;
      if (c == 0) wsc[r] = sabr / den;  // folds the softmax normaliser and sqrt(abar)
    }
    __syncthreads();
    // pass 2: score and target mean of this thread's group
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      if (R[r].live && own) {
        float ws[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c = 0; c < MAXC; ++c) {
          const float rc = resp[r][c];
          ws[0] = fmaf(rc, m4[c].x, ws[0]);
          ws[1] = fmaf(rc, m4[c].y, ws[1]);
          ws[2] = fmaf(rc, m4[c].z, ws[2]);
          ws[3] = fmaf(rc, m4[c].w, ws[3]);
        }
        const float w = wsc[r];
        const float zf[4] = {z[r].x, z[r].y, z[r].z, z[r].w};
        float sc[4], m[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          sc[e] = (w * ws[e] - zf[e]) * R[r].inv_v;
          m[e] = zf[e] + S.delta * (0.5f * R[r].be * zf[e] + cst * R[r].be * sc[e]);
        }
        reinterpret_cast<float4*>(R[r].score)[tid] = make_float4(sc[0], sc[1], sc[2], sc[3]);
        reinterpret_cast<float4*>(R[r].mq)[tid] = make_float4(m[0], m[1], m[2], m[3]);
      }
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) z[r] = zn[r];
    cur = nxt;
  }
}

// Free / Frozen drafter: gamma_b elementwise steps from y[b] with the cached score.
// One thread per group of four elements; VEC: d % 4 == 0 and 16-byte aligned rows
// (float4 loads and stores).  The Philox draws do not depend on the state, so the
// unrolled step loop overlaps the next step's draws with this step's stores.
template <bool VEC>
__global__ void __launch_bounds__(256)
k_draft(const float* __restrict__ y, const float* __restrict__ s_cache, const int32_t* __restrict__ kk,
        const int32_t* __restrict__ gam, int B, int L, int64_t d, Sched S, uint64_t seed_v,
        const uint64_t* __restrict__ seed_dev, float* __restrict__ x_draft, float* __restrict__ mu_draft,
        float* __restrict__ sigma) {
  const int64_t ng = (d + 3) / 4;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * ng) return;
  const int b = (int)(t / ng);
  const int64_t gi = t - (int64_t)b * ng;
  const int g = gam[b];
  if (g == 0) return;
  const uint64_t seed = seed_dev ? *seed_dev : seed_v;
  const int k = kk[b];
  const float cst = 0.5f * (1.0f + S.churn * S.churn);
  const int64_t i0 = 4 * gi;
  float cur[4], sc[4];
  if (VEC) {
    const float4 a = *reinterpret_cast<const float4*>(y + (int64_t)b * d + i0);
    const float4 c = *reinterpret_cast<const float4*>(s_cache + (int64_t)b * d + i0);
    cur[0] = a.x; cur[1] = a.y; cur[2] = a.z; cur[3] = a.w;
    sc[0] = c.x; sc[1] = c.y; sc[2] = c.z; sc[3] = c.w;
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      cur[q] = (i0 + q < d) ? y[(int64_t)b * d + i0 + q] : 0.f;
      sc[q] = (i0 + q < d) ? s_cache[(int64_t)b * d + i0 + q] : 0.f;
    }
  }
#pragma unroll 4
  for (int step = 1; step <= g; ++step) {
    const int kc = k + step - 1;
    const float be = S.beta(S.tfwd(kc));
    const float sg = S.sigma(kc);
    const float4 n4 = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamDraft, (uint32_t)(step - 1));
    const float nz[4] = {n4.x, n4.y, n4.z, n4.w};
    const int64_t row = ((int64_t)b * L + step - 1) * d;
    float m[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      m[q] = cur[q] + S.delta * (0.5f * be * cur[q] + cst * be * sc[q]);
      cur[q] = m[q] + sg * nz[q];
    }
    if (VEC) {
      *reinterpret_cast<float4*>(mu_draft + row + i0) = make_float4(m[0], m[1], m[2], m[3]);
      *reinterpret_cast<float4*>(x_draft + row + i0) = make_float4(cur[0], cur[1], cur[2], cur[3]);
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (i0 + q < d) {
          mu_draft[row + i0 + q] = m[q];
          x_draft[row + i0 + q] = cur[q];
        }
      }
    }
    if (gi == 0) sigma[(int64_t)b * L + step - 1] = sg;
  }
}

// Device-resident state of the round loop: the seed of the current round, the rounds
// run, and the chains k_round_update found still active in the current round.
struct SamplerCtl {
  uint64_t seed_r;
  int32_t r;
  uint32_t active;
  uint32_t done;  // k_round_update CTAs that finished this round
};

// End of a round (the k_round_update CTA holding the round's last ticket): advance the
// round counter and seed, reset the round's counters, and (inside the round graph)
// keep the loop going while a chain is active and fewer than max_rounds rounds ran.
__device__ __forceinline__ void close_round(SamplerCtl* ctl, uint64_t seed, int max_rounds, int in_loop,
                                            cudaGraphConditionalHandle h) {
  const int r = ctl->r + 1;
  ctl->r = r;
  ctl->seed_r = round_seed(seed, r);
  const bool more = ctl->active != 0u && r < max_rounds;
  ctl->active = 0u;
  ctl->done = 0u;
  if (in_loop) cudaGraphSetConditional(h, more ? 1u : 0u);
}

// Round bookkeeping, one warp per chain and kUpdateChains chains per CTA: the emitted
// state, the score cache, k, the next window length and the statistics; each CTA adds
// its chains that remain active with one atomic, and the CTA holding the round's last
// ticket closes the round (close_round).  (One CTA per chain made 1024 same-address
// atomics per round, and that serialisation cost most of the kernel's time.)
// VEC: d % 4 == 0 (workspace rows are then 16-byte aligned).
constexpr int kUpdateChains = 8;

template <bool VEC>
__global__ void __launch_bounds__(32 * kUpdateChains)
k_round_update(const int32_t* __restrict__ acc, const float* __restrict__ y_out,
               const float* __restrict__ x_draft, const float* __restrict__ sc_all, int B, int L, int64_t d,
               int K, float* y, float* s_cache, int32_t* kk, int32_t* gam, int32_t* rounds,
               int32_t* tau_sum, SamplerCtl* ctl, uint64_t seed, int max_rounds, int in_loop,
               cudaGraphConditionalHandle h) {
  __shared__ unsigned int act_s[kUpdateChains];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * kUpdateChains + w;
  unsigned int act = 0u;
  if (b < B) {
    const int g = gam[b];
    const int k = kk[b];
    __syncwarp();  // every lane has read k and gamma before lane 0 updates them
    const int tau = acc[b] + 1;
    if (g > 0) {
      const bool end = (tau == g + 1) && (k + g >= K);  // no bonus step past the end of sampling
      const float* ysrc = end ? x_draft + ((int64_t)b * L + g - 1) * d : y_out + (int64_t)b * d;
      const float* ssrc = sc_all + ((int64_t)b * (L + 1) + min(tau, g)) * d;
      if (VEC) {
        const float4* ys4 = reinterpret_cast<const float4*>(ysrc);
        const float4* ss4 = reinterpret_cast<const float4*>(ssrc);
        float4* yd4 = reinterpret_cast<float4*>(y + (int64_t)b * d);
        float4* sd4 = reinterpret_cast<float4*>(s_cache + (int64_t)b * d);
        for (int64_t i = lane; i < d / 4; i += 32) {
          yd4[i] = ys4[i];
          sd4[i] = ss4[i];
        }
      } else {
        for (int64_t i = lane; i < d; i += 32) {
          y[(int64_t)b * d + i] = ysrc[i];
          s_cache[(int64_t)b * d + i] = ssrc[i];
        }
      }
      if (lane == 0) {
        const int kn = min(k + tau, K);
        kk[b] = kn;
        const int gn = kn < K ? min(L, K - kn) : 0;
        gam[b] = gn;
        rounds[b] += 1;
        tau_sum[b] += tau;
        act = gn > 0 ? 1u : 0u;
      }
    }
  }
  if (lane == 0) act_s[w] = act;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int n = 0u;
#pragma unroll
    for (int i = 0; i < kUpdateChains; ++i) n += act_s[i];
    if (n) atomicAdd(&ctl->active, n);
    if (ticket_acq_rel(&ctl->done) == gridDim.x - 1) close_round(ctl, seed, max_rounds, in_loop, h);
  }
}

__global__ void __launch_bounds__(256)
k_sampler_init(int B, int L, int64_t d, int K, uint64_t seed, float* y, int32_t* kk, int32_t* gam,
               int32_t* rounds, int32_t* tau_sum, SamplerCtl* ctl) {
  const int64_t ng = (d + 3) / 4;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * ng) return;
  const int b = (int)(t / ng);
  const int64_t gi = t - (int64_t)b * ng;
  const float4 n4 = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamInit, 0u);
  const float nz[4] = {n4.x, n4.y, n4.z, n4.w};
#pragma unroll
  for (int q = 0; q < 4; ++q)
    if (4 * gi + q < d) y[(int64_t)b * d + 4 * gi + q] = nz[q];
  if (t == 0 && ctl != nullptr) {
    ctl->seed_r = round_seed(seed, 0);
    ctl->r = 0;
    ctl->active = 0u;
    ctl->done = 0u;
  }
  if (gi == 0 && kk != nullptr) {
    kk[b] = 0;
    gam[b] = min(L, K);
    rounds[b] = 0;
    tau_sum[b] = 0;
  }
}

// One plain Euler-Maruyama step for every chain, in place: y <- m^q_k(y) + sigma_k G_k;
// one warp per chain.
template <int MAXC, bool VEC>
__global__ void __launch_bounds__(kGmmThreads)
k_em_step(float* y, int B, int64_t d, int k, Sched S, Gmm G, bool use_smem, uint64_t seed) {
  const float* mu = stage_means(G, d, use_smem);
  const int warp = threadIdx.x >> 5;
  for (int b = blockIdx.x * kGmmWarps + warp; b < B; b += gridDim.x * kGmmWarps) {
    float* row = y + (int64_t)b * d;
    const GmmRow R[1] = {{row, row, nullptr, k, (uint32_t)b, S.sigma(k)}};
    gmm_rows_warp<MAXC, VEC, 1>(R, 1, d, S, G, mu, seed, kStreamEM);
  }
}

// Launch geometry of the one-warp-per-row kernels: dynamic shared memory for the means
// when they fit, the component bound, vector accesses, and the grid for n rows.
struct GmmLaunch {
  bool smem;
  size_t smem_bytes;
  bool vec;
  int maxc;
};

template <int MAXC, bool VEC>
static void gmm_set_smem(size_t bytes) {
  cudaFuncSetAttribute(k_gmm_rows<MAXC, VEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  cudaFuncSetAttribute(k_round_target<MAXC, VEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  cudaFuncSetAttribute(k_em_step<MAXC, VEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

// rows_aligned: every state / output row the kernel touches starts on a 16-byte boundary
static GmmLaunch gmm_launch(int C, int64_t d, const void* means, bool rows_aligned) {
  GmmLaunch g{};
  const size_t bytes = (size_t)C * (size_t)d * sizeof(float);
  g.smem = bytes <= kGmmSmemCap;
  g.smem_bytes = g.smem ? bytes : 0;
  g.vec = (d % 4 == 0) && (reinterpret_cast<uintptr_t>(means) % 16 == 0) && rows_aligned;
  g.maxc = C <= 8 ? 8 : 16;
  if (g.smem_bytes > 48 * 1024) {
    if (g.maxc == 8) { gmm_set_smem<8, true>(g.smem_bytes); gmm_set_smem<8, false>(g.smem_bytes); }
    else { gmm_set_smem<16, true>(g.smem_bytes); gmm_set_smem<16, false>(g.smem_bytes); }
  }
  return g;
}

static unsigned rows_grid(int n) { return (unsigned)std::max(1, (n + kGmmWarps - 1) / kGmmWarps); }

static int sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  if (cache[dev] == 0) {
    int n = 0;
    cache[dev] = (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0) ? n : 152;
  }
  return cache[dev];
}

// Grid of k_round_target: one warp per RB row slots, at most four CTAs per SM (each
// CTA stages the means once and strides over its share of the slots).
static unsigned round_target_grid(const GmmLaunch& gl, int B, int L) {
  const int64_t rb = gl.maxc <= 8 ? RoundRows<8>::value : RoundRows<16>::value;
  const int64_t need = ((int64_t)B * (L + 1) + kGmmWarps * rb - 1) / (kGmmWarps * rb);
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(need, 4 * (int64_t)sm_count()));
}

// Rows of up to 4 kGmmThreads elements with 16-byte aligned rows and means take the
// register-resident k_round_target_reg (grid-stride over its resident CTAs); others
// the shared-memory k_round_target.
static bool round_target_reg(const GmmLaunch& gl, int64_t d) { return gl.vec && d <= 4 * kGmmThreads; }

static unsigned round_target_reg_grid(const GmmLaunch& gl, int B, int L) {
  const int64_t rb = 32 / (gl.maxc <= 8 ? 8 : 16);
  const int64_t need = ((int64_t)B * (L + 1) + rb - 1) / rb;
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(need, round_reg_blocks(gl.maxc) * (int64_t)sm_count()));
}

#define SDV_GMM_DISPATCH(GL, KERNEL, GRID, STREAM, ...)                                          \
  do {                                                                                          \
    if ((GL).maxc == 8) {                                                                       \
      if ((GL).vec) KERNEL<8, true><<<GRID, kGmmThreads, (GL).smem_bytes, STREAM>>>(__VA_ARGS__);  \
      else KERNEL<8, false><<<GRID, kGmmThreads, (GL).smem_bytes, STREAM>>>(__VA_ARGS__);          \
    } else {                                                                                    \
      if ((GL).vec) KERNEL<16, true><<<GRID, kGmmThreads, (GL).smem_bytes, STREAM>>>(__VA_ARGS__); \
      else KERNEL<16, false><<<GRID, kGmmThreads, (GL).smem_bytes, STREAM>>>(__VA_ARGS__);         \
    }                                                                                           \
  } while (0)

static int launch_check() {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error((int)e);
    return SDV_ECUDA;
  }
  return SDV_OK;
}

static bool valid_sched(int K, float churn, float bmin, float bmax, float tfl) {
  return K >= 1 && std::isfinite(churn) && churn > 0.f && std::isfinite(bmin) && std::isfinite(bmax) &&
         bmin > 0.f && bmax >= bmin && tfl > 0.f && tfl <= 1.f;
}

static Sched make_sched(int K, float churn, float bmin, float bmax, float tfl) {
  Sched S;
  S.K = K; S.churn = churn; S.beta_min = bmin; S.beta_max = bmax; S.t_floor = tfl;
  S.delta = 1.0f / (float)K;
  return S;
}

struct SamplerLayout {
  size_t y, s, k, g, x, mp, mq, mqb, sg, sgb, sc, acc, yo, rounds, tausum, ctl, vws, total;
};

static SamplerLayout sampler_layout(int B, int L, int64_t d) {
  SamplerLayout w{};
  auto up = [](size_t v) { return (v + 255) & ~(size_t)255; };
  const size_t Bd = (size_t)B * d * sizeof(float);
  const size_t BLd = (size_t)B * L * d * sizeof(float);
  size_t o = 0;
  w.y = o; o = up(o + Bd);
  w.s = o; o = up(o + Bd);
  w.k = o; o = up(o + (size_t)B * 4);
  w.g = o; o = up(o + (size_t)B * 4);
  w.x = o; o = up(o + BLd);
  w.mp = o; o = up(o + BLd);
  w.mq = o; o = up(o + BLd);
  w.mqb = o; o = up(o + Bd);
  w.sg = o; o = up(o + (size_t)B * L * 4);
  w.sgb = o; o = up(o + (size_t)B * 4);
  w.sc = o; o = up(o + (size_t)B * (L + 1) * d * sizeof(float));
  w.acc = o; o = up(o + (size_t)B * 4);
  w.yo = o; o = up(o + Bd);
  w.rounds = o; o = up(o + (size_t)B * 4);
  w.tausum = o; o = up(o + (size_t)B * 4);
  w.ctl = o; o = up(o + sizeof(SamplerCtl));
  w.vws = o; o = up(o + sdv_workspace_bytes(B, L, d, SDV_F32));
  w.total = o;
  return w;
}

// A sampler problem and the views of its workspace.
struct SamplerRun {
  int B, L;
  int64_t d;
  int K, mode, drafter;
  uint64_t seed;
  Sched S;
  Gmm G;
  GmmLaunch gl;
  unsigned eg;
  float *y, *sc, *xd, *mpd, *mqd, *mqb, *sg, *sgb, *scall, *yo;
  int32_t *kk, *gam, *acc, *rounds, *tsum;
  SamplerCtl* ctl;
  void* vws;
  size_t vws_bytes;
};

static void sampler_views(const SamplerLayout& w, char* ws, SamplerRun* R) {
  R->y = (float*)(ws + w.y);
  R->sc = (float*)(ws + w.s);
  R->kk = (int32_t*)(ws + w.k);
  R->gam = (int32_t*)(ws + w.g);
  R->xd = (float*)(ws + w.x);
  R->mpd = (float*)(ws + w.mp);
  R->mqd = (float*)(ws + w.mq);
  R->mqb = (float*)(ws + w.mqb);
  R->sg = (float*)(ws + w.sg);
  R->sgb = (float*)(ws + w.sgb);
  R->scall = (float*)(ws + w.sc);
  R->acc = (int32_t*)(ws + w.acc);
  R->yo = (float*)(ws + w.yo);
  R->rounds = (int32_t*)(ws + w.rounds);
  R->tsum = (int32_t*)(ws + w.tausum);
  R->ctl = (SamplerCtl*)(ws + w.ctl);
  R->vws = ws + w.vws;
  R->vws_bytes = w.total - w.vws;
}

static int sampler_setup(int B, int L, int64_t d, const float* means, const float* log_weights, int C,
                         float comp_var, int K, float churn, float beta_min, float beta_max, float t_floor,
                         uint64_t seed, int mode, int drafter, void* workspace, size_t workspace_bytes,
                         SamplerRun* R) {
  if (!means || !log_weights) return SDV_EINVAL;
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1 || C < 1 || C > kSdvMaxComponents) return SDV_EINVAL;
  if (!(comp_var > 0.f) || !valid_sched(K, churn, beta_min, beta_max, t_floor)) return SDV_EINVAL;
  if (mode != SDV_MODE_SAMPLE && mode != SDV_MODE_BLOCK) return SDV_EINVAL;
  if (drafter != SDV_DRAFTER_FREE && drafter != SDV_DRAFTER_FROZEN) return SDV_EINVAL;
  const SamplerLayout w = sampler_layout(B, L, d);
  if (!workspace || workspace_bytes < w.total) return SDV_ENOWORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SDV_EALIGN;
  R->B = B; R->L = L; R->d = d; R->K = K; R->mode = mode; R->drafter = drafter; R->seed = seed;
  R->S = make_sched(K, churn, beta_min, beta_max, t_floor);
  R->G = Gmm{means, log_weights, C, comp_var};
  // workspace arrays start on 256-byte boundaries
  R->gl = gmm_launch(C, d, means, reinterpret_cast<uintptr_t>(workspace) % 16 == 0);
  R->eg = (unsigned)(((int64_t)B * ((d + 3) / 4) + 255) / 256);
  sampler_views(w, (char*)workspace, R);
  return SDV_OK;
}

// Initial states, bookkeeping and round state, and the only explicit target call: the
// score at Y_0 (step 0).
static int enqueue_begin(const SamplerRun& R, cudaStream_t s) {
  k_sampler_init<<<R.eg, 256, 0, s>>>(R.B, R.L, R.d, R.K, R.seed, R.y, R.kk, R.gam, R.rounds, R.tsum, R.ctl);
  int rc = launch_check();
  if (rc != SDV_OK) return rc;
  SDV_GMM_DISPATCH(R.gl, k_gmm_rows, rows_grid(R.B), s, R.y, R.kk, nullptr, R.B, R.d, R.S, R.G, R.gl.smem,
                   nullptr, R.sc);
  return launch_check();
}

// One round on stream cs (captured into the round graph's loop body when `loop`,
// whose condition the round's last update CTA then sets; launched directly
// otherwise).
static int enqueue_round(const SamplerRun& R, cudaStream_t cs, int max_rounds, bool loop,
                         cudaGraphConditionalHandle handle) {
  const int B = R.B, L = R.L;
  const int64_t d = R.d;
  const GmmLaunch& gl = R.gl;
  int rc = SDV_OK;
  if (R.drafter == SDV_DRAFTER_FROZEN) {  // a fresh score at the round's start state
    SDV_GMM_DISPATCH(gl, k_gmm_rows, rows_grid(B), cs, R.y, R.kk, R.gam, B, d, R.S, R.G, gl.smem, nullptr, R.sc);
    if ((rc = launch_check()) != SDV_OK) return rc;
  }
  if (gl.vec)
    k_draft<true><<<R.eg, 256, 0, cs>>>(R.y, R.sc, R.kk, R.gam, B, L, d, R.S, 0, &R.ctl->seed_r, R.xd, R.mpd, R.sg);
  else
    k_draft<false><<<R.eg, 256, 0, cs>>>(R.y, R.sc, R.kk, R.gam, B, L, d, R.S, 0, &R.ctl->seed_r, R.xd, R.mpd, R.sg);
  if ((rc = launch_check()) != SDV_OK) return rc;
  if (round_target_reg(gl, d)) {
    const unsigned grid = round_target_reg_grid(gl, B, L);
    if (gl.maxc == 8)
      k_round_target_reg<8><<<grid, kGmmThreads, 0, cs>>>(R.y, R.xd, R.kk, R.gam, B, L, d, R.S, R.G, R.mqd, R.mqb,
                                                         R.sgb, R.scall);
    else
      k_round_target_reg<16><<<grid, kGmmThreads, 0, cs>>>(R.y, R.xd, R.kk, R.gam, B, L, d, R.S, R.G, R.mqd, R.mqb,
                                                          R.sgb, R.scall);
  } else {
    SDV_GMM_DISPATCH(gl, k_round_target, round_target_grid(gl, B, L), cs, R.y, R.xd, R.kk, R.gam, B, L, d, R.S,
                     R.G, gl.smem, R.mqd, R.mqb, R.sgb, R.scall);
  }
  if ((rc = launch_check()) != SDV_OK) return rc;
  rc = verify_ex_impl(R.xd, R.mqd, R.mpd, R.sg, L, B, L, d, SDV_F32, 0, &R.ctl->seed_r, R.mode, R.gam, R.mqb,
                      R.sgb, SDV_RESIDUAL_DECOMPOSITION, 1.0f, R.acc, R.yo, nullptr, nullptr, nullptr, nullptr,
                      R.vws, R.vws_bytes, false, cs);
  if (rc != SDV_OK) return rc;
  if (d % 4 == 0)
    k_round_update<true><<<(B + kUpdateChains - 1) / kUpdateChains, 32 * kUpdateChains, 0, cs>>>(
        R.acc, R.yo, R.xd, R.scall, B, L, d, R.K, R.y, R.sc, R.kk, R.gam, R.rounds, R.tsum, R.ctl, R.seed,
        max_rounds, loop ? 1 : 0, handle);
  else
    k_round_update<false><<<(B + kUpdateChains - 1) / kUpdateChains, 32 * kUpdateChains, 0, cs>>>(
        R.acc, R.yo, R.xd, R.scall, B, L, d, R.K, R.y, R.sc, R.kk, R.gam, R.rounds, R.tsum, R.ctl, R.seed,
        max_rounds, loop ? 1 : 0, handle);
  return launch_check();
}

// Rounds run (host, after a synchronisation) and the chains' outputs (device copies).
static int read_results(const SamplerRun& R, float* y_out, int32_t* k_out, int32_t* chain_rounds_out,
                        int32_t* tau_sum_out, int32_t* rounds_out, cudaStream_t s) {
  const int B = R.B;
  int r = 0;
  if (cudaMemcpyAsync(&r, &R.ctl->r, sizeof(r), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  *rounds_out = r;
  if (cudaMemcpyAsync(y_out, R.y, (size_t)B * R.d * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  if (k_out && cudaMemcpyAsync(k_out, R.kk, (size_t)B * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  if (chain_rounds_out &&
      cudaMemcpyAsync(chain_rounds_out, R.rounds, (size_t)B * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  if (tau_sum_out && cudaMemcpyAsync(tau_sum_out, R.tsum, (size_t)B * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  return SDV_OK;
}

}  // namespace sdv

using namespace sdv;

extern "C" {

int sdv_gmm_target(const float* states, const int32_t* k, int n, int64_t d, const float* means,
                   const float* log_weights, int C, float comp_var, int K, float churn,
                   float beta_min, float beta_max, float t_floor, float* mq_out, float* score_out,
                   sdv_stream_t stream) {
  if (!states || !k || !means || !log_weights || (!mq_out && !score_out)) return SDV_EINVAL;
  if (n < 0 || d < 1 || C < 1 || C > kSdvMaxComponents || !(comp_var > 0.f)) return SDV_EINVAL;
  if (!valid_sched(K, churn, beta_min, beta_max, t_floor)) return SDV_EINVAL;
  if (n == 0) return SDV_OK;
  const Sched S = make_sched(K, churn, beta_min, beta_max, t_floor);
  const Gmm G{means, log_weights, C, comp_var};
  // float4 paths need 16-byte aligned rows in every array the kernel touches
  const bool al = ((reinterpret_cast<uintptr_t>(states) | reinterpret_cast<uintptr_t>(mq_out) |
                    reinterpret_cast<uintptr_t>(score_out)) % 16) == 0;
  const GmmLaunch gl = gmm_launch(C, d, means, al);
  SDV_GMM_DISPATCH(gl, k_gmm_rows, rows_grid(n), (cudaStream_t)stream, states, k, nullptr, n, d, S, G,
                   gl.smem, mq_out, score_out);
  return launch_check();
}

int sdv_free_draft(const float* y, const float* score, const int32_t* k, const int32_t* L_eff, int B,
                   int L, int64_t d, int K, float churn, float beta_min, float beta_max,
                   float t_floor, uint64_t seed, float* x_draft, float* mu_draft, float* sigma,
                   sdv_stream_t stream) {
  if (!y || !score || !k || !L_eff || !x_draft || !mu_draft || !sigma) return SDV_EINVAL;
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1) return SDV_EINVAL;
  if (!valid_sched(K, churn, beta_min, beta_max, t_floor)) return SDV_EINVAL;
  const Sched S = make_sched(K, churn, beta_min, beta_max, t_floor);
  const int64_t n = (int64_t)B * ((d + 3) / 4);
  const bool vec = (d % 4 == 0) && ((reinterpret_cast<uintptr_t>(y) | reinterpret_cast<uintptr_t>(score) |
                                      reinterpret_cast<uintptr_t>(x_draft) |
                                      reinterpret_cast<uintptr_t>(mu_draft)) % 16 == 0);
  const unsigned grid = (unsigned)((n + 255) / 256);
  if (vec) k_draft<true><<<grid, 256, 0, (cudaStream_t)stream>>>(y, score, k, L_eff, B, L, d, S, seed, nullptr, x_draft, mu_draft, sigma);
  else k_draft<false><<<grid, 256, 0, (cudaStream_t)stream>>>(y, score, k, L_eff, B, L, d, S, seed, nullptr, x_draft, mu_draft, sigma);
  return launch_check();
}

size_t sdv_sampler_workspace_bytes(int B, int L, int64_t d) {
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1) return 0;
  return sampler_layout(B, L, d).total;
}

int sdv_sampler_run(int B, int L, int64_t d, const float* means, const float* log_weights, int C,
                    float comp_var, int K, float churn, float beta_min, float beta_max,
                    float t_floor, uint64_t seed, int mode, int drafter, int max_rounds,
                    float* y_out, int32_t* k_out, int32_t* chain_rounds_out,
                    int32_t* tau_sum_out, int32_t* rounds_out, void* workspace,
                    size_t workspace_bytes, sdv_stream_t stream) {
  if (!y_out || !rounds_out) return SDV_EINVAL;
  if (max_rounds < 0) return SDV_EINVAL;
  SamplerRun R;
  int rc = sampler_setup(B, L, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max, t_floor, seed,
                         mode, drafter, workspace, workspace_bytes, &R);
  if (rc != SDV_OK) return rc;
  cudaStream_t s = (cudaStream_t)stream;
  if ((rc = enqueue_begin(R, s)) != SDV_OK) return rc;

  // The round loop is one CUDA graph: a while node whose body is one round, captured
  // once; the round's seed lives in device memory (SamplerCtl) and the round's last
  // update CTA ends the loop.  One graph launch runs every round with no host round trip.
  if (max_rounds > 0) {
    cudaGraph_t graph = nullptr, body = nullptr;
    cudaGraphExec_t exec = nullptr;
    cudaStream_t cs = nullptr;
    cudaGraphConditionalHandle handle = 0;
    cudaGraphNode_t loop = nullptr;
    bool ok = cudaGraphCreate(&graph, 0) == cudaSuccess &&
              cudaGraphConditionalHandleCreate(&handle, graph, 1u, cudaGraphCondAssignDefault) == cudaSuccess;
    if (ok) {
      cudaGraphNodeParams cp{};
      cp.type = cudaGraphNodeTypeConditional;
      cp.conditional.handle = handle;
      cp.conditional.type = cudaGraphCondTypeWhile;
      cp.conditional.size = 1;
      ok = cudaGraphAddNode(&loop, graph, nullptr, nullptr, 0, &cp) == cudaSuccess;
      if (ok) body = cp.conditional.phGraph_out[0];
    }
    ok = ok && cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) == cudaSuccess &&
         cudaStreamBeginCaptureToGraph(cs, body, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal) ==
             cudaSuccess;
    if (ok) {
      rc = enqueue_round(R, cs, max_rounds, true, handle);
      cudaGraph_t captured = nullptr;
      const bool ended = cudaStreamEndCapture(cs, &captured) == cudaSuccess;
      ok = rc == SDV_OK && ended && cudaGraphInstantiate(&exec, graph, 0) == cudaSuccess &&
           cudaGraphLaunch(exec, s) == cudaSuccess;
    }
    if (exec) cudaGraphExecDestroy(exec);
    if (graph) cudaGraphDestroy(graph);
    if (cs) cudaStreamDestroy(cs);
    if (!ok) {
      if (rc != SDV_OK) return rc;
      return launch_check(), SDV_ECUDA;
    }
  }
  return read_results(R, y_out, k_out, chain_rounds_out, tau_sum_out, rounds_out, s);
}

int sdv_sampler_begin(int B, int L, int64_t d, const float* means, const float* log_weights, int C,
                      float comp_var, int K, float churn, float beta_min, float beta_max, float t_floor,
                      uint64_t seed, void* workspace, size_t workspace_bytes, sdv_stream_t stream) {
  SamplerRun R;
  const int rc = sampler_setup(B, L, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max, t_floor,
                               seed, SDV_MODE_BLOCK, SDV_DRAFTER_FREE, workspace, workspace_bytes, &R);
  if (rc != SDV_OK) return rc;
  return enqueue_begin(R, (cudaStream_t)stream);
}

int sdv_sampler_round(int B, int L, int64_t d, const float* means, const float* log_weights, int C,
                      float comp_var, int K, float churn, float beta_min, float beta_max, float t_floor,
                      uint64_t seed, int mode, int drafter, void* workspace, size_t workspace_bytes,
                      sdv_stream_t stream) {
  SamplerRun R;
  const int rc = sampler_setup(B, L, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max, t_floor,
                               seed, mode, drafter, workspace, workspace_bytes, &R);
  if (rc != SDV_OK) return rc;
  return enqueue_round(R, (cudaStream_t)stream, 0, false, 0);
}

int sdv_sampler_end(int B, int L, int64_t d, void* workspace, size_t workspace_bytes, float* y_out,
                    int32_t* k_out, int32_t* chain_rounds_out, int32_t* tau_sum_out, int32_t* rounds_out,
                    sdv_stream_t stream) {
  if (!y_out || !rounds_out) return SDV_EINVAL;
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1) return SDV_EINVAL;
  const SamplerLayout w = sampler_layout(B, L, d);
  if (!workspace || workspace_bytes < w.total) return SDV_ENOWORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SDV_EALIGN;
  SamplerRun R{};
  R.B = B; R.L = L; R.d = d;
  sampler_views(w, (char*)workspace, &R);
  return read_results(R, y_out, k_out, chain_rounds_out, tau_sum_out, rounds_out, (cudaStream_t)stream);
}

int sdv_em_sample(int B, int64_t d, const float* means, const float* log_weights, int C,
                  float comp_var, int K, float churn, float beta_min, float beta_max,
                  float t_floor, uint64_t seed, float* y_out, sdv_stream_t stream) {
  if (!means || !log_weights || !y_out) return SDV_EINVAL;
  if (B < 1 || d < 1 || C < 1 || C > kSdvMaxComponents || !(comp_var > 0.f)) return SDV_EINVAL;
  if (!valid_sched(K, churn, beta_min, beta_max, t_floor)) return SDV_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  const Sched S = make_sched(K, churn, beta_min, beta_max, t_floor);
  const Gmm G{means, log_weights, C, comp_var};
  const int64_t ng = (int64_t)B * ((d + 3) / 4);
  // the initial state only needs y; the bookkeeping arrays of the init kernel are not used
  k_sampler_init<<<(unsigned)((ng + 255) / 256), 256, 0, s>>>(B, 1, d, K, seed, y_out, nullptr, nullptr,
                                                              nullptr, nullptr, nullptr);
  int rc = launch_check();
  if (rc != SDV_OK) return rc;
  const GmmLaunch gl = gmm_launch(C, d, means, reinterpret_cast<uintptr_t>(y_out) % 16 == 0);
  for (int k = 0; k < K; ++k) {
    SDV_GMM_DISPATCH(gl, k_em_step, rows_grid(B), s, y_out, B, d, k, S, G, gl.smem, seed);
    if ((rc = launch_check()) != SDV_OK) return rc;
  }
  return SDV_OK;
}

}  // extern "C"
