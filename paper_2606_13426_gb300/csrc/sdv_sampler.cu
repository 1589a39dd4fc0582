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

constexpr int kGmmThreads = 256;              // 8 warps, one state row per warp at a time
constexpr int kGmmWarps = kGmmThreads / 32;
constexpr size_t kGmmSmemCap = 96 * 1024;     // stage the means in shared memory up to this size

// m^q and the score for one state row z (generative step k), by one warp.  mu points to
// the means [C, d] (shared or global memory).  mq / score may be null; z may alias mq:
// each lane reads a group of four elements before it writes it, and no other lane
// touches that group.  add_sigma != 0 adds sigma * G (Philox stream noise_stream,
// sub-counter noise_sub; one Philox block per group of four) to mq.
// VEC: d % 4 == 0 and 16-byte aligned rows (float4 accesses); MAXC >= C components.
template <int MAXC, bool VEC>
__device__ __forceinline__ void gmm_row_warp(const float* z, int64_t d, int k, const Sched& S,
                                             const Gmm& G, const float* mu, float* mq, float* score,
                                             float add_sigma, uint64_t noise_seed,
                                             uint32_t noise_chain, uint32_t noise_stream,
                                             uint32_t noise_sub) {
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int C = G.C;
  const float tf = S.tfwd(k);
  const float ab = S.abar(tf);
  const float sab = sqrtf(ab);
  const float v = ab * G.comp_var + 1.0f - ab;
  const float b = S.beta(tf);
  const float cst = 0.5f * (1.0f + S.churn * S.churn);
  const int64_t ng = (d + 3) / 4;
  auto load_group = [&](const float* p, int64_t gi, float (&f)[4]) {
    if (VEC) {
      const float4 t = *reinterpret_cast<const float4*>(p + 4 * gi);
      f[0] = t.x; f[1] = t.y; f[2] = t.z; f[3] = t.w;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) f[q] = (4 * gi + q < d) ? p[4 * gi + q] : 0.f;
    }
  };
  // pass 1: squared distances to the scaled centres sqrt(abar) mu_c
  float acc[MAXC];
#pragma unroll
  for (int c = 0; c < MAXC; ++c) acc[c] = 0.f;
#pragma unroll 4
  for (int64_t gi = lane; gi < ng; gi += 32) {
    float zf[4];
    load_group(z, gi, zf);
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
      if (c < C) {
        float mf[4];
        load_group(mu + (int64_t)c * d, gi, mf);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float df = (4 * gi + q < d) ? zf[q] - sab * mf[q] : 0.f;
          acc[c] = fmaf(df, df, acc[c]);
        }
      }
    }
  }
  // responsibilities r_c = softmax(log w_c - d2_c / (2 v)), identical in every lane
  float r[MAXC];
  float mx = -INFINITY;
#pragma unroll
  for (int c = 0; c < MAXC; ++c) {
    float a = acc[c];
    if (c < C) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(FULL, a, o);
    }
    r[c] = (c < C) ? __ldg(G.log_w + c) - a / (2.0f * v) : -INFINITY;
    mx = fmaxf(mx, r[c]);
  }
  float den = 0.f;
#pragma unroll
  for (int c = 0; c < MAXC; ++c) {
    r[c] = (c < C) ? expf(r[c] - mx) : 0.f;
    den += r[c];
  }
  const float w_sc = sab / den;  // folds the softmax normaliser and sqrt(abar)
  // pass 2: score and target mean
#pragma unroll 4
  for (int64_t gi = lane; gi < ng; gi += 32) {
    float zf[4], wsum[4] = {0.f, 0.f, 0.f, 0.f};
    load_group(z, gi, zf);
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
      if (c < C) {
        float mf[4];
        load_group(mu + (int64_t)c * d, gi, mf);
#pragma unroll
        for (int q = 0; q < 4; ++q) wsum[q] = fmaf(r[c], mf[q], wsum[q]);
      }
    }
    float G4[4] = {0.f, 0.f, 0.f, 0.f};
    if (add_sigma != 0.f) {
      const float4 n4 = normals4(noise_seed, noise_chain, (uint32_t)gi, noise_stream, noise_sub);
      G4[0] = n4.x; G4[1] = n4.y; G4[2] = n4.z; G4[3] = n4.w;
    }
    float sc[4], m[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      sc[q] = (w_sc * wsum[q] - zf[q]) / v;
      m[q] = zf[q] + S.delta * (0.5f * b * zf[q] + cst * b * sc[q]) + add_sigma * G4[q];
    }
    if (VEC) {
      if (score) *reinterpret_cast<float4*>(score + 4 * gi) = make_float4(sc[0], sc[1], sc[2], sc[3]);
      if (mq) *reinterpret_cast<float4*>(mq + 4 * gi) = make_float4(m[0], m[1], m[2], m[3]);
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (4 * gi + q < d) {
          if (score) score[4 * gi + q] = sc[q];
          if (mq) mq[4 * gi + q] = m[q];
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
    gmm_row_warp<MAXC, VEC>(states + o, d, k[row], S, G, mu, mq ? mq + o : nullptr,
                            score ? score + o : nullptr, 0.f, 0, 0, 0, 0);
  }
}

// Parallel target call of a round, one CTA per chain: state j of chain b is y[b] (j = 0)
// or x_draft[b, j-1], at step k[b] + j, for j = 0 .. gamma_b.  Means go to mu_target[b, j]
// (j < gamma_b) or mu_bonus[b] (j = gamma_b, with sigma_bonus[b] = sigma_{k+gamma});
// scores to sc_all[b, j].
template <int MAXC, bool VEC>
__global__ void __launch_bounds__(kGmmThreads)
k_round_target(const float* __restrict__ y, const float* __restrict__ x_draft,
               const int32_t* __restrict__ kk, const int32_t* __restrict__ gam, int L, int64_t d,
               Sched S, Gmm G, bool use_smem, float* mu_target, float* mu_bonus, float* sigma_bonus,
               float* sc_all) {
  const int b = blockIdx.x;
  const int g = gam[b];
  if (g == 0) return;  // CTA-uniform: before any barrier
  const float* mu = stage_means(G, d, use_smem);
  const int warp = threadIdx.x >> 5;
  for (int j = warp; j <= g; j += kGmmWarps) {
    const float* z = (j == 0) ? y + (int64_t)b * d : x_draft + ((int64_t)b * L + j - 1) * d;
    float* mq = (j < g) ? mu_target + ((int64_t)b * L + j) * d : mu_bonus + (int64_t)b * d;
    gmm_row_warp<MAXC, VEC>(z, d, kk[b] + j, S, G, mu, mq, sc_all + ((int64_t)b * (L + 1) + j) * d,
                            0.f, 0, 0, 0, 0);
  }
  if (threadIdx.x == 0) sigma_bonus[b] = S.sigma(kk[b] + g);
}

// Free / Frozen drafter: gamma_b elementwise steps from y[b] with the cached score.
__global__ void __launch_bounds__(256)
k_draft(const float* __restrict__ y, const float* __restrict__ s_cache, const int32_t* __restrict__ kk,
        const int32_t* __restrict__ gam, int B, int L, int64_t d, Sched S, uint64_t seed,
        float* x_draft, float* mu_draft, float* sigma) {
  const int64_t ng = (d + 3) / 4;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * ng) return;
  const int b = (int)(t / ng);
  const int64_t gi = t - (int64_t)b * ng;
  const int g = gam[b];
  if (g == 0) return;
  const int k = kk[b];
  const float cst = 0.5f * (1.0f + S.churn * S.churn);
  float cur[4], sc[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int64_t i = 4 * gi + q;
    cur[q] = (i < d) ? y[(int64_t)b * d + i] : 0.f;
    sc[q] = (i < d) ? s_cache[(int64_t)b * d + i] : 0.f;
  }
  for (int step = 1; step <= g; ++step) {
    const int kc = k + step - 1;
    const float be = S.beta(S.tfwd(kc));
    const float sg = S.sigma(kc);
    const float4 n4 = normals4(seed, (uint32_t)b, (uint32_t)gi, kStreamDraft, (uint32_t)(step - 1));
    const float nz[4] = {n4.x, n4.y, n4.z, n4.w};
    const int64_t row = ((int64_t)b * L + step - 1) * d;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t i = 4 * gi + q;
      const float m = cur[q] + S.delta * (0.5f * be * cur[q] + cst * be * sc[q]);
      const float nx = m + sg * nz[q];
      if (i < d) {
        mu_draft[row + i] = m;
        x_draft[row + i] = nx;
      }
      cur[q] = nx;
    }
    if (gi == 0) sigma[(int64_t)b * L + step - 1] = sg;
  }
}

// Round bookkeeping, one CTA per chain: the emitted state, the score cache, k, the next
// window length and the statistics; counts the chains that remain active.
__global__ void __launch_bounds__(256)
k_round_update(const int32_t* __restrict__ acc, const float* __restrict__ y_out,
               const float* __restrict__ x_draft, const float* __restrict__ sc_all, int L, int64_t d,
               int K, float* y, float* s_cache, int32_t* kk, int32_t* gam, int32_t* rounds,
               int32_t* tau_sum, unsigned int* active) {
  const int b = blockIdx.x;
  const int g = gam[b];
  const int k = kk[b];
  __syncthreads();  // every thread has read k and gamma before thread 0 updates them
  if (g == 0) return;
  const int tau = acc[b] + 1;
  const bool end = (tau == g + 1) && (k + g >= K);  // no bonus step past the end of sampling
  const float* ysrc = end ? x_draft + ((int64_t)b * L + g - 1) * d : y_out + (int64_t)b * d;
  const float* ssrc = sc_all + ((int64_t)b * (L + 1) + min(tau, g)) * d;
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) {
    y[(int64_t)b * d + i] = ysrc[i];
    s_cache[(int64_t)b * d + i] = ssrc[i];
  }
  if (threadIdx.x == 0) {
    const int kn = min(k + tau, K);
    kk[b] = kn;
    const int gn = kn < K ? min(L, K - kn) : 0;
    gam[b] = gn;
    rounds[b] += 1;
    tau_sum[b] += tau;
    if (gn > 0) atomicAdd(active, 1u);
  }
}

__global__ void __launch_bounds__(256)
k_sampler_init(int B, int L, int64_t d, int K, uint64_t seed, float* y, int32_t* kk, int32_t* gam,
               int32_t* rounds, int32_t* tau_sum) {
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
    gmm_row_warp<MAXC, VEC>(row, d, k, S, G, mu, row, nullptr, S.sigma(k), seed, (uint32_t)b, kStreamEM,
                            (uint32_t)k);
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

static uint64_t splitmix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Seed of round r: the (r+1)-th SplitMix64 output of a stream started at `seed`.
static uint64_t round_seed(uint64_t seed, int r) {
  return splitmix64(seed + (uint64_t)(r + 1) * 0x9E3779B97F4A7C15ull);
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
  size_t y, s, k, g, x, mp, mq, mqb, sg, sgb, sc, acc, yo, rounds, tausum, active, vws, total;
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
  w.active = o; o = up(o + 4);
  w.vws = o; o = up(o + sdv_workspace_bytes(B, L, d, SDV_F32));
  w.total = o;
  return w;
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
  k_draft<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(y, score, k, L_eff, B, L, d, S, seed,
                                                                         x_draft, mu_draft, sigma);
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
  if (!means || !log_weights || !y_out || !rounds_out) return SDV_EINVAL;
  if (B < 1 || L < 1 || L > SDV_MAX_L || d < 1 || C < 1 || C > kSdvMaxComponents) return SDV_EINVAL;
  if (!(comp_var > 0.f) || !valid_sched(K, churn, beta_min, beta_max, t_floor)) return SDV_EINVAL;
  if (mode != SDV_MODE_SAMPLE && mode != SDV_MODE_BLOCK) return SDV_EINVAL;
  if (drafter != SDV_DRAFTER_FREE && drafter != SDV_DRAFTER_FROZEN) return SDV_EINVAL;
  if (max_rounds < 0) return SDV_EINVAL;
  const SamplerLayout w = sampler_layout(B, L, d);
  if (!workspace || workspace_bytes < w.total) return SDV_ENOWORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SDV_EALIGN;
  cudaStream_t s = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  float* y = (float*)(ws + w.y);
  float* sc = (float*)(ws + w.s);
  int32_t* kk = (int32_t*)(ws + w.k);
  int32_t* gam = (int32_t*)(ws + w.g);
  float* xd = (float*)(ws + w.x);
  float* mpd = (float*)(ws + w.mp);
  float* mqd = (float*)(ws + w.mq);
  float* mqb = (float*)(ws + w.mqb);
  float* sg = (float*)(ws + w.sg);
  float* sgb = (float*)(ws + w.sgb);
  float* scall = (float*)(ws + w.sc);
  int32_t* acc = (int32_t*)(ws + w.acc);
  float* yo = (float*)(ws + w.yo);
  int32_t* rounds = (int32_t*)(ws + w.rounds);
  int32_t* tsum = (int32_t*)(ws + w.tausum);
  unsigned int* active = (unsigned int*)(ws + w.active);
  void* vws = ws + w.vws;
  const size_t vws_bytes = w.total - w.vws;
  const Sched S = make_sched(K, churn, beta_min, beta_max, t_floor);
  const Gmm G{means, log_weights, C, comp_var};
  const int64_t ng = (int64_t)B * ((d + 3) / 4);
  const unsigned eg = (unsigned)((ng + 255) / 256);
  // workspace arrays start on 256-byte boundaries
  const GmmLaunch gl = gmm_launch(C, d, means, reinterpret_cast<uintptr_t>(workspace) % 16 == 0);

  int rc;
  k_sampler_init<<<eg, 256, 0, s>>>(B, L, d, K, seed, y, kk, gam, rounds, tsum);
  if ((rc = launch_check()) != SDV_OK) return rc;
  // the only explicit target call: the score at Y_0 (step 0)
  SDV_GMM_DISPATCH(gl, k_gmm_rows, rows_grid(B), s, y, kk, nullptr, B, d, S, G, gl.smem, nullptr, sc);
  if ((rc = launch_check()) != SDV_OK) return rc;

  int r = 0;
  const int check_every = 8;
  for (; r < max_rounds; ++r) {
    const uint64_t seed_r = round_seed(seed, r);
    if (drafter == SDV_DRAFTER_FROZEN) {  // a fresh score at the round's start state
      SDV_GMM_DISPATCH(gl, k_gmm_rows, rows_grid(B), s, y, kk, gam, B, d, S, G, gl.smem, nullptr, sc);
      if ((rc = launch_check()) != SDV_OK) return rc;
    }
    k_draft<<<eg, 256, 0, s>>>(y, sc, kk, gam, B, L, d, S, seed_r, xd, mpd, sg);
    if ((rc = launch_check()) != SDV_OK) return rc;
    SDV_GMM_DISPATCH(gl, k_round_target, B, s, y, xd, kk, gam, L, d, S, G, gl.smem, mqd, mqb, sgb, scall);
    if ((rc = launch_check()) != SDV_OK) return rc;
    rc = sdv_verify_ex(xd, mqd, mpd, sg, L, B, L, d, SDV_F32, seed_r, mode, gam, mqb, sgb,
                       SDV_RESIDUAL_DECOMPOSITION, 1.0f, acc, yo, nullptr, nullptr, nullptr, nullptr,
                       vws, vws_bytes, stream);
    if (rc != SDV_OK) return rc;
    if (cudaMemsetAsync(active, 0, sizeof(unsigned int), s) != cudaSuccess) return launch_check(), SDV_ECUDA;
    k_round_update<<<B, 256, 0, s>>>(acc, yo, xd, scall, L, d, K, y, sc, kk, gam, rounds, tsum, active);
    if ((rc = launch_check()) != SDV_OK) return rc;
    if ((r + 1) % check_every == 0 || r + 1 == max_rounds) {
      unsigned int h_active = 1;
      if (cudaMemcpyAsync(&h_active, active, sizeof(h_active), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
          cudaStreamSynchronize(s) != cudaSuccess)
        return launch_check(), SDV_ECUDA;
      if (h_active == 0) {
        ++r;
        break;
      }
    }
  }
  *rounds_out = r;
  if (cudaMemcpyAsync(y_out, y, (size_t)B * d * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  if (k_out && cudaMemcpyAsync(k_out, kk, (size_t)B * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  if (chain_rounds_out &&
      cudaMemcpyAsync(chain_rounds_out, rounds, (size_t)B * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  if (tau_sum_out && cudaMemcpyAsync(tau_sum_out, tsum, (size_t)B * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return launch_check(), SDV_ECUDA;
  return SDV_OK;
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
                                                              nullptr, nullptr);
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
