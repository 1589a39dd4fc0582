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

constexpr int kGmmThreads = 256;

// m^q and the score for one state row z (generative step k), by the whole CTA.
// mq / score may be null.  z may alias mq (each element is read before it is written
// by the same thread), which the in-place EM step uses.
__device__ void gmm_row(const float* z, int64_t d, int k, const Sched& S, const Gmm& G,
                        float* mq, float* score, float add_sigma, uint64_t noise_seed,
                        uint32_t noise_chain, uint32_t noise_stream, uint32_t noise_sub) {
  __shared__ float red[kGmmThreads / 32][kSdvMaxComponents];
  __shared__ float d2s[kSdvMaxComponents];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int C = G.C;
  const float tf = S.tfwd(k);
  const float ab = S.abar(tf);
  const float sab = sqrtf(ab);
  const float v = ab * G.comp_var + 1.0f - ab;
  const float b = S.beta(tf);
  const float cst = 0.5f * (1.0f + S.churn * S.churn);
  // pass 1: squared distances to the scaled centres
  float acc[kSdvMaxComponents];
#pragma unroll
  for (int c = 0; c < kSdvMaxComponents; ++c) acc[c] = 0.f;
  for (int64_t i = tid; i < d; i += kGmmThreads) {
    const float zi = z[i];
#pragma unroll
    for (int c = 0; c < kSdvMaxComponents; ++c) {
      if (c < C) {
        const float df = zi - sab * __ldg(G.means + (int64_t)c * d + i);
        acc[c] = fmaf(df, df, acc[c]);
      }
    }
  }
#pragma unroll
  for (int c = 0; c < kSdvMaxComponents; ++c) {
    if (c < C) {
      float a = acc[c];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
      if (lane == 0) red[warp][c] = a;
    }
  }
  __syncthreads();
  if (tid < C) {
    float a = 0.f;
    for (int w = 0; w < kGmmThreads / 32; ++w) a += red[w][tid];
    d2s[tid] = a;
  }
  __syncthreads();
  // responsibilities r_c = softmax(log w_c - d2_c / (2 v))
  float r[kSdvMaxComponents];
  float mx = -INFINITY;
#pragma unroll
  for (int c = 0; c < kSdvMaxComponents; ++c) {
    r[c] = (c < C) ? __ldg(G.log_w + c) - d2s[c] / (2.0f * v) : -INFINITY;
    mx = fmaxf(mx, r[c]);
  }
  float den = 0.f;
#pragma unroll
  for (int c = 0; c < kSdvMaxComponents; ++c) {
    r[c] = (c < C) ? expf(r[c] - mx) : 0.f;
    den += r[c];
  }
  const float inv = 1.0f / den;
  // pass 2: score and target mean (optionally plus sigma * noise)
  for (int64_t i0 = 4 * (int64_t)tid; i0 < d; i0 += 4 * kGmmThreads) {
    float G4[4] = {0.f, 0.f, 0.f, 0.f};
    if (add_sigma != 0.f) {
      const float4 n4 = normals4(noise_seed, noise_chain, (uint32_t)(i0 / 4), noise_stream, noise_sub);
      G4[0] = n4.x; G4[1] = n4.y; G4[2] = n4.z; G4[3] = n4.w;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t i = i0 + q;
      if (i >= d) break;
      const float zi = z[i];
      float wsum = 0.f;
#pragma unroll
      for (int c = 0; c < kSdvMaxComponents; ++c)
        if (c < C) wsum = fmaf(r[c], __ldg(G.means + (int64_t)c * d + i), wsum);
      const float sc = (sab * wsum * inv - zi) / v;
      const float m = zi + S.delta * (0.5f * b * zi + cst * b * sc);
      if (score) score[i] = sc;
      if (mq) mq[i] = m + add_sigma * G4[q];
    }
  }
}

// Target means and scores for rows of a [n, d] array at steps k[row]; rows whose
// window mask (if given) is 0 are skipped.
__global__ void __launch_bounds__(kGmmThreads)
k_gmm_rows(const float* __restrict__ states, const int32_t* __restrict__ k, const int32_t* __restrict__ mask,
           int64_t d, Sched S, Gmm G, float* mq, float* score) {
  const int row = blockIdx.x;
  if (mask && mask[row] == 0) return;
  const int64_t o = (int64_t)row * d;
  gmm_row(states + o, d, k[row], S, G, mq ? mq + o : nullptr, score ? score + o : nullptr, 0.f, 0,
          0, 0, 0);
}

// Parallel target call of a round: state j of chain b is y[b] (j = 0) or x_draft[b, j-1],
// at step k[b] + j, for j = 0 .. gamma_b.  Means go to mu_target[b, j] (j < gamma_b) or
// mu_bonus[b] (j = gamma_b, with sigma_bonus[b] = sigma_{k+gamma}); scores to sc_all[b, j].
__global__ void __launch_bounds__(kGmmThreads)
k_round_target(const float* __restrict__ y, const float* __restrict__ x_draft,
               const int32_t* __restrict__ kk, const int32_t* __restrict__ gam, int L, int64_t d,
               Sched S, Gmm G, float* mu_target, float* mu_bonus, float* sigma_bonus, float* sc_all) {
  const int b = blockIdx.x / (L + 1), j = blockIdx.x - b * (L + 1);
  const int g = gam[b];
  if (g == 0 || j > g) return;
  const float* z = (j == 0) ? y + (int64_t)b * d : x_draft + ((int64_t)b * L + j - 1) * d;
  float* mq = (j < g) ? mu_target + ((int64_t)b * L + j) * d : mu_bonus + (int64_t)b * d;
  gmm_row(z, d, kk[b] + j, S, G, mq, sc_all + ((int64_t)b * (L + 1) + j) * d, 0.f, 0, 0, 0, 0);
  if (j == g && threadIdx.x == 0) sigma_bonus[b] = S.sigma(kk[b] + g);
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

// One plain Euler-Maruyama step for every chain, in place: y <- m^q_k(y) + sigma_k G_k.
__global__ void __launch_bounds__(kGmmThreads)
k_em_step(float* y, int64_t d, int k, Sched S, Gmm G, uint64_t seed) {
  const int b = blockIdx.x;
  float* row = y + (int64_t)b * d;
  gmm_row(row, d, k, S, G, row, nullptr, S.sigma(k), seed, (uint32_t)b, kStreamEM, (uint32_t)k);
}

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
  k_gmm_rows<<<n, kGmmThreads, 0, (cudaStream_t)stream>>>(states, k, nullptr, d, S, G, mq_out, score_out);
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

  int rc;
  k_sampler_init<<<eg, 256, 0, s>>>(B, L, d, K, seed, y, kk, gam, rounds, tsum);
  if ((rc = launch_check()) != SDV_OK) return rc;
  // the only explicit target call: the score at Y_0 (step 0)
  k_gmm_rows<<<B, kGmmThreads, 0, s>>>(y, kk, nullptr, d, S, G, nullptr, sc);
  if ((rc = launch_check()) != SDV_OK) return rc;

  int r = 0;
  const int check_every = 8;
  for (; r < max_rounds; ++r) {
    const uint64_t seed_r = round_seed(seed, r);
    if (drafter == SDV_DRAFTER_FROZEN) {  // a fresh score at the round's start state
      k_gmm_rows<<<B, kGmmThreads, 0, s>>>(y, kk, gam, d, S, G, nullptr, sc);
      if ((rc = launch_check()) != SDV_OK) return rc;
    }
    k_draft<<<eg, 256, 0, s>>>(y, sc, kk, gam, B, L, d, S, seed_r, xd, mpd, sg);
    if ((rc = launch_check()) != SDV_OK) return rc;
    k_round_target<<<B * (L + 1), kGmmThreads, 0, s>>>(y, xd, kk, gam, L, d, S, G, mqd, mqb, sgb, scall);
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
  for (int k = 0; k < K; ++k) {
    k_em_step<<<B, kGmmThreads, 0, s>>>(y_out, d, k, S, G, seed);
    if ((rc = launch_check()) != SDV_OK) return rc;
  }
  return SDV_OK;
}

}  // extern "C"
