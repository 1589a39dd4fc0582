// sdv_device.cuh - device-side building blocks of the verification step (sm_103a).
//
//  * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) and the uniform /
//    Box-Muller transforms of the counter layout documented in specdiff.h.
//  * log Phi and the scaled log-CDF g(a) = log Phi(a) + a^2/2, its derivative
//    g'(s) = lambda(s) + s (lambda = phi/Phi, the inverse Mills ratio), and
//    differences g(hi) - g(hi - h) by 8-point Gauss-Legendre quadrature.
//  * The block-verification acceptance probability h_j (Algorithm
//    block-verification) in log form (App. "Density ratio calculations"), from
//    the same residual mass log v that the U-sampler's setup computes.
//  * The residual's 1-D draw U = Psi_alpha^{-1}(w) (Prop. decomposition,
//    Eq. u-cdf, Algorithm u-sample) as a one-warp multisection.
//
// Everything is fp32: GB300's fp64 rate is a small fraction of its fp32 rate.
// The special-function helpers are __noinline__: inlined at every call site they
// made the acceptance-scan kernel's code too large for the instruction cache.
// Inside gdiff, g' stays inline so that its eight quadrature nodes interleave.
// The forms below avoid the cancellations that fp32 would otherwise suffer:
//  - v = alpha Phi(a+) - Phi(a-) is written as alpha Phi(a+) (1 - e^{x0}) with
//    x0 = log(Phi(a-)/(alpha Phi(a+))) = g(a-) - g(a+), exact because
//    log alpha + a-^2/2 = a+^2/2 (a+- = log alpha / D +- D/2);
//  - Psi near its upper end a+ (where its density vanishes) is evaluated as a
//    complement, 1 - Psi(a+ - t) = int_0^t phi(a- - s) expm1(D s) ds / v,
//    which has a positive integrand (alpha phi(u) - phi(u - D) =
//    phi(u - D) expm1(D (a+ - u)));
//  - for s < -4, lambda(s) + s = 1/(x + 2/(x + 3/(x + ...))), x = -s, which is
//    Laplace's continued fraction for the Mills ratio with its first term
//    cancelled analytically.
#pragma once

// Linkage of the special-function helpers (see above); a translation unit may
// define SDV_HELPER before including this header.
#ifndef SDV_HELPER
#define SDV_HELPER __noinline__
#endif
// Unrolling of the quadrature nodes in gdiff.  The finishing path runs once per chain
// from a cold instruction cache, where every 128-byte line of straight-line code costs a
// fetch, but the eight nodes are independent: unrolled, their exponentials overlap, and
// that measured faster (the other once-run helpers stay out of line).
#ifndef SDV_GL_UNROLL
#define SDV_GL_UNROLL 8
#endif
namespace sdv {
constexpr int kGLUnroll = SDV_GL_UNROLL;
}

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

namespace sdv {

// ---------------------------------------------------------------- Philox
constexpr float kLn2Hi = 0.69314718055994531f;  // log 2 (fp32)
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

enum : uint32_t {
  kStreamCoin = 0,
  kStreamUSample = 1,
  kStreamResid = 2,
  kStreamBonus = 3,
  kStreamDraft = 4,
  kStreamInit = 5,
  kStreamEM = 6,
};

// Ten rounds of the Philox4x32 S-box: (c0,c1,c2,c3) -> (hi(M1 c2)^c1^k0,
// lo(M1 c2), hi(M0 c0)^c3^k1, lo(M0 c0)); the key is bumped by the Weyl
// constants between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += kPhiloxW0;
      k1 += kPhiloxW1;
    }
    const uint32_t lo0 = kPhiloxM0 * c.x;
    const uint32_t hi0 = __umulhi(kPhiloxM0, c.x);
    const uint32_t lo1 = kPhiloxM1 * c.z;
    const uint32_t hi1 = __umulhi(kPhiloxM1, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

__device__ __forceinline__ uint4 philox_block(uint64_t seed, uint32_t c0, uint32_t c1,
                                              uint32_t c2, uint32_t c3) {
  return philox4x32_10(make_uint4(c0, c1, c2, c3), (uint32_t)seed, (uint32_t)(seed >> 32));
}

// log u for u = (x + 1/2) 2^-32 with one logarithm: in the lower half, u = m 2^e with
// m in [1/2, 1) split off the exponent bits, so log u = (e - 1) log 2 + log1p(2m - 1),
// 2m - 1 exact; the upper half goes through 1 - u, exact in the integer domain, as
// log1p(-(1 - u)), so log u keeps full relative accuracy near 1.  The argument and the
// offset are selected first (no divergence between lanes), then one log1pf.
__device__ __forceinline__ float log_uniform(uint32_t x) {
  const float u = ((float)x + 0.5f) * 0x1p-32f;
  const uint32_t ub = __float_as_uint(u);
  const float m2 = __uint_as_float((ub & 0x007fffffu) | 0x3f800000u);   // 2m in [1, 2)
  const float e1 = (float)((int)(ub >> 23) - 127);                      // e - 1
  const float v = ((float)(0xFFFFFFFFu - x) + 0.5f) * 0x1p-32f;          // 1 - u
  const bool lower = x < 0x80000000u;
  const float arg = lower ? m2 - 1.0f : -v;
  const float base = lower ? e1 * kLn2Hi : 0.0f;
  return base + log1pf(arg);
}

// Box-Muller on two words: (r cos 2 pi u1, r sin 2 pi u1), r = sqrt(-2 ln u0).
__device__ __forceinline__ float2 box_muller(uint32_t w0, uint32_t w1) {
  const float r = sqrtf(-2.0f * log_uniform(w0));
  float s, c;
  sincospif(((float)w1 + 0.5f) * 0x1p-31f, &s, &c);
  return make_float2(r * c, r * s);
}

// Four normals of Philox block (b, blk, stream, sub): elements 4 blk .. 4 blk + 3.
__device__ __forceinline__ float4 normals4(uint64_t seed, uint32_t b, uint32_t blk,
                                           uint32_t stream, uint32_t sub) {
  const uint4 w = philox_block(seed, b, blk, stream, sub);
  const float2 z01 = box_muller(w.x, w.y);
  const float2 z23 = box_muller(w.z, w.w);
  return make_float4(z01.x, z01.y, z23.x, z23.y);
}

// normals4 as one shared copy, for the residual paths that run once per chain.
static __device__ SDV_HELPER float4 normals4_f(uint64_t seed, uint32_t b, uint32_t blk, uint32_t stream,
                                               uint32_t sub) {
  return normals4(seed, b, blk, stream, sub);
}

// ---------------------------------------------------------------- normal CDF helpers
constexpr float kSqrtHalf = 0.70710678118654752f;
constexpr float kHalfLog2Pi = 0.91893853320467274f;  // log(2 pi) / 2
constexpr float kLn2 = 0.69314718055994531f;

// Reciprocal without the IEEE slow path: the hardware approximation refined by one
// Newton step (about 1 ulp for finite non-zero x; +-inf gives 0 and 0 gives inf).
// IEEE division and __frcp_rn branch to a slow path, which keeps independent
// evaluations from overlapping; this form does not.
__device__ __forceinline__ float frcp_fast(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  const float e = fmaf(-x, r, 1.0f);
  return (r != 0.0f && isfinite(r)) ? fmaf(r, e, r) : r;
}

// 8-point Gauss-Legendre nodes / weights on [-1, 1] (positive half).
static __constant__ float kGLx[4] = {0.18343464249564978f, 0.52553240991632899f,
                                          0.79666647741362673f, 0.96028985649753618f};
static __constant__ float kGLw[4] = {0.36268378337836166f, 0.31370664587788688f,
                                          0.22238103445337443f, 0.10122853629037706f};

// The scaled complementary error function erfcx(z) = exp(z^2) erfc(z), branch-free and
// inline so that independent evaluations (the quadrature nodes below) overlap.  For
// z >= 0: erfcx(z) = t exp(f(t)), t = 1/(1 + z/2), with f(t) = log(erfcx(z)/t) a
// degree-11 polynomial in x = 2t - 1 (a Chebyshev fit of f, generated by
// gen_erfcx_coeffs.py; max relative error 1.4e-7 in fp32).  z = +inf gives t = 0 and 0.
__device__ __forceinline__ float erfcx_pos(float z) {
  const float t = frcp_fast(fmaf(0.5f, z, 1.0f));
  const float x = fmaf(2.0f, t, -1.0f);
  // f(t) = log(erfcx(z)/t) in the power basis of x = 2t - 1, degree 11 (Horner)
  float f = -8.728381024e-05f;
  f = fmaf(f, x, 8.000738166e-06f);
  f = fmaf(f, x, 5.737663720e-04f);
  f = fmaf(f, x, -2.279109660e-04f);
  f = fmaf(f, x, -2.288765239e-03f);
  f = fmaf(f, x, 1.794066250e-03f);
  f = fmaf(f, x, 8.808825369e-03f);
  f = fmaf(f, x, -9.880019324e-03f);
  f = fmaf(f, x, -4.689364056e-02f);
  f = fmaf(f, x, 4.734388761e-02f);
  f = fmaf(f, x, 6.726431548e-01f);
  f = fmaf(f, x, -6.717940917e-01f);
  return t * expf(f);
}

// erfcx of any sign: erfcx(-a) = 2 exp(a^2) - erfcx(a) (no cancellation: the first
// term is at least 2, the second at most 1), with a^2 split exactly (hi + lo) so that
// exp(a^2) keeps full relative accuracy; overflows to +inf for a above ~9.4.
__device__ __forceinline__ float erfcx_any(float z) {
  const float a = fabsf(z);
  const float e = erfcx_pos(a);
  const float hi = a * a, lo = fmaf(a, a, -hi);
  const float big = 2.0f * expf(hi) * (1.0f + lo);
  return (z >= 0.0f) ? e : big - e;
}

// (log Phi(a), g(a)) from one scaled complement E = erfcx(|a|/sqrt 2)/2 =
// Phi(-|a|) e^{a^2/2}: for a <= 0, log Phi(a) = log E - a^2/2 (no underflow); for
// a > 0, log Phi(a) = log(1 - E e^{-a^2/2}).  Both branches are computed and one is
// selected, so that lanes with different arguments do not diverge.
__device__ __forceinline__ float2 log_ndtr_g(float a) {
  const float E = 0.5f * erfcx_pos(fabsf(a) * kSqrtHalf);
  const float h = 0.5f * a * a;
  const float lneg = logf(E);                  // log Phi(-|a|) + a^2/2
  const float lpos = log1pf(-E * expf(-h));    // log Phi(|a|)
  return (a <= 0.0f) ? make_float2(lneg - h, lneg) : make_float2(lpos, lpos + h);
}

// log Phi(a).
static __device__ SDV_HELPER float log_ndtr(float a) { return log_ndtr_g(a).x; }

// g(a) = log Phi(a) + a^2/2 (moderate for a <= 0).
static __device__ SDV_HELPER float gfun(float a) { return log_ndtr_g(a).y; }

// g'(s) = lambda(s) + s > 0 in its two forms.  For s < -4 (x = -s) Laplace's
// continued fraction for the Mills ratio with its first term cancelled,
// lambda(s) + s = 1/(x + 2/(x + 3/(x + ... 16/x))), written as 1/(x c) with
// c = 1 + 2u/(1 + 3u/(1 + ... 16u)), u = 1/x^2 <= 1/16, and c evaluated by the
// forward three-term recurrence (fused multiply-adds on positive terms, one
// division); 15 levels give ~5e-10 relative at x = 4 and less beyond.  Elsewhere
// sqrt(2/pi)/erfcx(-s/sqrt 2) + s, which tends to s for large s as erfcx overflows.
__device__ __forceinline__ float gprime_cf(float s) {
  const float x = fmaxf(-s, 4.0f);
  const float u = frcp_fast(x * x);
  float a0 = 1.0f, a1 = 1.0f, b0 = 0.0f, b1 = 1.0f;  // A_{n-2}, A_{n-1}, B_{n-2}, B_{n-1}
#pragma unroll
  for (int n = 2; n <= 16; ++n) {
    const float an = (float)n * u;
    const float a2 = fmaf(an, a0, a1), b2 = fmaf(an, b0, b1);
    a0 = a1; a1 = a2; b0 = b1; b1 = b2;
  }
  return b1 * frcp_fast(x * a1);
}
__device__ __forceinline__ float gprime_ex(float s) {
  // lambda(s) = sqrt(2/pi) / erfcx(-s/sqrt 2); erfcx = +inf (s above ~13) gives 0
  const float e = erfcx_any(-s * kSqrtHalf);
  return (isinf(e) ? 0.0f : __fdividef(0.79788456080286536f, e)) + s;
}

// g(hi) - g(hi - h) for h >= 0; the interval length is exactly h.  The direct
// difference of two g values is accurate to a few 1e-7 absolute (|g| <= ~3 for
// arguments above -8); it is replaced by 8-point Gauss-Legendre quadrature of g'
// where the difference itself is small: short intervals and the deep left tail
// (g' ~ 1/|s| there).  The choice of form (and, inside the quadrature, of the
// form of g') is voted over the converged lanes, and every form that some lane
// needs is evaluated by all of them as straight-line code (the eight nodes
// interleave); lanes with different arguments therefore never diverge.
static __device__ SDV_HELPER float gdiff(float hi, float h) {
  const unsigned act = __activemask();
  const bool careful = ((h < 0.5f) || (hi < -2.0f)) && (h <= fmaxf(2.0f, 0.5f * fabsf(hi)));
  float quad = 0.0f, direct = 0.0f;
  if (__any_sync(act, careful)) {
    const float r = 0.5f * h, m = hi - r;
    float sv[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      sv[2 * i] = m + r * kGLx[i];
      sv[2 * i + 1] = m - r * kGLx[i];
    }
    // nodes lie in [hi - h, hi]
    const bool need_cf = __any_sync(act, careful && hi - h < -4.0f);
    const bool need_ex = __any_sync(act, careful && hi >= -4.0f);
    float gp[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) gp[i] = 0.0f;
    if (need_ex) {
#pragma unroll kGLUnroll
      for (int i = 0; i < 8; ++i) gp[i] = gprime_ex(sv[i]);
    }
    if (need_cf) {
#pragma unroll kGLUnroll
      for (int i = 0; i < 8; ++i) {
        const float cf = gprime_cf(sv[i]);
        gp[i] = (sv[i] < -4.0f) ? cf : gp[i];
      }
    }
    float acc = 0.0f;
#pragma unroll
    for (int i = 0; i < 4; ++i) acc += kGLw[i] * (gp[2 * i] + gp[2 * i + 1]);
    quad = r * acc;
  }
  if (__any_sync(act, !careful)) {
    const float lo = hi - h;
    const float2 ph = log_ndtr_g(hi), pl = log_ndtr_g(lo);
    direct = (hi <= 0.0f) ? ph.y - pl.y : (ph.x - pl.x) + h * (hi - 0.5f * h);
  }
  return careful ? quad : direct;
}

// log(1 - e^x), x <= 0 (both forms evaluated, one selected).
__device__ __forceinline__ float log1mexp(float x) {
  x = fminf(x, 0.0f);
  const float near0 = logf(-expm1f(x));
  const float far = log1pf(-expf(x));
  return (x > -kLn2) ? near0 : far;
}

// log(e^y - 1), y >= 0 (both forms evaluated, one selected).
__device__ __forceinline__ float logexpm1(float y) {
  const float big = y + log1pf(-expf(-y));
  const float small = logf(expm1f(fminf(y, 15.0f)));
  return (y > 15.0f) ? big : small;
}

__device__ __forceinline__ float logaddexp(float a, float b) {
  const float m = fmaxf(a, b);
  if (m == -INFINITY) return -INFINITY;
  return m + log1pf(expf(-fabsf(a - b)));
}

// log(Phi(b) - Phi(a)) for a < b.
static __device__ SDV_HELPER float log_ndtr_interval(float a, float b) {
  if (b <= 0.0f) return log_ndtr(b) + log1mexp(log_ndtr(a) - log_ndtr(b));
  if (a >= 0.0f) return log_ndtr(-a) + log1mexp(log_ndtr(-b) - log_ndtr(-a));
  return log1pf(-(expf(log_ndtr(a)) + expf(log_ndtr(-b))));
}

// ---------------------------------------------------------------- block verification
// log h_j, h_j = v_j / (v_j + 1 - alpha_j), from log alpha_j (<= 0), |Delta_{j+1}| and
// log v_j, the residual mass of step j + 1 at alpha_j (usample_setup(|Delta_{j+1}|,
// log alpha_j).lv).  Limits: alpha_j = 1 -> h = 1; alpha_j = 0 or |Delta_{j+1}| = 0
// (alpha_j < 1) -> h = 0.
__device__ __forceinline__ float block_log_h(float la, float Dn, float lv) {
  if (isnan(la) || isnan(Dn)) return -INFINITY;
  if (!(la < 0.0f)) return 0.0f;
  if (la == -INFINITY || !(Dn > 0.0f)) return -INFINITY;
  return lv - logaddexp(lv, log1mexp(la));
}

// log h_j from log alpha_j and |Delta_{j+1}| alone (evaluates log v_j).
static __device__ SDV_HELPER float block_log_h(float la, float Dn) {
  if (isnan(la) || isnan(Dn) || !(la < 0.0f) || la == -INFINITY || !(Dn > 0.0f))
    return block_log_h(la, Dn, 0.0f);  // the limits, which do not read log v
  const float ap = la * frcp_fast(Dn) + 0.5f * Dn;
  const float x0 = -gdiff(ap, Dn);              // log(Phi(a-) / (alpha Phi(a+)))
  const float lv = la + log_ndtr(ap) + log1mexp(x0);
  return block_log_h(la, Dn, lv);
}

// ---------------------------------------------------------------- residual U-sampler
struct UParams {
  float D, la, ap, am;
  float lv;      // log v
  float lvn;     // log v - log phi(a-)
  float lnd_ap;  // log Phi(a+)
  float g_ap;    // g(a+)
  float l1mx0;   // log(1 - e^{x0}) = log(v / (alpha Phi(a+)))
};

static __device__ SDV_HELPER UParams usample_setup(float D, float la) {
  UParams P;
  P.D = D;
  P.la = la;
  P.ap = la * frcp_fast(D) + 0.5f * D;
  P.am = P.ap - D;
  const float x0 = -gdiff(P.ap, D);
  const float2 lg = log_ndtr_g(P.ap);
  P.lnd_ap = lg.x;
  P.g_ap = lg.y;
  P.l1mx0 = log1mexp(x0);
  P.lv = la + P.lnd_ap + P.l1mx0;
  P.lvn = gfun(P.am) + kHalfLog2Pi + logexpm1(-x0);
  return P;
}

// log Psi(a+ - t), t > 0, as [log Phi(u) - log Phi(a+)] + log(1 - e^x) - log(1 - e^{x0}),
// u = a+ - t: Psi(u) = alpha Phi(u) (1 - e^x) / v and v = alpha Phi(a+) (1 - e^{x0}).
// The first bracket is g(u) - g(a+) + t (a+ + u)/2 for a+ <= 0 (no term larger than
// the result grows with |a+|) and a plain difference of log Phi otherwise.
static __device__ SDV_HELPER float usample_log_psi(float t, const UParams& P) {
  const float u = P.ap - t;
  const float x = -gdiff(u, P.D) - P.D * t;     // log(Phi(u - D) / (alpha Phi(u)))
  const float2 lg = log_ndtr_g(u);
  const float dl = (P.ap <= 0.0f) ? (lg.y - P.g_ap) + 0.5f * t * (P.ap + u) : lg.x - P.lnd_ap;
  return dl + log1mexp(x) - P.l1mx0;
}

// log(1 - Psi(a+ - t)), t > 0.
static __device__ SDV_HELPER float usample_log_1mpsi(float t, const UParams& P) {
  if (P.D * t <= 1.0f && -P.am * t <= 4.0f) {
    const float r = 0.5f * t;
    float acc = 0.0f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float s1 = r * (1.0f + kGLx[i]), s2 = r * (1.0f - kGLx[i]);
      acc += kGLw[i] * (expf(P.am * s1 - 0.5f * s1 * s1) * expm1f(P.D * s1) +
                        expf(P.am * s2 - 0.5f * s2 * s2) * expm1f(P.D * s2));
    }
    return logf(r * acc) - P.lvn;
  }
  const float u = P.ap - t;
  const float lA = P.la + log_ndtr_interval(u, P.ap);
  const float lB = log_ndtr_interval(u - P.D, P.am);
  return lA + log1mexp(lB - lA) - P.lv;
}

// log psi(a+ - t) (the residual's density at u = a+ - t), in the form whose terms do
// not cancel: a- t - t^2/2 + log expm1(D t) - (log v - log phi(a-)) keeps every term
// small when t is small (the deep left tail), while log alpha + log phi(u) +
// log(1 - e^{-D t}) - log v does when u is moderate and D t is large (large |Delta|,
// where the first form cancels terms of size D^2/2).
__device__ __forceinline__ float usample_log_density(float t, const UParams& P) {
  const float u = P.ap - t;
  const float mag1 = fmaxf(fabsf(P.am * t), fmaxf(0.5f * t * t, P.D * t));
  const float mag2 = fmaxf(0.5f * u * u, fmaxf(fabsf(P.la), fabsf(P.lv)));
  if (mag1 <= mag2) return P.am * t - 0.5f * t * t + logexpm1(P.D * t) - P.lvn;
  return P.la - 0.5f * u * u - kHalfLog2Pi + log1mexp(-P.D * t) - P.lv;
}

// Bracket widths (in t, i.e. in u) above which one Newton step from the bracket is not
// accurate enough: the residual's bulk has unit scale, so a bracket of 1e-2 leaves an
// error of ~1e-4 after one step and ~1e-8 after two.  The multisection leaves brackets
// of about 3.5e-4 t, wider than this only for t above ~30, i.e. |Delta| of ~60 and more.
constexpr float kUPolishWidth = 1e-2f;
constexpr int kUPolishIters = 8;

// Newton step from the end of [lo, hi] with the smaller |gap|, clamped to the bracket;
// returns u = a+ - t directly (u_e = fl(a+ - t_e) is the point the evaluator used, so
// the correction keeps U's rounding relative to |U| rather than to |a+|).
__device__ __forceinline__ float usample_newton(const UParams& P, bool upper, float target, float lo,
                                                float glo, float hi, float ghi) {
  const bool from_lo = isfinite(glo) && (-glo < ghi);
  const float te = from_lo ? lo : hi, ge = from_lo ? glo : ghi;
  const float lpsi = usample_log_density(te, P);
  const float lden = upper ? ge + target : target - ge;   // log(1 - Psi) or log Psi at te
  const float dg = expf(lpsi - lden);
  const float ue = P.ap - te;
  float step = (isfinite(dg) && dg > 0.0f && isfinite(ge)) ? ge * frcp_fast(dg) : 0.0f;
  step = fminf(fmaxf(step, te - hi), te - lo);   // stay inside the bracket
  return ue + step;
}

// While the bracket is wider than kUPolishWidth: evaluate the gap at the Newton point
// (the bracket's midpoint if that point is not strictly inside) and keep the half that
// holds the root (safeguarded Newton).  Every thread passes and gets the same values.
template <typename Gap>
__device__ __forceinline__ void usample_polish(const UParams& P, bool upper, float target, const Gap& gap,
                                               float& lo, float& glo, float& hi, float& ghi) {
#pragma unroll 1
  for (int it = 0; it < kUPolishIters && hi - lo > kUPolishWidth; ++it) {
    float t = P.ap - usample_newton(P, upper, target, lo, glo, hi, ghi);
    if (!(t > lo && t < hi)) t = 0.5f * (lo + hi);
    const float gt = gap(t);
    if (!(gt == gt)) break;
    if (gt >= 0.0f) { hi = t; ghi = gt; } else { lo = t; glo = gt; }
  }
}

// Shared scratch of usample_block.
struct USampleScratch {
  int first[32];
  float t[2];
  float g[2];
};

// U = Psi_alpha^{-1}(w), w = (wbits + 1/2) 2^-32, by all NT threads of a CTA (NT a
// multiple of 32, <= 1024) with the same arguments (P from usample_setup); every
// thread returns U.
// Work in t = a+ - u (Psi decreases in t) with the gap g(t) = log w - log Psi
// (lower half of w) or log(1 - Psi) - log(1 - w) (upper half), increasing in t
// and >= 0 exactly when Psi(a+ - t) <= w:
//  1. bracket: NT candidates t_k = s0 2^(k/8 - 8) (the paper's doubling of the
//     bracket, eight steps per octave, all at once), s0 = 1/max(1, |a-|) the
//     scale of the residual's spread;
//  2. one round of NT-way multisection;
//  3. while the bracket is wider than kUPolishWidth (large |Delta| only), safeguarded
//     Newton steps with the gap evaluated at each new point;
//  4. one Newton step from the bracket end with the smaller |g|, clamped to the
//     bracket.  g' = psi / Psi (or psi / (1 - Psi)) with the density in closed form
//     (usample_log_density).
template <int NT>
__device__ __forceinline__ float usample_block(const UParams& P, uint32_t wbits, uint32_t* status,
                                               USampleScratch* sm) {
  const unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool upper = wbits >= 0x80000000u;
  const float target = upper ? logf(((float)(0xFFFFFFFFu - wbits) + 0.5f) * 0x1p-32f)
                             : logf(((float)wbits + 0.5f) * 0x1p-32f);
  auto gap = [&](float t) -> float {
    if (upper) return usample_log_1mpsi(t, P) - target;
    return target - usample_log_psi(t, P);
  };
  auto first_true = [&](bool pred) -> int {  // smallest tid with pred (NT if none)
    const unsigned m = __ballot_sync(FULL, pred);
    if (lane == 0) sm->first[warp] = m ? warp * 32 + __ffs(m) - 1 : NT;
    __syncthreads();
    int f = NT;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) f = min(f, sm->first[w]);
    __syncthreads();
    return f;
  };
  const float s0 = frcp_fast(fmaxf(1.0f, fabsf(P.am)));
  const float tk = s0 * exp2f((float)tid * 0.125f - 8.0f);
  const float gk = gap(tk);
  int f = first_true(gk >= 0.0f);
  if (f == NT) {
    *status |= 4u;  // SDV_STATUS_USAMPLE_RANGE
    return P.ap - s0 * exp2f((float)NT * 0.125f - 8.0f);
  }
  if (tid == f) { sm->t[1] = tk; sm->g[1] = gk; }
  if (tid == f - 1) { sm->t[0] = tk; sm->g[0] = gk; }
  __syncthreads();
  float hi = sm->t[1], ghi = sm->g[1];
  float lo = (f == 0) ? 0.0f : sm->t[0];
  float glo = (f == 0) ? -INFINITY : sm->g[0];
  __syncthreads();
  {
    const float h = (hi - lo) * (1.0f / (float)NT);
    const float t = (tid < NT - 1) ? lo + (float)(tid + 1) * h : hi;
    const float gt = (tid < NT - 1) ? gap(t) : ghi;
    f = first_true(gt >= 0.0f);
    if (tid == f) { sm->t[1] = t; sm->g[1] = gt; }
    if (tid == f - 1) { sm->t[0] = t; sm->g[0] = gt; }
    __syncthreads();
    if (f > 0) { lo = sm->t[0]; glo = sm->g[0]; }
    hi = sm->t[1];
    ghi = sm->g[1];
    __syncthreads();
  }
  usample_polish(P, upper, target, gap, lo, glo, hi, ghi);
  return usample_newton(P, upper, target, lo, glo, hi, ghi);
}

// U = Psi_alpha^{-1}(w), w = (wbits + 1/2) 2^-32, by one converged warp: every lane
// passes the same P (from usample_setup) and wbits and returns U.  Work in
// t = a+ - u (Psi decreases in t) with the gap g(t) = log w - log Psi (lower half
// of w) or log(1 - Psi) - log(1 - w) (upper half), increasing in t and >= 0
// exactly when Psi(a+ - t) <= w:
//  1. bracket: the 32 candidates t_k = s0 2^(k - 8) (the paper's doubling of the
//     bracket, all steps at once), s0 = 1/max(1, |a-|) the residual's scale;
//  2. kURounds rounds of 32-way multisection (each shrinks the bracket 32-fold);
//  3. while the bracket is wider than kUPolishWidth (large |Delta| only), safeguarded
//     Newton steps with the gap evaluated at each new point;
//  4. one Newton step from the bracket end with the smaller |g|, clamped to the
//     bracket.  g' = psi / Psi (or psi / (1 - Psi)) with the density in closed form
//     (usample_log_density).
constexpr int kURounds = 3;

__device__ __forceinline__ float usample_warp(const UParams& P, uint32_t wbits, uint32_t* status) {
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const bool upper = wbits >= 0x80000000u;
  const float target = upper ? logf(((float)(0xFFFFFFFFu - wbits) + 0.5f) * 0x1p-32f)
                             : logf(((float)wbits + 0.5f) * 0x1p-32f);
  auto gap = [&](float t) -> float {
    if (upper) return usample_log_1mpsi(t, P) - target;
    return target - usample_log_psi(t, P);
  };
  const float s0 = frcp_fast(fmaxf(1.0f, fabsf(P.am)));
  const float tk = s0 * exp2f((float)lane - 8.0f);
  const float gk = gap(tk);
  unsigned m = __ballot_sync(FULL, gk >= 0.0f);
  if (m == 0u) {
    *status |= 4u;  // SDV_STATUS_USAMPLE_RANGE
    return P.ap - s0 * exp2f(24.0f);
  }
  int f = __ffs(m) - 1;
  float hi = __shfl_sync(FULL, tk, f), ghi = __shfl_sync(FULL, gk, f);
  const float tp = __shfl_sync(FULL, tk, (f + 31) & 31), gp = __shfl_sync(FULL, gk, (f + 31) & 31);
  float lo = (f == 0) ? 0.0f : tp;
  float glo = (f == 0) ? -INFINITY : gp;
#pragma unroll 1
  for (int r = 0; r < kURounds; ++r) {
    const float h = (hi - lo) * (1.0f / 32.0f);
    const float t = (lane < 31) ? lo + (float)(lane + 1) * h : hi;
    const float gt0 = gap(t);                 // every lane evaluates (converged votes)
    const float gt = (lane < 31) ? gt0 : ghi;  // the upper end keeps its known value
    m = __ballot_sync(FULL, gt >= 0.0f);       // lane 31 always votes true
    f = __ffs(m) - 1;
    const float nt = __shfl_sync(FULL, t, f), ng = __shfl_sync(FULL, gt, f);
    const float pt = __shfl_sync(FULL, t, (f + 31) & 31), pg = __shfl_sync(FULL, gt, (f + 31) & 31);
    if (f > 0) { lo = pt; glo = pg; }
    hi = nt;
    ghi = ng;
  }
  usample_polish(P, upper, target, gap, lo, glo, hi, ghi);
  return usample_newton(P, upper, target, lo, glo, hi, ghi);
}

// ---------------------------------------------------------------- tickets
// Fetch-and-add of 1 with acquire-release semantics at GPU scope: the release
// publishes this thread's earlier writes, and the holder of the last ticket
// acquires every write released before it.
__device__ __forceinline__ unsigned int ticket_acq_rel(unsigned int* p) {
  unsigned int old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(p) : "memory");
  return old;
}

// ---------------------------------------------------------------- element access
template <typename T> struct Elem;
template <> struct Elem<float> {
  static __device__ __forceinline__ float load(const float* p) { return __ldg(p); }
  static __device__ __forceinline__ void store(float* p, float v) { *p = v; }
};
template <> struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ float load(const __nv_bfloat16* p) {
    return __bfloat162float(__ldg(p));
  }
  static __device__ __forceinline__ void store(__nv_bfloat16* p, float v) {
    *p = __float2bfloat16_rn(v);
  }
};

}  // namespace sdv
