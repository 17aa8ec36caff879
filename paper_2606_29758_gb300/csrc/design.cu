// Cutoff-distribution design on the device (the step upstream of the sampler).
//
//  ps_lmhead_score_proxy: per token, the output-head score proxy of Appendix D,
//      gamma = ||h||^2 (1 - 2 p(o) + ||p||^2),
//  and log p(o), from one pass of the LM-head GEMM (the forward's schedule) whose epilogue keeps
//  two running exponential sums (||p||^2 from the two-logsumexp identity).
//  ps_design_cutoffs: per prompt, the group average of gamma at each step (Section 3.3), timestep
//  weights w = gamma_bar * u, the budgeted monotone xi of Appendix F (closed form + pooling of
//  adjacent violators + the xi <= 1 cap), or one of the Section 4 variants, and the integer
//  masses the sampler takes (the deficit is Pr(H = 0)).
//
// The design arithmetic is sequential float64 with explicitly rounded operations (no FMA
// contraction), so the masses are reproducible bit for bit.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <cstdint>

#include "ps_nvtx.h"
#include "internal.h"
#include "ps_common.cuh"
#include "psppo.h"

namespace psk {

static size_t al256(size_t x) { return (x + 255) / 256 * 256; }

// ================================================================== score proxy
__global__ void row_sqnorm_kernel(int64_t N, int d, int is_bf16, const void* __restrict__ H,
                                  float* __restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); i < N; i += warps) {
    float acc = 0.f;
    if (is_bf16) {
      const uint4* r = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(H) + i * d);
      for (int c = lane; c < d / 8; c += 32) {
        const uint4 v = r[c];
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float a = __uint_as_float(w4[k] << 16), b = __uint_as_float(w4[k] & 0xFFFF0000u);
          acc = fmaf(a, a, fmaf(b, b, acc));
        }
      }
    } else {
      const float* r = static_cast<const float*>(H) + i * d;
      for (int c = lane; c < d; c += 32) acc = fmaf(r[c], r[c], acc);
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) out[i] = acc;
  }
}

__global__ void proxy_finalize_kernel(int64_t N, int V, int splits, const float4* __restrict__ part,
                                      const float* __restrict__ ztok, const float* __restrict__ hn,
                                      const int32_t* __restrict__ tok, float* __restrict__ gamma,
                                      float* __restrict__ logp, int topk_k, const float2* __restrict__ topk_part,
                                      int32_t* __restrict__ top_idx, float* __restrict__ top_prob,
                                      uint32_t* status) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= N) return;
  float m = -INFINITY;
  for (int s = 0; s < splits; ++s) m = fmaxf(m, part[static_cast<int64_t>(s) * N + i].x);
  double S1 = 0.0, S2 = 0.0;
  for (int s = 0; s < splits; ++s) {
    const float4 pr = part[static_cast<int64_t>(s) * N + i];
    const double f = exp2(static_cast<double>(pr.x) - m);
    S1 += pr.y * f;
    S2 += pr.z * f * f;
  }
  const int t = tok[i];
  if (t < 0 || t >= V) {
    raise_status(status, PS_DEV_BAD_TOKEN);
    gamma[i] = NAN;
    if (logp) logp[i] = NAN;
    return;
  }
  // S1, S2: sums over the other columns; e_o = 2^(x_o - m) for the chosen one
  const double x = static_cast<double>(ztok[i]) * 1.4426950408889634 - m;
  const double eo = exp2(x);
  const double tot = eo + S1;
  gamma[i] = static_cast<float>(static_cast<double>(hn[i]) * ((S1 * S1 + S2) / (tot * tot)));
  if (logp) logp[i] = static_cast<float>((x - log2(tot)) * 0.6931471805599453);
  if (topk_k > 0) {
    // merge the ranges' lists (each descending, lower column first on ties), ranges in order
    float v[16];
    int id[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      v[j] = -INFINITY;
      id[j] = -1;
    }
    for (int sp = 0; sp < splits; ++sp) {
      const float2* lst = topk_part + (static_cast<int64_t>(sp) * N + i) * 16;
      for (int c = 0; c < 16; ++c) {
        const float2 e = lst[c];
        float xv = e.x;
        int xi = __float_as_int(e.y);
        if (!(xv > v[15])) continue;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const bool take = xv > v[j];
          const float tv = v[j];
          const int ti = id[j];
          v[j] = take ? xv : tv;
          id[j] = take ? xi : ti;
          xv = take ? tv : xv;
          xi = take ? ti : xi;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      if (j < topk_k) {
        top_idx[i * topk_k + j] = id[j];
        top_prob[i * topk_k + j] =
            static_cast<float>(exp2(static_cast<double>(v[j]) * 1.4426950408889634 - m) / tot);
      }
    }
  }
}

// ================================================================== reward uncertainty
// One warp per (prompt, step t): the group's completions that reach t contribute their top-k
// next-token probabilities with coefficient p_hat / |G_t| (success) or -(1 - p_hat) / |B_t|
// (failure); u_t = 1/2 - 1/2 (sum over distinct tokens |sum of contributions| + |other mass|).
constexpr int kUncWarps = 4;
__global__ void __launch_bounds__(kUncWarps * 32)
    uncertainty_kernel(int P, int K, int T_max, const int32_t* __restrict__ L, const float* __restrict__ R,
                       int topk, const int32_t* __restrict__ top_idx, const float* __restrict__ top_prob,
                       const int64_t* __restrict__ off, float* __restrict__ u) {
  extern __shared__ uint8_t smem[];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int cap = K * topk;
  int32_t* etok = reinterpret_cast<int32_t*>(smem) + wid * cap;
  double* eval = reinterpret_cast<double*>(smem + sizeof(int32_t) * kUncWarps * cap + 16) + wid * cap;
  const int64_t task = static_cast<int64_t>(blockIdx.x) * kUncWarps + wid;
  if (task >= static_cast<int64_t>(P) * T_max) return;
  const int p = static_cast<int>(task / T_max);
  const int t = static_cast<int>(task % T_max);   // 0-based step
  int nG = 0, gA = 0, bA = 0, Tp = 0;
  for (int j = 0; j < K; ++j) {
    const int k = p * K + j;
    const bool g = R[k] >= 0.5f;
    nG += g;
    gA += (g && L[k] > t);
    bA += (!g && L[k] > t);
    Tp = max(Tp, L[k]);
  }
  if (t >= Tp) {
    if (lane == 0) u[static_cast<int64_t>(p) * T_max + t] = 0.f;
    return;
  }
  const double phat = static_cast<double>(nG) / K;
  const double cg = gA > 0 ? phat / gA : 0.0, cb = bA > 0 ? -(1.0 - phat) / bA : 0.0;
  // entries of the alive completions, in completion order
  int E = 0;
  double other = 0.0;
  for (int j = 0; j < K; ++j) {
    const int k = p * K + j;
    if (L[k] <= t) continue;
    const double c = R[k] >= 0.5f ? cg : cb;
    const int64_t row = off[k] + t;
    double tot = 0.0;
    for (int i = lane; i < topk; i += 32) {
      etok[E + i] = top_idx[row * topk + i];
      const double pv = top_prob[row * topk + i];
      eval[E + i] = c * pv;
      tot += pv;
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    other += c * (1.0 - tot);
    E += topk;
  }
  __syncwarp();
  double acc = 0.0;
  for (int e = lane; e < E; e += 32) {
    const int tk = etok[e];
    bool first = true;
    for (int f = 0; f < e && first; ++f) first = etok[f] != tk;
    if (!first) continue;
    double sum = 0.0;
    for (int f = e; f < E; ++f)
      if (etok[f] == tk) sum += eval[f];
    acc += fabs(sum);
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) {
    const double l1 = acc + fabs(other);
    u[static_cast<int64_t>(p) * T_max + t] = static_cast<float>(fmin(0.5, fmax(0.0, 0.5 - 0.5 * l1)));
  }
}

__global__ void group_offsets_kernel(int B, const int32_t* __restrict__ L, int64_t* __restrict__ off) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    int64_t o = 0;
    for (int k = 0; k < B; ++k) {
      off[k] = o;
      o += L[k];
    }
  }
}

// ================================================================== design
// Lanes of the warp that tries saturated prefixes side by side in the capped design.
constexpr int kCapLanes = 32;

struct DesignWs {
  double* w;       // [P][T_max] weights
  double* xi;      // [P][T_max]
  double* bW;      // [P][T_max][kCapLanes] PAV block weights, one stack per lane (interleaved)
  double* bs;      // [P][T_max][kCapLanes] PAV block scores sqrt(W / n)
  int32_t* bn;     // [P][T_max][kCapLanes] PAV block lengths
  int64_t* off;    // [P][K] row offsets of the group's completions
};

// True when the block (Wc, nc) violates the order against the block (Wp, np) below it, i.e. when
// sqrt(Wp / np) < sqrt(Wc / nc) with both quotients and roots rounded to double, exactly as the
// sequential definition decides it. The cross products Wp nc and Wc np settle every case whose
// quotients differ by more than 2^-40 relative (then the rounded roots are ordered the same way);
// only near-ties pay for the two divisions and square roots, which are slow in double precision.
__device__ __forceinline__ bool pav_violates(double Wp, int np, double Wc, int nc) {
  const double a = __dmul_rn(Wp, static_cast<double>(nc));
  const double b = __dmul_rn(Wc, static_cast<double>(np));
  if (a > 0x1p-900 && b > 0x1p-900 && a < 0x1p900 && b < 0x1p900) {
    if (b > __dmul_rn(a, 1.0 + 0x1p-40)) return true;
    if (b < __dmul_rn(a, 1.0 - 0x1p-40)) return false;
  }
  return __dsqrt_rn(__ddiv_rn(Wp, static_cast<double>(np))) < __dsqrt_rn(__ddiv_rn(Wc, static_cast<double>(nc)));
}

// Pool adjacent violators over w[0..T) (Appendix F) into one lane's stack (element m of the stack
// at index m * kCapLanes): a new block is merged with the one below it while the block below has
// the smaller score sqrt(W / n); merged weights add as W_prev + W_last, in the order of the
// sequential definition, so every block sum is the same double. Returns the number of blocks (-1
// if *stop was set before the end).
__device__ int pav_stack_dev(const double* w, int T, double* bW, int32_t* bn, const volatile int* stop = nullptr) {
  // The top block stays in registers (Wt, nt); the blocks below it are in memory at [0, nb - 1).
  // Memory is read only when a merge uncovers the block below.
  int nb = 0;
  double Wt = 0.0;
  int nt = 0;
  double wnext = T > 0 ? w[0] : 0.0;
  for (int t0 = 0; t0 < T; t0 += 64) {
    if (stop != nullptr && *stop) return -1;   // abandoned: the caller needs no answer
    const int t1 = min(T, t0 + 64);
    for (int t = t0; t < t1; ++t) {
      if (t + 16 < T) asm volatile("prefetch.global.L1 [%0];" ::"l"(w + t + 16));
      double Wc = wnext;
      if (t + 1 < T) wnext = w[t + 1];
      int nc = 1;
      while (nb > 0 && pav_violates(Wt, nt, Wc, nc)) {
        Wc = __dadd_rn(Wt, Wc);
        nc += nt;
        --nb;
        if (nb > 0) {
          Wt = bW[(nb - 1) * kCapLanes];
          nt = bn[(nb - 1) * kCapLanes];
        }
      }
      if (nb > 0) {
        bW[(nb - 1) * kCapLanes] = Wt;
        bn[(nb - 1) * kCapLanes] = nt;
      }
      Wt = Wc;
      nt = nc;
      ++nb;
    }
  }
  if (nb > 0) {
    bW[(nb - 1) * kCapLanes] = Wt;
    bn[(nb - 1) * kCapLanes] = nt;
  }
  return nb;
}

// ---------------------------------------------------------------- capped design: locating the prefix
// The capped design saturates the smallest prefix s whose suffix design (w[s..T), budget B - s)
// starts at or below 1. Whether a prefix qualifies is not monotone in s, so it cannot be bisected;
// instead one pass of pooling from the right gives every suffix's first value at once: once w[t]
// has been pushed (and pooled with the blocks to its right while it violates the order), the stack
// holds the pooled blocks of the suffix w[t..T), because the pooled solution of a suffix is unique
// whatever order its violators are pooled in (only the rounding of the block sums depends on it).
// With D(t) = sum over those blocks of n_m s_m = sqrt(n_m W_m), the suffix design starts at
// g(t) = (B - t) s_front / D(t). The pass records whether g(t) is clearly above 1 (0), clearly
// below (2) or within kCapBand of 1 (1); only the last kind, and the first clear one, are then
// decided by the exact rounded sequence of the definition.
constexpr double kCapBand = 0x1p-16;
constexpr int kMaxNearCap = 64;        // prefixes within the band decided exactly (beyond: the full scan)
constexpr int kCapStackSmem = 8192;    // stack entries of the status pass held in shared memory

// Float-float numbers (an unevaluated sum hi + lo of two floats, about 44 significant bits): the
// status pass's block sums and D. Knuth's TwoSum and the Dekker renormalisation.
struct FF {
  float hi, lo;
};
__device__ __forceinline__ FF ff_add(FF a, FF b) {
  const float s = a.hi + b.hi;
  const float bb = s - a.hi;
  const float e = (a.hi - (s - bb)) + (b.hi - bb) + a.lo + b.lo;
  const float h = s + e;
  return FF{h, e - (h - s)};
}

// One thread: status[t] for t = T-1 down to 0 (see above), in float arithmetic (the FP64 units are
// far slower). ws[t] = w[t] / max_t w[t] as floats (g does not depend on the scale, and every
// n W then lies in [1e-12, T]); block sums and D as float-float numbers, roots and the comparison
// in float: g is within about 2e-7 relative of its exact value, far inside kCapBand. The stack keeps
// its front block in registers, the next kCapStackSmem entries in shared memory (W, n and the
// root r = sqrt(n W) of each block, so that a pooled block leaves D as it entered) and deeper ones
// in gW / gn / gr with stride kCapLanes. Stops early once *stop is set.
__device__ void cap_status_pass(const float* __restrict__ ws, int T, double B, float2* sW, int32_t* sn, float* sr,
                                double* gW, int32_t* gn, double* gr, float* status, const volatile int* stop) {
  int nb = 0;            // blocks below the front
  FF Wf{0.f, 0.f};       // front block
  int nf = 0;
  float rf = 0.f;
  FF D{0.f, 0.f};
  const float hi_band = static_cast<float>(1.0 + kCapBand), lo_band = static_cast<float>(1.0 - kCapBand);
  for (int t = T - 1; t >= 0; --t) {
    if ((t & 255) == 0 && *stop) return;   // the prefix s = 0 already qualifies: no status is needed
    if (t >= 32) asm volatile("prefetch.global.L1 [%0];" ::"l"(ws + t - 32));
    FF Wc{ws[t], 0.f};
    int nc = 1;
    // the new block sits left of the front: pool while its mean is below the front's
    while (nf > 0 && Wf.hi * static_cast<float>(nc) > Wc.hi * static_cast<float>(nf)) {
      D = ff_add(D, FF{-rf, 0.f});
      Wc = ff_add(Wc, Wf);
      nc += nf;
      if (nb > 0) {
        --nb;
        if (nb < kCapStackSmem) {
          const float2 v = sW[nb];
          Wf = FF{v.x, v.y};
          nf = sn[nb];
          rf = sr[nb];
        } else {
          const float2 v = reinterpret_cast<const float2*>(gW)[static_cast<int64_t>(nb) * kCapLanes];
          Wf = FF{v.x, v.y};
          nf = gn[static_cast<int64_t>(nb) * kCapLanes];
          rf = static_cast<float>(gr[static_cast<int64_t>(nb) * kCapLanes]);
        }
      } else {
        nf = 0;
      }
    }
    if (nf > 0) {
      if (nb < kCapStackSmem) {
        sW[nb] = make_float2(Wf.hi, Wf.lo);
        sn[nb] = nf;
        sr[nb] = rf;
      } else {
        reinterpret_cast<float2*>(gW)[static_cast<int64_t>(nb) * kCapLanes] = make_float2(Wf.hi, Wf.lo);
        gn[static_cast<int64_t>(nb) * kCapLanes] = nf;
        gr[static_cast<int64_t>(nb) * kCapLanes] = rf;
      }
      ++nb;
    }
    Wf = Wc;
    nf = nc;
    rf = sqrtf(static_cast<float>(nc) * Wc.hi);
    D = ff_add(D, FF{rf, 0.f});
    const float num = static_cast<float>(B - static_cast<double>(t)) * rf, den = D.hi * static_cast<float>(nc);
    status[t] = num > hi_band * den ? 0.f : (num < lo_band * den ? 2.f : 1.f);
  }
}

constexpr size_t kDesignDynSmem = kCapStackSmem * (sizeof(float2) + sizeof(int32_t) + sizeof(float));

constexpr int kDesignThreads = 256;

// One CTA per prompt (and 128 KB of shared memory each): registers are not what limits residency.
__global__ void __launch_bounds__(kDesignThreads, 1)
    design_kernel(int K, int T_max, const int32_t* __restrict__ L, const float* __restrict__ gamma,
                  const float* __restrict__ u, double budget, int strategy, double param, uint64_t* __restrict__ q,
                  double* __restrict__ xi_out, DesignWs ws, uint32_t* status) {
  const int p = blockIdx.x;
  const int tid = threadIdx.x;
  __shared__ int Tp_s;
  __shared__ double red_d[kDesignThreads / 32];
  __shared__ unsigned long long red_u[kDesignThreads / 32];
  __shared__ unsigned long long red_b[kDesignThreads / 32];
  __shared__ long long red_l[kDesignThreads / 32];
  __shared__ int red_i[kDesignThreads / 32];
  __shared__ double lam_s;
  __shared__ int found_s, found_lane_s, ncand_s, nnear_s, tdef_s;
  __shared__ volatile int s0_ok_s, s0_skip_s;
  __shared__ int cand_s[kMaxNearCap + 1];
  __shared__ int nb_s[kCapLanes];
  __shared__ double den_s[kCapLanes];
  extern __shared__ double dyn_smem[];    // the status pass's stack (kDesignDynSmem bytes)
  const int lane = tid & 31, wid = tid >> 5;
  double* w = ws.w + static_cast<int64_t>(p) * T_max;
  double* xi = ws.xi + static_cast<int64_t>(p) * T_max;
  int64_t* off = ws.off + static_cast<int64_t>(p) * K;

  // horizon of the group, and the row offset of its first completion
  long long base = 0;
  for (int k = tid; k < p * K; k += kDesignThreads) base += L[k];
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) base += __shfl_xor_sync(0xffffffffu, base, o);
  if (lane == 0) red_l[wid] = base;
  __syncthreads();
  if (tid == 0) {
    long long b = 0;
    for (int i = 0; i < kDesignThreads / 32; ++i) b += red_l[i];
    int Tp = 0;
    for (int j = 0; j < K; ++j) {
      off[j] = b;
      b += L[p * K + j];
      Tp = max(Tp, L[p * K + j]);
    }
    if (Tp < 1 || Tp > T_max) raise_status(status, PS_DEV_BAD_LENGTH);
    Tp_s = Tp < 1 ? 1 : (Tp > T_max ? T_max : Tp);
  }
  __syncthreads();
  const int Tp = Tp_s;
  const double Bp = fmin(budget, static_cast<double>(Tp));

  if (strategy == PS_DESIGN_OPTIMIZED || strategy == PS_DESIGN_HEURISTIC) {
    // w_t = gamma_bar_t * u_t; gamma_bar_t = (1/K) sum over the completions that reach t
    double wmax = 0.0;
    for (int t = tid; t < Tp; t += kDesignThreads) {
      double acc = 0.0;
      for (int j = 0; j < K; ++j)
        if (t < L[p * K + j]) acc = __dadd_rn(acc, static_cast<double>(gamma[off[j] + t]));
      double v = __ddiv_rn(acc, static_cast<double>(K));
      if (u) v = __dmul_rn(v, static_cast<double>(u[static_cast<int64_t>(p) * T_max + t]));
      if (!isfinite(v)) raise_status(status, PS_DEV_NONFINITE);
      w[t] = v;
      wmax = fmax(wmax, v);
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) wmax = fmax(wmax, __shfl_xor_sync(0xffffffffu, wmax, o));
    if (lane == 0) red_d[wid] = wmax;
    __syncthreads();
    double wm = 0.0;
    for (int i = 0; i < kDesignThreads / 32; ++i) wm = fmax(wm, red_d[i]);
    const double fl = __dmul_rn(1e-12, wm);
    for (int t = tid; t < Tp; t += kDesignThreads) w[t] = wm > 0.0 ? (w[t] > fl ? w[t] : fl) : 1.0;
    __syncthreads();
    if (strategy == PS_DESIGN_OPTIMIZED) {
      // The smallest saturated prefix s whose suffix design (budget B - s) starts at or below 1,
      // decided by the definition's exact rounded sequence: for a candidate s, a lane of warp 0 pools
      // w[s..T) into its own stack; all threads take the blocks' scores s_m = sqrt(W_m / n_m); the
      // lane sums den = sum_m n_m s_m in block order and tests (B - s) s_1 / den <= 1. Candidates:
      // the prefixes the status pass puts within the band of 1, then the first clearly below it, in
      // increasing order; the first that passes is the answer. (If the band holds too many, or none
      // passes, the search falls back to trying every prefix in order, 32 at a time.)
      const int64_t sbase = static_cast<int64_t>(p) * T_max * kCapLanes;
      double* bW = ws.bW + sbase;
      double* bs = ws.bs + sbase;
      int32_t* bn = ws.bn + sbase;
      // xi is written last; meanwhile its 8 Tp bytes hold the scaled weights of the status pass
      // (floats, [0, Tp)) and the statuses (floats, [Tp, 2 Tp))
      float* wsc = reinterpret_cast<float*>(xi);
      float* status = wsc + Tp;
      {
        const double inv = 1.0 / (wm > 0.0 ? wm : 1.0);
        for (int t = tid; t < Tp; t += kDesignThreads) wsc[t] = static_cast<float>(w[t] * inv);
      }
      // s = 0 first, exactly (small budgets end here), on warp 0; meanwhile warp 1 runs the status
      // pass for every other prefix on a stack of its own (shared memory, then lane 31's slots), and
      // stops as soon as s = 0 has qualified.
      if (tid == 0) {
        found_s = -1;
        nnear_s = 0;
        ncand_s = 0;
        s0_ok_s = 0;
        s0_skip_s = 0;
      }
      __syncthreads();
      if (wid == 0) {
        // (abandoned when the status pass, finished first, puts s = 0 clearly above the cap)
        if (lane == 0) nb_s[0] = pav_stack_dev(w, Tp, bW, bn, &s0_skip_s);
        __syncwarp();
        const int nb0 = nb_s[0];
        for (int m = lane; m < nb0; m += 32)
          bs[m * kCapLanes] = __dsqrt_rn(__ddiv_rn(bW[m * kCapLanes], static_cast<double>(bn[m * kCapLanes])));
        __syncwarp();
        if (lane == 0) {
          double den = 0.0;
          for (int m = 0; m < nb0; ++m)
            den = __dadd_rn(den, __dmul_rn(static_cast<double>(bn[m * kCapLanes]), bs[m * kCapLanes]));
          den_s[0] = den;
          if (nb0 > 0 && __ddiv_rn(__dmul_rn(Bp, bs[0]), den) <= 1.0) {
            found_s = 0;
            found_lane_s = 0;
            s0_ok_s = 1;
          }
        }
      }
      if (wid == 1 && lane == 0) {
        float2* sW = reinterpret_cast<float2*>(dyn_smem);
        int32_t* sn = reinterpret_cast<int32_t*>(sW + kCapStackSmem);
        float* sr = reinterpret_cast<float*>(sn + kCapStackSmem);
        cap_status_pass(wsc, Tp, Bp, sW, sn, sr, bW + (kCapLanes - 1), bn + (kCapLanes - 1),
                        bs + (kCapLanes - 1), status, &s0_ok_s);
        if (!s0_ok_s && status[0] == 0.f) s0_skip_s = 1;
      }
      __syncthreads();
      int td = Tp;
      for (int t = 1 + tid; t < Tp; t += kDesignThreads)
        if (status[t] == 2.f) {
          td = t;
          break;
        }
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) td = min(td, __shfl_xor_sync(0xffffffffu, td, o));
      if (lane == 0) red_i[wid] = td;
      __syncthreads();
      if (tid == 0) {
        int m = Tp;
        for (int i = 0; i < kDesignThreads / 32; ++i) m = min(m, red_i[i]);
        tdef_s = m;
      }
      __syncthreads();
      const int tdef = tdef_s;
      if (found_s < 0)
        for (int t = 1 + tid; t < tdef; t += kDesignThreads)
          if (status[t] == 1.f) {
            const int i = atomicAdd(&nnear_s, 1);
            if (i < kMaxNearCap) cand_s[i] = t;
          }
      __syncthreads();
      if (tid == 0 && found_s < 0) {
        const int n = min(nnear_s, kMaxNearCap);
        for (int i = 1; i < n; ++i) {          // the few near-band prefixes, in increasing order
          const int v = cand_s[i];
          int j = i - 1;
          while (j >= 0 && cand_s[j] > v) {
            cand_s[j + 1] = cand_s[j];
            --j;
          }
          cand_s[j + 1] = v;
        }
        ncand_s = nnear_s > kMaxNearCap ? 0 : n + (tdef < Tp ? 1 : 0);
        if (tdef < Tp && nnear_s <= kMaxNearCap) cand_s[n] = tdef;
      }
      __syncthreads();
      // One round: lanes l < width try the prefixes start(l); sets found_s / found_lane_s.
      auto try_prefixes = [&](int width, auto start) {
        if (wid == 0) {
          const int st = lane < width ? start(lane) : Tp;
          nb_s[lane] = st < Tp ? pav_stack_dev(w + st, Tp - st, bW + lane, bn + lane) : 0;
        }
        __syncthreads();
        for (int l = 0; l < width; ++l)
          for (int m = tid; m < nb_s[l]; m += kDesignThreads)
            bs[m * kCapLanes + l] =
                __dsqrt_rn(__ddiv_rn(bW[m * kCapLanes + l], static_cast<double>(bn[m * kCapLanes + l])));
        __syncthreads();
        if (wid == 0) {
          const int st = lane < width ? start(lane) : Tp;
          bool ok = false;
          if (st < Tp) {
            double den = 0.0;
            for (int m = 0; m < nb_s[lane]; ++m)
              den = __dadd_rn(den, __dmul_rn(static_cast<double>(bn[m * kCapLanes + lane]), bs[m * kCapLanes + lane]));
            den_s[lane] = den;
            ok = __ddiv_rn(__dmul_rn(__dsub_rn(Bp, static_cast<double>(st)), bs[lane]), den) <= 1.0;
          }
          const unsigned m = __ballot_sync(0xffffffffu, ok);
          if (lane == 0 && m != 0u) {
            found_lane_s = __ffs(m) - 1;
            found_s = start(found_lane_s);
          }
        }
        __syncthreads();
      };
      const int ncand = ncand_s;
      for (int c0 = 0; c0 < ncand && found_s < 0; c0 += kCapLanes)
        try_prefixes(min(kCapLanes, ncand - c0), [&](int l) { return cand_s[c0 + l]; });
      // the exact scan over every prefix: only when the band held too many prefixes or no candidate
      // passed, which the status pass's accuracy rules out in practice
      for (int base = 1; found_s < 0 && base < Tp; base += kCapLanes)
        try_prefixes(kCapLanes, [&](int l) { return base + l; });
      const int found = found_s;
      if (found < 0) {
        for (int t = tid; t < Tp; t += kDesignThreads) xi[t] = 1.0;
      } else {
        // the design of the lane that found it: block starts by a scan, then every block in parallel
        const int l = found_lane_s;
        const int nb = nb_s[l];
        const double Bs = __dsub_rn(Bp, static_cast<double>(found));
        const double den = den_s[l];
        for (int t = tid; t < found; t += kDesignThreads) xi[t] = 1.0;
        if (tid == 0) {
          int t0 = found;
          for (int m = 0; m < nb; ++m) {
            const int n = bn[m * kCapLanes + l];
            bn[m * kCapLanes + l] = t0;          // the block's first step replaces its length
            t0 += n;
          }
        }
        __syncthreads();
        for (int m = tid; m < nb; m += kDesignThreads) {
          const double v = __ddiv_rn(__dmul_rn(Bs, bs[m * kCapLanes + l]), den);
          const int t_end = m + 1 < nb ? bn[(m + 1) * kCapLanes + l] : Tp;
          for (int t = bn[m * kCapLanes + l]; t < t_end; ++t) xi[t] = v;
        }
      }
    } else {
      // Heuristic: closed form B sqrt(w_t) / sum_j sqrt(w_j) (the sum in step order), a running
      // minimum, then the cap at 1. The roots and quotients are taken in parallel.
      for (int t = tid; t < Tp; t += kDesignThreads) xi[t] = __dsqrt_rn(w[t]);
      __syncthreads();
      if (tid == 0) {
        double tot = 0.0;
        for (int t = 0; t < Tp; ++t) tot = __dadd_rn(tot, xi[t]);
        den_s[0] = tot;
      }
      __syncthreads();
      const double tot = den_s[0];
      for (int t = tid; t < Tp; t += kDesignThreads) xi[t] = __ddiv_rn(__dmul_rn(Bp, xi[t]), tot);
      __syncthreads();
      if (tid == 0)
        for (int t = 1; t < Tp; ++t) xi[t] = fmin(xi[t - 1], xi[t]);
      __syncthreads();
      for (int t = tid; t < Tp; t += kDesignThreads) xi[t] = fmin(xi[t], 1.0);
    }
  } else if (strategy == PS_DESIGN_UNIFORM) {
    for (int t = tid; t < Tp; t += kDesignThreads)
      xi[t] = __ddiv_rn(static_cast<double>(Tp - t), static_cast<double>(Tp));
  } else if (strategy == PS_DESIGN_FIXED) {
    for (int t = tid; t < Tp; t += kDesignThreads) xi[t] = (t + 1 <= param) ? 1.0 : 0.0;
  } else {  // PS_DESIGN_TIME_PRIOR: xi_t = exp(-lam t), sum_t xi_t = budget, lam by bisection
    auto budget_at = [&](double lam) {
      double part = 0.0;
      for (int t = tid; t < Tp; t += kDesignThreads) part += exp(-lam * t);
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      __syncthreads();
      if (lane == 0) red_d[wid] = part;
      __syncthreads();
      double tot = 0.0;
      for (int i = 0; i < kDesignThreads / 32; ++i) tot += red_d[i];
      return tot;
    };
    if (static_cast<double>(Tp) <= Bp) {
      if (tid == 0) lam_s = 0.0;
    } else {
      double lo = 0.0, hi = 1.0;
      for (int it = 0; it < 64 && budget_at(hi) > Bp; ++it) hi *= 2.0;
      for (int it = 0; it < 200; ++it) {
        const double mid = 0.5 * (lo + hi);
        if (mid <= lo || mid >= hi) break;   // lo and hi are adjacent doubles: nothing changes any more
        if (budget_at(mid) > Bp) lo = mid;
        else hi = mid;
      }
      if (tid == 0) lam_s = hi;
    }
    __syncthreads();
    for (int t = tid; t < Tp; t += kDesignThreads) xi[t] = exp(-lam_s * t);
  }
  __syncthreads();

  // masses q_h = floor((xi_h - xi_{h+1}) 2^62); excess over 2^62 comes off the largest mass
  uint64_t* qp = q + static_cast<int64_t>(p) * T_max;
  unsigned long long sum = 0, best = 0;
  int besti = INT_MAX;
  for (int t = tid; t < T_max; t += kDesignThreads) {
    uint64_t v = 0;
    if (t < Tp) {
      const double d = __dsub_rn(xi[t], t + 1 < Tp ? xi[t + 1] : 0.0);
      v = d > 0.0 ? __double2ull_rz(floor(__dmul_rn(d, 4611686018427387904.0))) : 0ull;
    }
    qp[t] = v;
    if (xi_out) xi_out[static_cast<int64_t>(p) * T_max + t] = t < Tp ? xi[t] : 0.0;
    sum += v;
    if (v > best || (v == best && t < besti)) {
      best = v;
      besti = t;
    }
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const unsigned long long ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, besti, o);
    if (ob > best || (ob == best && oi < besti)) {
      best = ob;
      besti = oi;
    }
  }
  __syncthreads();
  if (lane == 0) {
    red_u[wid] = sum;
    red_b[wid] = best;
    red_i[wid] = besti;
  }
  __syncthreads();
  if (tid == 0) {
    unsigned long long s = 0, b = 0;
    int bi = INT_MAX;
    for (int i = 0; i < kDesignThreads / 32; ++i) {
      s += red_u[i];
      const unsigned long long v = red_b[i];
      if (v > b || (v == b && red_i[i] < bi)) {
        b = v;
        bi = red_i[i];
      }
    }
    if (s > kOne62 && bi < T_max) qp[bi] -= (s - kOne62);
  }
}

// ---------------------------------------------------------------- reward binarisation (Appendix G)
constexpr uint64_t kRewardKeyTag = 0x5053505052574431ull;  // "PSPPRWD1"
constexpr double kLn2d = 0.6931471805599453;              // the double nearest ln 2
constexpr double kTwo53 = 9007199254740992.0;

// sigma(r) = 1 / (1 + e^-r) by one fixed sequence of correctly rounded double operations:
// z = -r clamped to [-40, 40], k = floor(z / ln2 + 1/2), f = z - k ln2, e^f by Horner's rule
// over its Taylor series to degree 16, e^z = e^f 2^k (exact scaling), sigma = 1 / (1 + e^z).
// No step is left to the compiler's choice (no contraction into FMAs), so the value is the
// same double wherever the sequence is repeated. The clamp moves sigma by less than 4.3e-18.
__device__ double sigmoid_fixed_dev(double r) {
  if (r != r) return 0.0;
  double z = -r;
  z = z > 40.0 ? 40.0 : (z < -40.0 ? -40.0 : z);
  const double k = floor(__dadd_rn(__ddiv_rn(z, kLn2d), 0.5));
  const double f = __dsub_rn(z, __dmul_rn(k, kLn2d));
  double p = 1.0;
  for (int n = 16; n >= 1; --n) p = __dadd_rn(1.0, __ddiv_rn(__dmul_rn(f, p), static_cast<double>(n)));
  const double two_k = __longlong_as_double(static_cast<long long>(static_cast<int>(k) + 1023) << 52);
  return __ddiv_rn(1.0, __dadd_rn(1.0, __dmul_rn(p, two_k)));
}

// y_k = 1 when the trajectory's 53-bit Philox uniform lies below sigma(R_k), else 0.
__global__ void binarize_rewards_kernel(int B, const float* __restrict__ R, uint64_t seed, uint64_t step,
                                        int64_t traj_base, float* __restrict__ y) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= B) return;
  uint64_t c[4] = {static_cast<uint64_t>(traj_base + k), step, 0ull, 0ull};
  philox4x64_10(c, seed, kRewardKeyTag);
  const double m = static_cast<double>(c[0] >> 11);
  const double s = sigmoid_fixed_dev(static_cast<double>(R[k]));
  y[k] = m < __dmul_rn(s, kTwo53) ? 1.0f : 0.0f;
}

}  // namespace psk

using namespace psk;

extern "C" {

// Score-proxy workspace: header | ztok [N] f32 | hn [N] f32 | part [S][N] float4 (S as many as fit,
// up to one per 256-column vocabulary tile) -- with top-k: part [S][N] float4 and topk [S][N][16]
// float2 for S <= 16 contiguous vocabulary ranges.
static size_t proxy_fixed(int64_t N) { return kWsHeader + al256(sizeof(float) * N) * 2; }
static size_t proxy_per_split(int64_t N, int topk) {
  return (sizeof(float4) + (topk > 0 ? sizeof(float2) * 16 : 0)) * static_cast<size_t>(N);
}
static int proxy_max_splits(int V, int topk) { return topk > 0 ? 16 : fwd_tile_splits_bf16(V); }

size_t ps_lmhead_score_proxy_workspace_size(int64_t N, int d, int V, int dtype, int topk) {
  if (N < 0 || V < 1 || d < 8 || dtype != PS_DTYPE_BF16 || topk < 0 || topk > 16) return 0;
  int S = proxy_max_splits(V, topk);
  if (S > fwd_tile_splits_bf16(V)) S = fwd_tile_splits_bf16(V);
  return proxy_fixed(N) + proxy_per_split(N, topk) * S;
}

int ps_lmhead_score_proxy(int64_t N, int d, int V, int dtype, const void* Hrows, const void* W, const int32_t* tok,
                          float* gamma, float* logp, int topk, int32_t* top_idx, float* top_prob, void* ws,
                          size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_score_proxy");
  if (N < 0 || N > INT32_MAX || V < 1 || d < 8 || d % 8 || topk < 0 || topk > 16) return PS_ERR_INVALID_ARG;
  if (dtype != PS_DTYPE_BF16) return PS_ERR_UNSUPPORTED;
  if (N > 0 && (!Hrows || !W || !tok || !gamma)) return PS_ERR_INVALID_ARG;
  if (N > 0 && topk > 0 && (!top_idx || !top_prob)) return PS_ERR_INVALID_ARG;
  if (N > 0 && ((reinterpret_cast<uintptr_t>(Hrows) & 15) || (reinterpret_cast<uintptr_t>(W) & 15)))
    return PS_ERR_INVALID_ARG;
  if (!device_is_sm103()) return PS_ERR_UNSUPPORTED;
  if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) & 255)) return PS_ERR_WORKSPACE;
  const size_t fixed = proxy_fixed(N);
  int S = proxy_max_splits(V, topk);
  if (S > fwd_tile_splits_bf16(V)) S = fwd_tile_splits_bf16(V);
  if (N > 0) {
    const size_t room = ws_bytes > fixed ? ws_bytes - fixed : 0;
    const size_t fit = room / proxy_per_split(N, topk);
    if (fit < static_cast<size_t>(S)) S = static_cast<int>(fit);
    if (S < 1) return PS_ERR_WORKSPACE;
  }
  if (ws_bytes < fixed) return PS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, s) != cudaSuccess) return PS_ERR_CUDA;
  if (N == 0) return PS_OK;
  uint8_t* base = static_cast<uint8_t*>(ws);
  float* ztok = reinterpret_cast<float*>(base + kWsHeader);
  float* hn = reinterpret_cast<float*>(base + kWsHeader + al256(sizeof(float) * N));
  float4* part = reinterpret_cast<float4*>(base + fixed);
  float2* tpart = reinterpret_cast<float2*>(base + fixed + sizeof(float4) * static_cast<size_t>(S) * N);
  uint32_t* status = static_cast<uint32_t*>(ws);
  row_sqnorm_kernel<<<num_sms_current() * 8, 256, 0, s>>>(N, d, 1, Hrows, hn);
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  // With the top-k lists, as many vocabulary ranges as the workspace holds (up to 16): shorter
  // ranges keep the CTAs of a band closer together along W (16 ranges measured 4% faster than
  // the 11 the forward's chooser picks at 7B). Without them, the forward's per-tile schedule.
  const int splits = topk > 0 ? S : choose_fwd_splits_bf16(N, d, V, num_sms_current(), S);
  int rc = topk > 0 ? proxy_topk_gemm_bf16(N, d, V, Hrows, W, tok, part, tpart, ztok, splits, status, s)
                    : proxy_gemm_bf16(N, d, V, Hrows, W, tok, part, ztok, splits, status, s);
  if (rc != PS_OK) return rc;
  proxy_finalize_kernel<<<static_cast<unsigned>((N + 127) / 128), 128, 0, s>>>(
      N, V, splits, part, ztok, hn, tok, gamma, logp, topk, tpart, top_idx, top_prob, status);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

size_t ps_reward_uncertainty_workspace_size(int P, int K) {
  if (P < 1 || K < 1) return 0;
  return kWsHeader + al256(sizeof(int64_t) * static_cast<size_t>(P) * K);
}

int ps_binarize_rewards(int B, const float* R, uint64_t seed, uint64_t step, int64_t traj_base, float* y,
                        ps_stream_t stream) {
  NvtxRange nvtx_range("ps_binarize_rewards");
  if (B < 1 || traj_base < 0 || !R || !y) return PS_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  binarize_rewards_kernel<<<(B + 255) / 256, 256, 0, s>>>(B, R, seed, step, traj_base, y);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

int ps_reward_uncertainty(int P, int K, int T_max, const int32_t* L, const float* R, int topk,
                          const int32_t* top_idx, const float* top_prob, float* u, void* ws, size_t ws_bytes,
                          ps_stream_t stream) {
  NvtxRange nvtx_range("ps_reward_uncertainty");
  if (P < 1 || K < 1 || K > 64 || T_max < 1 || topk < 1 || topk > 16) return PS_ERR_INVALID_ARG;
  if (!L || !R || !top_idx || !top_prob || !u) return PS_ERR_INVALID_ARG;
  if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) & 255) ||
      ws_bytes < ps_reward_uncertainty_workspace_size(P, K))
    return PS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, s) != cudaSuccess) return PS_ERR_CUDA;
  int64_t* off = reinterpret_cast<int64_t*>(static_cast<uint8_t*>(ws) + kWsHeader);
  group_offsets_kernel<<<1, 32, 0, s>>>(P * K, L, off);
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  const size_t smem = (sizeof(int32_t) + sizeof(double)) * kUncWarps * K * topk + 16;
  if (cudaFuncSetAttribute(uncertainty_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return PS_ERR_CUDA;
  const int64_t tasks = static_cast<int64_t>(P) * T_max;
  uncertainty_kernel<<<static_cast<unsigned>((tasks + kUncWarps - 1) / kUncWarps), kUncWarps * 32, smem, s>>>(
      P, K, T_max, L, R, topk, top_idx, top_prob, off, u);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

static DesignWs design_ws(void* ws, int P, int K, int T_max) {
  uint8_t* b = static_cast<uint8_t*>(ws) + kWsHeader;
  const size_t pt = static_cast<size_t>(P) * T_max;
  DesignWs d;
  d.w = reinterpret_cast<double*>(b);
  b += al256(sizeof(double) * pt);
  d.xi = reinterpret_cast<double*>(b);
  b += al256(sizeof(double) * pt);
  d.bW = reinterpret_cast<double*>(b);
  b += al256(sizeof(double) * pt * kCapLanes);
  d.bs = reinterpret_cast<double*>(b);
  b += al256(sizeof(double) * pt * kCapLanes);
  d.bn = reinterpret_cast<int32_t*>(b);
  b += al256(sizeof(int32_t) * pt * kCapLanes);
  d.off = reinterpret_cast<int64_t*>(b);
  return d;
}

size_t ps_design_cutoffs_workspace_size(int P, int K, int T_max) {
  if (P < 1 || K < 1 || T_max < 1) return 0;
  const size_t pt = static_cast<size_t>(P) * T_max;
  return kWsHeader + al256(sizeof(double) * pt) * 2 + al256(sizeof(double) * pt * kCapLanes) * 2 +
         al256(sizeof(int32_t) * pt * kCapLanes) + al256(sizeof(int64_t) * static_cast<size_t>(P) * K);
}

int ps_design_cutoffs(int P, int K, int T_max, const int32_t* L, const float* gamma_full, const float* u,
                      double budget, int strategy, double param, uint64_t* q, double* xi, void* ws, size_t ws_bytes,
                      ps_stream_t stream) {
  NvtxRange nvtx_range("ps_design_cutoffs");
  if (P < 1 || K < 1 || T_max < 1 || T_max > (1 << 24) || !L || !q) return PS_ERR_INVALID_ARG;
  if (static_cast<int64_t>(P) * K > INT32_MAX) return PS_ERR_INVALID_ARG;
  if (strategy < PS_DESIGN_OPTIMIZED || strategy > PS_DESIGN_FIXED) return PS_ERR_INVALID_ARG;
  const bool uses_gamma = strategy == PS_DESIGN_OPTIMIZED || strategy == PS_DESIGN_HEURISTIC;
  if (uses_gamma && !gamma_full) return PS_ERR_INVALID_ARG;
  if ((uses_gamma || strategy == PS_DESIGN_TIME_PRIOR) && !(budget > 0.0)) return PS_ERR_INVALID_ARG;
  if (strategy == PS_DESIGN_FIXED && !(param >= 1.0)) return PS_ERR_INVALID_ARG;
  if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) & 255) ||
      ws_bytes < ps_design_cutoffs_workspace_size(P, K, T_max))
    return PS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, s) != cudaSuccess) return PS_ERR_CUDA;
  if (cudaFuncSetAttribute(design_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kDesignDynSmem)) != cudaSuccess)
    return PS_ERR_CUDA;
  design_kernel<<<P, kDesignThreads, kDesignDynSmem, s>>>(K, T_max, L, gamma_full, u, budget, strategy, param, q, xi,
                                              design_ws(ws, P, K, T_max), static_cast<uint32_t*>(ws));
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

}  // extern "C"
