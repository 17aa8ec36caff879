// C ABI of libpsppo: argument checks, workspace layout, and the SIMT kernels of the
// pass (cutoff sampling, packing, forward finalisation). The GEMM-shaped steps live
// in lmhead_bf16.cu (tensor cores) and lmhead_f32.cu (CUDA cores).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <cstdint>

#include "ps_nvtx.h"
#include "internal.h"
#include "ps_common.cuh"
#include "psppo.h"
#include "psppo_diag.h"

namespace psk {

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int num_sms_current() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 1;
  return n;
}

int device_is_sm103() {
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return major == 10 && minor == 3;
}

static int begin_call(void* ws, size_t ws_bytes, size_t need, cudaStream_t s) {
  if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) & 255)) return PS_ERR_WORKSPACE;
  if (ws_bytes < need) return PS_ERR_WORKSPACE;
  if (cudaMemsetAsync(ws, 0, kWsHeader, s) != cudaSuccess) return PS_ERR_CUDA;
  return PS_OK;
}

static uint32_t* status_word(void* ws) { return static_cast<uint32_t*>(ws); }

constexpr uint64_t kCutoffKeyTag = 0x5053505030303031ull;  // "PSPP0001"

// ================================================================== K1: cutoff sampler
// One CTA per prompt. Saturating block scan of the masses gives U[h]; S[t] = 2^62 - U[t-1];
// the thread that owns h decides every completion whose draw x lies in [U[h-1], U[h]).
constexpr int kSampThreads = 1024;
constexpr uint64_t kSatCap = kOne62 + 1;   // any prefix above 2^62 is invalid; saturate just past it

__device__ __forceinline__ uint64_t sat_add(uint64_t a, uint64_t b) {
  const uint64_t s = a + b;  // a, b <= kSatCap so no wrap
  return s > kSatCap ? kSatCap : s;
}

__global__ void __launch_bounds__(kSampThreads)
    sample_cutoffs_kernel(int K, int T_max, const uint64_t* __restrict__ q, const int32_t* __restrict__ L,
                          uint64_t seed, uint64_t step, int64_t traj_base, int mode, int32_t* __restrict__ H,
                          int32_t* __restrict__ n, float* __restrict__ w_tab, uint32_t* status) {
  extern __shared__ uint64_t xs[];  // [K] draws
  __shared__ uint64_t warp_tot[32];
  __shared__ uint64_t carry_s, total_s;
  const int p = blockIdx.x;
  const int tid = threadIdx.x;
  const int64_t wrow = static_cast<int64_t>(p) * T_max;

  for (int j = tid; j < K; j += blockDim.x) {
    const int k = p * K + j;
    const int Lk = L[k];
    if (Lk < 1 || Lk > T_max) raise_status(status, PS_DEV_BAD_LENGTH);
    if (mode == PS_MODE_FULL) {
      H[k] = Lk;
      n[k] = Lk;
    } else {
      H[k] = 0;
      n[k] = 0;
      uint64_t c[4] = {static_cast<uint64_t>(traj_base + k), step, 0ull, 0ull};
      philox4x64_10(c, seed, kCutoffKeyTag);
      xs[j] = c[0] >> 2;
    }
  }
  if (mode == PS_MODE_FULL) {
    for (int t = tid; t < T_max; t += blockDim.x) w_tab[wrow + t] = 1.0f;
    return;
  }
  const int lane = tid & 31, wid = tid >> 5;
  // Total mass U[T] (saturating). Exact mode requires 2^62; in the H = 0 mode the deficit
  // 2^62 - U[T] is Pr(H = 0) and the survival is S[t] = U[T] - U[t-1].
  {
    uint64_t part = 0;
    for (int t = tid; t < T_max; t += blockDim.x) {
      const uint64_t m = q[wrow + t];
      part = sat_add(part, m > kOne62 ? kSatCap : m);
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) part = sat_add(part, __shfl_xor_sync(0xffffffffu, part, o));
    if (lane == 0) warp_tot[wid] = part;
    __syncthreads();
    if (tid == 0) {
      uint64_t tot = 0;
      for (int w = 0; w < kSampThreads / 32; ++w) tot = sat_add(tot, warp_tot[w]);
      total_s = tot;
      if (tot > kOne62 || (mode == PS_MODE_TRUNC && tot != kOne62)) raise_status(status, PS_DEV_BAD_PMF);
    }
  }
  if (tid == 0) carry_s = 0;
  __syncthreads();
  const uint64_t total = total_s > kOne62 ? kOne62 : total_s;

  for (int base = 0; base < T_max; base += kSampThreads) {
    const int t = base + tid;  // 0-based: bucket h = t + 1
    uint64_t m = t < T_max ? q[wrow + t] : 0ull;
    if (m > kOne62) {
      raise_status(status, PS_DEV_BAD_PMF);
      m = kSatCap;
    }
    uint64_t v = m;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t y = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v = sat_add(v, y);
    }
    if (lane == 31) warp_tot[wid] = v;
    __syncthreads();
    if (wid == 0) {
      uint64_t w = warp_tot[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint64_t y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w = sat_add(w, y);
      }
      warp_tot[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const uint64_t carry = carry_s;
    const uint64_t before = wid > 0 ? warp_tot[wid - 1] : 0ull;
    const uint64_t incl = sat_add(carry, sat_add(before, v));  // U[h]
    const uint64_t excl = sat_add(carry, sat_add(before, v - m > kSatCap ? kSatCap : v - m));
    if (t < T_max) {
      // S[t+1] = U[T] - U[t]; weight 2^62 / S (f64 divide, rounded once to f32)
      float wt;
      if (excl >= total) {
        wt = INFINITY;
        if (excl > kOne62) raise_status(status, PS_DEV_BAD_PMF);
      } else {
        const double S = __ull2double_rn(total - excl);
        wt = __double2float_rn(__ddiv_rn(4611686018427387904.0, S));
      }
      w_tab[wrow + t] = wt;
      if (m > 0 && incl <= kOne62) {
        for (int j = 0; j < K; ++j) {
          const uint64_t x = xs[j];
          if (x >= excl && x < incl) {
            const int k = p * K + j;
            H[k] = t + 1;
            n[k] = min(t + 1, L[k]);
          }
        }
      }
    }
    __syncthreads();
    if (tid == kSampThreads - 1) carry_s = incl;
    __syncthreads();
  }
  // (the total was checked before the scan; a draw at or above U[T] leaves H = n = 0)
}

// ================================================================== K2: packing
// Workspace after the header: off_L [B+1] int64, A [B] f64, N (int64).
struct PackWs {
  int64_t* off_L;
  double* A;
  int64_t* N;
};
static PackWs pack_ws(void* ws, int B) {
  uint8_t* base = static_cast<uint8_t*>(ws) + kWsHeader;
  PackWs w;
  w.off_L = reinterpret_cast<int64_t*>(base);
  base += align_up(sizeof(int64_t) * (B + 1), 256);
  w.A = reinterpret_cast<double*>(base);
  base += align_up(sizeof(double) * B, 256);
  w.N = reinterpret_cast<int64_t*>(base);
  return w;
}

// One CTA: scans of L and n, group advantages (sequential f64 sums per group, no FMA
// contraction, so the result is the correctly rounded sequence of the stated operations).
__global__ void __launch_bounds__(1024)
    pack_meta_kernel(int P, int K, int T_max, const int32_t* __restrict__ L, const int32_t* __restrict__ n,
                     const float* __restrict__ R, int adv_mode, int64_t capacity, int32_t* __restrict__ cu_seqlens,
                     PackWs w, uint32_t* status) {
  const int B = P * K;
  __shared__ int64_t sl[1024], sn[1024];
  __shared__ int64_t carry_l, carry_n;
  if (threadIdx.x == 0) {
    carry_l = 0;
    carry_n = 0;
  }
  __syncthreads();
  for (int base = 0; base < B; base += 1024) {
    const int k = base + threadIdx.x;
    int64_t lk = 0, nk = 0;
    if (k < B) {
      lk = L[k];
      nk = n[k];
      if (lk < 1 || lk > T_max || nk < 0 || nk > lk) {
        raise_status(status, PS_DEV_BAD_LENGTH);
        lk = lk < 0 ? 0 : lk;
        nk = nk < 0 ? 0 : (nk > lk ? lk : nk);
      }
    }
    sl[threadIdx.x] = lk;
    sn[threadIdx.x] = nk;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {  // Hillis-Steele inclusive scan
      const int64_t al = threadIdx.x >= o ? sl[threadIdx.x - o] : 0;
      const int64_t an = threadIdx.x >= o ? sn[threadIdx.x - o] : 0;
      __syncthreads();
      sl[threadIdx.x] += al;
      sn[threadIdx.x] += an;
      __syncthreads();
    }
    if (k < B) {
      w.off_L[k] = carry_l + sl[threadIdx.x] - lk;
      const int64_t cu = carry_n + sn[threadIdx.x] - nk;
      cu_seqlens[k] = static_cast<int32_t>(cu > INT32_MAX ? INT32_MAX : cu);
    }
    __syncthreads();
    if (threadIdx.x == 1023) {
      carry_l += sl[1023];
      carry_n += sn[1023];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    w.off_L[B] = carry_l;
    int64_t N = carry_n;
    if (N > capacity || N > INT32_MAX || carry_l > INT32_MAX) {
      raise_status(status, PS_DEV_CAPACITY);
      N = 0;  // write no rows
    }
    cu_seqlens[B] = static_cast<int32_t>(carry_n > INT32_MAX ? INT32_MAX : carry_n);
    *w.N = N;
  }
  for (int p = threadIdx.x; p < P; p += blockDim.x) {
    double s = 0.0;
    for (int j = 0; j < K; ++j) s = __dadd_rn(s, static_cast<double>(R[p * K + j]));
    const double mu = __ddiv_rn(s, static_cast<double>(K));
    if (adv_mode == PS_ADV_CENTERED) {
      for (int j = 0; j < K; ++j) w.A[p * K + j] = __dsub_rn(static_cast<double>(R[p * K + j]), mu);
      continue;
    }
    double ss = 0.0;
    for (int j = 0; j < K; ++j) {
      const double dv = __dsub_rn(static_cast<double>(R[p * K + j]), mu);
      ss = __dadd_rn(ss, __dmul_rn(dv, dv));
    }
    const double sigma = __dsqrt_rn(__ddiv_rn(ss, static_cast<double>(K)));
    const double den = __dadd_rn(sigma, 1e-6);
    for (int j = 0; j < K; ++j)
      w.A[p * K + j] = __ddiv_rn(__dsub_rn(static_cast<double>(R[p * K + j]), mu), den);
  }
}

// One warp per packed row: lane 0 locates (k, t) by binary search over cu_seqlens and
// writes the row's scalars; the warp copies the hidden row with 16-byte accesses.
constexpr int kPackThreads = 256;
__global__ void __launch_bounds__(kPackThreads)
    pack_rows_kernel(int B, int K, int T_max, const int32_t* __restrict__ cu_seqlens, PackWs w,
                     const float* __restrict__ w_tab, const int32_t* __restrict__ tok_full,
                     const float* __restrict__ oldlogp_full, const uint4* __restrict__ hid_full, int64_t row_vec,
                     int32_t* __restrict__ src_row, int32_t* __restrict__ row_traj, int32_t* __restrict__ row_pos,
                     int32_t* __restrict__ tok, float* __restrict__ oldlogp, float* __restrict__ wout,
                     float* __restrict__ adv, uint4* __restrict__ hid_packed) {
  const int64_t N = *w.N;
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); i < N; i += warps) {
    int64_t src = 0;
    if (lane == 0) {
      int lo = 0, hi = B - 1;  // largest k with cu_seqlens[k] <= i
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (cu_seqlens[mid] <= i) lo = mid;
        else hi = mid - 1;
      }
      const int k = lo;
      const int t = static_cast<int>(i - cu_seqlens[k]) + 1;
      src = w.off_L[k] + t - 1;
      if (src_row) src_row[i] = static_cast<int32_t>(src);
      if (row_traj) row_traj[i] = k;
      if (row_pos) row_pos[i] = t;
      tok[i] = tok_full[src];
      oldlogp[i] = oldlogp_full[src];
      wout[i] = w_tab[static_cast<int64_t>(k / K) * T_max + (t - 1)];
      adv[i] = __double2float_rn(w.A[k]);
    }
    if (hid_full == nullptr) continue;
    src = __shfl_sync(0xffffffffu, src, 0);
    const uint4* s = hid_full + src * row_vec;
    uint4* d = hid_packed + i * row_vec;
    int64_t c = lane;
    for (; c + 96 < row_vec; c += 128) {
      const uint4 v0 = s[c], v1 = s[c + 32], v2 = s[c + 64], v3 = s[c + 96];
      d[c] = v0;
      d[c + 32] = v1;
      d[c + 64] = v2;
      d[c + 96] = v3;
    }
    for (; c < row_vec; c += 32) d[c] = s[c];
  }
}

// ================================================================== K4: forward finalize
constexpr int kFinThreads = 256;

// One packed row of the forward (Eq. 1 through the head, the loss of Eq. truncated_update_Ghat):
// from the row's logsumexp in base 2, lse2 = m + log2(S) (m the base-2 maximum, S the sum of
// 2^(x - m) over the vocabulary), and its chosen logit zt. Returns the row's loss term.
__device__ __forceinline__ double finalize_row(int64_t i, float m, float S, float zt, int t, int V,
                                               const float* __restrict__ oldlogp, const float* __restrict__ adv,
                                               const float* __restrict__ w, double eps, double loss_scale,
                                               float* __restrict__ lse, float* __restrict__ logp,
                                               float* __restrict__ ratio, float* __restrict__ coef,
                                               float* __restrict__ row_loss, uint32_t* status) {
  const double l = (static_cast<double>(m) + log2(static_cast<double>(S))) * 0.6931471805599453;
  double lp;
  if (t < 0 || t >= V) {
    raise_status(status, PS_DEV_BAD_TOKEN);
    lp = NAN;
  } else {
    lp = static_cast<double>(zt) - l;
  }
  const double r = exp(lp - static_cast<double>(oldlogp[i]));
  const double A = adv[i], wt = w[i];
  // min and clip as the definition has them: a NaN ratio (a non-finite input or a bad token
  // id) gives a NaN surrogate, which fmin / fmax alone would replace by the other operand
  const double clipped = r != r ? r : fmin(fmax(r, 1.0 - eps), 1.0 + eps);
  const double ra = r * A, ca = clipped * A;
  const double sur = (ra != ra || ca != ca) ? NAN : fmin(ra, ca);
  const double rl = -loss_scale * wt * sur;
  const bool bind = (A > 0.0 && r > 1.0 + eps) || (A < 0.0 && r < 1.0 - eps);
  lse[i] = static_cast<float>(l);
  logp[i] = static_cast<float>(lp);
  ratio[i] = static_cast<float>(r);
  coef[i] = bind ? 0.f : static_cast<float>(-loss_scale * wt * A * r);
  if (row_loss) row_loss[i] = static_cast<float>(rl);
  return rl;
}

// The (max, sum) pairs of `count` parts of a row's vocabulary (stride `stride` between parts),
// merged into one pair: m = max m_s, S = sum S_s 2^(m_s - m).
__device__ __forceinline__ float2 merge_parts(const float2* __restrict__ part, int count, int64_t stride) {
  float m = -INFINITY;
  for (int s = 0; s < count; ++s) m = fmaxf(m, part[static_cast<int64_t>(s) * stride].x);
  float S = 0.f;
  for (int s = 0; s < count; ++s) {
    const float2 pr = part[static_cast<int64_t>(s) * stride];
    S += pr.y * exp2f(pr.x - m);
  }
  return make_float2(m, S);
}

// Fixed-order block sum of the rows' loss terms: warp shuffles, then warp 0 over the warp sums.
__device__ __forceinline__ void block_loss_sum(double rl, double* __restrict__ block_loss) {
  __shared__ double ws_sum[kFinThreads / 32];
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) rl += __shfl_down_sync(0xffffffffu, rl, o);
  if ((threadIdx.x & 31) == 0) ws_sum[threadIdx.x >> 5] = rl;
  __syncthreads();
  if (threadIdx.x < 32) {
    double v = threadIdx.x < kFinThreads / 32 ? ws_sum[threadIdx.x] : 0.0;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) block_loss[blockIdx.x] = v;
  }
}

__global__ void __launch_bounds__(kFinThreads)
    fwd_finalize_kernel(int64_t N, int V, int splits, const float2* __restrict__ part, const float* __restrict__ ztok,
                        const int32_t* __restrict__ tok, const float* __restrict__ oldlogp,
                        const float* __restrict__ adv, const float* __restrict__ w, double eps, double loss_scale,
                        float* __restrict__ lse, float* __restrict__ logp, float* __restrict__ ratio,
                        float* __restrict__ coef, float* __restrict__ row_loss, double* __restrict__ block_loss,
                        uint32_t* status) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * kFinThreads + threadIdx.x;
  double rl = 0.0;
  if (i < N) {
    const float2 ms = merge_parts(part + i, splits, N);
    rl = finalize_row(i, ms.x, ms.y, ztok[i], tok[i], V, oldlogp, adv, w, eps, loss_scale, lse, logp, ratio, coef,
                      row_loss, status);
  }
  block_loss_sum(rl, block_loss);
}

// A vocabulary shard's statistics: its vocabulary tiles' (max, sum) pairs merged per row, and the
// chosen logit where the row's token lies in the shard ([tok_base, tok_base + Vs)), -inf elsewhere.
__global__ void __launch_bounds__(kFinThreads)
    stats_merge_kernel(int64_t N, int splits, const float2* __restrict__ part, const float* __restrict__ ztok_ws,
                       const int32_t* __restrict__ tok, int64_t tok_base, int Vs, float2* __restrict__ stats,
                       float* __restrict__ ztok) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * kFinThreads + threadIdx.x;
  if (i >= N) return;
  stats[i] = merge_parts(part + i, splits, N);
  const int64_t t = static_cast<int64_t>(tok[i]) - tok_base;
  ztok[i] = (t >= 0 && t < Vs) ? ztok_ws[i] : -INFINITY;
}

// The forward finalize from the statistics of S vocabulary shards ([S][ld] each): their (max, sum)
// pairs merged as one row's tiles are, and the chosen logit from the shard that holds the token (the
// largest of the S values, the others being -inf).
__global__ void __launch_bounds__(kFinThreads)
    stats_finalize_kernel(int64_t N, int S, int64_t ld, int V, const float2* __restrict__ stats,
                          const float* __restrict__ ztok,
                          const int32_t* __restrict__ tok, const float* __restrict__ oldlogp,
                          const float* __restrict__ adv, const float* __restrict__ w, double eps, double loss_scale,
                          float* __restrict__ lse, float* __restrict__ logp, float* __restrict__ ratio,
                          float* __restrict__ coef, float* __restrict__ row_loss, double* __restrict__ block_loss,
                          uint32_t* status) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * kFinThreads + threadIdx.x;
  double rl = 0.0;
  if (i < N) {
    const float2 ms = merge_parts(stats + i, S, ld);
    float zt = -INFINITY;
    for (int r = 0; r < S; ++r) zt = fmaxf(zt, ztok[static_cast<int64_t>(r) * ld + i]);
    rl = finalize_row(i, ms.x, ms.y, zt, tok[i], V, oldlogp, adv, w, eps, loss_scale, lse, logp, ratio, coef,
                      row_loss, status);
  }
  block_loss_sum(rl, block_loss);
}

__global__ void __launch_bounds__(1024) loss_reduce_kernel(int64_t nblocks, const double* __restrict__ part,
                                                           double* __restrict__ loss) {
  double v = 0.0;
  for (int64_t b = threadIdx.x; b < nblocks; b += 1024) v += part[b];
  __shared__ double s[32];
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0) s[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x < 32) {
    double u = s[threadIdx.x];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) u += __shfl_down_sync(0xffffffffu, u, o);
    if (threadIdx.x == 0) *loss = u;
  }
}

// Forward workspace: header | ztok [N] f32 | block_loss [nb] f64 | part [S][N] float2. The
// (max, sum of exp) partials come last: S is as many as the workspace holds, up to two per
// 256-column vocabulary tile (bf16: one per column group of the forward's epilogue, so the
// vocabulary ranges per row are S / 2; at one range per tile every unit of the forward GEMM is one
// tile, the schedule that keeps W traffic lowest). f32 always uses one partial per 64-column tile.
struct FwdWs {
  float2* part;
  float* ztok;
  double* block_loss;
  int splits;       // S that fits (0 if not even one)
  size_t bytes;     // bytes used with that S
};
static int fwd_full_splits(int V, int dtype) {
  return dtype == PS_DTYPE_BF16 ? fwd_tile_splits_bf16(V) * fwd_partials_per_split_bf16() : fwd_splits_f32(V);
}
// Partials per vocabulary range, and the fewest partials a forward can run with.
static int fwd_group(int dtype) { return dtype == PS_DTYPE_BF16 ? fwd_partials_per_split_bf16() : 1; }
static size_t fwd_fixed_bytes(int64_t N) {
  const int64_t nb = (N + kFinThreads - 1) / kFinThreads;
  return kWsHeader + align_up(sizeof(float) * N, 256) + align_up(sizeof(double) * (nb > 0 ? nb : 1), 256);
}
// the partials are the last region: no padding after them, so S partials need exactly this much
static size_t fwd_part_bytes(int64_t N, int S) { return sizeof(float2) * static_cast<size_t>(S) * N; }
// Layout for a workspace of ws_bytes (SIZE_MAX: the full-size layout).
static FwdWs fwd_ws(void* ws, int64_t N, int V, int dtype, size_t ws_bytes) {
  const int full = fwd_full_splits(V, dtype);
  const size_t fixed = fwd_fixed_bytes(N);
  FwdWs f;
  uint8_t* base = static_cast<uint8_t*>(ws);
  f.ztok = reinterpret_cast<float*>(base + kWsHeader);
  f.block_loss = reinterpret_cast<double*>(base + kWsHeader + align_up(sizeof(float) * N, 256));
  f.part = reinterpret_cast<float2*>(base + fixed);
  const int g = fwd_group(dtype);
  int S = full;
  if (ws_bytes != SIZE_MAX && N > 0) {
    const size_t room = ws_bytes > fixed ? ws_bytes - fixed : 0;
    const size_t fit = room / (sizeof(float2) * static_cast<size_t>(N));
    if (fit < static_cast<size_t>(S)) S = static_cast<int>(fit) / g * g;   // whole vocabulary ranges
    if (dtype != PS_DTYPE_BF16 && S < full) S = 0;   // the f32 kernel needs every partial
  }
  f.splits = S;
  f.bytes = fixed + fwd_part_bytes(N, S > 0 ? S : g);
  return f;
}

static size_t elem_size(int dtype) { return dtype == PS_DTYPE_BF16 ? 2 : 4; }
static bool dtype_ok(int dtype) { return dtype == PS_DTYPE_BF16 || dtype == PS_DTYPE_F32; }
static bool d_ok(int d, int dtype) { return d >= 8 && (dtype == PS_DTYPE_BF16 ? d % 8 == 0 : d % 4 == 0); }
static bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
static int64_t ldz_for(int V) { return (static_cast<int64_t>(V) + 7) / 8 * 8; }

}  // namespace psk

using namespace psk;

// ============================================================================= C ABI
extern "C" {

const char* ps_status_string(int status) {
  switch (status) {
    case PS_OK: return "ok";
    case PS_ERR_INVALID_ARG: return "invalid argument";
    case PS_ERR_UNSUPPORTED: return "unsupported dtype, shape or device";
    case PS_ERR_WORKSPACE: return "workspace too small or misaligned";
    case PS_ERR_CAPACITY: return "packed rows exceed capacity";
    case PS_ERR_DEVICE_DATA: return "invalid device data (masses, lengths or token ids)";
    case PS_ERR_TIMEOUT: return "a bounded wait inside a kernel ran out";
    case PS_ERR_CUDA: return "CUDA runtime error";
    default: return "unknown status";
  }
}

int ps_version(void) { return 100; }

int ps_workspace_status(const void* ws, ps_stream_t stream, uint32_t* bits) {
  if (ws == nullptr) return PS_ERR_INVALID_ARG;
  uint32_t v = 0;
  if (cudaMemcpyAsync(&v, ws, sizeof(v), cudaMemcpyDeviceToHost, stream) != cudaSuccess) return PS_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return PS_ERR_CUDA;
  if (bits) *bits = v;
  if (v & PS_DEV_TIMEOUT) return PS_ERR_TIMEOUT;
  if (v & PS_DEV_CAPACITY) return PS_ERR_CAPACITY;
  if (v) return PS_ERR_DEVICE_DATA;
  return PS_OK;
}

size_t ps_sample_cutoffs_workspace_size(int, int, int) { return kWsHeader; }

int ps_sample_cutoffs(int P, int K, int T_max, const uint64_t* q, const int32_t* L, uint64_t seed, uint64_t step,
                      int64_t traj_base, int mode, int32_t* H, int32_t* n, float* w_tab, void* ws, size_t ws_bytes,
                      ps_stream_t stream) {
  NvtxRange nvtx_range("ps_sample_cutoffs");
  if (P < 1 || K < 1 || K > 8192 || T_max < 1 || T_max > (1 << 24) || traj_base < 0) return PS_ERR_INVALID_ARG;
  if (static_cast<int64_t>(P) * K > INT32_MAX) return PS_ERR_INVALID_ARG;
  if (mode != PS_MODE_TRUNC && mode != PS_MODE_FULL && mode != PS_MODE_TRUNC_ZERO) return PS_ERR_INVALID_ARG;
  if ((mode != PS_MODE_FULL && q == nullptr) || !L || !H || !n || !w_tab) return PS_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, ps_sample_cutoffs_workspace_size(P, K, T_max), s);
  if (rc != PS_OK) return rc;
  const size_t smem = sizeof(uint64_t) * K;
  if (cudaFuncSetAttribute(sample_cutoffs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return PS_ERR_CUDA;
  sample_cutoffs_kernel<<<P, kSampThreads, smem, s>>>(K, T_max, q, L, seed, step, traj_base, mode, H, n, w_tab,
                                                      status_word(ws));
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

size_t ps_pack_prefixes_workspace_size(int P, int K) {
  const int B = P * K;
  return kWsHeader + align_up(sizeof(int64_t) * (B + 1), 256) + align_up(sizeof(double) * B, 256) + 256;
}

int ps_pack_prefixes(int P, int K, int T_max, int d, int dtype, const int32_t* L, const int32_t* n, const float* R,
                     int adv_mode, const float* w_tab, const int32_t* tok_full, const float* oldlogp_full,
                     const void* hid_full, int64_t capacity, int32_t* cu_seqlens, int32_t* src_row,
                     int32_t* row_traj, int32_t* row_pos, int32_t* tok, float* oldlogp, float* w, float* adv,
                     void* hid_packed, int64_t* h_num_rows, void* ws, size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_pack_prefixes");
  if (P < 1 || K < 1 || T_max < 1 || capacity < 0 || !dtype_ok(dtype)) return PS_ERR_INVALID_ARG;
  if (static_cast<int64_t>(P) * K > (1 << 24)) return PS_ERR_INVALID_ARG;
  if (adv_mode != PS_ADV_CENTERED && adv_mode != PS_ADV_GROUP_NORM) return PS_ERR_INVALID_ARG;
  if (!L || !n || !R || !w_tab || !tok_full || !oldlogp_full || !cu_seqlens || !tok || !oldlogp || !w || !adv)
    return PS_ERR_INVALID_ARG;
  if (hid_full != nullptr) {
    if (!hid_packed || !d_ok(d, dtype) || !al16(hid_full) || !al16(hid_packed)) return PS_ERR_INVALID_ARG;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, ps_pack_prefixes_workspace_size(P, K), s);
  if (rc != PS_OK) return rc;
  const int B = P * K;
  PackWs pw = pack_ws(ws, B);
  pack_meta_kernel<<<1, 1024, 0, s>>>(P, K, T_max, L, n, R, adv_mode, capacity, cu_seqlens, pw, status_word(ws));
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  const int64_t row_vec = hid_full ? static_cast<int64_t>(d) * elem_size(dtype) / 16 : 0;
  const int grid = num_sms_current() * 8;
  pack_rows_kernel<<<grid, kPackThreads, 0, s>>>(B, K, T_max, cu_seqlens, pw, w_tab, tok_full, oldlogp_full,
                                                 static_cast<const uint4*>(hid_full), row_vec, src_row, row_traj,
                                                 row_pos, tok, oldlogp, w, adv, static_cast<uint4*>(hid_packed));
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  if (h_num_rows) {
    int32_t nr = 0;
    if (cudaMemcpyAsync(&nr, cu_seqlens + B, sizeof(nr), cudaMemcpyDeviceToHost, s) != cudaSuccess) return PS_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return PS_ERR_CUDA;
    *h_num_rows = nr;
  }
  return PS_OK;
}

size_t ps_lmhead_ppo_fwd_workspace_size(int64_t N, int d, int V, int dtype) {
  if (N < 0 || V < 1 || !dtype_ok(dtype)) return 0;
  (void)d;
  return fwd_ws(nullptr, N, V, dtype, SIZE_MAX).bytes;
}

}  // extern "C"

// Layout of the logit store of N rows: [N][ldz] 2-byte values (f16 e after the forward, bf16 dZ after
// the backward's conversion), then the slice maxima [ceil(V / 32)][N] f32 at a 256-byte boundary.
struct StoreLayout {
  int64_t ldz;
  size_t scale_off;
  size_t bytes;
};
static StoreLayout store_layout(int64_t N, int V) {
  StoreLayout L;
  L.ldz = ldz_for(V);
  L.scale_off = align_up(static_cast<size_t>(N) * static_cast<size_t>(L.ldz) * 2, 256);
  L.bytes = L.scale_off + sizeof(float) * static_cast<size_t>((V + 31) / 32) * static_cast<size_t>(N);
  return L;
}

static int lmhead_fwd_impl(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W, const int32_t* tok,
                           const float* oldlogp, const float* adv, const float* w, double eps, double loss_scale,
                           double* loss, float* lse, float* logp, float* ratio, float* coef, float* row_loss,
                           void* store, size_t store_bytes, void* ws, size_t ws_bytes, ps_stream_t stream) {
  if (N < 0 || N > INT32_MAX || V < 1 || !dtype_ok(dtype) || !d_ok(d, dtype)) return PS_ERR_INVALID_ARG;
  if (!(eps >= 0.0) || !loss || (N > 0 && (!Hpk || !W || !tok || !oldlogp || !adv || !w || !lse || !logp ||
                                           !ratio || !coef)))
    return PS_ERR_INVALID_ARG;
  if (N > 0 && (!al16(Hpk) || !al16(W))) return PS_ERR_INVALID_ARG;
  if (store != nullptr) {
    if (dtype != PS_DTYPE_BF16) return PS_ERR_UNSUPPORTED;
    if (!al16(store)) return PS_ERR_INVALID_ARG;
    if (store_bytes < store_layout(N, V).bytes) return PS_ERR_WORKSPACE;
  }
  if (dtype == PS_DTYPE_BF16 && !device_is_sm103()) return PS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  FwdWs f = fwd_ws(ws, N, V, dtype, ws_bytes);
  if (N > 0 && f.splits < 1) return PS_ERR_WORKSPACE;
  int rc = begin_call(ws, ws_bytes, f.bytes, s);
  if (rc != PS_OK) return rc;
  if (N == 0) return cudaMemsetAsync(loss, 0, sizeof(double), s) == cudaSuccess ? PS_OK : PS_ERR_CUDA;
  int splits;
  if (dtype == PS_DTYPE_BF16) {
    const int g = fwd_partials_per_split_bf16();
    const int ranges = choose_fwd_splits_bf16(N, d, V, num_sms_current(), f.splits / g);
    if (store) {
      const StoreLayout L = store_layout(N, V);
      float* scale = reinterpret_cast<float*>(static_cast<uint8_t*>(store) + L.scale_off);
      rc = fwd_gemm_store_bf16(N, d, V, Hpk, W, tok, f.part, f.ztok, ranges, store, L.ldz, scale, status_word(ws),
                               s);
    } else {
      rc = fwd_gemm_bf16(N, d, V, Hpk, W, tok, f.part, f.ztok, ranges, status_word(ws), s);
    }
    splits = ranges * g;   // the partials the finalize merges
  } else {
    splits = fwd_splits_f32(V);
    rc = fwd_gemm_f32(N, d, V, static_cast<const float*>(Hpk), static_cast<const float*>(W), tok, f.part, f.ztok,
                      status_word(ws), s);
  }
  if (rc != PS_OK) return rc;
  const int64_t nb = (N + kFinThreads - 1) / kFinThreads;
  fwd_finalize_kernel<<<static_cast<unsigned>(nb), kFinThreads, 0, s>>>(N, V, splits, f.part, f.ztok, tok, oldlogp,
                                                                       adv, w, eps, loss_scale, lse, logp, ratio,
                                                                       coef, row_loss, f.block_loss, status_word(ws));
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  loss_reduce_kernel<<<1, 1024, 0, s>>>(nb, f.block_loss, loss);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

// The backward from a logit store of V vocabulary columns whose first is global token id tok_base.
static int bwd_from_store_impl(int64_t N, int d, int V, int64_t tok_base, int dtype, const void* Hpk, const void* W,
                               const int32_t* tok, const float* lse, const float* logp, const float* coef,
                               void* store, size_t store_bytes, float* dH, float* dW, int flags, void* ws,
                               size_t ws_bytes, ps_stream_t stream) {
  if (N < 0 || N > INT32_MAX || V < 1 || !dtype_ok(dtype) || !d_ok(d, dtype)) return PS_ERR_INVALID_ARG;
  if (flags & ~(PS_DW_ACCUMULATE | PS_DH_ACCUMULATE)) return PS_ERR_INVALID_ARG;
  if (dtype != PS_DTYPE_BF16) return PS_ERR_UNSUPPORTED;
  if (N > 0 && (!Hpk || !W || !tok || !lse || !logp || !coef || !store)) return PS_ERR_INVALID_ARG;
  if ((N > 0 && (!al16(Hpk) || !al16(W) || !al16(store))) || (dH && !al16(dH)) || (dW && !al16(dW)))
    return PS_ERR_INVALID_ARG;
  if (N > 0 && store_bytes < store_layout(N, V).bytes) return PS_ERR_WORKSPACE;
  if (!device_is_sm103()) return PS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, kWsHeader, s);
  if (rc != PS_OK) return rc;
  if (N == 0) {
    if (dW && !(flags & PS_DW_ACCUMULATE))
      return cudaMemsetAsync(dW, 0, sizeof(float) * static_cast<size_t>(V) * d, s) == cudaSuccess ? PS_OK
                                                                                                : PS_ERR_CUDA;
    return PS_OK;
  }
  // the conversion into dZ (HBM-bound), then dH and dW over all rows. Running the conversion of later
  // rows on a second stream under the dH GEMM of earlier rows (the GEMM's one CTA per SM leaves room
  // for conversion blocks) measured 1-2% slower at the 7B workload (backward 272.7 / 273.0 against
  // 267.3 / 269.2 ms, back to back), so the parts run in turn.
  const StoreLayout L = store_layout(N, V);
  const float* scale = reinterpret_cast<const float*>(static_cast<const uint8_t*>(store) + L.scale_off);
  rc = dz_from_store_bf16(N, V, store, L.ldz, scale, N, tok, lse, logp, coef, s, static_cast<int>(tok_base));
  if (rc != PS_OK) return rc;
  return bwd_grads_bf16(N, d, V, Hpk, W, dH, dW, (flags & PS_DW_ACCUMULATE) ? 1 : 0, store, L.ldz, status_word(ws),
                        s, (flags & PS_DH_ACCUMULATE) ? 1 : 0);
}

extern "C" {

int ps_lmhead_ppo_fwd(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W, const int32_t* tok,
                      const float* oldlogp, const float* adv, const float* w, double eps, double loss_scale,
                      double* loss, float* lse, float* logp, float* ratio, float* coef, float* row_loss, void* ws,
                      size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_fwd");
  return lmhead_fwd_impl(N, d, V, dtype, Hpk, W, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp, ratio, coef,
                         row_loss, nullptr, 0, ws, ws_bytes, stream);
}

size_t ps_lmhead_logit_store_size(int64_t N, int V) {
  if (N < 0 || N > INT32_MAX || V < 1) return 0;
  return store_layout(N, V).bytes;
}

int ps_lmhead_ppo_fwd_store(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W, const int32_t* tok,
                            const float* oldlogp, const float* adv, const float* w, double eps, double loss_scale,
                            double* loss, float* lse, float* logp, float* ratio, float* coef, float* row_loss,
                            void* store, size_t store_bytes, void* ws, size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_fwd_store");
  if (store == nullptr) return PS_ERR_INVALID_ARG;
  return lmhead_fwd_impl(N, d, V, dtype, Hpk, W, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp, ratio, coef,
                         row_loss, store, store_bytes, ws, ws_bytes, stream);
}

size_t ps_lmhead_ppo_bwd_from_store_workspace_size(void) { return kWsHeader; }

int ps_lmhead_ppo_bwd_from_store(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W,
                                 const int32_t* tok, const float* lse, const float* logp, const float* coef,
                                 void* store, size_t store_bytes, float* dH, float* dW, int flags, void* ws,
                                 size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_bwd_from_store");
  return bwd_from_store_impl(N, d, V, 0, dtype, Hpk, W, tok, lse, logp, coef, store, store_bytes, dH, dW, flags, ws,
                             ws_bytes, stream);
}

int ps_lmhead_ppo_bwd_vocab_shard_from_store(int64_t N, int d, int Vs, int64_t v0, int V, int dtype, const void* Hpk,
                                             const void* W_shard, const int32_t* tok, const float* lse,
                                             const float* logp, const float* coef, void* store, size_t store_bytes,
                                             float* dH, float* dW_shard, int flags, void* ws, size_t ws_bytes,
                                             ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_bwd_vocab_shard_from_store");
  if (Vs < 1 || v0 < 0 || V < 1 || v0 + Vs > V) return PS_ERR_INVALID_ARG;
  return bwd_from_store_impl(N, d, Vs, v0, dtype, Hpk, W_shard, tok, lse, logp, coef, store, store_bytes, dH,
                             dW_shard, flags, ws, ws_bytes, stream);
}

size_t ps_lmhead_logit_stats_workspace_size(int64_t N, int d, int Vs, int dtype) {
  return ps_lmhead_ppo_fwd_workspace_size(N, d, Vs, dtype);
}

}  // extern "C"

static int logit_stats_impl(int64_t N, int d, int Vs, int64_t v0, int dtype, const void* Hpk, const void* W_shard,
                            const int32_t* tok, float* stats, float* ztok, void* store, size_t store_bytes, void* ws,
                            size_t ws_bytes, ps_stream_t stream) {
  if (N < 0 || N > INT32_MAX || Vs < 1 || v0 < 0 || v0 + Vs > INT32_MAX || !dtype_ok(dtype) || !d_ok(d, dtype))
    return PS_ERR_INVALID_ARG;
  if (N > 0 && (!Hpk || !W_shard || !tok || !stats || !ztok)) return PS_ERR_INVALID_ARG;
  if (N > 0 && (!al16(Hpk) || !al16(W_shard) || (reinterpret_cast<uintptr_t>(stats) & 7))) return PS_ERR_INVALID_ARG;
  if (store != nullptr) {
    if (dtype != PS_DTYPE_BF16) return PS_ERR_UNSUPPORTED;
    if (!al16(store)) return PS_ERR_INVALID_ARG;
    if (store_bytes < store_layout(N, Vs).bytes) return PS_ERR_WORKSPACE;
  }
  if (dtype == PS_DTYPE_BF16 && !device_is_sm103()) return PS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  FwdWs f = fwd_ws(ws, N, Vs, dtype, ws_bytes);
  if (N > 0 && f.splits < 1) return PS_ERR_WORKSPACE;
  int rc = begin_call(ws, ws_bytes, f.bytes, s);
  if (rc != PS_OK || N == 0) return rc;
  int splits;
  if (dtype == PS_DTYPE_BF16) {
    const int g = fwd_partials_per_split_bf16();
    const int ranges = choose_fwd_splits_bf16(N, d, Vs, num_sms_current(), f.splits / g);
    if (store) {
      const StoreLayout L = store_layout(N, Vs);
      float* scale = reinterpret_cast<float*>(static_cast<uint8_t*>(store) + L.scale_off);
      rc = fwd_gemm_store_bf16(N, d, Vs, Hpk, W_shard, tok, f.part, f.ztok, ranges, store, L.ldz, scale,
                               status_word(ws), s, static_cast<int>(v0));
    } else {
      rc = fwd_gemm_bf16(N, d, Vs, Hpk, W_shard, tok, f.part, f.ztok, ranges, status_word(ws), s,
                         static_cast<int>(v0));
    }
    splits = ranges * g;   // the partials the merge reads
  } else {
    splits = fwd_splits_f32(Vs);
    rc = fwd_gemm_f32(N, d, Vs, static_cast<const float*>(Hpk), static_cast<const float*>(W_shard), tok, f.part,
                      f.ztok, status_word(ws), s, static_cast<int>(v0));
  }
  if (rc != PS_OK) return rc;
  const int64_t nb = (N + kFinThreads - 1) / kFinThreads;
  stats_merge_kernel<<<static_cast<unsigned>(nb), kFinThreads, 0, s>>>(N, splits, f.part, f.ztok, tok, v0, Vs,
                                                                        reinterpret_cast<float2*>(stats), ztok);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

extern "C" {

int ps_lmhead_logit_stats(int64_t N, int d, int Vs, int64_t v0, int dtype, const void* Hpk, const void* W_shard,
                          const int32_t* tok, float* stats, float* ztok, void* ws, size_t ws_bytes,
                          ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_logit_stats");
  return logit_stats_impl(N, d, Vs, v0, dtype, Hpk, W_shard, tok, stats, ztok, nullptr, 0, ws, ws_bytes, stream);
}

int ps_lmhead_logit_stats_store(int64_t N, int d, int Vs, int64_t v0, int dtype, const void* Hpk,
                                const void* W_shard, const int32_t* tok, float* stats, float* ztok, void* store,
                                size_t store_bytes, void* ws, size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_logit_stats_store");
  if (store == nullptr) return PS_ERR_INVALID_ARG;
  return logit_stats_impl(N, d, Vs, v0, dtype, Hpk, W_shard, tok, stats, ztok, store, store_bytes, ws, ws_bytes,
                          stream);
}

size_t ps_lmhead_ppo_fwd_from_stats_workspace_size(int64_t N) {
  if (N < 0) return 0;
  const int64_t nb = (N + kFinThreads - 1) / kFinThreads;
  return kWsHeader + align_up(sizeof(double) * static_cast<size_t>(nb > 0 ? nb : 1), 256);
}

int ps_lmhead_ppo_fwd_from_stats(int64_t N, int S, int64_t ld, int V, const float* stats, const float* ztok,
                                 const int32_t* tok,
                                 const float* oldlogp, const float* adv, const float* w, double eps,
                                 double loss_scale, double* loss, float* lse, float* logp, float* ratio, float* coef,
                                 float* row_loss, void* ws, size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_fwd_from_stats");
  if (N < 0 || N > INT32_MAX || S < 1 || ld < N || V < 1 || !(eps >= 0.0) || !loss) return PS_ERR_INVALID_ARG;
  if (N > 0 && (!stats || !ztok || !tok || !oldlogp || !adv || !w || !lse || !logp || !ratio || !coef))
    return PS_ERR_INVALID_ARG;
  if (N > 0 && (reinterpret_cast<uintptr_t>(stats) & 7)) return PS_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, ps_lmhead_ppo_fwd_from_stats_workspace_size(N), s);
  if (rc != PS_OK) return rc;
  if (N == 0) return cudaMemsetAsync(loss, 0, sizeof(double), s) == cudaSuccess ? PS_OK : PS_ERR_CUDA;
  const int64_t nb = (N + kFinThreads - 1) / kFinThreads;
  double* block_loss = reinterpret_cast<double*>(static_cast<uint8_t*>(ws) + kWsHeader);
  stats_finalize_kernel<<<static_cast<unsigned>(nb), kFinThreads, 0, s>>>(
      N, S, ld, V, reinterpret_cast<const float2*>(stats), ztok, tok, oldlogp, adv, w, eps, loss_scale, lse, logp, ratio,
      coef, row_loss, block_loss, status_word(ws));
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  loss_reduce_kernel<<<1, 1024, 0, s>>>(nb, block_loss, loss);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

size_t ps_lmhead_ppo_bwd_workspace_size(int64_t N, int d, int V, int dtype, int64_t chunk_rows) {
  if (N < 0 || V < 1 || !dtype_ok(dtype)) return 0;
  (void)d;
  int64_t rows = chunk_rows <= 0 ? N : chunk_rows;
  if (rows > N) rows = N;
  rows = (rows + 127) / 128 * 128;
  if (rows < 128) rows = 128;
  return kWsHeader + static_cast<size_t>(rows) * ldz_for(V) * elem_size(dtype);
}

}  // extern "C"

// The backward over a head of V vocabulary rows whose first is global token id tok_base (0 for the
// whole head, v0 for one shard of a vocabulary-parallel head).
static int lmhead_bwd_impl(int64_t N, int d, int V, int64_t tok_base, int dtype, const void* Hpk, const void* W,
                           const int32_t* tok, const float* lse, const float* coef, float* dH, float* dW, int flags,
                           void* ws, size_t ws_bytes, ps_stream_t stream) {
  if (N < 0 || N > INT32_MAX || V < 1 || !dtype_ok(dtype) || !d_ok(d, dtype)) return PS_ERR_INVALID_ARG;
  if (flags & ~(PS_DW_ACCUMULATE | PS_DH_ACCUMULATE)) return PS_ERR_INVALID_ARG;
  if (N > 0 && (!Hpk || !W || !tok || !lse || !coef)) return PS_ERR_INVALID_ARG;
  if ((N > 0 && (!al16(Hpk) || !al16(W))) || (dH && !al16(dH)) || (dW && !al16(dW))) return PS_ERR_INVALID_ARG;
  if (dtype == PS_DTYPE_BF16 && !device_is_sm103()) return PS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, ps_lmhead_ppo_bwd_workspace_size(N, d, V, dtype, 128), s);
  if (rc != PS_OK) return rc;
  if (N == 0) {
    if (dW && !(flags & PS_DW_ACCUMULATE))
      return cudaMemsetAsync(dW, 0, sizeof(float) * static_cast<size_t>(V) * d, s) == cudaSuccess ? PS_OK
                                                                                                : PS_ERR_CUDA;
    return PS_OK;
  }
  const int64_t ldz = ldz_for(V);
  const size_t es = elem_size(dtype);
  int64_t chunk = static_cast<int64_t>((ws_bytes - kWsHeader) / (static_cast<size_t>(ldz) * es)) / 128 * 128;
  if (chunk < 1) return PS_ERR_WORKSPACE;
  // As few chunks as the workspace allows, of equal size (a multiple of 128 rows): a short last
  // chunk would cost a whole pass over dW for little work.
  const int64_t nchunks = (N + chunk - 1) / chunk;
  chunk = ((N + nchunks - 1) / nchunks + 127) / 128 * 128;
  if (chunk >= N) chunk = N;
  void* dz = static_cast<uint8_t*>(ws) + kWsHeader;
  for (int64_t r0 = 0; r0 < N; r0 += chunk) {
    const int64_t rcn = (N - r0) < chunk ? (N - r0) : chunk;
    const int acc = (r0 > 0 || (flags & PS_DW_ACCUMULATE)) ? 1 : 0;
    const int hacc = (flags & PS_DH_ACCUMULATE) ? 1 : 0;
    if (dtype == PS_DTYPE_BF16) {
      const uint16_t* h = static_cast<const uint16_t*>(Hpk) + r0 * d;
      rc = bwd_chunk_bf16(rcn, d, V, h, W, tok + r0, lse + r0, coef + r0, dH ? dH + r0 * d : nullptr, dW, acc, dz,
                          ldz, status_word(ws), s, static_cast<int>(tok_base), hacc);
    } else {
      const float* h = static_cast<const float*>(Hpk) + r0 * d;
      rc = bwd_chunk_f32(rcn, d, V, h, static_cast<const float*>(W), tok + r0, lse + r0, coef + r0,
                         dH ? dH + r0 * d : nullptr, dW, acc, static_cast<float*>(dz), ldz, status_word(ws), s,
                         static_cast<int>(tok_base), hacc);
    }
    if (rc != PS_OK) return rc;
  }
  return PS_OK;
}

extern "C" {

int ps_lmhead_ppo_bwd(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W, const int32_t* tok,
                      const float* lse, const float* coef, float* dH, float* dW, int flags, void* ws,
                      size_t ws_bytes, ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_bwd");
  return lmhead_bwd_impl(N, d, V, 0, dtype, Hpk, W, tok, lse, coef, dH, dW, flags, ws, ws_bytes, stream);
}

int ps_lmhead_ppo_bwd_vocab_shard(int64_t N, int d, int Vs, int64_t v0, int V, int dtype, const void* Hpk,
                                  const void* W_shard, const int32_t* tok, const float* lse, const float* coef,
                                  float* dH, float* dW_shard, int flags, void* ws, size_t ws_bytes,
                                  ps_stream_t stream) {
  NvtxRange nvtx_range("ps_lmhead_ppo_bwd_vocab_shard");
  if (Vs < 1 || v0 < 0 || V < 1 || v0 + Vs > V) return PS_ERR_INVALID_ARG;
  return lmhead_bwd_impl(N, d, Vs, v0, dtype, Hpk, W_shard, tok, lse, coef, dH, dW_shard, flags, ws, ws_bytes,
                         stream);
}

// ----------------------------------------------------------------------------- diagnostics
int ps_diag_gemm_bf16(int M, int N, int K, int a_mn_major, int b_mn_major, const void* A, int64_t lda,
                      const void* B, int64_t ldb, float* C, int64_t ldc, int accumulate, int variant, void* ws,
                      size_t ws_bytes, ps_stream_t stream) {
  if (M < 1 || N < 1 || K < 1 || !A || !B || !C || ldc < N || ldc % 4 || !al16(C)) return PS_ERR_INVALID_ARG;
  if (lda < (a_mn_major ? M : K) || ldb < (b_mn_major ? N : K) || lda % 8 || ldb % 8) return PS_ERR_INVALID_ARG;
  if (!device_is_sm103()) return PS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, kWsHeader, s);
  if (rc != PS_OK) return rc;
  return gemm_bf16(M, N, K, a_mn_major, b_mn_major, A, lda, B, ldb, C, ldc, accumulate, variant, status_word(ws), s);
}

int ps_diag_wait_timeout(uint64_t timeout_ns, void* ws, size_t ws_bytes, ps_stream_t stream) {
  if (timeout_ns > 10000000000ull) return PS_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = begin_call(ws, ws_bytes, kWsHeader, s);
  if (rc != PS_OK) return rc;
  return wait_timeout_probe(timeout_ns, status_word(ws), s);
}

}  // extern "C"
