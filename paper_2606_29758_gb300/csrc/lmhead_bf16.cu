// bf16 LM-head forward/backward on the tcgen05 tensor cores (sm_103a).
//
// Forward (Eq. 1 through the head of Appendix D): Z = Hpk W^T tile by tile; the
// epilogue folds each 32-column slice into a per-row running (max, sum of exp) in
// log2 units and captures the chosen token's logit, so the N x V logits never leave
// TMEM. Backward: the same product is recomputed per chunk of rows and turned into
// dZ = coef (onehot - softmax) in bf16; dH = dZ W and dW = dZ^T Hpk are two more
// tensor-core products over that chunk.
#include <mutex>

#include <cuda_bf16.h>

#include "internal.h"
#include "umma_gemm.cuh"

namespace psk {

// ============================================================================= epilogues
// Value j of a 32-column slice of accumulator registers, picked by a select tree on the bits of j
// (a dynamic index into the registers would move them to local memory).
static __device__ __forceinline__ float pick32(const uint32_t (&r)[32], int j) {
  float a[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) a[i] = __uint_as_float((j & 1) ? r[2 * i + 1] : r[2 * i]);
#pragma unroll
  for (int i = 0; i < 8; ++i) a[i] = (j & 2) ? a[2 * i + 1] : a[2 * i];
#pragma unroll
  for (int i = 0; i < 4; ++i) a[i] = (j & 4) ? a[2 * i + 1] : a[2 * i];
#pragma unroll
  for (int i = 0; i < 2; ++i) a[i] = (j & 8) ? a[2 * i + 1] : a[2 * i];
  return (j & 16) ? a[1] : a[0];
}

struct FwdLseEpi {
  static constexpr int kEpiWarps = 8;   // two column groups per row: two (max, sum) partials per unit
  static constexpr bool kTmaStore = false;
  struct Params {
    const int32_t* tok;
    int M, N;
    float2* part;
    float* ztok;
    int tok_base;   // token ids are global; W holds vocabulary rows [tok_base, tok_base + N)
  };
  struct State {
    float m2, s;
    int tok;
  };
  static __device__ __forceinline__ void begin_unit(const Params& p, State& st, int row, int) {
    st.m2 = -INFINITY;
    st.s = 0.f;
    st.tok = row < p.M ? __ldg(p.tok + row) - p.tok_base : -1;
  }
  static __device__ __forceinline__ void chunk(const Params& p, State& st, int row, int col0,
                                               const uint32_t (&r)[32]) {
    if (col0 >= p.N) return;
    float x[32];
    if (col0 + 32 <= p.N) {
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] = __uint_as_float(r[j]) * kLog2e;
    } else {   // the vocabulary's ragged last slice
      const int nv = p.N - col0;
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] = (j < nv) ? __uint_as_float(r[j]) * kLog2e : -INFINITY;
    }
    float c0 = fmaxf(x[0], x[1]), c1 = fmaxf(x[2], x[3]);
#pragma unroll
    for (int j = 4; j < 32; j += 4) {
      c0 = fmaxf(c0, fmaxf(x[j], x[j + 1]));
      c1 = fmaxf(c1, fmaxf(x[j + 2], x[j + 3]));
    }
    const int rel = st.tok - col0;
    if (static_cast<unsigned>(rel) < 32u) p.ztok[row] = pick32(r, rel);
    const float mn = fmaxf(st.m2, fmaxf(c0, c1));
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
    for (int j = 0; j < 32; j += 4) {
      a0 += ex2_ftz(x[j] - mn);
      a1 += ex2_ftz(x[j + 1] - mn);
      a2 += ex2_ftz(x[j + 2] - mn);
      a3 += ex2_ftz(x[j + 3] - mn);
    }
    st.s = st.s * ex2_ftz(st.m2 - mn) + ((a0 + a1) + (a2 + a3));
    st.m2 = mn;
  }
  static __device__ __forceinline__ void end_unit(const Params& p, State& st, int row, int split) {
    if (row < p.M) p.part[static_cast<size_t>(split) * p.M + row] = make_float2(st.m2, st.s);
  }
};

// FwdLseEpi that also keeps the logits for the backward (the logit store): for every 32-column
// slice of a row, with m the running maximum after the slice (log2 units), it writes the slice's
// e_v = 2^(x_v - m) in f16 (in (0, 1], relative precision 2^-11 down to 2^-14) through TMA and m to
// scale[slice][row]. The sums use the same e_v, in the same order as FwdLseEpi, so lse is the same.
// The backward turns e into dZ = coef (1[v = o] - e 2^(m - lse log2 e)) in place.
struct FwdLseStoreEpi {
  static constexpr int kEpiWarps = 8;   // as FwdLseEpi
  static constexpr bool kTmaStore = true;
  struct Params {
    const int32_t* tok;
    int M, N;
    float2* part;
    float* ztok;
    float* scale;   // [ceil(N / 32)][lds]
    int64_t lds;
    int tok_base;   // token ids are global; W holds vocabulary rows [tok_base, tok_base + N)
  };
  using State = FwdLseEpi::State;
  static __device__ __forceinline__ int cols(const Params& p) { return p.N; }
  static __device__ __forceinline__ void begin_unit(const Params& p, State& st, int row, int) {
    st.m2 = -INFINITY;
    st.s = 0.f;
    st.tok = row < p.M ? __ldg(p.tok + row) - p.tok_base : -1;
  }
  static __device__ __forceinline__ void chunk_to_smem(const Params& p, State& st, int row, int col0,
                                                       const uint32_t (&r)[32], uint8_t* buf, int lane) {
    float x[32];
    if (col0 + 32 <= p.N) {
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] = __uint_as_float(r[j]) * kLog2e;
    } else {   // the vocabulary's ragged last slice
      const int nv = p.N - col0;
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] = (j < nv) ? __uint_as_float(r[j]) * kLog2e : -INFINITY;
    }
    float c0 = fmaxf(x[0], x[1]), c1 = fmaxf(x[2], x[3]);
#pragma unroll
    for (int j = 4; j < 32; j += 4) {
      c0 = fmaxf(c0, fmaxf(x[j], x[j + 1]));
      c1 = fmaxf(c1, fmaxf(x[j + 2], x[j + 3]));
    }
    const int rel = st.tok - col0;
    if (static_cast<unsigned>(rel) < 32u) p.ztok[row] = pick32(r, rel);
    const float mn = fmaxf(st.m2, fmaxf(c0, c1));
#pragma unroll
    for (int j = 0; j < 32; ++j) x[j] = ex2_ftz(x[j] - mn);
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
    for (int j = 0; j < 32; j += 4) {
      a0 += x[j];
      a1 += x[j + 1];
      a2 += x[j + 2];
      a3 += x[j + 3];
    }
    st.s = st.s * ex2_ftz(st.m2 - mn) + ((a0 + a1) + (a2 + a3));
    st.m2 = mn;
    if (row < p.M) p.scale[static_cast<int64_t>(col0 >> 5) * p.lds + row] = mn;
    uint4* dst = reinterpret_cast<uint4*>(buf + lane * 64);
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      dst[q ^ sw] = make_uint4(pack_f16x2(x[8 * q], x[8 * q + 1]), pack_f16x2(x[8 * q + 2], x[8 * q + 3]),
                               pack_f16x2(x[8 * q + 4], x[8 * q + 5]), pack_f16x2(x[8 * q + 6], x[8 * q + 7]));
  }
  static __device__ __forceinline__ void end_unit(const Params& p, State& st, int row, int split) {
    if (row < p.M) p.part[static_cast<size_t>(split) * p.M + row] = make_float2(st.m2, st.s);
  }
};

// Score proxy of the cutoff design (Appendix D): besides the running max m (log2 units, over all
// columns) keep r1 = sum_{v != o} 2^(x_v - m) and r2 = sum_{v != o} 4^(x_v - m) -- the two
// logsumexp reductions of ||p||^2 = exp(LSE(2z) - 2 LSE(z)) with the chosen column o left out, so
// that ||e_o - p||^2 = (r1^2 + r2) / (e_o + r1)^2 keeps its relative accuracy when p(o) -> 1
// (1 - 2 p(o) + ||p||^2 would cancel there).
struct FwdProxyEpi {
  static constexpr int kEpiWarps = 4;
  static constexpr bool kTmaStore = false;
  struct Params {
    const int32_t* tok;
    int M, N;
    float4* part;   // [splits][M] (m2, s1, s2, 0)
    float* ztok;
  };
  struct State {
    float m2, s1, s2;
    int tok;
  };
  static __device__ __forceinline__ void begin_unit(const Params& p, State& st, int row, int) {
    st.m2 = -INFINITY;
    st.s1 = 0.f;
    st.s2 = 0.f;
    st.tok = row < p.M ? __ldg(p.tok + row) : -1;
  }
  static __device__ __forceinline__ void chunk(const Params& p, State& st, int row, int col0,
                                               const uint32_t (&r)[32]) {
    if (col0 >= p.N) return;
    float x[32];
    if (col0 + 32 <= p.N) {
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] = __uint_as_float(r[j]) * kLog2e;
    } else {   // the vocabulary's ragged last slice
      const int nv = p.N - col0;
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] = (j < nv) ? __uint_as_float(r[j]) * kLog2e : -INFINITY;
    }
    float c0 = fmaxf(x[0], x[1]), c1 = fmaxf(x[2], x[3]);
#pragma unroll
    for (int j = 4; j < 32; j += 4) {
      c0 = fmaxf(c0, fmaxf(x[j], x[j + 1]));
      c1 = fmaxf(c1, fmaxf(x[j + 2], x[j + 3]));
    }
    const float mn = fmaxf(st.m2, fmaxf(c0, c1));
    const int rel = st.tok - col0;
    if (static_cast<unsigned>(rel) < 32u) {
      float zt = 0.f;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j == rel) {
          zt = __uint_as_float(r[j]);
          x[j] = -INFINITY;   // the chosen column stays out of r1 and r2
        }
      p.ztok[row] = zt;
    }
    float a0 = 0.f, a1 = 0.f, b0 = 0.f, b1 = 0.f;
#pragma unroll
    for (int j = 0; j < 32; j += 2) {
      const float e0 = ex2_ftz(x[j] - mn), e1 = ex2_ftz(x[j + 1] - mn);
      a0 += e0;
      a1 += e1;
      b0 = fmaf(e0, e0, b0);
      b1 = fmaf(e1, e1, b1);
    }
    const float f = ex2_ftz(st.m2 - mn);
    st.s1 = st.s1 * f + (a0 + a1);
    st.s2 = st.s2 * (f * f) + (b0 + b1);
    st.m2 = mn;
  }
  static __device__ __forceinline__ void end_unit(const Params& p, State& st, int row, int split) {
    if (row < p.M) p.part[static_cast<size_t>(split) * p.M + row] = make_float4(st.m2, st.s1, st.s2, 0.f);
  }
};

// FwdProxyEpi plus the 16 largest logits of the unit's vocabulary range (Appendix I: u_t uses
// the top 16 next tokens). The list stays sorted (descending, lower column first on ties) in
// registers; only the values of a 32-column slice above the current 16th value are inserted.
constexpr int kTopK = 16;
struct FwdProxyTopkEpi {
  static constexpr int kEpiWarps = 4;
  static constexpr bool kTmaStore = false;
  struct Params {
    const int32_t* tok;
    int M, N;
    float4* part;     // [splits][M] (m2, r1, r2, 0)
    float2* topk;     // [splits][M][16] (logit, column as float bits)
    float* ztok;
  };
  struct State {
    FwdProxyEpi::State base;
    float v[kTopK];
    int id[kTopK];
  };
  static __device__ __forceinline__ void begin_unit(const Params& p, State& st, int row, int split) {
    FwdProxyEpi::Params bp{p.tok, p.M, p.N, p.part, p.ztok};
    FwdProxyEpi::begin_unit(bp, st.base, row, split);
#pragma unroll
    for (int j = 0; j < kTopK; ++j) {
      st.v[j] = -INFINITY;
      st.id[j] = -1;
    }
  }
  static __device__ __forceinline__ void chunk(const Params& p, State& st, int row, int col0,
                                               const uint32_t (&r)[32]) {
    if (col0 >= p.N) return;
    const int nv = p.N - col0;
    // Mask of the slice's values above the current 16th largest; after the first slices of a
    // range it is almost always empty. The candidates are then inserted one at a time by one
    // compact loop (a fully unrolled insertion per column overflows the instruction cache).
    const float tau = st.v[kTopK - 1];
    uint32_t m = 0;
#pragma unroll
    for (int j = 0; j < 32; ++j) m |= (j < nv && __uint_as_float(r[j]) > tau) ? (1u << j) : 0u;
#pragma unroll 1
    while (m != 0u) {
      const int j = __ffs(m) - 1;
      m &= m - 1u;
      float x = pick32(r, j);
      if (!(x > st.v[kTopK - 1])) continue;   // the threshold rose since the mask was taken
      int c = col0 + j;
#pragma unroll
      for (int i = 0; i < kTopK; ++i) {
        const bool take = x > st.v[i];
        const float tv = st.v[i];
        const int ti = st.id[i];
        st.v[i] = take ? x : tv;
        st.id[i] = take ? c : ti;
        x = take ? tv : x;
        c = take ? ti : c;
      }
    }
    FwdProxyEpi::Params bp{p.tok, p.M, p.N, p.part, p.ztok};
    FwdProxyEpi::chunk(bp, st.base, row, col0, r);
  }
  static __device__ __forceinline__ void end_unit(const Params& p, State& st, int row, int split) {
    FwdProxyEpi::Params bp{p.tok, p.M, p.N, p.part, p.ztok};
    FwdProxyEpi::end_unit(bp, st.base, row, split);
    if (row < p.M) {
      float2* dst = p.topk + (static_cast<size_t>(split) * p.M + row) * kTopK;
#pragma unroll
      for (int j = 0; j < kTopK; ++j) dst[j] = make_float2(st.v[j], __int_as_float(st.id[j]));
    }
  }
};

// Recomputed logits -> dZ = coef (onehot - softmax) in bf16, stored through TMA: each epilogue warp
// writes its 32 rows x 32 columns of a slice into a staging buffer and one lane issues the tensor
// store (coalesced 64-byte row segments; rows beyond the chunk and columns beyond V are clipped by
// the store itself).
struct BwdDzEpi {
  static constexpr int kEpiWarps = 8;   // no per-row state: the two column groups store their own slices
  static constexpr bool kTmaStore = true;
  struct Params {
    const int32_t* tok;
    const float* lse;
    const float* coef;
    int M, N;
    int tok_base;   // token ids are global; W holds vocabulary rows [tok_base, tok_base + N)
  };
  struct State {
    float lse2, coef;
    int tok;
  };
  static __device__ __forceinline__ int cols(const Params& p) { return p.N; }
  static __device__ __forceinline__ void begin_unit(const Params& p, State& st, int row, int) {
    if (row < p.M) {
      st.tok = __ldg(p.tok + row) - p.tok_base;
      st.lse2 = __ldg(p.lse + row) * kLog2e;
      st.coef = __ldg(p.coef + row);
    } else {
      st.tok = -1;
      st.lse2 = 0.f;
      st.coef = 0.f;   // rows past the chunk: zeros, which the store clips anyway
    }
  }
  // This lane's row of the slice: 32 bf16 = four 16-byte units, unit u at position u ^ ((lane >> 1) & 3)
  // of the lane's 64-byte row in `buf` (the 64-byte swizzle of the dZ tensor map).
  static __device__ __forceinline__ void chunk_to_smem(const Params& p, State& st, int, int col0,
                                                       const uint32_t (&r)[32], uint8_t* buf, int lane) {
    uint32_t pk[16];
    if (st.coef == 0.f) {
#pragma unroll
      for (int j = 0; j < 16; ++j) pk[j] = 0u;
    } else {
      // dZ_v = coef (1[v = o] - p_v). The chosen column o lies in one slice of the ~600 a row has:
      // every other slice is -coef p_v, without the test per column.
      const float nc = -st.coef;
      const int rel = st.tok - col0;
      if (static_cast<unsigned>(rel) < 32u) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float p0 = ex2_ftz(fmaf(__uint_as_float(r[2 * j]), kLog2e, -st.lse2));
          const float p1 = ex2_ftz(fmaf(__uint_as_float(r[2 * j + 1]), kLog2e, -st.lse2));
          pk[j] = pack_bf16x2(fmaf(nc, p0, rel == 2 * j ? st.coef : 0.f), fmaf(nc, p1, rel == 2 * j + 1 ? st.coef : 0.f));
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float p0 = ex2_ftz(fmaf(__uint_as_float(r[2 * j]), kLog2e, -st.lse2));
          const float p1 = ex2_ftz(fmaf(__uint_as_float(r[2 * j + 1]), kLog2e, -st.lse2));
          pk[j] = pack_bf16x2(nc * p0, nc * p1);
        }
      }
    }
    uint4* dst = reinterpret_cast<uint4*>(buf + lane * 64);
    const int x = (lane >> 1) & 3;
#pragma unroll
    for (int q = 0; q < 4; ++q) dst[q ^ x] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
  }
  static __device__ __forceinline__ void end_unit(const Params&, State&, int, int) {}
};

struct StoreF32Epi {
  static constexpr int kEpiWarps = 4;   // its K loops are long: the epilogue is a small share
  static constexpr bool kTmaStore = false;
  struct Params {
    float* out;
    int64_t ld;
    int M, N;
    int accumulate;
  };
  struct State {};
  static __device__ __forceinline__ void begin_unit(const Params&, State&, int, int) {}
  static __device__ __forceinline__ void chunk(const Params& p, State&, int row, int col0, const uint32_t (&r)[32]) {
    if (row >= p.M || col0 >= p.N) return;
    float* dst = p.out + static_cast<int64_t>(row) * p.ld + col0;
    if (col0 + 32 <= p.N) {
      float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v = make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                               __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
        if (p.accumulate) {
          const float4 o = d4[q];
          v.x += o.x;
          v.y += o.y;
          v.z += o.z;
          v.w += o.w;
        }
        d4[q] = v;
      }
    } else {
      const int nv = p.N - col0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j < nv) dst[j] = (p.accumulate ? dst[j] : 0.f) + __uint_as_float(r[j]);
    }
  }
  static __device__ __forceinline__ void end_unit(const Params&, State&, int, int) {}
};

// ============================================================================= logit store -> dZ
// One block turns a 32-row x 1024-column tile of the logit store into dZ in place: the f16
// e_v = 2^(x_v - m) of a 32-column slice (m its scale, log2 units) becomes bf16
// dZ_v = coef (1[v = o] - p_v) with p_v = e_v 2^(m - lse log2 e), the softmax of Eq. 1's gradient
// (Appendix D). The chosen column o takes 1 - p_o = -expm1(logp) from the forward's f32 logp
// rather than from its f16 e, so it keeps its relative accuracy as p_o -> 1. HBM-bound: 4 bytes
// moved per element plus 4 per 32-element slice.
constexpr int kDzRows = 32;
constexpr int kDzCols = 1024;
constexpr int kDzThreads = 256;

__global__ void __launch_bounds__(kDzThreads) dz_from_store_kernel(int64_t N, int V, uint16_t* z, int64_t ldz,
                                                                   const float* scale, int64_t lds,
                                                                   const int32_t* tok, int tok_base,
                                                                   const float* lse, const float* logp,
                                                                   const float* coef) {
  __shared__ float f_s[kDzCols / 32][kDzRows];   // -coef 2^(m - lse log2 e) per slice and row
  __shared__ float one_s[kDzRows];               // coef (1 - p_o)
  __shared__ int tok_s[kDzRows];
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * kDzRows;
  const int c0 = blockIdx.y * kDzCols;
  const int t = threadIdx.x;
#pragma unroll
  for (int k = 0; k < kDzCols / 32 * kDzRows / kDzThreads; ++k) {
    const int idx = t + k * kDzThreads;
    const int sl = idx >> 5, rr = idx & 31;
    const int64_t row = r0 + rr;
    const int col = c0 + sl * 32;
    float f = 0.f;
    if (row < N && col < V)
      f = -__ldg(coef + row) * exp2f(__ldg(scale + static_cast<int64_t>(col >> 5) * lds + row) - __ldg(lse + row) * kLog2e);
    f_s[sl][rr] = f;
  }
  if (t < kDzRows) {
    const int64_t row = r0 + t;
    tok_s[t] = row < N ? __ldg(tok + row) - tok_base : -1;   // outside [0, V): no one-hot term here
    one_s[t] = row < N ? -__ldg(coef + row) * expm1f(__ldg(logp + row)) : 0.f;
  }
  __syncthreads();
  const int warp = t >> 5, lane = t & 31;
#pragma unroll 1
  for (int cs = 0; cs < kDzCols; cs += 256) {
    const int col = c0 + cs + lane * 8;   // this lane's 8 columns, inside slice col / 32
    if (col >= V) break;
    uint4 v[kDzRows / 8];
#pragma unroll
    for (int k = 0; k < kDzRows / 8; ++k) {
      const int64_t row = r0 + warp + 8 * k;
      if (row < N) v[k] = *reinterpret_cast<const uint4*>(z + row * ldz + col);
    }
#pragma unroll
    for (int k = 0; k < kDzRows / 8; ++k) {
      const int rr = warp + 8 * k;
      const int64_t row = r0 + rr;
      if (row >= N) break;
      const float f = f_s[(cs + lane * 8) >> 5][rr];
      const uint32_t w[4] = {v[k].x, v[k].y, v[k].z, v[k].w};
      float o[8];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 e = unpack_f16x2(w[q]);
        o[2 * q] = e.x * f;
        o[2 * q + 1] = e.y * f;
      }
      const int rel = tok_s[rr] - col;
      if (static_cast<unsigned>(rel) < 8u) {
#pragma unroll
        for (int j = 0; j < 8; ++j)
          if (j == rel) o[j] = one_s[rr];
      }
      *reinterpret_cast<uint4*>(z + row * ldz + col) =
          make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]), pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
    }
  }
}

// ============================================================================= host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// 2-D tensor of 2-byte elements (bf16 unless `type` says f16) [outer][inner] with row pitch
// `pitch_bytes`, 128-byte swizzled boxes unless `swizzle` says otherwise.
static bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
                     uint32_t box_inner, uint32_t box_outer,
                     CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B,
                     CUtensorMapDataType type = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (pitch_bytes & 15)) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {pitch_bytes};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, type, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Operand maps. K-major [rows][K]: box 64 (K) x rows_box. MN-major [K][MN]: box 64 x 64.
static bool map_kmajor(CUtensorMap* m, const void* base, int64_t rows, int64_t K, int64_t pitch_elems,
                       uint32_t rows_box) {
  return make_map(m, base, K, rows, pitch_elems * 2, kBK, rows_box);
}
static bool map_mnmajor(CUtensorMap* m, const void* base, int64_t K, int64_t MN, int64_t pitch_elems) {
  return make_map(m, base, MN, K, pitch_elems * 2, 64, kBK);
}

template <bool A_MN, bool B_MN, class Epi, int HALVES = 1>
static int launch_gemm_single(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc, int64_t M,
                              int64_t N, int64_t K, int splits, int band_m, const typename Epi::Params& ep,
                              uint32_t* status, cudaStream_t s) {
  Sched sc;
  sc.m_blocks = static_cast<int>((M + kBM * HALVES - 1) / (kBM * HALVES));
  sc.n_blocks = static_cast<int>((N + kBN - 1) / kBN);
  sc.splits = splits > 0 ? splits : sc.n_blocks;
  sc.band_m = band_m > 0 ? band_m : 1;
  sc.num_units = sc.m_blocks * sc.splits;
  sc.num_kb = static_cast<int>((K + kBK - 1) / kBK);
  if (sc.num_units == 0) return PS_OK;
  if (sc.num_kb == 0) return PS_ERR_INVALID_ARG;
  auto kern = umma_gemm_kernel<A_MN, B_MN, Epi, HALVES>;
  constexpr int EW = EpiWarps<Epi>::value;
  constexpr size_t smem = gemm_smem_bytes<HALVES, EW>();
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
      cudaSuccess)
    return PS_ERR_CUDA;
  const int grid = sc.num_units < num_sms_current() ? sc.num_units : num_sms_current();
  kern<<<grid, 64 + 32 * EW, smem, s>>>(ta, tb, tc, sc, ep, status, kDefaultTimeoutNs);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

// Number of CTA pairs of the pair kernel that fit on the device at once.
template <class K>
static int resident_pairs(K kern) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(2 * (num_sms_current() / 2), 1, 1);
  cfg.blockDim = dim3(kGemmThreads, 1, 1);
  cfg.dynamicSmemBytes = kGemmPairSmemBytes;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kern), &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = num_sms_current() / 2;
  }
  return n;
}

template <bool A_MN, bool B_MN, class Epi>
static int launch_gemm_pair(const CUtensorMap& ta, const CUtensorMap& tb, int64_t M, int64_t N, int64_t K,
                            int splits, int band_m, const typename Epi::Params& ep, uint32_t* status,
                            cudaStream_t s) {
  Sched sc;
  sc.m_blocks = static_cast<int>((M + 255) / 256);
  sc.n_blocks = static_cast<int>((N + kBN - 1) / kBN);
  sc.splits = splits > 0 ? splits : sc.n_blocks;
  sc.band_m = band_m > 0 ? band_m : 1;
  sc.num_units = sc.m_blocks * sc.splits;
  sc.num_kb = static_cast<int>((K + kBK - 1) / kBK);
  if (sc.num_units == 0) return PS_OK;
  if (sc.num_kb == 0) return PS_ERR_INVALID_ARG;
  auto kern = umma_gemm_pair_kernel<A_MN, B_MN, Epi>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kGemmPairSmemBytes)) != cudaSuccess)
    return PS_ERR_CUDA;
  const int pairs = sc.num_units < resident_pairs(kern) ? sc.num_units : resident_pairs(kern);
  kern<<<2 * pairs, kGemmThreads, kGemmPairSmemBytes, s>>>(ta, tb, sc, ep, status, kDefaultTimeoutNs);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

// Row blocks of 128 rows per CTA (single) or 256 rows per CTA pair.
template <bool A_MN, bool B_MN, class Epi>
static int launch_gemm(bool pair, const CUtensorMap& ta, const CUtensorMap& tb, int64_t M, int64_t N, int64_t K,
                       int splits, int band_m, const typename Epi::Params& ep, uint32_t* status, cudaStream_t s) {
  return pair ? launch_gemm_pair<A_MN, B_MN, Epi>(ta, tb, M, N, K, splits, band_m, ep, status, s)
              : launch_gemm_single<A_MN, B_MN, Epi>(ta, tb, ta, M, N, K, splits, band_m, ep, status, s);
}

int fwd_tile_splits_bf16(int V) { return (V + kBN - 1) / kBN; }
int fwd_partials_per_split_bf16() {
  static_assert(FwdLseEpi::kEpiWarps == FwdLseStoreEpi::kEpiWarps, "the two forwards write the same partials");
  return FwdLseEpi::kEpiWarps / 4;
}

// Pick the number of vocabulary ranges per row block (at most max_splits): the makespan of a
// static round-robin over `workers`, in tiles, is rounds x tiles per unit. Among the split
// counts within 1% of the best makespan, take the smallest: fewer ranges mean wider bands of
// row blocks and fewer passes over W.
static int choose_splits(int64_t m_blocks, int64_t n_blocks, int workers, int min_splits, int max_splits) {
  auto cost = [&](int s) {
    const int64_t units = m_blocks * s;
    return ((units + workers - 1) / workers) * ((n_blocks + s - 1) / s);
  };
  const int hi = static_cast<int>(n_blocks < max_splits ? n_blocks : max_splits);
  if (min_splits > hi) return hi;
  int64_t best = INT64_MAX;
  for (int s = min_splits; s <= hi; ++s) best = cost(s) < best ? cost(s) : best;
  for (int s = min_splits; s <= hi; ++s)
    if (cost(s) * 100 <= best * 101) return s;
  return min_splits;
}

// Rows of the K-major B box in the library's GEMMs, which all run one CTA per tile: the whole
// 256-row B tile. (The CTA-pair kernel, reached only through the GEMM test hook, has each CTA
// load half of it, 128 rows; see gemm_bf16.)
constexpr uint32_t kBRowsBox = kBN;
// Tile height of the logit recompute in 128-row halves (see GemmCfg). The wide tile moves a third
// fewer operand bytes per FLOP (about 0.8 vs 0.95 pJ per FLOP at the power cap) but does not overlap
// its epilogue with the next tile; with dZ stored through TMA it is the faster of the two (7B-shaped
// backward 381.4 vs 382.8 ms, and 387.7 ms with per-thread stores of 128-row tiles, back to back).
constexpr int kRecHalves = 2;
// The forward's (and score proxy's) tile height depends on the hidden size: its K loop is d long,
// while the epilogue of a wide tile overlaps the next tile only in part (one TMEM half at a time).
// Measured back to back with the current epilogue: at d = 1536 the wide tile is 3% faster (56.5 vs
// 58.2 ms per 191k-row forward); below d = 1024 the K loop is short enough to keep 128-row tiles.
static int fwd_halves(int d) { return d < 1024 ? 1 : 2; }

// The forward keeps one band of row blocks in flight; every CTA re-reads its row block for
// every vocabulary tile, so the band's hidden rows must stay in L2 (129 MB) next to the W
// tiles being streamed: they get about a quarter of it (30 MB measured 2% faster on the 7B-shaped
// forward than 20 MB or 43 MB, and 64-86 MB were slower still).
constexpr double kFwdBandL2Bytes = 30e6;

static int fwd_band_max(int d) {
  const double block_bytes = static_cast<double>(kBM * fwd_halves(d)) * d * 2.0;
  const int b = static_cast<int>(kFwdBandL2Bytes / block_bytes);
  return b < 1 ? 1 : b;
}

// With a partial per vocabulary tile (splits = tiles) every unit is one tile and the band of
// row blocks walks the vocabulary in lockstep, tile by tile. With fewer partials, units are
// contiguous vocabulary ranges, and the number of ranges is at least what keeps the band in
// its L2 share.
int choose_fwd_splits_bf16(int64_t N, int d, int V, int num_sms, int max_splits) {
  const int nb = fwd_tile_splits_bf16(V);
  if (max_splits >= nb) return nb;
  const int rows = kBM * fwd_halves(d);
  int lo = (num_sms + fwd_band_max(d) - 1) / fwd_band_max(d);
  if (lo > max_splits) lo = max_splits;
  return choose_splits((N + rows - 1) / rows, nb, num_sms, lo, max_splits);
}

int fwd_gemm_bf16(int64_t N, int d, int V, const void* Hpk, const void* W, const int32_t* tok, float2* part,
                  float* ztok, int splits, uint32_t* status, cudaStream_t s, int tok_base) {
  const int halves = fwd_halves(d);
  CUtensorMap ta, tb;
  if (!map_kmajor(&ta, Hpk, N, d, d, kBM * halves) || !map_kmajor(&tb, W, V, d, d, kBRowsBox))
    return PS_ERR_INVALID_ARG;
  FwdLseEpi::Params ep{tok, static_cast<int>(N), V, part, ztok, tok_base};
  const int workers = num_sms_current();
  const int band = splits == fwd_tile_splits_bf16(V) ? fwd_band_max(d) : (workers + splits - 1) / splits;
  if (halves == 1)
    return launch_gemm_single<false, false, FwdLseEpi, 1>(ta, tb, ta, N, V, d, splits, band, ep, status, s);
  return launch_gemm_single<false, false, FwdLseEpi, 2>(ta, tb, ta, N, V, d, splits, band, ep, status, s);
}

// The forward that keeps its logits: f16 e [N][ldz] through TMA (32 x 32 boxes from 64-byte-swizzled
// staging) and the slice maxima scale [ceil(V / 32)][N], on the plain forward's tiles and schedule.
// With 8 epilogue warps the wide tile's epilogue, which also stages and stores every slice, holds
// each TMEM half for half as long: 131.4 / 131.7 ms per 7B forward against 135.9 / 136.8 ms for 4
// epilogue warps on 128-row tiles (back to back).
int fwd_gemm_store_bf16(int64_t N, int d, int V, const void* Hpk, const void* W, const int32_t* tok, float2* part,
                        float* ztok, int splits, void* store, int64_t ldz, float* scale, uint32_t* status,
                        cudaStream_t s, int tok_base) {
  const int halves = fwd_halves(d);
  CUtensorMap ta, tb, tc;
  if (!map_kmajor(&ta, Hpk, N, d, d, kBM * halves) || !map_kmajor(&tb, W, V, d, d, kBRowsBox)) return PS_ERR_INVALID_ARG;
  if (!make_map(&tc, store, V, N, ldz * 2, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_DATA_TYPE_FLOAT16))
    return PS_ERR_INVALID_ARG;
  FwdLseStoreEpi::Params ep{tok, static_cast<int>(N), V, part, ztok, scale, N, tok_base};
  const int workers = num_sms_current();
  const int band = splits == fwd_tile_splits_bf16(V) ? fwd_band_max(d) : (workers + splits - 1) / splits;
  if (halves == 1)
    return launch_gemm_single<false, false, FwdLseStoreEpi, 1>(ta, tb, tc, N, V, d, splits, band, ep, status, s);
  return launch_gemm_single<false, false, FwdLseStoreEpi, 2>(ta, tb, tc, N, V, d, splits, band, ep, status, s);
}

// Bands (row blocks walked together) of the backward GEMMs. Recompute: 32 row blocks of 128 rows
// (16 of its 256-row tiles) share each W tile; their hidden rows, 29 MB at d = 3584, stay in L2
// beside the W tiles in flight and the streamed dZ (44 MB bands read 46% more DRAM). dH and dW: bands of 4 row
// blocks, whose column tiles run side by side, so each panel of dZ (the large operand) is read
// from DRAM about once and the small operand once per wave (measured on the 7B-shaped step:
// bands of 4 beat 1, 2, 8 and 16 by 0.3-1.8% of the backward).
constexpr int kBandRecompute = 32;
constexpr int kBandGrad = 4;

int proxy_gemm_bf16(int64_t N, int d, int V, const void* Hrows, const void* W, const int32_t* tok, float4* part,
                    float* ztok, int splits, uint32_t* status, cudaStream_t s) {
  const int halves = fwd_halves(d);
  CUtensorMap ta, tb;
  if (!map_kmajor(&ta, Hrows, N, d, d, kBM * halves) || !map_kmajor(&tb, W, V, d, d, kBRowsBox))
    return PS_ERR_INVALID_ARG;
  FwdProxyEpi::Params ep{tok, static_cast<int>(N), V, part, ztok};
  const int workers = num_sms_current();
  const int band = splits == fwd_tile_splits_bf16(V) ? fwd_band_max(d) : (workers + splits - 1) / splits;
  if (halves == 1)
    return launch_gemm_single<false, false, FwdProxyEpi, 1>(ta, tb, ta, N, V, d, splits, band, ep, status, s);
  return launch_gemm_single<false, false, FwdProxyEpi, 2>(ta, tb, ta, N, V, d, splits, band, ep, status, s);
}

int proxy_topk_gemm_bf16(int64_t N, int d, int V, const void* Hrows, const void* W, const int32_t* tok,
                         float4* part, float2* topk, float* ztok, int splits, uint32_t* status, cudaStream_t s) {
  CUtensorMap ta, tb;
  if (!map_kmajor(&ta, Hrows, N, d, d, kBM) || !map_kmajor(&tb, W, V, d, d, kBRowsBox)) return PS_ERR_INVALID_ARG;
  FwdProxyTopkEpi::Params ep{tok, static_cast<int>(N), V, part, topk, ztok};
  // Units are contiguous vocabulary ranges; a band of row blocks whose rows fill the forward's L2
  // share walks them range by range, so W is read from DRAM about once per band.
  const int workers = num_sms_current();
  int band = static_cast<int>(kFwdBandL2Bytes / (static_cast<double>(kBM) * d * 2.0));
  if (band < (workers + splits - 1) / splits) band = (workers + splits - 1) / splits;
  return launch_gemm_single<false, false, FwdProxyTopkEpi, 1>(ta, tb, ta, N, V, d, splits, band, ep, status, s);
}

int bwd_chunk_bf16(int64_t rc, int d, int V, const void* Hpk, const void* W, const int32_t* tok,
                   const float* lse, const float* coef, float* dH, float* dW, int dw_accumulate, void* dz,
                   int64_t ldz, uint32_t* status, cudaStream_t s, int tok_base, int dh_accumulate) {
  int rcode;
  {
    CUtensorMap ta, tb;
    if (!map_kmajor(&ta, Hpk, rc, d, d, kBM * kRecHalves) || !map_kmajor(&tb, W, V, d, d, kBRowsBox))
      return PS_ERR_INVALID_ARG;
    // dZ [rc][ldz] bf16, written in 32 x 32 boxes from 64-byte-swizzled staging
    CUtensorMap tz;
    if (!make_map(&tz, dz, V, rc, ldz * 2, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B)) return PS_ERR_INVALID_ARG;
    BwdDzEpi::Params ep{tok, lse, coef, static_cast<int>(rc), V, tok_base};
    rcode = launch_gemm_single<false, false, BwdDzEpi, kRecHalves>(ta, tb, tz, rc, V, d, 0,
                                                                    kBandRecompute / kRecHalves, ep, status, s);
    if (rcode != PS_OK) return rcode;
  }
  return bwd_grads_bf16(rc, d, V, Hpk, W, dH, dW, dw_accumulate, dz, ldz, status, s, dh_accumulate);
}

// dH = dZ W and dW (+)= dZ^T H over rc rows of dZ [rc][ldz] bf16. Both have long K loops (V and rc):
// one CTA computes a 256 x 256 tile as two M = 128 halves that share each B stage (a third fewer
// operand bytes per FLOP).
int bwd_grads_bf16(int64_t rc, int d, int V, const void* Hpk, const void* W, float* dH, float* dW, int dw_accumulate,
                   const void* dz, int64_t ldz, uint32_t* status, cudaStream_t s, int dh_accumulate) {
  int rcode;
  if (dH) {
    CUtensorMap ta, tb;
    if (!map_kmajor(&ta, dz, rc, V, ldz, 2 * kBM) || !map_mnmajor(&tb, W, V, d, d)) return PS_ERR_INVALID_ARG;
    StoreF32Epi::Params ep{dH, d, static_cast<int>(rc), d, dh_accumulate};
    rcode = launch_gemm_single<false, true, StoreF32Epi, 2>(ta, tb, ta, rc, d, V, 0, kBandGrad, ep, status, s);
    if (rcode != PS_OK) return rcode;
  }
  if (dW) {
    CUtensorMap ta, tb;
    if (!map_mnmajor(&ta, dz, rc, V, ldz) || !map_mnmajor(&tb, Hpk, rc, d, d)) return PS_ERR_INVALID_ARG;
    StoreF32Epi::Params ep{dW, d, V, d, dw_accumulate};
    rcode = launch_gemm_single<true, true, StoreF32Epi, 2>(ta, tb, ta, V, d, rc, 0, kBandGrad, ep, status, s);
    if (rcode != PS_OK) return rcode;
  }
  return PS_OK;
}

int dz_from_store_bf16(int64_t N, int V, void* store, int64_t ldz, const float* scale, int64_t lds,
                       const int32_t* tok, const float* lse, const float* logp, const float* coef, cudaStream_t s,
                       int tok_base) {
  if (N == 0) return PS_OK;
  const dim3 grid(static_cast<unsigned>((N + kDzRows - 1) / kDzRows), static_cast<unsigned>((V + kDzCols - 1) / kDzCols));
  dz_from_store_kernel<<<grid, kDzThreads, 0, s>>>(N, V, static_cast<uint16_t*>(store), ldz, scale, lds, tok,
                                                   tok_base, lse, logp, coef);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

int gemm_bf16(int M, int N, int K, int a_mn, int b_mn, const void* A, int64_t lda, const void* B, int64_t ldb,
              float* C, int64_t ldc, int accumulate, int variant, uint32_t* status, cudaStream_t s) {
  if (variant < 0 || variant > 2) return PS_ERR_INVALID_ARG;
  CUtensorMap ta, tb;
  const uint32_t a_rows = variant == 2 ? 2 * kBM : kBM;     // K-major A box rows
  const uint32_t b_rows = variant == 1 ? 128 : kBN;         // K-major B box rows (half per CTA of a pair)
  const bool oka = a_mn ? map_mnmajor(&ta, A, K, M, lda) : map_kmajor(&ta, A, M, K, lda, a_rows);
  const bool okb = b_mn ? map_mnmajor(&tb, B, K, N, ldb) : map_kmajor(&tb, B, N, K, ldb, b_rows);
  if (!oka || !okb) return PS_ERR_INVALID_ARG;
  StoreF32Epi::Params ep{C, ldc, M, N, accumulate};
  using E = StoreF32Epi;
  if (variant == 2) {
    if (!a_mn && !b_mn) return launch_gemm_single<false, false, E, 2>(ta, tb, ta, M, N, K, 0, 16, ep, status, s);
    if (!a_mn && b_mn) return launch_gemm_single<false, true, E, 2>(ta, tb, ta, M, N, K, 0, 16, ep, status, s);
    if (a_mn && b_mn) return launch_gemm_single<true, true, E, 2>(ta, tb, ta, M, N, K, 0, 16, ep, status, s);
    return launch_gemm_single<true, false, E, 2>(ta, tb, ta, M, N, K, 0, 16, ep, status, s);
  }
  const bool p = variant == 1;
  if (!a_mn && !b_mn) return launch_gemm<false, false, E>(p, ta, tb, M, N, K, 0, 16, ep, status, s);
  if (!a_mn && b_mn) return launch_gemm<false, true, E>(p, ta, tb, M, N, K, 0, 16, ep, status, s);
  if (a_mn && b_mn) return launch_gemm<true, true, E>(p, ta, tb, M, N, K, 0, 16, ep, status, s);
  return launch_gemm<true, false, E>(p, ta, tb, M, N, K, 0, 16, ep, status, s);
}

// ----------------------------------------------------------------------------- wait probe
__global__ void wait_probe_kernel(uint64_t timeout_ns, uint32_t* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0, timeout_ns, nullptr)) raise_status(status, PS_DEV_TIMEOUT);
}

int wait_timeout_probe(uint64_t timeout_ns, uint32_t* status, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(timeout_ns, status);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

}  // namespace psk
