// f32 LM-head forward/backward on the CUDA cores.
//
// The tensor cores have no full-f32 mode (tf32 keeps a 10-bit mantissa), so f32
// inputs run here with exact f32 products and f32 accumulation. One tiled kernel
// computes C(m, n) = sum_k A(m, k) B(k, n) for arbitrary element strides of A and B
// (so the same kernel serves Z = H W^T, dH = dZ W and dW = dZ^T H) and hands its
// 64 x 64 tile to an epilogue: the forward's per-row (max, sum of exp) over the
// tile (rows reduced across the 16 threads that share them with warp shuffles), the
// backward's dZ, or a plain store.
#include "internal.h"
#include "ps_common.cuh"

namespace psk {

constexpr int kSB = 64;   // tile edge
constexpr int kSK = 16;   // k depth per stage
constexpr int kSThreads = 256;

struct Operand {
  const float* p;
  int64_t s0, s1;  // element strides: A(m, k) = p[m*s0 + k*s1]; B(k, n) = p[k*s0 + n*s1]
};

// Each thread owns rows ty*4+i and columns tx*4+j (i, j < 4) of the 64 x 64 tile, with
// tx = threadIdx % 16 and ty = threadIdx / 16: the 16 threads of a row group sit in one
// half-warp.
template <class Epi>
__global__ void __launch_bounds__(kSThreads)
    simt_gemm_kernel(int64_t M, int64_t N, int64_t K, Operand A, Operand B, typename Epi::Params ep) {
  __shared__ float As[kSK][kSB + 4];
  __shared__ float Bs[kSK][kSB + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int64_t m0 = static_cast<int64_t>(blockIdx.y) * kSB;
  const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kSB;
  float acc[4][4] = {};
  for (int64_t k0 = 0; k0 < K; k0 += kSK) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = tid + e * kSThreads;   // 0..1023
      const int kk = idx & 15, mm = idx >> 4;  // A: 64 rows x 16 k
      const int64_t gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < M && gk < K) ? A.p[gm * A.s0 + gk * A.s1] : 0.f;
      const int nn = idx & 63, kb = idx >> 6;  // B: 16 k x 64 cols
      const int64_t gn = n0 + nn, gkb = k0 + kb;
      Bs[kb][nn] = (gn < N && gkb < K) ? B.p[gkb * B.s0 + gn * B.s1] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kSK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  Epi::tile(ep, M, N, m0 + ty * 4, n0 + tx * 4, blockIdx.x, tx, acc);
}

struct SimtFwdEpi {
  struct Params {
    const int32_t* tok;
    float2* part;   // [n_tiles][M]
    float* ztok;
    int tok_base;   // token ids are global; W holds vocabulary rows [tok_base, tok_base + N)
  };
  static __device__ __forceinline__ void tile(const Params& p, int64_t M, int64_t N, int64_t r0, int64_t c0,
                                              int ntile, int tx, float (&acc)[4][4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t row = r0 + i;
      float x[4];
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        x[j] = (c0 + j < N) ? acc[i][j] * kLog2e : -INFINITY;
        mx = fmaxf(mx, x[j]);
      }
      const int t = row < M ? __ldg(p.tok + row) - p.tok_base : -1;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (c0 + j < N && c0 + j == t) p.ztok[row] = acc[i][j];
#pragma unroll
      for (int o = 8; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float s = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) s += exp2f(x[j] - mx);
#pragma unroll
      for (int o = 8; o >= 1; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if (tx == 0 && row < M) p.part[static_cast<int64_t>(ntile) * M + row] = make_float2(mx, s);
    }
  }
};

struct SimtDzEpi {
  struct Params {
    const int32_t* tok;
    const float* lse;
    const float* coef;
    float* dz;
    int64_t ldz;
    int tok_base;
  };
  static __device__ __forceinline__ void tile(const Params& p, int64_t M, int64_t N, int64_t r0, int64_t c0, int,
                                              int, float (&acc)[4][4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t row = r0 + i;
      if (row >= M) continue;
      const int t = __ldg(p.tok + row) - p.tok_base;
      const float l = __ldg(p.lse + row), c = __ldg(p.coef + row);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t col = c0 + j;
        if (col >= N) continue;
        const float pr = expf(acc[i][j] - l);
        p.dz[row * p.ldz + col] = c * ((col == t ? 1.f : 0.f) - pr);
      }
    }
  }
};

struct SimtStoreEpi {
  struct Params {
    float* out;
    int64_t ld;
    int accumulate;
  };
  static __device__ __forceinline__ void tile(const Params& p, int64_t M, int64_t N, int64_t r0, int64_t c0, int,
                                              int, float (&acc)[4][4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t row = r0 + i;
      if (row >= M) continue;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t col = c0 + j;
        if (col >= N) continue;
        float* d = p.out + row * p.ld + col;
        *d = (p.accumulate ? *d : 0.f) + acc[i][j];
      }
    }
  }
};

template <class Epi>
static int launch_simt(int64_t M, int64_t N, int64_t K, Operand A, Operand B, const typename Epi::Params& ep,
                       cudaStream_t s) {
  if (M == 0 || N == 0) return PS_OK;
  const int64_t gy = (M + kSB - 1) / kSB, gx = (N + kSB - 1) / kSB;
  if (gy > 65535 || gx > 2147483647) return PS_ERR_UNSUPPORTED;
  dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(gy));
  simt_gemm_kernel<Epi><<<grid, kSThreads, 0, s>>>(M, N, K, A, B, ep);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

int fwd_splits_f32(int V) { return (V + kSB - 1) / kSB; }

int fwd_gemm_f32(int64_t N, int d, int V, const float* Hpk, const float* W, const int32_t* tok, float2* part,
                 float* ztok, uint32_t*, cudaStream_t s, int tok_base) {
  Operand A{Hpk, d, 1};  // A(m, k) = H[m][k]
  Operand B{W, 1, d};    // B(k, n) = W[n][k]
  return launch_simt<SimtFwdEpi>(N, V, d, A, B, SimtFwdEpi::Params{tok, part, ztok, tok_base}, s);
}

int bwd_chunk_f32(int64_t rc, int d, int V, const float* Hpk, const float* W, const int32_t* tok,
                  const float* lse, const float* coef, float* dH, float* dW, int dw_accumulate, float* dz,
                  int64_t ldz, uint32_t*, cudaStream_t s, int tok_base, int dh_accumulate) {
  int r = launch_simt<SimtDzEpi>(rc, V, d, Operand{Hpk, d, 1}, Operand{W, 1, d},
                                 SimtDzEpi::Params{tok, lse, coef, dz, ldz, tok_base}, s);
  if (r != PS_OK) return r;
  if (dH) {  // dH(m=i, n=c) = sum_v dz[i][v] W[v][c]
    r = launch_simt<SimtStoreEpi>(rc, d, V, Operand{dz, ldz, 1}, Operand{W, d, 1}, SimtStoreEpi::Params{dH, d, dh_accumulate},
                                  s);
    if (r != PS_OK) return r;
  }
  if (dW) {  // dW(m=v, n=c) = sum_i dz[i][v] H[i][c]
    r = launch_simt<SimtStoreEpi>(V, d, rc, Operand{dz, 1, ldz}, Operand{Hpk, d, 1},
                                  SimtStoreEpi::Params{dW, d, dw_accumulate}, s);
  }
  return r;
}

}  // namespace psk
