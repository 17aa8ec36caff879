// Internal interfaces between the translation units of libpsppo (not exported).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace psk {

int num_sms_current();
int device_is_sm103();

// Forward GEMM with the online-logsumexp epilogue. part: [splits * fwd_partials_per_split_bf16()][N]
// (max2, sum) pairs (max in log2 units); ztok: [N] chosen-token logit, written only for rows whose token id minus
// tok_base falls in [0, V) (W holding vocabulary rows [tok_base, tok_base + V) of a sharded head).
int fwd_tile_splits_bf16(int V);   // one vocabulary range per 256-column vocabulary tile
// (max, sum) partials per vocabulary range of the bf16 forward (one per column group of its
// epilogue): part holds [splits * this][N] entries.
int fwd_partials_per_split_bf16();
// Vocabulary ranges per row block, at most max_splits (the ranges whose partials the workspace
// holds); the score proxy uses the same chooser.
int choose_fwd_splits_bf16(int64_t N, int d, int V, int num_sms, int max_splits);
int fwd_gemm_bf16(int64_t N, int d, int V, const void* Hpk, const void* W, const int32_t* tok, float2* part,
                  float* ztok, int splits, uint32_t* status, cudaStream_t s, int tok_base = 0);
// The same forward keeping its logits (the logit store): store [N][ldz] f16 with e = 2^(x - m) per
// 32-column slice, m the running row maximum after the slice (log2 units), in scale [ceil(V/32)][N].
int fwd_gemm_store_bf16(int64_t N, int d, int V, const void* Hpk, const void* W, const int32_t* tok, float2* part,
                        float* ztok, int splits, void* store, int64_t ldz, float* scale, uint32_t* status,
                        cudaStream_t s, int tok_base = 0);
int fwd_splits_f32(int V);
int fwd_gemm_f32(int64_t N, int d, int V, const float* Hpk, const float* W, const int32_t* tok, float2* part,
                 float* ztok, uint32_t* status, cudaStream_t s, int tok_base = 0);

// Score-proxy GEMM (the forward's schedule): part [splits][N] (max2, s1, s2, 0), ztok [N].
int proxy_gemm_bf16(int64_t N, int d, int V, const void* Hrows, const void* W, const int32_t* tok, float4* part,
                    float* ztok, int splits, uint32_t* status, cudaStream_t s);

// Score proxy plus the 16 largest logits per row and vocabulary range (contiguous ranges, at most
// 16): topk [splits][N][16] (logit, column bits).
int proxy_topk_gemm_bf16(int64_t N, int d, int V, const void* Hrows, const void* W, const int32_t* tok,
                         float4* part, float2* topk, float* ztok, int splits, uint32_t* status, cudaStream_t s);

// Backward for one chunk of rows [0, rc) of already offset pointers: recompute dZ into
// dz ([rc][ldz], operand dtype), then dH = dZ W and dW (+)= dZ^T Hpk. With tok_base, W holds
// vocabulary rows [tok_base, tok_base + V) and the one-hot term applies where tok - tok_base is in [0, V);
// dh_accumulate adds dH to what the buffer holds.
int bwd_chunk_bf16(int64_t rc, int d, int V, const void* Hpk, const void* W, const int32_t* tok,
                   const float* lse, const float* coef, float* dH, float* dW, int dw_accumulate, void* dz,
                   int64_t ldz, uint32_t* status, cudaStream_t s, int tok_base = 0, int dh_accumulate = 0);
// dH = dZ W and dW (+)= dZ^T Hpk from dZ [rc][ldz] bf16 already in memory.
int bwd_grads_bf16(int64_t rc, int d, int V, const void* Hpk, const void* W, float* dH, float* dW, int dw_accumulate,
                   const void* dz, int64_t ldz, uint32_t* status, cudaStream_t s, int dh_accumulate);
// The logit store of the forward turned into dZ in place (f16 e -> bf16 dZ), rows [0, N) of already
// offset pointers; scale [c][lds] (lds: the store's row count, the pitch of its slice maxima). With
// tok_base, the store holds vocabulary columns [tok_base, tok_base + V) and the one-hot term applies
// where tok - tok_base is in [0, V).
int dz_from_store_bf16(int64_t N, int V, void* store, int64_t ldz, const float* scale, int64_t lds,
                       const int32_t* tok, const float* lse, const float* logp, const float* coef, cudaStream_t s,
                       int tok_base = 0);
int bwd_chunk_f32(int64_t rc, int d, int V, const float* Hpk, const float* W, const int32_t* tok,
                  const float* lse, const float* coef, float* dH, float* dW, int dw_accumulate, float* dz,
                  int64_t ldz, uint32_t* status, cudaStream_t s, int tok_base = 0, int dh_accumulate = 0);

// Plain tensor-core GEMM (test hook): C[M][N] (+)= sum_k A(m,k) B(k,n), f32 out. variant: 0 one
// CTA per 128 x 256 tile, 1 a CTA pair per 256 x 256 tile, 2 one CTA per 256 x 256 tile.
int gemm_bf16(int M, int N, int K, int a_mn, int b_mn, const void* A, int64_t lda, const void* B, int64_t ldb,
              float* C, int64_t ldc, int accumulate, int variant, uint32_t* status, cudaStream_t s);

// Bounded-wait self test: waits on an mbarrier nobody arrives at.
int wait_timeout_probe(uint64_t timeout_ns, uint32_t* status, cudaStream_t s);

}  // namespace psk
