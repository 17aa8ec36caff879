/*
 * psppo.h -- C ABI of the GB300 (sm_103a) PS-PPO LM-head update pass.
 *
 * The update pass of Prefix-Sampling PPO (Algorithm 1, steps 6 and 10-11) over the
 * LM head: per-completion cutoffs H ~ xi with inverse-survival weights 1/xi_t
 * (Section 3.2), ragged packing of the retained prefixes with group-normalised
 * advantages (Section 3.1), the weighted clipped PPO surrogate through the head
 * (Eq. 1, Eq. truncated_update_Ghat) and its gradients dH and dW (Appendix D).
 *
 * Conventions shared by every entry point:
 *  - All array pointers are DEVICE pointers owned by the caller, except where an
 *    argument is documented as a host pointer. The library allocates no device
 *    memory; scratch is the caller's workspace `ws` of `ws_bytes` bytes (at least
 *    the matching *_workspace_size(); 256-byte aligned).
 *  - Every call is asynchronous and ordered on `stream` (a cudaStream_t; NULL is
 *    the legacy default stream), unless a host output is requested.
 *  - Every call returns a ps_status (0 = PS_OK). Arguments are checked on the host
 *    before anything is launched; a failed check launches nothing.
 *  - Data that can only be checked on the device (masses that do not sum to 2^62,
 *    a length out of range, a token id outside [0, V), more rows than capacity, a
 *    barrier wait that ran out of time) set bits in a status word at the start of
 *    the call's workspace. Each call clears that word when it starts;
 *    ps_workspace_status() synchronises the stream and reports it.
 *  - Row-major layouts. "bf16" is IEEE bfloat16, "f32" IEEE binary32.
 *  - No global state: calls on different streams with different workspaces may
 *    run concurrently.
 */
#ifndef PSPPO_H_
#define PSPPO_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* ps_stream_t; /* identical to cudaStream_t */

typedef enum {
  PS_OK = 0,
  PS_ERR_INVALID_ARG = 1,   /* a host-checked argument is out of range or NULL */
  PS_ERR_UNSUPPORTED = 2,   /* dtype, shape or device not supported (e.g. not sm_103) */
  PS_ERR_WORKSPACE = 3,     /* ws_bytes smaller than the required size, or ws misaligned */
  PS_ERR_CAPACITY = 4,      /* (device) more packed rows than the given capacity */
  PS_ERR_DEVICE_DATA = 5,   /* (device) bad masses, lengths or token ids */
  PS_ERR_TIMEOUT = 6,       /* (device) a bounded wait inside a kernel ran out */
  PS_ERR_CUDA = 7           /* a CUDA runtime call failed */
} ps_status;

enum { PS_MODE_TRUNC = 0, PS_MODE_FULL = 1, PS_MODE_TRUNC_ZERO = 2 };
enum { PS_DTYPE_BF16 = 0, PS_DTYPE_F32 = 1 };
enum { PS_ADV_CENTERED = 0, PS_ADV_GROUP_NORM = 1 };
/* Backward flags (bits): dW overwritten (0) or added to (PS_DW_ACCUMULATE); dH likewise
 * (PS_DH_ACCUMULATE, e.g. to sum the terms of vocabulary shards run on one device). */
enum { PS_DW_OVERWRITE = 0, PS_DW_ACCUMULATE = 1, PS_DH_ACCUMULATE = 2 };

/* Device status bits (the word at offset 0 of every workspace). */
enum {
  PS_DEV_BAD_PMF = 1, PS_DEV_BAD_LENGTH = 2, PS_DEV_CAPACITY = 4,
  PS_DEV_BAD_TOKEN = 8, PS_DEV_TIMEOUT = 16,
  PS_DEV_NONFINITE = 32   /* ps_design_cutoffs: a timestep weight gamma_bar * u is NaN or infinite */
};

/* Static string for a ps_status value. */
const char* ps_status_string(int status);

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int ps_version(void);

/*
 * Synchronise `stream`, read the device status word of a workspace used by a
 * previous call on that stream, and map it to a ps_status (PS_OK if clear). If
 * `bits` is not NULL (host pointer) the raw PS_DEV_* bits are stored there.
 */
int ps_workspace_status(const void* ws, ps_stream_t stream, uint32_t* bits);

/* ---------------------------------------------------------------------------
 * ps_sample_cutoffs -- cutoffs and inverse-survival weights.
 *
 * Section 3.2: the cutoff H of a completion has survival xi_t = Pr(H >= t | x);
 * tokens t <= H are kept and reweighted by 1/xi_t (Eq. truncated_update_Ghat,
 * Algorithm 1 steps 10-11, unbiased by Appendix B).
 *
 * q      [P][T_max] uint64 masses: Pr(H = h) = q[p][h-1] / 2^62 for prompt p; each
 *        row must sum to exactly 2^62 (checked on the device: PS_DEV_BAD_PMF).
 * L      [B] int32 completion lengths, 1 <= L <= T_max (PS_DEV_BAD_LENGTH), B = P*K;
 *        completion k belongs to prompt k / K.
 * seed, step, traj_base: the cutoff of completion k is decided by the 62-bit
 *        uniform x = (Philox4x64-10(counter = (traj_base + k, step, 0, 0),
 *        key = (seed, 0x5053505030303031))[0]) >> 2, as H = min{h : x < U[h]},
 *        U[h] = q[p][0] + ... + q[p][h-1]. traj_base is the global index of the
 *        first completion, so a batch split across ranks draws the same cutoffs.
 * mode   PS_MODE_TRUNC, PS_MODE_FULL (H = L, weights 1: the untruncated control), or
 *        PS_MODE_TRUNC_ZERO: the masses may sum to less than 2^62 and the deficit is
 *        Pr(H = 0) (the design of Appendix F allows xi_1 < 1); a draw x >= U[T] gives H = 0
 *        and n = 0, and S_p[t] = U_p[T] - U_p[t-1]. A sum above 2^62 sets PS_DEV_BAD_PMF.
 * H, n   [B] int32 outputs: the cutoff and the prefix length n = min(H, L).
 * w_tab  [P][T_max] f32 output: w_tab[p][t-1] = 2^62 / S_p[t] rounded to f32, with
 *        S_p[t] = 2^62 - U_p[t-1] (so 1/w = xi_t exactly before rounding); +inf
 *        where S_p[t] = 0 (never read); 1 in full mode.
 * Limits: 1 <= K <= 8192, 1 <= T_max <= 2^24, P >= 1.
 * ------------------------------------------------------------------------- */
size_t ps_sample_cutoffs_workspace_size(int P, int K, int T_max);
int ps_sample_cutoffs(int P, int K, int T_max, const uint64_t* q, const int32_t* L,
                      uint64_t seed, uint64_t step, int64_t traj_base, int mode,
                      int32_t* H, int32_t* n, float* w_tab,
                      void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_pack_prefixes -- group advantages and the packed prefix rows.
 *
 * Section 3.1: one advantage per completion, A = R - mean_group(R)
 * (PS_ADV_CENTERED) or (R - mean) / (std + 1e-6) with the population std
 * (PS_ADV_GROUP_NORM); group sums run sequentially in f64. Algorithm 1 step 11:
 * only tokens t <= n_k are kept; rows (k, t), k = 0..B-1, t = 1..n_k are laid out
 * back to back in that order.
 *
 * Inputs: L, n [B] int32 (as from ps_sample_cutoffs; 0 <= n <= L), R [B] f32
 * rewards, w_tab [P][T_max] f32, tok_full [sum L] int32, oldlogp_full [sum L] f32,
 * hid_full [sum L][d] (dtype; may be NULL to skip the hidden-state gather).
 * capacity: rows available in every per-row output. If sum n > capacity the call
 * writes no rows and sets PS_DEV_CAPACITY.
 * Outputs: cu_seqlens [B+1] int32 (exclusive scan of n; cu_seqlens[B] = N);
 * per row i < N: tok, oldlogp, w (= w_tab[k/K][t-1]), adv (= A_k, f32),
 * hid_packed [N][d]; optional (may be NULL): src_row (row of the unpacked batch),
 * row_traj (k), row_pos (t, 1-based).
 * h_num_rows: HOST pointer; if not NULL the call synchronises the stream and
 * stores N there.
 * Limits: d >= 8 and d % 8 == 0 (bf16) or d % 4 == 0 (f32); sum L < 2^31.
 * ------------------------------------------------------------------------- */
size_t ps_pack_prefixes_workspace_size(int P, int K);
int ps_pack_prefixes(int P, int K, int T_max, int d, int dtype,
                     const int32_t* L, const int32_t* n, const float* R, int adv_mode,
                     const float* w_tab, const int32_t* tok_full, const float* oldlogp_full,
                     const void* hid_full, int64_t capacity,
                     int32_t* cu_seqlens, int32_t* src_row, int32_t* row_traj, int32_t* row_pos,
                     int32_t* tok, float* oldlogp, float* w, float* adv, void* hid_packed,
                     int64_t* h_num_rows, void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_lmhead_ppo_fwd -- fused LM-head forward: loss without materialised logits.
 *
 * For each packed row i (Appendix D head, Eq. 1 surrogate):
 *   z_i = W h_i (W stored [V][d]; f32 accumulation), lse_i = log sum_v exp(z_iv),
 *   logp_i = z_{i,tok_i} - lse_i, ratio_i = exp(logp_i - oldlogp_i),
 *   s_i = min(ratio_i adv_i, clip(ratio_i, 1-eps, 1+eps) adv_i),
 *   row_loss_i = -loss_scale * w_i * s_i,   loss = sum_i row_loss_i (f64, fixed order),
 *   coef_i = d loss / d logp_i = -loss_scale * w_i * adv_i * ratio_i, or 0 where the
 *   clip binds ((adv > 0 and ratio > 1+eps) or (adv < 0 and ratio < 1-eps)).
 * loss_scale is 1/(P*K) for the paper's estimator (1/K per prompt, mean over prompts).
 * Data-parallel use: split the batch by whole prompt groups (advantages are per group),
 * give every shard's ps_sample_cutoffs the global index of its first completion as
 * traj_base and every shard's forward the whole batch's 1/(P*K); the sums of the shards'
 * losses and dW (an all-reduce across devices, or PS_DW_ACCUMULATE for shards run one
 * after another on one device) are then the whole batch's (Eq. full_update_G).
 *
 * Hpk [N][d], W [V][d]: dtype PS_DTYPE_BF16 (tcgen05 tensor cores) or PS_DTYPE_F32
 * (f32 CUDA cores). tok [N] int32 (0 <= tok < V, else PS_DEV_BAD_TOKEN), oldlogp,
 * adv, w [N] f32. Outputs: loss [1] f64 (device), lse, logp, ratio, coef [N] f32,
 * row_loss [N] f32 (may be NULL). Only O(N) values are written; the N x V logits
 * are never stored (ps_lmhead_ppo_fwd_store below keeps them).
 * Workspace: ps_lmhead_ppo_fwd_workspace_size() bytes hold the (max, sum) partials of
 * every row for every 256-column vocabulary tile, the fastest schedule: bf16 two per tile
 * (one per half of the tile's columns: 16 B x ceil(V/256) per row), f32 one per 64-column
 * tile, plus 4 B per row and a few KB. A smaller bf16 workspace is accepted down to one
 * vocabulary range per row (16 B); the forward then splits the vocabulary into as many
 * ranges as fit (more passes over W). f32 needs the full size. Too small:
 * PS_ERR_WORKSPACE, nothing launched.
 * Limits: N >= 0 (N = 0 writes loss = 0), 1 <= V < 2^31, d >= 8 and d % 8 == 0 (bf16)
 * or d % 4 == 0 (f32); 16-byte aligned Hpk and W.
 * ------------------------------------------------------------------------- */
size_t ps_lmhead_ppo_fwd_workspace_size(int64_t N, int d, int V, int dtype);
int ps_lmhead_ppo_fwd(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W,
                      const int32_t* tok, const float* oldlogp, const float* adv, const float* w,
                      double eps, double loss_scale,
                      double* loss, float* lse, float* logp, float* ratio, float* coef,
                      float* row_loss, void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_lmhead_ppo_bwd -- fused LM-head backward over recomputed logit tiles.
 *
 * Appendix D: d logp / dz = e_o - p. With coef from the forward:
 *   dZ_iv = coef_i (1[v = tok_i] - exp(z_iv - lse_i)),
 *   dH = dZ W            [N][d] f32 (overwritten, or added to with PS_DH_ACCUMULATE),
 *   dW = dZ^T Hpk        [V][d] f32 (overwritten, or added to with PS_DW_ACCUMULATE).
 * The logits are recomputed tile by tile; dZ is held, in the operand dtype, only
 * for one chunk of rows at a time inside the workspace: the rows are split into as
 * few chunks as the workspace holds (ws_bytes), of equal size rounded up to a
 * multiple of 128 rows, so a larger workspace means fewer chunks. dH or dW may be
 * NULL to skip that product.
 * Limits as for the forward; ws_bytes >= ps_lmhead_ppo_bwd_workspace_size(N, d, V,
 * dtype, 128) (one chunk of 128 rows).
 * ------------------------------------------------------------------------- */
size_t ps_lmhead_ppo_bwd_workspace_size(int64_t N, int d, int V, int dtype, int64_t chunk_rows);
int ps_lmhead_ppo_bwd(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W,
                      const int32_t* tok, const float* lse, const float* coef,
                      float* dH, float* dW, int flags,
                      void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * Logit store: the forward keeps the head's logits for the backward, which then
 * executes 4NdV instead of 6NdV FLOPs (no recomputation), at the price of N x V
 * 2-byte values of device memory (about 60 GB for 2e5 rows of a 152k vocabulary).
 * The same loss and gradients as ps_lmhead_ppo_fwd / ps_lmhead_ppo_bwd (Eq. 1,
 * the head of Appendix D); bf16 only (PS_DTYPE_F32: PS_ERR_UNSUPPORTED).
 *
 * ps_lmhead_logit_store_size(N, V): bytes of the store of N rows (0 for bad args).
 * Layout (owned by the caller, 16-byte aligned, written by the forward and
 * consumed by the backward of the same N, Hpk, W and tok):
 *   [N][ldz] 2-byte values, ldz = V rounded up to a multiple of 8: after the forward
 *   f16 e_iv = 2^(x_iv - m_ic) with x = z log2(e), for the 32-column slice c = v / 32,
 *   where m_ic is a running maximum of row i's x over the forward's sweep, at least
 *   the largest x of slice c (so e is in [0, 1]; relative precision 2^-11 above 2^-14);
 *   then, from byte offset ceil(N * ldz * 2 / 256) * 256, f32 m [ceil(V/32)][N].
 * ps_lmhead_ppo_fwd_store: ps_lmhead_ppo_fwd (same arguments, outputs, workspace,
 *   limits and errors) that also fills the store. store_bytes below
 *   ps_lmhead_logit_store_size(N, V): PS_ERR_WORKSPACE, nothing launched.
 * ps_lmhead_ppo_bwd_from_store: the backward of ps_lmhead_ppo_bwd from the store,
 *   which it overwrites in place with dZ [N][ldz] bf16:
 *     dZ_iv = coef_i (1[v = tok_i] - e_iv 2^(m_ic - lse_i log2(e))) for v != tok_i,
 *     dZ_i,tok_i = coef_i (1 - exp(logp_i)) from the forward's logp,
 *   then dH = dZ W and dW = dZ^T Hpk over all N rows (flags PS_DW_ACCUMULATE,
 *   PS_DH_ACCUMULATE as for ps_lmhead_ppo_bwd; dH or dW may be NULL). lse, logp and
 *   coef are the forward's outputs. Workspace: the status header,
 *   ps_lmhead_ppo_bwd_from_store_workspace_size() bytes. Calling it twice on one
 *   store is an error the library cannot see (the second call reads dZ as e).
 * ------------------------------------------------------------------------- */
size_t ps_lmhead_logit_store_size(int64_t N, int V);
int ps_lmhead_ppo_fwd_store(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W,
                            const int32_t* tok, const float* oldlogp, const float* adv,
                            const float* w, double eps, double loss_scale,
                            double* loss, float* lse, float* logp, float* ratio, float* coef,
                            float* row_loss, void* store, size_t store_bytes,
                            void* ws, size_t ws_bytes, ps_stream_t stream);
size_t ps_lmhead_ppo_bwd_from_store_workspace_size(void);
int ps_lmhead_ppo_bwd_from_store(int64_t N, int d, int V, int dtype, const void* Hpk,
                                 const void* W, const int32_t* tok, const float* lse,
                                 const float* logp, const float* coef,
                                 void* store, size_t store_bytes, float* dH, float* dW,
                                 int flags, void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * Vocabulary-parallel head: W split by vocabulary rows across devices.
 *
 * The same loss and gradients as ps_lmhead_ppo_fwd / ps_lmhead_ppo_bwd (Eq. 1 through
 * the head of Appendix D) when each device holds a shard W_shard = rows [v0, v0 + Vs)
 * of W [V][d] and every packed row. Per step:
 *   1. every shard: ps_lmhead_logit_stats -> its per-row statistics (12 bytes a row);
 *   2. gather the S shards' statistics on every device ([S][N] each, shard order);
 *   3. every device: ps_lmhead_ppo_fwd_from_stats -> loss, lse, logp, ratio, coef,
 *      row_loss, identical on all devices;
 *   4. every shard: ps_lmhead_ppo_bwd_vocab_shard -> its dW rows and its part of dH;
 *   5. sum the S parts of dH.
 * The steps run on one device too, shard after shard (a head larger than one launch
 * should take, or a test of the split).
 *
 * ps_lmhead_logit_stats: for every row i, with z_iv = W[v] . Hpk[i] over the shard,
 *   stats[i] = (m_i, s_i), m_i = max_v z_iv log2(e), s_i = sum_v 2^(z_iv log2(e) - m_i),
 *   ztok[i]  = z_{i, tok_i} if v0 <= tok_i < v0 + Vs, else -inf.
 *   stats is [N][2] f32 (8-byte aligned), ztok [N] f32; tok holds global token ids and
 *   is not range-checked here (a shard does not know the others' range).
 *   ws_bytes >= ps_lmhead_logit_stats_workspace_size(N, d, Vs, dtype); fewer bytes
 *   than that give fewer vocabulary ranges, as for the forward.
 * ps_lmhead_ppo_fwd_from_stats: stats [S][ld][2] and ztok [S][ld] of the S shards (ld >= N
 *   rows between shards; rows [0, N) of each are read); per
 *   row, m = max_r m_r, s = sum_r s_r 2^(m_r - m), lse = (m + log2 s) ln 2, the chosen
 *   logit from the shard that holds it, then the forward's outputs exactly as defined
 *   under ps_lmhead_ppo_fwd (a token id outside [0, V) sets PS_DEV_BAD_TOKEN and gives
 *   NaN in its row and the loss). ws_bytes >= ps_lmhead_ppo_fwd_from_stats_workspace_size(N).
 * ps_lmhead_ppo_bwd_vocab_shard: ps_lmhead_ppo_bwd over the shard, with global token ids
 *   (the one-hot term applies where tok_i - v0 is in [0, Vs)) and the lse and coef of
 *   step 3: dW_shard [Vs][d] is the shard's rows of dW; dH [N][d] is the shard's term of
 *   dH (the S terms sum to dH; with PS_DH_ACCUMULATE it is added to dH, which sums the
 *   shards run one after another on one device). Requires 0 <= v0, v0 + Vs <= V; workspace as for
 *   ps_lmhead_ppo_bwd_workspace_size(N, d, Vs, dtype, chunk_rows).
 * ------------------------------------------------------------------------- */
size_t ps_lmhead_logit_stats_workspace_size(int64_t N, int d, int Vs, int dtype);
int ps_lmhead_logit_stats(int64_t N, int d, int Vs, int64_t v0, int dtype, const void* Hpk,
                          const void* W_shard, const int32_t* tok, float* stats, float* ztok,
                          void* ws, size_t ws_bytes, ps_stream_t stream);
size_t ps_lmhead_ppo_fwd_from_stats_workspace_size(int64_t N);
int ps_lmhead_ppo_fwd_from_stats(int64_t N, int S, int64_t ld, int V, const float* stats, const float* ztok,
                                 const int32_t* tok, const float* oldlogp, const float* adv,
                                 const float* w, double eps, double loss_scale, double* loss,
                                 float* lse, float* logp, float* ratio, float* coef,
                                 float* row_loss, void* ws, size_t ws_bytes, ps_stream_t stream);
int ps_lmhead_ppo_bwd_vocab_shard(int64_t N, int d, int Vs, int64_t v0, int V, int dtype,
                                  const void* Hpk, const void* W_shard, const int32_t* tok,
                                  const float* lse, const float* coef, float* dH, float* dW_shard,
                                  int flags, void* ws, size_t ws_bytes, ps_stream_t stream);

/* The vocabulary-parallel steps with a logit store per shard (bf16 only):
 * ps_lmhead_logit_stats_store: ps_lmhead_logit_stats (same arguments, outputs, workspace and
 *   errors) that also fills the shard's store, laid out as for ps_lmhead_ppo_fwd_store with
 *   Vs columns (store_bytes >= ps_lmhead_logit_store_size(N, Vs), else PS_ERR_WORKSPACE).
 * ps_lmhead_ppo_bwd_vocab_shard_from_store: ps_lmhead_ppo_bwd_vocab_shard from the shard's
 *   store, which it overwrites with the shard's dZ [N][ldz] (ldz = Vs rounded up to 8), as
 *   ps_lmhead_ppo_bwd_from_store does; lse, logp and coef from step 3 (the one-hot column
 *   takes 1 - exp(logp_i) where tok_i - v0 is in [0, Vs)). Workspace: the status header,
 *   ps_lmhead_ppo_bwd_from_store_workspace_size() bytes.
 */
int ps_lmhead_logit_stats_store(int64_t N, int d, int Vs, int64_t v0, int dtype, const void* Hpk,
                                const void* W_shard, const int32_t* tok, float* stats, float* ztok,
                                void* store, size_t store_bytes, void* ws, size_t ws_bytes,
                                ps_stream_t stream);
int ps_lmhead_ppo_bwd_vocab_shard_from_store(int64_t N, int d, int Vs, int64_t v0, int V, int dtype,
                                             const void* Hpk, const void* W_shard, const int32_t* tok,
                                             const float* lse, const float* logp, const float* coef,
                                             void* store, size_t store_bytes, float* dH,
                                             float* dW_shard, int flags, void* ws, size_t ws_bytes,
                                             ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_lmhead_score_proxy -- per-token output-head score proxy (cutoff design input).
 *
 * Appendix D: for a softmax head the squared norm of the head score is
 *   gamma_i = ||h_i||^2 (1 - 2 p_i(o_i) + ||p_i||^2),  p_i = softmax(W h_i),
 * i.e. ||h_i||^2 ||e_o - p_i||^2. The epilogue keeps two running sums over the row's
 * logits other than the chosen one, r1 = sum_v e^(z_v - m) and r2 = sum_v e^(2 (z_v - m)),
 * and evaluates ||e_o - p||^2 = (r1^2 + r2) / (e^(z_o - m) + r1)^2, which does not cancel as
 * p(o) -> 1. One pass of the head GEMM over the rows (e.g. every token of the rollouts,
 * with the old-policy head) gives gamma [N] f32 and, if logp is not NULL, log p_i(o_i) [N] f32.
 * Hrows [N][d] bf16, W [V][d] bf16 (bf16 only: other dtypes return PS_ERR_UNSUPPORTED),
 * tok [N] int32 (PS_DEV_BAD_TOKEN and NaN outputs for ids outside [0, V)).
 * topk (0..16): if > 0, the same pass also returns each row's topk most likely next tokens,
 * top_idx [N][topk] int32 (descending probability, lower id first on ties) and their
 * probabilities top_prob [N][topk] f32 -- the input of ps_reward_uncertainty (Appendix I
 * uses 16).
 * Workspace: as many vocabulary partials per row as fit (16 B each; with topk > 0, 144 B each
 * and at most 16), up to ps_lmhead_score_proxy_workspace_size(); at least one per row.
 * ------------------------------------------------------------------------- */
size_t ps_lmhead_score_proxy_workspace_size(int64_t N, int d, int V, int dtype, int topk);
int ps_lmhead_score_proxy(int64_t N, int d, int V, int dtype, const void* Hrows, const void* W,
                          const int32_t* tok, float* gamma, float* logp,
                          int topk, int32_t* top_idx, float* top_prob,
                          void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_reward_uncertainty -- the reward-uncertainty proxy u_t of each prompt and step.
 *
 * Appendix E (Eq. ut_def): u_t = 1/2 - 1/2 || p pi_G(.|t) - (1 - p) pi_B(.|t) ||_1, an upper
 * bound on E[Var(R | S_t) | x] for binary rewards, estimated from the group's K completions:
 * p = fraction with R >= 0.5; pi_G / pi_B average the old-policy next-token distributions at
 * step t over the successful / unsuccessful completions that reach t (an empty class adds 0).
 * Each distribution is its top-k tokens plus one "other" symbol with its remaining mass
 * (the top-k approximation of Appendix I). Output u [P][T_max] f32, 0 beyond a group's
 * horizon. Inputs: L [B], R [B] f32, top_idx [sum L][topk] int32 and top_prob [sum L][topk]
 * f32 in completion order (as from ps_lmhead_score_proxy). Limits: K <= 64, 1 <= topk <= 16.
 * ------------------------------------------------------------------------- */
size_t ps_reward_uncertainty_workspace_size(int P, int K);
int ps_reward_uncertainty(int P, int K, int T_max, const int32_t* L, const float* R, int topk,
                          const int32_t* top_idx, const float* top_prob, float* u,
                          void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_binarize_rewards -- binary labels of continuous rewards, for u_t only.
 *
 * Appendix G: to use the u_t estimate with a continuous reward r, each completion's reward is
 * turned into a label y ~ Bernoulli(sigma(r)), sigma(r) = 1 / (1 + e^-r); the labels feed
 * ps_reward_uncertainty (as R), while the update keeps the continuous rewards. Completion k
 * (global index traj_base + k) draws u = m 2^-53 from Philox4x64-10 with key (seed,
 * 0x5053505052574431 "PSPPRWD1") and counter (traj_base + k, step, 0, 0), m = first output
 * word >> 11, and y_k = 1 if u < sigma(R_k), else 0 (a NaN reward gives 0). sigma is taken by
 * a fixed sequence of double operations (|r| clamped to 40, exp by range reduction and a
 * degree-16 Taylor polynomial), so the labels are reproducible bit for bit. Binary rewards
 * in {0, 1} need no binarisation: pass them to ps_reward_uncertainty directly.
 * R [B] f32 in, y [B] f32 out (0 or 1). No workspace; asynchronous on `stream`.
 * ------------------------------------------------------------------------- */
int ps_binarize_rewards(int B, const float* R, uint64_t seed, uint64_t step, int64_t traj_base,
                        float* y, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_design_cutoffs -- the per-prompt cutoff distribution and its integer masses.
 *
 * Section 3.3 / Algorithm 1 steps 7-9, Appendix F, and the Section 4 variants. For prompt p
 * with horizon T_p = max of its group's lengths and budget B_p = min(budget, T_p):
 *  PS_DESIGN_OPTIMIZED: gamma_bar_t = (1/K) sum of gamma over the group's completions that
 *    reach step t (shorter ones count as 0); w_t = gamma_bar_t * u_t (u_t = 1 if u is NULL),
 *    raised to at least 1e-12 * max_t w_t; xi minimises sum_t w_t / xi_t subject to
 *    sum_t xi_t = B_p and 1 >= xi_1 >= ... >= xi_T_p: pooled blocks with
 *    xi_m = B s_m / sum_j L_j s_j, s_m = sqrt(W_m / L_m) (adjacent violators merged), and the
 *    smallest saturated prefix xi = 1 whose remaining design starts at or below 1.
 *  PS_DESIGN_HEURISTIC: xi_t = B sqrt(w_t) / sum_j sqrt(w_j), then xi_t <- min(xi_{t-1}, xi_t),
 *    then min(xi_t, 1).
 *  PS_DESIGN_UNIFORM: xi_t = (T_p - t + 1) / T_p (cutoff uniform on 1..T_p; budget unused).
 *  PS_DESIGN_TIME_PRIOR: xi_t = exp(-lambda (t - 1)), lambda >= 0 with sum_t xi_t = B_p.
 *  PS_DESIGN_FIXED: xi_t = 1 for t <= param, 0 after (the biased fixed-prefix control).
 * Outputs: q [P][T_max] uint64 masses, q[p][h-1] = floor((xi_h - xi_{h+1}) 2^62) (xi_{T+1} = 0;
 * an excess over 2^62 from rounding is taken off the largest mass), zero beyond T_p; the
 * deficit 2^62 - sum_h q[p][h-1] is Pr(H = 0): sample with PS_MODE_TRUNC_ZERO. xi [P][T_max]
 * f64 (may be NULL). Inputs: L [B] int32, gamma_full [sum L] f32 in completion order (needed
 * by OPTIMIZED and HEURISTIC, may be NULL otherwise), u [P][T_max] f32 or NULL. A weight
 * that is NaN or infinite sets PS_DEV_NONFINITE (the design is then undefined).
 * The arithmetic is f64 in the order of the sequential definition (the parallel parts change
 * no rounding), so the masses are reproducible bit for bit.
 * ------------------------------------------------------------------------- */
enum {
  PS_DESIGN_OPTIMIZED = 0, PS_DESIGN_HEURISTIC = 1, PS_DESIGN_UNIFORM = 2,
  PS_DESIGN_TIME_PRIOR = 3, PS_DESIGN_FIXED = 4
};
size_t ps_design_cutoffs_workspace_size(int P, int K, int T_max);
int ps_design_cutoffs(int P, int K, int T_max, const int32_t* L, const float* gamma_full,
                      const float* u, double budget, int strategy, double param,
                      uint64_t* q, double* xi, void* ws, size_t ws_bytes, ps_stream_t stream);

/* ---------------------------------------------------------------------------
 * ps_lmhead_ppo_fwd_noalloc -- ps_lmhead_ppo_fwd for callers that cannot allocate.
 *
 * The paper has no counterpart: this is a deployment variant of the forward above.
 * Some callers cannot allocate device memory for a workspace -- a plugin inside a
 * framework that owns the GPU's memory pool and forbids cudaMalloc, or a deployment
 * whose device memory plan is fixed at start-up. This call computes exactly what
 * ps_lmhead_ppo_fwd computes (same arguments and outputs, same kernels), but takes
 * its scratch from a static 64 MiB device array inside the library instead of a
 * caller workspace. It allocates nothing (no cudaMalloc, no cudaFree, no allocating
 * library routine).
 *  - Memory: every GPU that loads the library holds the 64 MiB array until the
 *    process exits.
 *  - Limit: the forward takes as many vocabulary ranges per row as 64 MiB hold. For bf16
 *    it needs at least one (20 bytes per packed row plus a few KB: about 3.3 million
 *    rows); all ceil(V/256) of them, the fastest schedule, fit up to about 7,000 rows at
 *    V = 152064. For f32, N * ceil(V/64) * 8 bytes must fit. Larger problems return
 *    PS_ERR_UNSUPPORTED and launch nothing.
 *  - Set-up: the first call in each device context looks up the array's device
 *    address (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture. The address is kept per context: after
 *    cudaDeviceReset, or with another context current, the next call looks it up
 *    again (so that call, too, belongs before any capture).
 *  - Sharing: every call on a device uses the same array, which keeps the last call's
 *    contents. Calls that overlap on the GPU (e.g. on two streams without ordering)
 *    race on it; order them. Each call clears the status word it uses.
 *  - Device-side errors (e.g. a token id outside [0, V)) are still detected, but no
 *    workspace is returned to read them from; a bad token id shows as NaN in logp and
 *    loss.
 * ------------------------------------------------------------------------- */
int ps_lmhead_ppo_fwd_noalloc(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W,
                              const int32_t* tok, const float* oldlogp, const float* adv, const float* w,
                              double eps, double loss_scale,
                              double* loss, float* lse, float* logp, float* ratio, float* coef,
                              float* row_loss, ps_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* PSPPO_H_ */
