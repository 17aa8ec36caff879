// Persistent, warp-specialised tcgen05 GEMM for sm_103a with pluggable epilogues.
//
//   D[M, N] = sum_k A[m, k] B[n, k]      (bf16 operands, f32 accumulation in TMEM)
//
// A is K-major ([M][K] in memory) or MN-major ([K][M]); likewise B ([N][K] or [K][N]).
// Tiles of 128 x 256 or 256 x 256 outputs (HALVES, below), 64-deep K blocks, a shared-memory
// ring fed by TMA with 128-byte swizzle. Roles (64 + 32 x Epi::kEpiWarps threads):
//   warp 0      TMA producer (one lane)
//   warp 1      TMEM allocator + MMA issuer (one lane)
//   warps 2..   epilogue: each thread owns one accumulator row (TMEM lane) and reads its
//               256 columns in chunks of 32 with tcgen05.ld; with 8 epilogue warps two warps
//               share each TMEM lane quarter, one reading columns 0..127 and one 128..255
// An epilogue either stores from registers itself or (Epi::kTmaStore) stages 32 x 32 slices in
// shared memory for TMA tensor stores through a third map. Every wait is bounded; on expiry the
// kernel sets PS_DEV_TIMEOUT, waits (bounded) for its own loads in flight, frees TMEM and returns.
//
// Work is split into units: unit u is (m block, range of n blocks [n0, n1)), walked in
// order by one CTA, so an epilogue can keep per-row state across a unit's tiles (the
// forward's running logsumexp). Units are enumerated in bands of `band_m` m-blocks;
// inside a band the split index is the slow coordinate, so CTAs that run at the same
// time share B panels (and A panels) through L2.
#pragma once

#include "ps_common.cuh"

namespace psk {

constexpr int kBM = 128;
constexpr int kBN = 256;
constexpr int kBK = 64;
constexpr int kGemmThreads = 192;                 // the CTA-pair kernel: 4 epilogue warps
constexpr uint32_t kTileABytes = kBM * kBK * 2;   // 16 KB
constexpr uint32_t kTileBBytes = kBN * kBK * 2;   // 32 KB
constexpr uint32_t kTmemCols = 512;               // two 256-column f32 accumulators

struct Sched {
  int m_blocks;   // ceil(M / 128)
  int n_blocks;   // ceil(N / 256)
  int splits;     // n-ranges per m block (n_blocks: one tile per unit)
  int band_m;     // m blocks per band
  int num_units;  // m_blocks * splits
  int num_kb;     // ceil(K / 64)

  __device__ __forceinline__ void unit(int u, int& m_blk, int& split, int& n0, int& n1) const {
    const int per_band = band_m * splits;
    const int band = u / per_band;
    const int r = u - band * per_band;
    const int m_first = band * band_m;
    const int this_band = min(band_m, m_blocks - m_first);
    split = r / this_band;
    m_blk = m_first + (r - split * this_band);
    n0 = static_cast<int>((static_cast<long long>(split) * n_blocks) / splits);
    n1 = static_cast<int>((static_cast<long long>(split + 1) * n_blocks) / splits);
  }
};

// HALVES = 1: 128 x 256 tiles, two TMEM accumulators (double-buffered, all 512 columns), so the
// epilogue of one tile overlaps the main loop of the next; 4-stage 48 KB ring.
// HALVES = 2: 256 x 256 tiles computed as two M = 128 MMAs that share each B stage, one
// accumulator pair filling TMEM, 3-stage 64 KB ring. The wide tile reads a third fewer operand
// bytes per FLOP. Its epilogue hands TMEM back half by half and the next tile runs ahead on the
// first half for as many k-blocks as the ring holds, so the epilogue overlaps the next tile only
// in part. Each epilogue thread owns one row of each half (two epilogue states).
template <int HALVES>
struct GemmCfg {
  static constexpr int kStagesH = HALVES == 1 ? 4 : 3;
  static constexpr int kRows = kBM * HALVES;                  // rows per tile
  static constexpr uint32_t kABytes = kTileABytes * HALVES;   // A bytes per stage
  static constexpr int kAccBufs = HALVES == 1 ? 2 : 1;        // accumulator buffers in TMEM
};

// Epilogues that store through TMA (Epi::kTmaStore) stage each 32-row x 32-column 2-byte slice of a
// warp in shared memory, 64-byte swizzled (a 64-byte row per TMEM lane, its 16-byte units permuted
// by row bits 1-2, so a warp's stores hit every bank group): two buffers per warp with 4 epilogue
// warps, one with 8 (two fit beside the wide-tile ring, 230.5 KB, but measured no faster).
constexpr int kStageBytes = 32 * 64;

// Epilogue warps per CTA: Epi::kEpiWarps, 4 or 8. With 8, each accumulator row is read by two
// warps (columns 0..127 and 128..255 of every tile), which halves the time an epilogue holds a
// TMEM half; an epilogue with per-row state then keeps one state per column group, and its
// per-unit results (the forward's partials) come in two parts.
template <class Epi>
struct EpiWarps {
  static_assert(Epi::kEpiWarps == 4 || Epi::kEpiWarps == 8, "4 or 8 epilogue warps");
  static constexpr int value = Epi::kEpiWarps;
};
template <int EW>
struct StageBufs { static constexpr int value = EW == 8 ? 1 : 2; };

template <int HALVES, int EW = 4>
struct GemmSmemT {
  // 1024-byte aligned tile ring first (128-byte swizzle atoms repeat every 1 KB)
  uint8_t a[GemmCfg<HALVES>::kStagesH][GemmCfg<HALVES>::kABytes];
  uint8_t b[GemmCfg<HALVES>::kStagesH][kTileBBytes];
  uint8_t stage[EW][StageBufs<EW>::value][kStageBytes];   // store staging of the epilogue warps
  uint64_t full[GemmCfg<HALVES>::kStagesH];
  uint64_t empty[GemmCfg<HALVES>::kStagesH];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
template <int HALVES, int EW = 4>
constexpr size_t gemm_smem_bytes() { return sizeof(GemmSmemT<HALVES, EW>) + 1024; }  // + alignment slack

// tmC: the output map of epilogues that store through TMA (unused by the others). An epilogue's
// begin_unit / end_unit see the unit's split index times the column groups (1 with 4 epilogue
// warps, 2 with 8) plus the thread's column group.
template <bool A_MN, bool B_MN, class Epi, int HALVES = 1>
__global__ void __launch_bounds__(64 + 32 * EpiWarps<Epi>::value, 1)
    umma_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmC, const Sched sched, const typename Epi::Params ep,
                     uint32_t* status, uint64_t timeout_ns) {
  using Cfg = GemmCfg<HALVES>;
  constexpr int S = Cfg::kStagesH;
  constexpr int NB = Cfg::kAccBufs;
  constexpr int EW = EpiWarps<Epi>::value;
  constexpr int G = EW / 4;                 // column groups per TMEM lane quarter
  constexpr int CPG = (kBN / 32) / G;       // 32-column chunks per group
  constexpr int SB = StageBufs<EW>::value;
  extern __shared__ uint8_t smem_raw[];
  GemmSmemT<HALVES, EW>& sm =
      *reinterpret_cast<GemmSmemT<HALVES, EW>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.tfull[a], 1);
      mbar_init(&sm.tempty[a], 32 * EW);
    }
    mbar_init(&sm.drain, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t kc = 0;  // k blocks issued by this CTA
      bool ok = true;
      for (int u = blockIdx.x; ok && u < sched.num_units; u += gridDim.x) {
        int m_blk, split, n0, n1;
        sched.unit(u, m_blk, split, n0, n1);
        for (int nb = n0; ok && nb < n1; ++nb) {
          for (int kb = 0; kb < sched.num_kb; ++kb, ++kc) {
            const int s = kc % S;
            const uint32_t ph = (kc / S) & 1u;
            if (!mbar_wait(&sm.empty[s], ph ^ 1u, timeout_ns, abort)) { ok = false; break; }
            mbar_arrive_expect_tx(&sm.full[s], Cfg::kABytes + kTileBBytes);
            const int m0 = m_blk * Cfg::kRows, nn0 = nb * kBN, k0 = kb * kBK;
            if (A_MN) {
              for (int i = 0; i < Cfg::kRows / 64; ++i)
                tma_load_2d(sm.a[s] + i * (kBK * 128), &tmA, &sm.full[s], m0 + i * 64, k0);
            } else {
              tma_load_2d(sm.a[s], &tmA, &sm.full[s], k0, m0);   // box of kRows rows
            }
            if (B_MN) {
              for (int i = 0; i < kBN / 64; ++i)
                tma_load_2d(sm.b[s] + i * (kBK * 128), &tmB, &sm.full[s], nn0 + i * 64, k0);
            } else {
              tma_load_2d(sm.b[s], &tmB, &sm.full[s], k0, nn0);
            }
          }
        }
      }
      if (!ok) {
        *abort = 1;
        raise_status(status, PS_DEV_TIMEOUT);
        // let the loads already issued land before the CTA can exit
        const uint32_t first = kc > static_cast<uint32_t>(S) ? kc - S : 0;
        for (uint32_t j = first; j < kc; ++j) mbar_wait(&sm.full[j % S], (j / S) & 1u, timeout_ns, nullptr);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, A_MN, B_MN);
      // K-major: 8-row groups 1024 B apart; a 16-deep K step is 32 B inside the swizzle atom.
      // MN-major: 64-element atoms kBK*128 B apart (LBO); 8-row K groups 1024 B apart (SBO);
      //           a 16-deep K step is 16 rows = 2048 B.
      // The second half of a wide tile (rows 128..255) starts 16 KB into the A stage in both
      // layouts (128 K-major rows of 128 B, or two MN-major atoms of 8 KB).
      constexpr uint32_t a_lbo = A_MN ? kBK * 128 : 16, a_step = A_MN ? 2048 : 32;
      constexpr uint32_t b_lbo = B_MN ? kBK * 128 : 16, b_step = B_MN ? 2048 : 32;
      uint32_t kc = 0, tile = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < sched.num_units; u += gridDim.x) {
        int m_blk, split, n0, n1;
        sched.unit(u, m_blk, split, n0, n1);
        for (int nb = n0; ok && nb < n1; ++nb, ++tile) {
          const uint32_t acc = tile % NB;
          const uint32_t aph = (tile / NB) & 1u;
          if (!mbar_wait(&sm.tempty[acc], aph ^ 1u, timeout_ns, abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * kBN;  // NB = 1: halves at columns 0 and 256
          // the MMAs of half h of k-block kb, from stage s (each half accumulates in k order)
          auto issue_half = [&](int h, int s, int kb) {
            const uint32_t a_base = smem_addr(sm.a[s]);
            const uint32_t b_base = smem_addr(sm.b[s]);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) {
              const uint64_t bd = smem_desc_sw128(b_base + k * b_step, b_lbo, 1024);
              const uint64_t ad = smem_desc_sw128(a_base + h * kTileABytes + k * a_step, a_lbo, 1024);
              umma_bf16(d_tmem + h * kBN, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
            }
          };
          if constexpr (HALVES == 1) {
            for (int kb = 0; kb < sched.num_kb; ++kb, ++kc) {
              const int s = kc % S;
              const uint32_t ph = (kc / S) & 1u;
              if (!mbar_wait(&sm.full[s], ph, timeout_ns, abort)) { ok = false; break; }
              tc_fence_after();
              issue_half(0, s, kb);
              umma_commit(&sm.empty[s]);  // frees the stage once these MMAs have read it
            }
          } else {
            // A wide tile's two halves own TMEM columns [0, 256) and [256, 512), and the epilogue
            // hands each back as soon as it has read it (tempty[0], then tempty[1]). The tile starts
            // once half 0 is free; while the epilogue still reads half 1 of the previous tile, the
            // leading k-blocks run on half 0 only and keep their stages; their half-1 MMAs follow, in
            // k order, as soon as half 1 is free -- at the latest when every stage is held.
            bool h1_free = false;
            const uint32_t kc0 = kc;
            for (int kb = 0; kb < sched.num_kb; ++kb, ++kc) {
              const int s = kc % S;
              const uint32_t ph = (kc / S) & 1u;
              if (!mbar_wait(&sm.full[s], ph, timeout_ns, abort)) { ok = false; break; }
              tc_fence_after();
              issue_half(0, s, kb);
              if (h1_free) {
                issue_half(1, s, kb);
                umma_commit(&sm.empty[s]);
                continue;
              }
              if (!mbar_try_wait(&sm.tempty[1], aph ^ 1u)) {
                if (kb + 1 < S && kb + 1 < sched.num_kb) continue;   // a stage is left: run ahead on half 0
                if (!mbar_wait(&sm.tempty[1], aph ^ 1u, timeout_ns, abort)) { ok = false; break; }
              }
              h1_free = true;
              tc_fence_after();
              for (int j = 0; j <= kb; ++j) {          // the held k-blocks' half 1, in order
                const int sj = (kc0 + j) % S;
                issue_half(1, sj, j);
                umma_commit(&sm.empty[sj]);
              }
            }
          }
          if (ok) umma_commit(&sm.tfull[acc]);  // accumulator ready for the epilogue
        }
      }
      if (!ok) {
        *abort = 1;
        raise_status(status, PS_DEV_TIMEOUT);
        // wait (bounded) until the MMAs already issued have finished with TMEM
        umma_commit(&sm.drain);
        mbar_wait(&sm.drain, 0, timeout_ns, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    const int quad = warp & 3;                  // TMEM lanes 32*quad .. 32*quad+31
    const int ew = warp - 2;                    // epilogue warp
    const int grp = ew >> 2;                    // column group: chunks [grp * CPG, grp * CPG + CPG)
    const int row_in_tile = quad * 32 + lane;
    typename Epi::State st[HALVES];             // a thread owns row r of each half
    uint32_t tile = 0;
    uint32_t nstore = 0;                        // TMA-stored slices of this warp
    bool ok = true;
    for (int u = blockIdx.x; ok && u < sched.num_units; u += gridDim.x) {
      int m_blk, split, n0, n1;
      sched.unit(u, m_blk, split, n0, n1);
      const int row0 = m_blk * Cfg::kRows + row_in_tile;
#pragma unroll
      for (int h = 0; h < HALVES; ++h) Epi::begin_unit(ep, st[h], row0 + h * kBM, split * G + grp);
      for (int nb = n0; nb < n1; ++nb, ++tile) {
        const uint32_t acc = tile % NB;
        const uint32_t aph = (tile / NB) & 1u;
        // one lane waits; the warp follows it, so tcgen05.ld always runs on a converged warp
        int got = 0;
        if (lane == 0) got = mbar_wait(&sm.tfull[acc], aph, timeout_ns, abort) ? 1 : 0;
        got = __shfl_sync(0xffffffffu, got, 0);
        if (!got) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int h = 0; h < HALVES; ++h) {
          const int row = row0 + h * kBM;
          const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + acc * kBN + h * kBN;
#pragma unroll 1
          for (int c = grp * CPG; c < grp * CPG + CPG; ++c) {
            uint32_t r[32];
            tmem_ld32(t_row + c * 32, r);
            tmem_ld_wait();
            if (c == grp * CPG + CPG - 1) {
              // this half of the accumulator has been read: hand it back to the MMA warp (a wide
              // tile returns its two halves one after the other, tempty[0] and tempty[1])
              tc_fence_before();
              mbar_arrive(&sm.tempty[HALVES == 2 ? h : acc]);
            }
            const int col0 = nb * kBN + c * 32;
            if constexpr (Epi::kTmaStore) {
              // the slice goes to a staging buffer, then one lane stores the warp's 32 x 32 box
              if (col0 < Epi::cols(ep)) {
                uint8_t* buf = sm.stage[ew][nstore % SB];
                if (lane == 0) bulk_wait_group_read<SB - 1>();   // the store that last used it has read it
                __syncwarp();
                Epi::chunk_to_smem(ep, st[h], row, col0, r, buf, lane);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                  tma_store_2d(&tmC, buf, col0, m_blk * Cfg::kRows + h * kBM + quad * 32);
                  bulk_commit_group();
                }
                ++nstore;
              }
            } else {
              Epi::chunk(ep, st[h], row, col0, r);
            }
          }
        }
      }
      if (ok) {
#pragma unroll
        for (int h = 0; h < HALVES; ++h) Epi::end_unit(ep, st[h], row0 + h * kBM, split * G + grp);
      }
    }
    if (!ok) {
      *abort = 1;
      raise_status(status, PS_DEV_TIMEOUT);
    }
    // the staged stores must finish reading shared memory (and reach global memory) before exit
    if (Epi::kTmaStore && lane == 0) bulk_wait_group_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// =============================================================================================
// CTA-pair variant (tcgen05 cta_group::2). A cluster of two CTAs computes 256 x 256 output
// tiles: each CTA loads its own 128 rows of A and one half (128 rows or columns) of B, so
// a stage is 32 KB per CTA instead of 48 KB and six stages fit. The even CTA ("leader")
// issues the MMAs for the pair (M = 256 split across the two CTAs' TMEM) and owns the
// barriers that gate them:
//   full[s]   (leader)  2 arrivals with expect-tx (one producer per CTA) + 64 KB of TMA bytes
//   empty[s]  (both)    1 arrival: the leader's commit multicast to both CTAs
//   tfull[a]  (both)    1 arrival: the leader's commit multicast to both CTAs
//   tempty[a] (leader)  8 arrivals: one per epilogue warp of either CTA
// Both CTAs walk the same sequence of units; every CTA reads its own TMEM lanes, i.e.
// output rows 256 * m_pair + 128 * rank + lane.
// =============================================================================================
constexpr int kStagesPair = 6;
constexpr uint32_t kHalfBBytes = 128 * kBK * 2;   // 16 KB: one CTA's half of the B tile

struct GemmPairSmem {
  uint8_t a[kStagesPair][kTileABytes];
  uint8_t b[kStagesPair][kHalfBBytes];
  uint64_t full[kStagesPair];
  uint64_t empty[kStagesPair];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
constexpr size_t kGemmPairSmemBytes = sizeof(GemmPairSmem) + 1024;

template <bool A_MN, bool B_MN, class Epi>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    umma_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                          const Sched sched, const typename Epi::Params ep, uint32_t* status,
                          uint64_t timeout_ns) {
  extern __shared__ uint8_t smem_raw[];
  GemmPairSmem& sm =
      *reinterpret_cast<GemmPairSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1;
  const int npairs = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesPair; ++s) {
      mbar_init(&sm.full[s], 2);
      mbar_init(&sm.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.tfull[a], 1);
      mbar_init(&sm.tempty[a], 8);
    }
    mbar_init(&sm.drain, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc_pair(&sm.tmem_base, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();  // barriers of both CTAs initialised before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      uint32_t kc = 0;
      bool ok = true;
      for (int u = pair; ok && u < sched.num_units; u += npairs) {
        int m_blk, split, n0, n1;
        sched.unit(u, m_blk, split, n0, n1);
        for (int nb = n0; ok && nb < n1; ++nb) {
          for (int kb = 0; kb < sched.num_kb; ++kb, ++kc) {
            const int s = kc % kStagesPair;
            const uint32_t ph = (kc / kStagesPair) & 1u;
            if (!mbar_wait(&sm.empty[s], ph ^ 1u, timeout_ns, abort)) { ok = false; break; }
            const uint32_t lfull = mapa_shared(smem_addr(&sm.full[s]), 0);
            mbar_arrive_expect_tx_cluster(lfull, kTileABytes + kHalfBBytes);
            const int m0 = m_blk * 256 + static_cast<int>(rank) * 128;
            const int nn0 = nb * kBN + static_cast<int>(rank) * 128;
            const int k0 = kb * kBK;
            if (A_MN) {
              for (int i = 0; i < 2; ++i) tma_load_2d_pair(sm.a[s] + i * (kBK * 128), &tmA, lfull, m0 + i * 64, k0);
            } else {
              tma_load_2d_pair(sm.a[s], &tmA, lfull, k0, m0);
            }
            if (B_MN) {
              for (int i = 0; i < 2; ++i) tma_load_2d_pair(sm.b[s] + i * (kBK * 128), &tmB, lfull, nn0 + i * 64, k0);
            } else {
              tma_load_2d_pair(sm.b[s], &tmB, lfull, k0, nn0);
            }
          }
        }
      }
      if (!ok) {
        *abort = 1;
        raise_status(status, PS_DEV_TIMEOUT);
        // the leader can see its stages land; the peer's barriers are remote, so it gives
        // its own loads in flight a bounded grace period instead
        if (leader) {
          const uint32_t first = kc > kStagesPair ? kc - kStagesPair : 0;
          for (uint32_t j = first; j < kc; ++j)
            mbar_wait(&sm.full[j % kStagesPair], (j / kStagesPair) & 1u, timeout_ns, nullptr);
        } else {
          const uint64_t t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < 2000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer (leader only)
    if (lane == 0 && leader) {
      constexpr uint32_t idesc = idesc_bf16_f32(256, kBN, A_MN, B_MN);
      constexpr uint32_t a_lbo = A_MN ? kBK * 128 : 16, a_step = A_MN ? 2048 : 32;
      constexpr uint32_t b_lbo = B_MN ? kBK * 128 : 16, b_step = B_MN ? 2048 : 32;
      uint32_t kc = 0, tile = 0;
      bool ok = true;
      for (int u = pair; ok && u < sched.num_units; u += npairs) {
        int m_blk, split, n0, n1;
        sched.unit(u, m_blk, split, n0, n1);
        for (int nb = n0; ok && nb < n1; ++nb, ++tile) {
          const uint32_t acc = tile & 1u;
          const uint32_t aph = (tile >> 1) & 1u;
          if (!mbar_wait(&sm.tempty[acc], aph ^ 1u, timeout_ns, abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * kBN;
          for (int kb = 0; kb < sched.num_kb; ++kb, ++kc) {
            const int s = kc % kStagesPair;
            const uint32_t ph = (kc / kStagesPair) & 1u;
            if (!mbar_wait(&sm.full[s], ph, timeout_ns, abort)) { ok = false; break; }
            tc_fence_after();
            const uint32_t a_base = smem_addr(sm.a[s]);
            const uint32_t b_base = smem_addr(sm.b[s]);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) {
              const uint64_t ad = smem_desc_sw128(a_base + k * a_step, a_lbo, 1024);
              const uint64_t bd = smem_desc_sw128(b_base + k * b_step, b_lbo, 1024);
              umma_bf16_pair(d_tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
            }
            umma_commit_pair_multicast(&sm.empty[s], 0x3);
          }
          if (ok) umma_commit_pair_multicast(&sm.tfull[acc], 0x3);
        }
      }
      if (!ok) {
        *abort = 1;
        raise_status(status, PS_DEV_TIMEOUT);
        umma_commit_pair_multicast(&sm.drain, 0x1);
        mbar_wait(&sm.drain, 0, timeout_ns, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue (both CTAs)
    const int quad = warp & 3;
    const int row_in_tile = quad * 32 + lane;
    const uint32_t ltempty0 = mapa_shared(smem_addr(&sm.tempty[0]), 0);
    const uint32_t ltempty1 = mapa_shared(smem_addr(&sm.tempty[1]), 0);
    typename Epi::State st;
    uint32_t tile = 0;
    bool ok = true;
    for (int u = pair; ok && u < sched.num_units; u += npairs) {
      int m_blk, split, n0, n1;
      sched.unit(u, m_blk, split, n0, n1);
      const int row = m_blk * 256 + static_cast<int>(rank) * 128 + row_in_tile;
      Epi::begin_unit(ep, st, row, split);
      for (int nb = n0; nb < n1; ++nb, ++tile) {
        const uint32_t acc = tile & 1u;
        const uint32_t aph = (tile >> 1) & 1u;
        int got = 0;
        if (lane == 0) got = mbar_wait(&sm.tfull[acc], aph, timeout_ns, abort) ? 1 : 0;
        got = __shfl_sync(0xffffffffu, got, 0);
        if (!got) { ok = false; break; }
        tc_fence_after();
        const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + acc * kBN;
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(t_row + c * 32, r);
          tmem_ld_wait();
          if (c == kBN / 32 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(acc ? ltempty1 : ltempty0);
          }
          Epi::chunk(ep, st, row, nb * kBN + c * 32, r);
        }
      }
      if (ok) Epi::end_unit(ep, st, row, split);
    }
    if (!ok) {
      *abort = 1;
      raise_status(status, PS_DEV_TIMEOUT);
    }
  }

  tc_fence_before();
  cluster_sync_all();  // no remote arrival or multicast commit can target an exited CTA
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

}  // namespace psk
