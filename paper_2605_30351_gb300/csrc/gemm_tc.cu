// Dense bf16 GEMMs around the attention (tcgen05, TMEM accumulator, TMA):
// (at large M the 256-wide tiles run as paired-SM MMAs, see GemmShape)
// the query prologue (Eqs. cq, qnope, qrope with App. E's absorbed weights)
// and the output projection (Eq. absorb-v). C[M x N] = A[M x K] B[N x K]^T,
// both operands K-major, fp32 accumulation, one 128 x BN tile per CTA:
//   warp 0     TMA producer (A [128 x 64], B [BN x 64] per stage, SW128;
//              B in two boxes when BN > 256)
//   warp 1     TMEM allocation; one lane issues tcgen05.mma (N = BN, or two
//              MMAs of N = BN/2 when BN > 256)
//   warps 2-5  epilogue, thread i = row i: TMEM -> registers -> bf16 staged
//              in shared memory, then one bulk copy per row (two when the row
//              straddles kRowScale's split between C and C2).
// Epilogues:
//   kStore      plain bf16 C
//   kStoreSq    bf16 C plus, per row, the sum of squares of this tile's fp32
//               columns (RMSNorm's statistics, App. D.2)
//   kRowScale   every row scaled by 1/sqrt(mean of the squares + eps) before
//               rounding, columns [0, split) to C and [split, N) to C2.
// RMSNorm's per-row scale commutes with the following linear map, so the
// query latent is normalised in the next GEMM's epilogue: q = (W diag(gamma))
// c~ / rms(c~), with gamma folded into W when the weights are absorbed.
#include <cmath>
#include <mutex>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;

// PAIR: paired-SM MMAs (cta_group::2). Two CTAs of a cluster take M tiles
// 2i and 2i + 1 of the same N tile as one M = 256 MMA; each holds its 128
// rows of A and BN/2 of the B rows, so each SM streams half of the B tile.
template <int BN, int MAXST, bool PAIR = false>
struct GemmShape {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBRows = PAIR ? BN / 2 : BN;
  static constexpr int kBBytes = kBRows * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  // bytes a stage's full barrier counts (PAIR: in the even CTA, both CTAs')
  static constexpr int kTxBytes = PAIR ? 2 * kStageBytes : kStageBytes;
  static constexpr int kBarBytes = 256;
  static constexpr int kFit = (232448 - 1024 - kBarBytes) / kStageBytes;
  static constexpr int kStages = kFit > MAXST ? MAXST : kFit;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kBarBytes;
  static constexpr uint32_t kTmemCols = BN <= 128 ? 128 : (BN <= 256 ? 256 : 512);
  static constexpr int kHalves = BN > 256 ? 2 : 1;  // MMAs (and B boxes) per K step
  static constexpr int kBN1 = BN / kHalves;         // columns of one MMA
  static constexpr int kBBox = PAIR ? BN / 2 : kBN1;  // rows of one B box
  static constexpr uint32_t kIdesc = idesc_bf16_f32(PAIR ? 2 * kBM : kBM, kBN1, false, false);
  static_assert(!PAIR || (BN <= 256 && BN % 32 == 0), "paired MMA: one N <= 256 MMA, 16-row B halves");
  static_assert(BN % 32 == 0 && BN <= 512 && kBN1 % 32 == 0, "tile width");
  static_assert(kStageBytes % 1024 == 0, "swizzle-atom alignment");
  static_assert(kBM * BN * 2 <= kStages * kStageBytes, "staging fits in the ring");
  static_assert(BN % 64 == 0, "rows staged in 64-column segments");
};

struct GemmKParams {
  __nv_bfloat16* c;       // [M][ldc] (columns [0, split) when kRowScale)
  __nv_bfloat16* c2;      // kRowScale: [M][ld2] for columns [split, N)
  float* sq;              // kStoreSq: out [n_tiles][M]; kRowScale: in [sq_tiles][M]
  int M, N, K, ldc, ld2, split, sq_tiles;
  float sq_dim, eps;
  int* status;
};

enum { kStore = 0, kStoreSq = 1, kRowScale = 2 };

template <int BN, int EPI, int MAXST, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1)
    mla_gemm_tc_kernel(const __grid_constant__ CUtensorMap tm_a,
                       const __grid_constant__ CUtensorMap tm_b, const GemmKParams p) {
  using S = GemmShape<BN, MAXST, PAIR>;
  constexpr int NST = S::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_smem_1024(smem_raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NST * S::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + NST;
  uint64_t* acc_full = bars + 2 * NST;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // N tiles run fastest (blockIdx.x), so the N tiles of one row tile of A
  // follow one another and A comes from HBM once; B stays in L2. PAIR: the
  // two CTAs of an x-cluster take M tiles 2y and 2y + 1 of the same N tile.
  const int n_tile = PAIR ? blockIdx.x / 2 : blockIdx.x;
  const int m0 = (PAIR ? 2 * blockIdx.y + (blockIdx.x & 1) : blockIdx.y) * kBM;
  const int n0 = n_tile * BN;
  const int k_blocks = p.K / kBK;
  const WaitCtx wc{abort_flag, p.status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (PAIR) {
      tmem_alloc_pair(tmem_slot, S::kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, S::kTmemCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int crank = PAIR ? static_cast<int>(cluster_ctarank()) : 0;
  // the peer's barriers exist before the pair's copies and commits signal them
  if constexpr (PAIR) cluster_sync();
  grid_dep_sync();

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tm_a);
      tma_prefetch_desc(&tm_b);
      int issued = 0;
      for (int kb = 0; kb < k_blocks; ++kb) {
        const int st = kb % NST;
        if (kb >= NST && !mbar_wait(&empty[st], ((kb / NST) - 1) & 1, wc)) break;
        uint8_t* a = smem + st * S::kStageBytes;
        if constexpr (PAIR) {
          // this CTA's A rows and its half of the B rows; the even CTA's full
          // barrier counts both CTAs' bytes
          const uint32_t bar = dsmem_addr(smem_u32(&full[st]), 0);
          if (crank == 0) mbar_arrive_expect_tx(&full[st], S::kTxBytes);
          tma_load_2d_pair(a, &tm_a, bar, kb * kBK, m0);
          tma_load_2d_pair(a + S::kABytes, &tm_b, bar, kb * kBK, n0 + crank * S::kBBox);
        } else {
          mbar_arrive_expect_tx(&full[st], S::kTxBytes);
          tma_load_2d(a, &tm_a, &full[st], kb * kBK, m0);
#pragma unroll
          for (int h = 0; h < S::kHalves; ++h)
            tma_load_2d(a + S::kABytes + h * S::kBN1 * 128, &tm_b, &full[st], kb * kBK,
                        n0 + h * S::kBN1);
        }
        issued = kb + 1;
      }
      if constexpr (PAIR) {
        // the even CTA's MMAs release this CTA's stages: their last releases
        // must have landed before the CTA may exit
        for (int st = 0; st < NST && st < k_blocks && !*abort_flag; ++st)
          mbar_wait(&empty[st], (((k_blocks - st + NST - 1) / NST) - 1) & 1, wc);
      }
      if (*abort_flag && (!PAIR || crank == 0))
        for (int u = issued > NST ? issued - NST : 0; u < issued; ++u)
          mbar_wait_drain(&full[u % NST], (u / NST) & 1, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && crank == 0) {
      bool ok = true;
      for (int kb = 0; kb < k_blocks; ++kb) {
        const int st = kb % NST;
        if (!mbar_wait(&full[st], (kb / NST) & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t aa = smem_u32(smem + st * S::kStageBytes);
        const uint32_t ba = aa + S::kABytes;
        if constexpr (PAIR) {
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_pair_ss(tmem, sdesc(aa + k * 32, 16, 1024, kSw128),
                         sdesc(ba + k * 32, 16, 1024, kSw128), S::kIdesc, (kb | k) != 0 ? 1u : 0u);
          umma_pair_commit_mc(&empty[st], 3);
        } else {
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
#pragma unroll
            for (int h = 0; h < S::kHalves; ++h)
              umma_ss(tmem + h * S::kBN1, sdesc(aa + k * 32, 16, 1024, kSw128),
                      sdesc(ba + h * S::kBN1 * 128 + k * 32, 16, 1024, kSw128), S::kIdesc,
                      (kb | k) != 0 ? 1u : 0u);
          umma_commit(&empty[st]);
        }
      }
      if constexpr (PAIR)
        umma_pair_commit_mc(acc_full, 3);
      else
        umma_commit(acc_full);
      if (!ok) mbar_wait_drain(acc_full, 0, p.status);
    }
    __syncwarp();
  } else {
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t t_row = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int m = m0 + r;
    const int n_valid = min(BN, p.N - n0);
    // kRowScale: the row's statistics (written by the previous GEMM) are
    // fetched while the MMAs run, so no global load follows the accumulator
    float scale = 1.f;
    if constexpr (EPI == kRowScale) {
      float ss = 0.f;
      if (m < p.M)
        for (int t = 0; t < p.sq_tiles; ++t) ss += p.sq[static_cast<size_t>(t) * p.M + m];
      scale = rsqrtf(ss / p.sq_dim + p.eps);
    }
    const bool have_acc = mbar_wait(acc_full, 0, wc) && !*abort_flag;
    // Each thread stages its row densely in shared memory ([128][BN] bf16,
    // the ring being free once the accumulator is complete; chunk order
    // rotated per row so the quarter warp's rows hit distinct banks) and
    // hands it to the bulk-copy engine, one copy per destination matrix.
    uint8_t* srow = smem + r * BN * 2;
    if (have_acc) {
      tc_fence_after();
      float ss_own = 0.f;
#pragma unroll 1
      for (int sg = 0; sg < BN / 64; ++sg) {
        uint32_t va[32], vb[32];
        tmem_ld32(t_row + sg * 64, va);
        tmem_ld32(t_row + sg * 64 + 32, vb);
        tmem_wait_ld();
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const uint32_t* v = i < 16 ? va : vb;
          const int j = i & 15;
          const float a0 = __uint_as_float(v[2 * j]), a1 = __uint_as_float(v[2 * j + 1]);
          if constexpr (EPI == kStoreSq) {
            const int col = sg * 64 + 2 * i;
            if (col < n_valid) ss_own = fmaf(a0, a0, ss_own);
            if (col + 1 < n_valid) ss_own = fmaf(a1, a1, ss_own);
          }
          pk[i] = pack_bf16x2(a0 * scale, a1 * scale);
        }
        stage_row<8>(srow + sg * 128, pk, r & 7);
      }
      if constexpr (EPI == kStoreSq)
        if (m < p.M) p.sq[static_cast<size_t>(n_tile) * p.M + m] = ss_own;
      if (m < p.M) {
        // columns [n0, n0 + n_valid) of row m: below `split` to C, from it to
        // C2; addresses and sizes are multiples of 16 bytes (N, split, the
        // leading dimensions and n0 are multiples of 8)
        int c_end = n_valid;
        if constexpr (EPI == kRowScale) c_end = max(0, min(n_valid, p.split - n0));
        fence_proxy_async_smem();
        if (c_end > 0) bulk_store(p.c + static_cast<size_t>(m) * p.ldc + n0, srow, c_end * 2);
        if constexpr (EPI == kRowScale)
          if (c_end < n_valid)
            bulk_store(p.c2 + static_cast<size_t>(m) * p.ld2 + (n0 + c_end - p.split),
                       srow + c_end * 2, (n_valid - c_end) * 2);
        bulk_commit();
        bulk_wait_read_all();  // the staged row must outlive the copies' reads
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) {
    cluster_sync();  // both CTAs are done with the pair's TMEM and shared memory
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc_pair(tmem, S::kTmemCols);
    }
  } else if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, S::kTmemCols);
  }
}

// Persistent paired-SM form, for large M. One CTA per SM; each cluster of
// two (an SM pair) walks the pair tiles t = cluster, cluster + clusters, ...
// (a pair tile: M tiles 2i and 2i + 1 of one N tile, N tiles fastest, so the
// pairs working at one moment share their A rows in L2). The stage ring runs
// on across tile boundaries, and two TMEM accumulators of BN columns let the
// epilogue warps drain one tile while the MMAs fill the next; a non-
// persistent CTA instead pays its set-up, pipeline fill and epilogue once
// per tile. The staged output rows have their own shared memory, apart from
// the ring.
template <int BN>
struct PGemmShape {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBox = BN / 2;  // B rows per CTA
  static constexpr int kBBytes = kBBox * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kTxBytes = 2 * kStageBytes;  // the even CTA's full barrier counts both
  static constexpr int kStagingBytes = kBM * BN * 2;
  static constexpr int kBarBytes = 256;
  static constexpr int kFit = (232448 - 1024 - kBarBytes - kStagingBytes) / kStageBytes;
  static constexpr int kStages = kFit > 8 ? 8 : kFit;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kStagingBytes + kBarBytes;
  static constexpr uint32_t kAccStride = 256;  // TMEM columns per accumulator
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(2 * kBM, BN, false, false);
  static_assert(BN % 64 == 0 && BN <= 256, "one N <= 256 MMA, rows staged in 64-column segments");
  static_assert(kStages >= 3, "ring depth");
  static_assert(kStageBytes % 1024 == 0 && kStagingBytes % 1024 == 0, "swizzle-atom alignment");
  static_assert(2 * kStages + 5 <= kBarBytes / 8 - 1, "barriers, TMEM slot and abort flag");
};

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    mla_gemm_tc_persistent_kernel(const __grid_constant__ CUtensorMap tm_a,
                                  const __grid_constant__ CUtensorMap tm_b, const GemmKParams p) {
  using S = PGemmShape<BN>;
  constexpr int NST = S::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_smem_1024(smem_raw);
  uint8_t* staging = smem + NST * S::kStageBytes;  // [128][BN] bf16
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging + S::kStagingBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + NST;
  uint64_t* acc_full = bars + 2 * NST;  // [2]
  uint64_t* acc_empty = acc_full + 2;   // [2], used in the even CTA
  uint64_t* mma_drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int cluster = blockIdx.x / 2;
  const int clusters = gridDim.x / 2;
  const int n_tiles = (p.N + BN - 1) / BN;
  const int m_pairs = ((p.M + kBM - 1) / kBM + 1) / 2;
  const int total = n_tiles * m_pairs;
  const int k_blocks = p.K / kBK;
  const WaitCtx wc{abort_flag, p.status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 2 * 128);  // every epilogue thread of both CTAs
    }
    mbar_init(mma_drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, S::kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int crank = static_cast<int>(cluster_ctarank());
  cluster_sync();  // the peer's barriers exist before copies, commits and arrivals reach them
  grid_dep_sync();

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tm_a);
      tma_prefetch_desc(&tm_b);
      int it = 0;  // k blocks issued so far, over all tiles
      bool ok = true;
      for (int t = cluster; t < total && ok; t += clusters) {
        const int n0 = (t % n_tiles) * BN;
        const int m0 = (2 * (t / n_tiles) + crank) * kBM;
        for (int kb = 0; kb < k_blocks; ++kb) {
          const int st = it % NST;
          if (it >= NST && !mbar_wait(&empty[st], ((it / NST) - 1) & 1, wc)) {
            ok = false;
            break;
          }
          uint8_t* a = smem + st * S::kStageBytes;
          const uint32_t bar = dsmem_addr(smem_u32(&full[st]), 0);
          if (crank == 0) mbar_arrive_expect_tx(&full[st], S::kTxBytes);
          tma_load_2d_pair(a, &tm_a, bar, kb * kBK, m0);
          tma_load_2d_pair(a + S::kABytes, &tm_b, bar, kb * kBK, n0 + crank * S::kBBox);
          ++it;
        }
      }
      // the even CTA's MMAs release this CTA's stages: the last releases must
      // have landed before the CTA may exit
      for (int u = it > NST ? it - NST : 0; u < it && !*abort_flag; ++u)
        mbar_wait(&empty[u % NST], (u / NST) & 1, wc);
      if (*abort_flag && crank == 0)
        for (int u = it > NST ? it - NST : 0; u < it; ++u)
          mbar_wait_drain(&full[u % NST], (u / NST) & 1, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && crank == 0) {
      int it = 0, tl = 0;
      bool ok = true;
      for (int t = cluster; t < total && ok; t += clusters, ++tl) {
        const int buf = tl & 1;
        // both CTAs' epilogues have drained this accumulator (two tiles ago)
        if (tl >= 2 && !mbar_wait_cluster(&acc_empty[buf], ((tl >> 1) - 1) & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + buf * S::kAccStride;
        for (int kb = 0; kb < k_blocks; ++kb, ++it) {
          const int st = it % NST;
          if (!mbar_wait(&full[st], (it / NST) & 1, wc)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t aa = smem_u32(smem + st * S::kStageBytes);
          const uint32_t ba = aa + S::kABytes;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_pair_ss(acc, sdesc(aa + k * 32, 16, 1024, kSw128),
                         sdesc(ba + k * 32, 16, 1024, kSw128), S::kIdesc, (kb | k) != 0 ? 1u : 0u);
          umma_pair_commit_mc(&empty[st], 3);
        }
        if (ok) umma_pair_commit_mc(&acc_full[buf], 3);
      }
      if (!ok) {  // every MMA issued must be done before the CTA moves on
        umma_pair_commit_mc(mma_drain, 1);
        mbar_wait_drain(mma_drain, 0, p.status);
      }
    }
    __syncwarp();
  } else {
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t t_lane = static_cast<uint32_t>(quarter * 32) << 16;
    uint8_t* srow = staging + r * BN * 2;
    int tl = 0;
    for (int t = cluster; t < total; t += clusters, ++tl) {
      const int buf = tl & 1;
      const int n_tile = t % n_tiles;
      const int n0 = n_tile * BN;
      const int m = (2 * (t / n_tiles) + crank) * kBM + r;
      const int n_valid = min(BN, p.N - n0);
      // kRowScale: the row's statistics (from the previous GEMM), fetched
      // before the accumulator is ready
      float scale = 1.f;
      if constexpr (EPI == kRowScale) {
        float ss = 0.f;
        if (m < p.M)
          for (int q = 0; q < p.sq_tiles; ++q) ss += p.sq[static_cast<size_t>(q) * p.M + m];
        scale = rsqrtf(ss / p.sq_dim + p.eps);
      }
      if (!mbar_wait(&acc_full[buf], (tl >> 1) & 1, wc)) break;
      tc_fence_after();
      float ss_own = 0.f;
      const uint32_t acc = tmem + t_lane + buf * S::kAccStride;
      // the whole row into registers as bf16 pairs first, so that the
      // accumulator goes back to the MMA issuer before the staged rows wait
      // for the previous tile's copies
      uint32_t pk[BN / 64][32];
#pragma unroll
      for (int sg = 0; sg < BN / 64; ++sg) {
        uint32_t va[32], vb[32];
        tmem_ld32(acc + sg * 64, va);
        tmem_ld32(acc + sg * 64 + 32, vb);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const uint32_t* v = i < 16 ? va : vb;
          const int j = i & 15;
          const float a0 = __uint_as_float(v[2 * j]), a1 = __uint_as_float(v[2 * j + 1]);
          if constexpr (EPI == kStoreSq) {
            const int col = sg * 64 + 2 * i;
            if (col < n_valid) ss_own = fmaf(a0, a0, ss_own);
            if (col + 1 < n_valid) ss_own = fmaf(a1, a1, ss_own);
          }
          pk[sg][i] = pack_bf16x2(a0 * scale, a1 * scale);
        }
      }
      // this thread's reads of the accumulator are done: release it to the
      // MMA issuer (in the even CTA)
      tc_fence_before();
      mbar_arrive_cluster(dsmem_addr(smem_u32(&acc_empty[buf]), 0));
      bulk_wait_read_all();  // the previous tile's copy of this row has read it
#pragma unroll
      for (int sg = 0; sg < BN / 64; ++sg) stage_row<8>(srow + sg * 128, pk[sg], r & 7);
      if constexpr (EPI == kStoreSq)
        if (m < p.M) p.sq[static_cast<size_t>(n_tile) * p.M + m] = ss_own;
      if (m < p.M) {
        // columns [n0, n0 + n_valid) of row m: below `split` to C, from it to
        // C2 (16-byte aligned and sized, as in the non-persistent form)
        int c_end = n_valid;
        if constexpr (EPI == kRowScale) c_end = max(0, min(n_valid, p.split - n0));
        fence_proxy_async_smem();
        if (c_end > 0) bulk_store(p.c + static_cast<size_t>(m) * p.ldc + n0, srow, c_end * 2);
        if constexpr (EPI == kRowScale)
          if (c_end < n_valid)
            bulk_store(p.c2 + static_cast<size_t>(m) * p.ld2 + (n0 + c_end - p.split),
                       srow + c_end * 2, (n_valid - c_end) * 2);
        bulk_commit();
      }
    }
    bulk_wait_read_all();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs are done with the pair's TMEM and barriers
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, S::kTmemCols);
  }
}

template <int BN, int EPI>
int launch_gemm_persistent(const void* a, const void* b, int M, int N, int K, GemmKParams kp,
                           cudaStream_t stream) {
  using S = PGemmShape<BN>;
  if (K % kBK != 0 || N % 8 != 0) return MLA_ERR_UNSUPPORTED;
  CUtensorMap tm_a, tm_b;
  if (!encode_map_2d_bf16(&tm_a, a, K, M, K * 2ull, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_b, b, K, N, K * 2ull, kBK, S::kBBox, CU_TENSOR_MAP_SWIZZLE_128B))
    return MLA_ERR_CUDA;
  auto kern = mla_gemm_tc_persistent_kernel<BN, EPI>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmemBytes);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  kp.M = M;
  kp.N = N;
  kp.K = K;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = S::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_sync
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  // as many clusters as are resident at once (one CTA per SM), at most one
  // per pair tile
  static int resident = -1;  // per process, for this instantiation
  if (resident < 0) {
    int n = 0;
    cudaLaunchConfig_t oc = cfg;
    oc.gridDim = dim3(2, 1, 1);
    oc.numAttrs = 2;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &oc) != cudaSuccess) {
      cudaGetLastError();
      n = 0;
    }
    resident = n;
  }
  if (resident < 1) return MLA_ERR_UNSUPPORTED;
  const long long m_pairs = ((M + kBM - 1) / kBM + 1) / 2;
  const long long total = m_pairs * ((N + BN - 1) / BN);
  const int clusters = static_cast<int>(total < resident ? total : resident);
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  e = cudaLaunchKernelEx(&cfg, kern, tm_a, tm_b, kp);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

template <int BN, int EPI, int MAXST = 6, bool PAIR = false>
int launch_gemm(const void* a, const void* b, int M, int N, int K, GemmKParams kp,
                cudaStream_t stream) {
  using S = GemmShape<BN, MAXST, PAIR>;
  if (K % kBK != 0 || N % 8 != 0) return MLA_ERR_UNSUPPORTED;
  CUtensorMap tm_a, tm_b;
  if (!encode_map_2d_bf16(&tm_a, a, K, M, K * 2ull, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_b, b, K, N, K * 2ull, kBK, S::kBBox, CU_TENSOR_MAP_SWIZZLE_128B))
    return MLA_ERR_CUDA;
  auto kern = mla_gemm_tc_kernel<BN, EPI, MAXST, PAIR>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmemBytes);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  kp.M = M;
  kp.N = N;
  kp.K = K;
  cudaLaunchConfig_t cfg = {};
  // PAIR: M tiles rounded up to pairs (a last tile past M loads zeros and
  // stores nothing)
  const int m_tiles = (M + kBM - 1) / kBM;
  if (m_tiles > 65534) return MLA_ERR_UNSUPPORTED;  // row tiles index the grid's y dimension
  const int n_tiles = (N + BN - 1) / BN;
  cfg.gridDim = PAIR ? dim3(2 * n_tiles, (m_tiles + 1) / 2) : dim3(n_tiles, m_tiles);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = S::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_sync
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;  // PAIR: M tiles 2y, 2y + 1
  attr[1].val.clusterDim.x = PAIR ? 2 : 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, kern, tm_a, tm_b, kp);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

// ---- load-time weight absorption (App. E), fp32 accumulation, bf16 out ----
// w_qcat row (h, c) for c < d_c: sum_e W_uq[h][e][q] W_uk[h][e][c] * gamma_q[q]
//        row H*d_c + (h, j):     W_qr[h][j][q] * gamma_q[q]
__global__ void absorb_query_kernel(const __nv_bfloat16* __restrict__ w_uq,
                                    const __nv_bfloat16* __restrict__ w_uk,
                                    const __nv_bfloat16* __restrict__ w_qr,
                                    const __nv_bfloat16* __restrict__ gamma_q,
                                    __nv_bfloat16* __restrict__ w_qcat, int H, int dn, int dc,
                                    int dr, int dq) {
  const long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  const long long rows = static_cast<long long>(H) * (dc + dr);
  if (idx >= rows * dq) return;
  const int row = static_cast<int>(idx / dq), q = static_cast<int>(idx % dq);
  const float g = gamma_q ? __bfloat162float(gamma_q[q]) : 1.f;
  float acc = 0.f;
  if (row < H * dc) {
    const int h = row / dc, c = row % dc;
    for (int e = 0; e < dn; ++e)
      acc = fmaf(__bfloat162float(w_uq[(static_cast<size_t>(h) * dn + e) * dq + q]),
                 __bfloat162float(w_uk[(static_cast<size_t>(h) * dn + e) * dc + c]), acc);
  } else {
    const int rr = row - H * dc;  // (h, j) -> w_qr[h][j][q]
    acc = __bfloat162float(w_qr[static_cast<size_t>(rr) * dq + q]);
  }
  w_qcat[idx] = __float2bfloat16_rn(acc * g);
}

// w_b[i][(h, c)] = sum_v W_o[i][h*dh + v] W_uv[h][v][c]
__global__ void absorb_output_kernel(const __nv_bfloat16* __restrict__ w_uv,
                                     const __nv_bfloat16* __restrict__ w_o,
                                     __nv_bfloat16* __restrict__ w_b, int d, int H, int dh,
                                     int dc) {
  const long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (idx >= static_cast<long long>(d) * H * dc) return;
  const int i = static_cast<int>(idx / (H * dc));
  const int hc = static_cast<int>(idx % (H * dc));
  const int h = hc / dc, c = hc % dc;
  float acc = 0.f;
  for (int v = 0; v < dh; ++v)
    acc = fmaf(__bfloat162float(w_o[static_cast<size_t>(i) * H * dh + h * dh + v]),
               __bfloat162float(w_uv[(static_cast<size_t>(h) * dh + v) * dc + c]), acc);
  w_b[idx] = __float2bfloat16_rn(acc);
}

}  // namespace

int launch_absorb(const AbsorbArgs& a) {
  const long long nq = static_cast<long long>(a.heads) * (a.d_c + a.d_r) * a.d_q;
  const long long nb = static_cast<long long>(a.hidden) * a.heads * a.d_c;
  absorb_query_kernel<<<static_cast<unsigned>((nq + 255) / 256), 256, 0, a.stream>>>(
      static_cast<const __nv_bfloat16*>(a.w_uq), static_cast<const __nv_bfloat16*>(a.w_uk),
      static_cast<const __nv_bfloat16*>(a.w_qr), static_cast<const __nv_bfloat16*>(a.gamma_q),
      static_cast<__nv_bfloat16*>(a.w_qcat), a.heads, a.head_dim - a.d_r, a.d_c, a.d_r, a.d_q);
  absorb_output_kernel<<<static_cast<unsigned>((nb + 255) / 256), 256, 0, a.stream>>>(
      static_cast<const __nv_bfloat16*>(a.w_uv), static_cast<const __nv_bfloat16*>(a.w_o),
      static_cast<__nv_bfloat16*>(a.w_b), a.hidden, a.heads, a.head_dim, a.d_c);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

int launch_query_prologue(const QueryArgs& a) {
  const int M = a.rows;  // batch * Nq tokens
  // c~ = x W_dq^T (bf16) with per-row partial sums of squares. 192-wide tiles
  // when 256-wide ones would not give every SM a CTA (one chunk: 37 row tiles
  // x 4 = 148 CTAs, 47.5 -> 46.0 us); 256-wide otherwise (four chunks: 138 vs
  // 141 us). The workspace holds ceil(d_q / 192) partial sums per row, enough
  // for either.
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long row_tiles = (M + kBM - 1) / kBM;
  const bool narrow = row_tiles * ((a.d_q + 255) / 256) < sms;
  const int sq_tiles = narrow ? (a.d_q + kQuerySqTile - 1) / kQuerySqTile : (a.d_q + 255) / 256;
  GemmKParams k1 = {};
  k1.c = static_cast<__nv_bfloat16*>(a.c_tilde);
  k1.ldc = a.d_q;
  k1.sq = a.sq;
  k1.status = a.status;
  // large M (e.g. four chunks): paired-SM 256-wide tiles, two pairs per SM
  // pair of SMs (three 32 KB stages each): each SM streams half of every B
  // tile (four Wan chunks: 132.8 -> 129.3 us for both GEMMs, same outputs)
  int rc = narrow ? launch_gemm<kQuerySqTile, kStoreSq>(a.x, a.w_dq, M, a.d_q, a.hidden, k1, a.stream)
                  : launch_gemm_persistent<256, kStoreSq>(a.x, a.w_dq, M, a.d_q, a.hidden, k1,
                                                          a.stream);
  if (rc == MLA_ERR_UNSUPPORTED && !narrow)
    rc = launch_gemm<256, kStoreSq, 3, true>(a.x, a.w_dq, M, a.d_q, a.hidden, k1, a.stream);
  if (rc != MLA_OK) return rc;
  // [q_c | q_r] = (c~ / rms(c~)) [W_qc ; W_qr]^T with gamma folded into the weights
  GemmKParams k2 = {};
  k2.c = static_cast<__nv_bfloat16*>(a.q_c);
  k2.ldc = a.heads * a.d_c;
  k2.c2 = static_cast<__nv_bfloat16*>(a.q_r);
  k2.ld2 = a.heads * a.d_r;
  k2.split = a.heads * a.d_c;
  k2.sq = a.sq;
  k2.sq_tiles = sq_tiles;
  k2.sq_dim = static_cast<float>(a.d_q);
  k2.eps = a.eps;
  k2.status = a.status;
  // The persistent paired-SM form at every M: its clusters walk more than one
  // pair tile each even at one Wan chunk (19 x 11 pair tiles), so each
  // tile's epilogue runs under the next one's MMAs (one chunk: query prologue
  // 37.7 -> 32.4 us against the two-CTAs-per-SM form; four chunks: 131 ->
  // 87 us against the non-persistent paired form). If its clusters cannot be
  // co-resident, the non-persistent forms: a two-stage ring with two CTAs per
  // SM at small M, paired-SM MMAs at large M.
  const int nq = a.heads * (a.d_c + a.d_r);
  rc = launch_gemm_persistent<256, kRowScale>(a.c_tilde, a.w_qcat, M, nq, a.d_q, k2, a.stream);
  if (rc != MLA_ERR_UNSUPPORTED) return rc;
  if (!narrow)
    return launch_gemm<256, kRowScale, 3, true>(a.c_tilde, a.w_qcat, M, nq, a.d_q, k2, a.stream);
  return launch_gemm<256, kRowScale, 2>(a.c_tilde, a.w_qcat, M, nq, a.d_q, k2, a.stream);
}

// ---- fixed scratch for mla_query_prologue_noalloc ----
// The library's only device memory of its own: a file-scope array every GPU
// that loads the library holds until the process exits. Host code must not
// pass the symbol itself to a kernel (on the host it names a host-side
// stand-in); query_scratch_address() looks up the device address instead,
// once per device. The cached address belongs to the device's primary
// context: after cudaDeviceReset it would be stale, and the library does not
// support a reset within the process.
namespace {
static __device__ __align__(256) unsigned char g_query_scratch[MLA_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxScratchDevices = 64;
void* g_scratch_addr[kMaxScratchDevices] = {nullptr};
std::mutex g_scratch_mu;
}  // namespace

int query_scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxScratchDevices) return MLA_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_addr[dev]) {  // once per device, with that device current
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_query_scratch);
    if (e != cudaSuccess || !p) {
      set_last_cuda_error(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
      return MLA_ERR_CUDA;
    }
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return MLA_OK;
}

int launch_output_projection(const OutProjArgs& a) {
  GemmKParams k = {};
  k.c = static_cast<__nv_bfloat16*>(a.y);
  k.ldc = a.hidden;
  k.status = a.status;
  // 384-wide tiles, one CTA per SM with three 64 KB stages, when they fit in
  // one wave (one Wan chunk: 37 x 4 = 148 CTAs); otherwise two CTAs per SM
  // (two-stage ring): 192-wide tiles when 256-wide ones would leave the GPU
  // less than two CTAs per SM (one chunk: 29 vs 35 us), 256-wide otherwise
  // (four chunks: 100 vs 119 us).
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long row_tiles = (a.rows + kBM - 1) / kBM;
  if (a.hidden % 384 == 0 && row_tiles * (a.hidden / 384) <= sms)
    return launch_gemm<384, kStore, 3>(a.o_lat, a.w_b, a.rows, a.hidden, a.heads * a.d_c, k,
                                       a.stream);
  const long long ctas256 = row_tiles * ((a.hidden + 255) / 256);
  if (ctas256 < 2ll * sms && a.hidden % 192 == 0)
    return launch_gemm<192, kStore, 2>(a.o_lat, a.w_b, a.rows, a.hidden, a.heads * a.d_c, k,
                                       a.stream);
  // large M: paired-SM MMAs (each SM streams half of every B tile; four Wan
  // chunks: 97.3 -> 85.9 us, same output)
  const int rc = launch_gemm_persistent<256, kStore>(a.o_lat, a.w_b, a.rows, a.hidden,
                                                     a.heads * a.d_c, k, a.stream);
  if (rc != MLA_ERR_UNSUPPORTED) return rc;
  return launch_gemm<256, kStore, 3, true>(a.o_lat, a.w_b, a.rows, a.hidden, a.heads * a.d_c, k,
                                           a.stream);
}

}  // namespace vmla
