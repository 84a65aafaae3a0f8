// Absorbed-form MLA attention on the sm_103a tensor cores (tcgen05 + TMEM + TMA).
//
// Paper: Eq. (score) and App. E (Eqs. absorb-q, absorb-v). Every query row is
// one (token, head) pair; all rows of a batch element score the SAME cached
// latents, so the n_h heads simply stack along M and each KV tile is loaded
// once per 128 rows:
//     S   = [q_c | RoPE(q_r)] . [c | k]^T          K = d_c + d_r (224)
//     P   = exp2(S * log2(e)/sqrt(d_h) - m)        online, fp32
//     O  += P . c                                  N = d_c (192), latent output
// One CTA owns 128 rows (one TMEM lane each) and walks the window in blocks
// of BN keys (128; 64 for d_c = 512):
//   warp 0     TMA producer: [c | k] tiles into a ring of shared-memory
//              stages (c with 128-byte swizzle, k with 64-byte swizzle).
//              CTAs run in pairs (a cluster of two consecutive row tiles of
//              the same batch element): each CTA fetches half of every key
//              tile from L2 and multicasts it into both CTAs' stage, halving
//              the L2-to-SM traffic, which otherwise bounds the kernel.
//   warp 1     allocates TMEM; one lane issues the score MMAs
//              S_j = Q K_j^T with Q read from TMEM, so they read only the key
//              tile from shared memory. S_{j+1} is issued as soon as the
//              softmax has copied S_j into registers.
//   warp 6     one lane issues O += P_j V_j with P read from TMEM. Two issuing
//              threads keep the tensor pipe fed while either one waits on a
//              barrier: the MMA queue is shallow, so a single issuer's
//              bookkeeping between groups would leave the pipe idle.
//   warps 2-5  load q_c, rotate q_r and store both into TMEM; then the online
//              softmax: thread i owns row i, copies S_j out of TMEM (releasing
//              it), writes P_j (bf16) once PV_{j-1} has read the previous P,
//              rescales O in TMEM only when its running max grows by more
//              than 2^8, and finally writes O / l as bf16.
// TMEM columns: S [0,BN) P [BN,3BN/2) O [3BN/2,3BN/2+d_c) Q [3BN/2+d_c, +(d_c+d_r)/2).
// When Q does not fit there (d_c = 256) it stays in shared memory (TMA-loaded
// q_c plus the rotated q_r stored by the softmax warps) and QK reads it there;
// where that leaves room for fewer than two key stages ((256, 64)), the first
// q_c columns go to the TMEM left after O and QK mixes TMEM and shared-memory
// A operands.
// d_c = 512: a 512-column fp32 O alone fills TMEM, so each 128-row tile runs
// on a cluster of two CTAs, each owning 256 output columns (DV). Both score
// the full [c | k] tile (QK is computed twice, PV once: 2112 useful of 3200
// issued FLOP per row-key pair) and share every key tile through the same
// multicast as the row-tile pairs above; each keeps the q_c columns that fit
// next to S, P and its O half in TMEM (320) and the rest of Q in shared
// memory, so QK mixes TMEM- and shared-memory A operands.
// The V operand is the first d_c columns of the same key tile read MN-major,
// so the cache is never expanded into per-head keys or values.
#include <cmath>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kBM = 128;       // rows per CTA = TMEM lanes
constexpr int kThreads = 224;  // 7 warps
constexpr float kRescaleLog2 = 8.0f;

template <int DC, int DR, int BN, int DV = DC>
struct AttnShape {
  static constexpr int kBN = BN;                   // keys per block
  static constexpr int DK = DC + DR;
  static constexpr int kSplit = DC / DV;           // CTAs per row tile, DV output columns each
  static constexpr int kTileBytes = kBN * DK * 2;  // one key stage
  static constexpr int kCBox = kBN * 128;          // one [BN keys x 64 columns] box of c
  static constexpr int kKrOff = DC * kBN * 2;      // byte offset of the d_r columns in a tile
  static constexpr int kTmemS = 0;
  static constexpr int kTmemP = kBN;               // bf16 P: two values per column
  static constexpr int kTmemO = kBN + kBN / 2;
  static constexpr int kTmemQ = kTmemO + DV;
  static constexpr int kBarBytes = 256;
  static constexpr int kSmemCap = 232448;
  static constexpr bool kQinTmem = kTmemQ + DK / 2 <= 512;
  // Where Q lives when it does not fit in TMEM: all of it in shared memory
  // if two key stages still fit beside it (SS score MMAs measured faster
  // than a TS/SS mix there), else the leading 64-column boxes of q_c that
  // fit go to TMEM and the rest of Q to shared memory
  static constexpr bool kQSmemFits = 1024 + kBarBytes + kBM * DK * 2 + 2 * kTileBytes <= kSmemCap;
  static constexpr int kQcTmem =
      kQinTmem ? DC : (kQSmemFits ? 0 : ((512 - kTmemQ) * 2 / 64) * 64);
  static constexpr int kQcSmem = DC - kQcTmem;
  // shared-memory Q tile: [128 rows x 64 columns] boxes of q_c, then q_r
  static constexpr int kQKrOff = kQcSmem * kBM * 2;
  static constexpr int kQBytes = kQinTmem ? 0 : kQKrOff + kBM * DR * 2;
  static constexpr int kFit = (kSmemCap - 1024 - kBarBytes - kQBytes) / kTileBytes;
  static constexpr int kMaxStages = BN == 128 ? 4 : 6;
  static constexpr int kStages = kFit > kMaxStages ? kMaxStages : kFit;
  static constexpr int kSmemBytes = 1024 + kQBytes + kTileBytes * kStages + kBarBytes;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kKrSw = DR == 32 ? kSw64 : kSw128;
  static constexpr uint32_t kKrRow = DR * 2;      // bytes per row of the d_r block
  static constexpr uint32_t kKrSbo = 8 * kKrRow;  // one 8-row swizzle atom
  static constexpr uint32_t kIdescQK = idesc_bf16_f32(kBM, kBN, false, false);
  static constexpr uint32_t kIdescPV = idesc_bf16_f32(kBM, DV, false, true);
  static_assert(BN == 128 || BN == 64, "key block: 128 or 64");
  static_assert(DC % 64 == 0 && DC >= 64 && DV % 64 == 0 && DV <= 256 && DC % DV == 0,
                "d_c: multiple of 64; each CTA's output columns: multiple of 64 up to 256");
  static_assert(kSplit == 1 || kSplit == 2, "output split over at most two CTAs");
  static_assert(DR == 32 || DR == 64, "d_r: 32 or 64");
  static_assert(kTmemO + DV <= 512 && kTmemQ + kQcTmem / 2 <= 512,
                "S, P, O and the TMEM part of Q must fit in 512 TMEM columns");
  static_assert(kStages >= 2, "at least two key stages must fit in shared memory");
  static_assert(kTileBytes % 1024 == 0 && kKrOff % 1024 == 0 && kQKrOff % 1024 == 0,
                "swizzle-atom alignment");
};

struct AttnKParams {
  const __nv_bfloat16* q_c;
  const __nv_bfloat16* q_r;
  const int* q_pos;
  const float2* rope;
  __nv_bfloat16* o;
  int rows, heads, n_valid, rope_len, pairs_t, pairs_h;
  float scale_log2;
  int* status;
};

template <int DC, int DR, int CL, int BN, int DV>
__global__ void __launch_bounds__(kThreads, 1)
    mla_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_qc,
                       const __grid_constant__ CUtensorMap tm_c,
                       const __grid_constant__ CUtensorMap tm_kr, const AttnKParams p) {
  using S = AttnShape<DC, DR, BN, DV>;
  constexpr int kBN = S::kBN;
  constexpr int NST = S::kStages;
  constexpr uint16_t kPair = static_cast<uint16_t>((1u << CL) - 1u);  // every CTA of the cluster
  static_assert(CL == 1 || CL == 2, "clusters of one or two CTAs");
  // a split row tile's CTAs form the cluster: both read every key tile
  static_assert(S::kSplit == 1 || CL == S::kSplit, "split CTAs share one cluster");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_smem_1024(smem_raw);
  uint8_t* sQ = smem;  // only when Q stays in shared memory
  uint8_t* sKV = smem + S::kQBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sKV + NST * S::kTileBytes);
  uint64_t* q_tma_full = bars + 0;
  uint64_t* q_ready = bars + 1;
  uint64_t* kv_full = bars + 2;
  uint64_t* kv_empty = kv_full + NST;
  uint64_t* s_full = kv_empty + NST;
  uint64_t* s_free = s_full + 1;
  uint64_t* p_full = s_free + 1;
  uint64_t* pv_done = p_full + 1;
  uint64_t* mma_drain = pv_done + 1;  // [2]: one per issuing thread
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_drain + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.y;
  const int tile = blockIdx.x / S::kSplit;
  const int vpart = blockIdx.x - tile * S::kSplit;  // which DV output columns
  const int row0 = tile * kBM;
  const int nblk = (p.n_valid + kBN - 1) / kBN;
  const WaitCtx wc{abort_flag, p.status};

  if (threadIdx.x == 0) {
    mbar_init(q_tma_full, 1);
    mbar_init(q_ready, kBM);
    for (int s = 0; s < NST; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], CL);  // released by the MMA of every CTA that reads it
    }
    mbar_init(s_full, 1);
    mbar_init(s_free, kBM);
    mbar_init(p_full, kBM);
    mbar_init(pv_done, 1);
    mbar_init(&mma_drain[0], 1);
    mbar_init(&mma_drain[1], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, S::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the peer's barriers must be initialised before any multicast lands
  if constexpr (CL > 1) cluster_sync();
  grid_dep_sync();
  const int crank = CL > 1 ? static_cast<int>(cluster_ctarank()) : 0;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_c);
      tma_prefetch_desc(&tm_kr);
      if constexpr (!S::kQinTmem) {
        tma_prefetch_desc(&tm_qc);
        mbar_arrive_expect_tx(q_tma_full, S::kQcSmem * kBM * 2);
        for (int cb = 0; cb < S::kQcSmem / 64; ++cb)
          tma_load_3d(sQ + cb * 16384, &tm_qc, q_tma_full, S::kQcTmem + cb * 64, row0, b);
      }
      int issued = 0;
      for (int j = 0; j < nblk; ++j) {
        const int st = j % NST;
        if (j >= NST && !mbar_wait(&kv_empty[st], ((j / NST) - 1) & 1, wc)) break;
        uint8_t* kv = sKV + st * S::kTileBytes;
        mbar_arrive_expect_tx(&kv_full[st], S::kTileBytes);
        if constexpr (CL == 1) {
          for (int cb = 0; cb < DC / 64; ++cb)
            tma_load_3d(kv + cb * S::kCBox, &tm_c, &kv_full[st], cb * 64, j * kBN, b);
          tma_load_3d(kv + S::kKrOff, &tm_kr, &kv_full[st], 0, j * kBN, b);
        } else {
          // each CTA fetches every other box once and multicasts it to both
          for (int bx = crank; bx <= DC / 64; bx += CL) {
            if (bx < DC / 64)
              tma_load_3d_mc(kv + bx * S::kCBox, &tm_c, &kv_full[st], bx * 64, j * kBN, b, kPair);
            else
              tma_load_3d_mc(kv + S::kKrOff, &tm_kr, &kv_full[st], 0, j * kBN, b, kPair);
          }
        }
        issued = j + 1;
      }
      // every stage's last use must be released before the CTA may exit
      for (int st = 0; st < NST && st < nblk && !*abort_flag; ++st)
        mbar_wait(&kv_empty[st], (((nblk - st + NST - 1) / NST) - 1) & 1, wc);
      if (*abort_flag) {  // let every copy this CTA started land before exit
        if constexpr (!S::kQinTmem) mbar_wait_drain(q_tma_full, 0, p.status);
        for (int u = issued > NST ? issued - NST : 0; u < issued; ++u)
          mbar_wait_drain(&kv_full[u % NST], (u / NST) & 1, p.status);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------ QK^T issuer
    if (lane == 0) {
      bool ok = mbar_wait(q_ready, 0, wc);
      if constexpr (!S::kQinTmem) ok = ok && mbar_wait(q_tma_full, 0, wc);
      tc_fence_after();
      const uint32_t qa = smem_u32(sQ);
      for (int j = 0; ok && j < nblk; ++j) {
        // S = Q K_j^T; S's previous contents (block j-1) must have been read
        if (j >= 1 && !mbar_wait(s_free, (j - 1) & 1, wc)) {
          ok = false;
          break;
        }
        const int st = j % NST;
        if (!mbar_wait(&kv_full[st], (j / NST) & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t ka = smem_u32(sKV) + st * S::kTileBytes;
#pragma unroll
        for (int cb = 0; cb < DC / 64; ++cb)
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint64_t bd = sdesc(ka + cb * S::kCBox + k * 32, 16, 1024, kSw128);
            const uint32_t acc = (cb | k) != 0 ? 1u : 0u;
            if (cb < S::kQcTmem / 64)  // resolved at compile time (unrolled)
              umma_ts(tmem + S::kTmemS, tmem + S::kTmemQ + (cb * 4 + k) * 8, bd, S::kIdescQK, acc);
            else
              umma_ss(tmem + S::kTmemS,
                      sdesc(qa + (cb - S::kQcTmem / 64) * 16384 + k * 32, 16, 1024, kSw128), bd,
                      S::kIdescQK, acc);
          }
#pragma unroll
        for (int k = 0; k < DR / 16; ++k) {
          const uint64_t bd = sdesc(ka + S::kKrOff + k * 32, 16, S::kKrSbo, S::kKrSw);
          if constexpr (S::kQinTmem)
            umma_ts(tmem + S::kTmemS, tmem + S::kTmemQ + DC / 2 + k * 8, bd, S::kIdescQK, 1u);
          else
            umma_ss(tmem + S::kTmemS, sdesc(qa + S::kQKrOff + k * 32, 16, S::kKrSbo, S::kKrSw),
                    bd, S::kIdescQK, 1u);
        }
        umma_commit(s_full);
      }
      if (!ok) {  // wait for every MMA this thread issued before TMEM is freed
        umma_commit(&mma_drain[0]);
        mbar_wait_drain(&mma_drain[0], 0, p.status);
      }
    }
    __syncwarp();
  } else if (warp == 6) {
    // --------------------------------------------------------- PV issuer
    if (lane == 0) {
      bool ok = true;
      for (int i = 0; ok && i < nblk; ++i) {
        // O += P_i V_i, V = this CTA's DV of the first d_c columns of block
        // i's stage (MN-major)
        if (!mbar_wait(p_full, i & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int st = i % NST;
        const uint32_t va = smem_u32(sKV) + st * S::kTileBytes + vpart * (DV / 64) * S::kCBox;
#pragma unroll
        for (int s = 0; s < kBN / 16; ++s)
          umma_ts(tmem + S::kTmemO, tmem + S::kTmemP + s * 8,
                  sdesc(va + s * 2048, S::kCBox, 1024, kSw128), S::kIdescPV,
                  (i > 0 || s > 0) ? 1u : 0u);
        if constexpr (CL == 1)
          umma_commit(&kv_empty[st]);
        else
          umma_commit_mc(&kv_empty[st], kPair);
        umma_commit(pv_done);
      }
      if (!ok) {
        umma_commit(&mma_drain[1]);
        mbar_wait_drain(&mma_drain[1], 0, p.status);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ softmax (warps 2..5)
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int r = quarter * 32 + lane;
    const uint32_t t_lane = static_cast<uint32_t>(quarter * 32) << 16;
    const int grow = row0 + r;
    const bool row_ok = grow < p.rows;

    // Q: q_c as is, q_r rotated by the query position (RoPE3D), both bf16.
    {
      uint32_t w[DR / 2];
#pragma unroll
      for (int i = 0; i < DR / 2; ++i) w[i] = 0u;
      if (row_ok) {
        const uint4* src = reinterpret_cast<const uint4*>(
            p.q_r + (static_cast<size_t>(b) * p.rows + grow) * DR);
#pragma unroll
        for (int i = 0; i < DR / 8; ++i) {
          const uint4 v = __ldg(src + i);
          w[4 * i + 0] = v.x;
          w[4 * i + 1] = v.y;
          w[4 * i + 2] = v.z;
          w[4 * i + 3] = v.w;
        }
        const int nq = p.rows / p.heads;
        const int* pp = p.q_pos + (static_cast<size_t>(b) * nq + grow / p.heads) * 3;
        int pa[3] = {__ldg(pp), __ldg(pp + 1), __ldg(pp + 2)};
#pragma unroll
        for (int a = 0; a < 3; ++a)
          if (pa[a] < 0 || pa[a] >= p.rope_len) {
            record_status(p.status, MLA_ERR_RANGE);
            pa[a] = 0;
          }
#pragma unroll
        for (int i = 0; i < DR / 2; ++i) {
          const int pos = i < p.pairs_t ? pa[0] : (i < p.pairs_t + p.pairs_h ? pa[1] : pa[2]);
          const float2 cs = __ldg(p.rope + static_cast<size_t>(pos) * (DR / 2) + i);
          const float x0 = bf16_lo(w[i]), x1 = bf16_hi(w[i]);
          w[i] = pack_bf16x2(x0 * cs.x - x1 * cs.y, x0 * cs.y + x1 * cs.x);
        }
      }
      if constexpr (S::kQcTmem > 0) {
        // TMEM holds the MMA's A operand row-major: column c = elements 2c, 2c+1
        const uint4* qsrc = reinterpret_cast<const uint4*>(
            p.q_c + (static_cast<size_t>(b) * p.rows + (row_ok ? grow : 0)) * DC);
#pragma unroll
        for (int c = 0; c < S::kQcTmem / 64; ++c) {
          uint32_t qw[32];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const uint4 v = row_ok ? __ldg(qsrc + c * 8 + i) : make_uint4(0u, 0u, 0u, 0u);
            qw[4 * i + 0] = v.x;
            qw[4 * i + 1] = v.y;
            qw[4 * i + 2] = v.z;
            qw[4 * i + 3] = v.w;
          }
          tmem_st32(tmem + t_lane + S::kTmemQ + c * 32, qw);
        }
      }
      if constexpr (S::kQinTmem) {
#pragma unroll
        for (int c = 0; c < DR / 32; ++c)
          tmem_st16(tmem + t_lane + S::kTmemQ + DC / 2 + c * 16, w + c * 16);
      } else {
        // the same 16-byte-chunk swizzle the TMA applies to the q_c part
        uint8_t* krow = sQ + S::kQKrOff + r * S::kKrRow;
#pragma unroll
        for (int c = 0; c < DR / 8; ++c) {
          const int phys = DR == 32 ? (c ^ ((r >> 1) & 3)) : (c ^ (r & 7));
          *reinterpret_cast<uint4*>(krow + phys * 16) =
              make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
        }
        fence_proxy_async_smem();
      }
      if constexpr (S::kQcTmem > 0) {
        tmem_wait_st();
        tc_fence_before();
      }
      mbar_arrive(q_ready);
    }

    float m_run = -INFINITY;
    float l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      if (!mbar_wait(s_full, j & 1, wc)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sr[kBN];
#pragma unroll
      for (int c = 0; c < kBN / 32; ++c)
        tmem_ld32(tmem + t_lane + S::kTmemS + c * 32,
                  *reinterpret_cast<uint32_t(*)[32]>(&sr[c * 32]));
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(s_free);  // S_j is in registers: the next block's scores may land
      float sv[kBN];
#pragma unroll
      for (int c = 0; c < kBN; ++c) sv[c] = __uint_as_float(sr[c]);
      const int valid = p.n_valid - j * kBN;
      if (valid < kBN) {
#pragma unroll
        for (int c = 0; c < kBN; ++c)
          if (c >= valid) sv[c] = -INFINITY;
      }
      // row max as 8 independent chains + a 3-level tree (short dependency path)
      // (three-input max: two new scores per instruction)
      float m8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) m8[i] = sv[i];
#pragma unroll
      for (int c = 8; c + 16 <= kBN; c += 16)
#pragma unroll
        for (int i = 0; i < 8; ++i) m8[i] = fmax3(m8[i], sv[c + i], sv[c + 8 + i]);
      if constexpr ((kBN - 8) % 16 != 0) {
#pragma unroll
        for (int i = 0; i < 8; ++i) m8[i] = fmaxf(m8[i], sv[kBN - 8 + i]);
      }
      const float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                             fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
      const float m_blk = mx * p.scale_log2;
      // lazy rescale: keep the running max unless this block's max exceeds it
      // by more than 2^8 (P <= 256 then, harmless in bf16 / fp32)
      float alpha = 1.f;
      bool need = false;
      if (j == 0) {
        m_run = m_blk;
      } else if (m_blk > m_run + kRescaleLog2) {
        need = true;
        alpha = ex2_approx(m_run - m_blk);
        m_run = m_blk;
      }
      debug_count_rescale(need && row_ok, p.status);
      l_run *= alpha;
      // P_j in registers before waiting on PV_{j-1}: only the TMEM store
      // below is serialised with the previous PV
      const float neg_m = -m_run;
      // scale-and-shift and the row sum two scores per instruction (paired
      // fp32: the same IEEE roundings as the scalar forms, same 8 sum chains)
      const uint64_t scale2 = f32x2_pack(p.scale_log2, p.scale_log2);
      const uint64_t negm2 = f32x2_pack(neg_m, neg_m);
      uint64_t l4[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) l4[i] = 0ull;
      uint32_t pk[kBN / 2];
#pragma unroll
      for (int i = 0; i < kBN / 2; ++i) {
        float t0, t1;
        f32x2_unpack(f32x2_fma(f32x2_pack(sv[2 * i], sv[2 * i + 1]), scale2, negm2), t0, t1);
        const float p0 = ex2_approx(t0);
        const float p1 = ex2_approx(t1);
        l4[i & 3] = f32x2_add(l4[i & 3], f32x2_pack(p0, p1));
        pk[i] = pack_bf16x2(p0, p1);
      }
      float l8[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) f32x2_unpack(l4[i], l8[2 * i], l8[2 * i + 1]);
      l_run += ((l8[0] + l8[1]) + (l8[2] + l8[3])) + ((l8[4] + l8[5]) + (l8[6] + l8[7]));
      if (j > 0) {
        // PV_{j-1} must have read P (and finished with O) before P_j is
        // written or O is rescaled
        if (!mbar_wait(pv_done, (j - 1) & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xffffffffu, need)) {
#pragma unroll 1
          for (int c = 0; c < DV / 32; ++c) {
            uint32_t ov[32];
            tmem_ld32(tmem + t_lane + S::kTmemO + c * 32, ov);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * alpha);
            tmem_st32(tmem + t_lane + S::kTmemO + c * 32, ov);
          }
          tmem_wait_st();
        }
      }
#pragma unroll
      for (int c = 0; c < kBN / 64; ++c)
        tmem_st32(tmem + t_lane + S::kTmemP + c * 32,
                  *reinterpret_cast<uint32_t(*)[32]>(&pk[c * 32]));
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(p_full);
    }

    // O / l as bf16: each thread stages its row densely in the key stages
    // (free once the last PV is done: every key tile, the peer's multicast
    // halves included, has landed and been read) and the rows leave shared
    // memory by bulk copy, the whole tile at once when its rows are
    // consecutive rows of o (DV = d_c).
    const bool have_o = ok && mbar_wait(pv_done, (nblk - 1) & 1, wc);
    uint8_t* srow = sKV + r * DV * 2;
    if (have_o) {
      tc_fence_after();
      const float inv_l = 1.f / l_run;
#pragma unroll 1
      for (int sg = 0; sg < DV / 64; ++sg) {
        uint32_t va[32], vb[32];
        tmem_ld32(tmem + t_lane + S::kTmemO + sg * 64, va);
        tmem_ld32(tmem + t_lane + S::kTmemO + sg * 64 + 32, vb);
        tmem_wait_ld();
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const uint32_t* v = i < 16 ? va : vb;
          const int j = i & 15;
          pk[i] = pack_bf16x2(__uint_as_float(v[2 * j]) * inv_l,
                              __uint_as_float(v[2 * j + 1]) * inv_l);
        }
        stage_row<8>(srow + sg * 128, pk, r & 7);
      }
    }
    fence_proxy_async_smem();
    if constexpr (DV == DC) {
      asm volatile("bar.sync 1, 128;" ::: "memory");  // the four softmax warps
      // the tile's rows below p.rows; none in the CTA that only pads the grid
      // to whole clusters (an odd number of row tiles)
      const int valid = min(kBM, p.rows - row0);
      if (r == 0 && have_o && !*abort_flag && valid > 0) {
        bulk_store(p.o + (static_cast<size_t>(b) * p.rows + row0) * DC, sKV, valid * DC * 2);
        bulk_commit();
        bulk_wait_read_all();  // the staged rows must outlive the copy's reads
      }
    } else if (have_o && row_ok) {
      bulk_store(p.o + (static_cast<size_t>(b) * p.rows + grow) * DC + vpart * DV, srow, DV * 2);
      bulk_commit();
      bulk_wait_read_all();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, S::kTmemCols);
  }
  // neither CTA leaves while the other may still write into its shared memory
  if constexpr (CL > 1) cluster_sync();
}

template <int DC, int DR, int CL, int BN, int DV = DC>
int launch_tc(const AttnArgs& a) {
  using S = AttnShape<DC, DR, BN, DV>;
  CUtensorMap tm_qc, tm_c, tm_kr;
  const unsigned long long rows = a.rows, slots = a.slots;
  if (!encode_map_3d_bf16(&tm_qc, a.q_c, DC, rows, a.batch, DC * 2ull, rows * DC * 2ull, 64,
                          kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_3d_bf16(&tm_c, a.c, DC, a.n_valid, a.batch, DC * 2ull, slots * DC * 2ull, 64,
                          S::kBN, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_3d_bf16(&tm_kr, a.kr, DR, a.n_valid, a.batch, DR * 2ull, slots * DR * 2ull, DR,
                          S::kBN,
                          DR == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B))
    return MLA_ERR_CUDA;
  auto kern = mla_attn_tc_kernel<DC, DR, CL, BN, DV>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmemBytes);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  AttnKParams kp;
  kp.q_c = static_cast<const __nv_bfloat16*>(a.q_c);
  kp.q_r = static_cast<const __nv_bfloat16*>(a.q_r);
  kp.q_pos = a.q_pos;
  kp.rope = reinterpret_cast<const float2*>(a.rope);
  kp.o = static_cast<__nv_bfloat16*>(a.o);
  kp.rows = a.rows;
  kp.heads = a.heads;
  kp.n_valid = a.n_valid;
  kp.rope_len = a.rope_len;
  kp.pairs_t = a.pairs_t;
  kp.pairs_h = a.pairs_h;
  kp.scale_log2 = a.scale_log2;
  kp.status = a.status;
  const int tiles = (a.rows + kBM - 1) / kBM;
  cudaLaunchConfig_t cfg = {};
  // pairs stay within a batch row; a split tile's CTAs are adjacent
  cfg.gridDim = dim3((tiles * S::kSplit + CL - 1) / CL * CL, a.batch, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = S::kSmemBytes;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_sync
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, kern, tm_qc, tm_c, tm_kr, kp);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

// Pairs of CTAs share every key tile through TMA multicast; a single row tile
// per batch element runs alone.
template <int DC, int DR, int BN = 128>
int launch_tc_pick(const AttnArgs& a) {
  return (a.rows + kBM - 1) / kBM >= 2 ? launch_tc<DC, DR, 2, BN>(a) : launch_tc<DC, DR, 1, BN>(a);
}

}  // namespace

int launch_attention_tc(const AttnArgs& a) {
  if (a.d_r == 32) {
    switch (a.d_c) {
      case 64: return launch_tc_pick<64, 32>(a);
      case 128: return launch_tc_pick<128, 32>(a);
      case 192: return launch_tc_pick<192, 32>(a);
      case 256: return launch_tc_pick<256, 32>(a);  // Q in shared memory (faster than 64-key blocks)
      case 512: return launch_tc<512, 32, 2, 64, 256>(a);  // output split over a CTA pair
      default: break;
    }
  } else if (a.d_r == 64) {
    switch (a.d_c) {
      case 64: return launch_tc_pick<64, 64>(a);
      case 128: return launch_tc_pick<128, 64>(a);
      case 192: return launch_tc_pick<192, 64>(a);
      case 256: return launch_tc_pick<256, 64>(a);  // Q split between TMEM and shared memory
      case 512: return launch_tc<512, 64, 2, 64, 256>(a);
      default: break;
    }
  }
  return MLA_ERR_UNSUPPORTED;
}

}  // namespace vmla
