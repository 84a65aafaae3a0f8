// Fused cache append on the sm_103a tensor cores.
//
// Paper: Eq. (ckv) c = W_dn^KV x, RMSNorm on c (App. D.2), Eq. (krope)
// k = RoPE3D(W_R^K x), FIFO ring write (App. D.4). One CTA takes 128 tokens:
//   warp 0     TMA producer: x tile [128 x 64] and the matching 64 columns of
//              [W_dkv ; W_kr] ([d_c + d_r] x 64) per stage, SW128.
//   warp 1     allocates TMEM; one lane issues tcgen05.mma into one
//              [128 x (d_c + d_r)] fp32 accumulator (a single N = 224 MMA per
//              K step at the paper's shape).
//   warps 2-5  epilogue, thread i = token i: RMSNorm over the d_c columns in
//              fp32, gamma, RoPE3D on the d_r columns (skipped when the
//              cache keeps k^R unrotated), bf16, staged in shared memory and
//              bulk-copied into the token's slot: (f mod W) * T + k, or with S
//              sink frames f * T + k for f < S and (S + (f - S) mod (W - S)) * T
//              + k after them.
// For d_c = 512 the [128 x (d_c + d_r)] accumulator does not fit the 512
// TMEM columns; the launch then runs two CTAs per token tile (blockIdx.z):
// one accumulates c (two N = 256 MMAs per K step) and applies RMSNorm, the
// other accumulates k^R and applies RoPE. Both stream the same x tile.
// When one CTA per token tile would leave most SMs idle (one chunk at batch
// 1), a cluster of d_c/64 CTAs shares each token tile, one per 64 columns of
// c (see AppendShape). When the tiles exceed one wave, two CTAs with fewer
// stages share each SM, so that one's start-up and epilogue overlap the
// other's K loop.
#include <cmath>
#include <type_traits>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;
// dynamic shared memory of a CTA that has an SM to itself, and of one of two
// CTAs sharing an SM (228 KB per SM, 1 KB of it reserved per CTA)
constexpr int kSmemOne = 232448;
constexpr int kSmemHalf = (233472 - 2 * 1024) / 2;
// K blocks of x a CTA of the first wave warms into L2 before its wait for
// the previous kernel (those CTAs start while that kernel finishes, HBM being
// mostly idle; later ones start under this kernel's own K loops and warm
// nothing). The two-CTAs-per-SM form holds two stages per CTA and profits
// from a deeper prefetch.
constexpr int kPrefetchOne = 4;
constexpr int kPrefetchX2 = 12;

// What one CTA computes: NC columns of c, from column c0 (given at run time),
// and NK columns of k^R, into one [128 x (NC + NK)] TMEM accumulator:
//  - both parts, NC = d_c and NK = d_r (d_c <= 256);
//  - d_c = 512, whose [d_c + d_r] accumulator exceeds TMEM: c alone or k^R
//    alone, two CTAs per token tile that need nothing from each other
//    (RMSNorm runs over c alone);
//  - a grid too small to occupy the SMs (one chunk at batch 1): a cluster
//    of CL = d_c/64 CTAs per token tile, one per 64 columns of c, the last
//    also computing k^R, so that each SM streams the token tile and only its
//    share of the weights. Every CTA fetches the whole x box (from L2 after
//    the first), so the CTAs' K loops do not wait on one another; they
//    exchange their partial RMSNorm sums of squares through distributed
//    shared memory.
template <int DC, int DR, int NC, int NK, int CL = 1, int BUDGET = kSmemOne>
struct AppendShape {
  static constexpr int N = NC + NK;
  static constexpr bool kSplitN = N > 256;  // then MMAs of at most 256: c part(s), k part
  static constexpr int kWcBox = NC == 0 ? 64 : (NC < 256 ? NC : 256);  // W_dkv rows per TMA box
  static constexpr int kABytes = kBM * kBK * 2;
  // rows of a stage's weight region: in a cluster every CTA takes the widest
  // slice's layout (one shared-memory size for the launch, and the partial
  // sums at the same offset in every CTA)
  static constexpr int kBRows = CL > 1 ? 64 + DR : N;
  static constexpr int kBBytes = kBRows * kBK * 2;
  static constexpr int kTxBytes = kABytes + N * kBK * 2;  // lands in this CTA per stage
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kBarBytes = 256;
  // [CL][128] partial sums of squares at the front of shared memory: the same
  // offset in every CTA of a cluster, whichever slice it computes
  static constexpr int kRedOff = CL > 1 ? (CL * kBM * 4 + 1023) / 1024 * 1024 : 0;
  // this CTA's gamma columns, fetched by the epilogue warps during the K loop
  static constexpr int kGammaBytes = NC * 2;
  static constexpr int kFit = (BUDGET - 1024 - kBarBytes - kGammaBytes - kRedOff) / kStageBytes;
  static constexpr int kStages = kFit > 6 ? 6 : kFit;
  static constexpr int kSmemBytes = 1024 + kRedOff + kStages * kStageBytes + kBarBytes + kGammaBytes;
  static constexpr uint32_t kTmemCols = N <= 32 ? 32 : (N <= 64 ? 64 : (N <= 256 ? 256 : 512));
  // output staging: dense c rows, dense k^R rows, then the rows' slots
  static_assert(kBM * N * 2 + kBM * 8 + 16 <= kStages * kStageBytes, "staging fits in the ring");
  static_assert(NC % 64 == 0 && (NK == 0 || NK == 32 || NK == 64), "staged row segments");
  static_assert(DC % 32 == 0 && DR % 32 == 0 && DR <= 64 && (DC <= 256 || DC % 256 == 0),
                "shape");
  static_assert(N > 0 && NC % 32 == 0 && (NK == 0 || NK == DR), "parts");
  static_assert((NC == DC && NK == DR && CL == 1) || (DC > 256 && CL == 1) ||
                    (CL == DC / 64 && CL >= 2 && DC <= 256 && NC == 64),
                "parts are split for d_c > 256, or over a cluster of 64-column slices");
  static_assert(N <= 512, "accumulator must fit in TMEM");
  static_assert(kStageBytes % 1024 == 0 && kWcBox > 0, "swizzle-atom alignment");
  static_assert(kStages >= 2, "smem");
};

struct AppendKParams {
  const __nv_bfloat16* gamma;
  const int* pos;
  const float2* rope;
  __nv_bfloat16* c;
  __nv_bfloat16* kr;
  int n_tok, k_blocks, slots, T, W, S;
  long long first_frame;
  int rope_len, pairs_t, pairs_h, use_rmsnorm, rotate;
  float eps;
  int* status;
  int first_wave;  // CTAs resident at once (a linear block index below it: the first wave)
  int pf_blocks;   // x K blocks a first-wave CTA warms into L2
};

// tile: the token tile (128 tokens) of this CTA; c0: its first column of c
template <int DC, int DR, int NC, int NK, int CL, int BUDGET = kSmemOne>
__device__ __forceinline__ void append_body(const CUtensorMap* tm_x, const CUtensorMap* tm_wc,
                                            const CUtensorMap* tm_wk, const AppendKParams& p,
                                            int tile, int c0) {
  using S = AppendShape<DC, DR, NC, NK, CL, BUDGET>;
  constexpr int NST = S::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = align_smem_1024(smem_raw);
  // [CL][128] partial sums of squares, written by every CTA of the cluster
  float* ss_all = reinterpret_cast<float*>(base);
  uint8_t* smem = base + S::kRedOff;  // the stage ring
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NST * S::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + NST;
  uint64_t* acc_full = bars + 2 * NST;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.y;
  const int row0 = tile * kBM;
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
    tmem_alloc(tmem_slot, S::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int crank = CL > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  // While the previous kernel in the stream finishes, HBM is mostly idle:
  // a CTA of the first wave warms the first x boxes of its tile (its part of
  // them in a cluster) into L2 then, so that the K loop starts on L2 hits.
  // Only the copies into shared memory wait for the previous kernel. The
  // weights are shared by every tile: each first-wave CTA also warms its
  // slice's rows of one K block, so that the first copies do not all miss
  // together.
  const long long lin =
      blockIdx.x + static_cast<long long>(gridDim.x) * (blockIdx.y + gridDim.y * blockIdx.z);
  const bool first_wave = lin < p.first_wave;
  if (first_wave && warp == 0 && lane == 0 && crank == 0) {
    const int kpf = p.k_blocks < p.pf_blocks ? p.k_blocks : p.pf_blocks;
    for (int kb = 0; kb < kpf; ++kb) tma_prefetch_l2_3d(tm_x, kb * kBK, row0, b);
  }
  if (first_wave && warp == 0 && lane == 1) {
    const int kb = (tile + static_cast<int>(gridDim.x) * b) % p.k_blocks;
    if constexpr (NC > 0)
      for (int h = 0; h < NC / S::kWcBox; ++h)
        tma_prefetch_l2_2d(tm_wc, kb * kBK, c0 + h * S::kWcBox);
    if constexpr (NK > 0) tma_prefetch_l2_2d(tm_wk, kb * kBK, 0);
  }
  // every CTA of the cluster has started before a peer writes its shared
  // memory (the partial sums of squares)
  if constexpr (CL > 1) cluster_sync();
  grid_dep_sync();

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(tm_x);
      if constexpr (NC > 0) tma_prefetch_desc(tm_wc);
      if constexpr (NK > 0) tma_prefetch_desc(tm_wk);
      int issued = 0;
      for (int kb = 0; kb < p.k_blocks; ++kb) {
        const int st = kb % NST;
        if (kb >= NST && !mbar_wait(&empty[st], ((kb / NST) - 1) & 1, wc)) break;
        uint8_t* a = smem + st * S::kStageBytes;
        uint8_t* bm = a + S::kABytes;
        mbar_arrive_expect_tx(&full[st], S::kTxBytes);
        tma_load_3d(a, tm_x, &full[st], kb * kBK, row0, b);
        if constexpr (NC > 0)
          for (int h = 0; h < NC / S::kWcBox; ++h)
            tma_load_2d(bm + h * S::kWcBox * 128, tm_wc, &full[st], kb * kBK,
                        c0 + h * S::kWcBox);
        if constexpr (NK > 0) tma_load_2d(bm + NC * 128, tm_wk, &full[st], kb * kBK, 0);
        issued = kb + 1;
      }
      if (*abort_flag)
        for (int u = issued > NST ? issued - NST : 0; u < issued; ++u)
          mbar_wait_drain(&full[u % NST], (u / NST) & 1, p.status);
    }
    __syncwarp();
    if constexpr (CL > 1) {  // the cluster's second barrier phase (see the epilogue)
      cluster_arrive_release();
      cluster_wait_acquire();
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      for (int kb = 0; kb < p.k_blocks; ++kb) {
        const int st = kb % NST;
        if (!mbar_wait(&full[st], (kb / NST) & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t aa = smem_u32(smem + st * S::kStageBytes);
        const uint32_t ba = aa + S::kABytes;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k) {
          const uint32_t acc = (kb | k) != 0 ? 1u : 0u;
          const uint64_t ad = sdesc(aa + k * 32, 16, 1024, kSw128);
          if constexpr (!S::kSplitN) {
            constexpr uint32_t idesc = idesc_bf16_f32(kBM, S::N, false, false);
            umma_ss(tmem, ad, sdesc(ba + k * 32, 16, 1024, kSw128), idesc, acc);
          } else {
            constexpr int kHc = NC < 256 ? NC : 256;  // columns per c MMA
            constexpr uint32_t idesc_c = idesc_bf16_f32(kBM, kHc, false, false);
#pragma unroll
            for (int h = 0; h < NC / kHc; ++h)
              umma_ss(tmem + h * kHc, ad, sdesc(ba + h * kHc * 128 + k * 32, 16, 1024, kSw128),
                      idesc_c, acc);
            if constexpr (NK > 0) {
              constexpr uint32_t idesc_k = idesc_bf16_f32(kBM, NK, false, false);
              umma_ss(tmem + NC, ad, sdesc(ba + NC * 128 + k * 32, 16, 1024, kSw128), idesc_k,
                      acc);
            }
          }
        }
        umma_commit(&empty[st]);
      }
      umma_commit(acc_full);
      if (!ok) mbar_wait_drain(acc_full, 0, p.status);
    }
    __syncwarp();
    if constexpr (CL > 1) {  // the cluster's second barrier phase
      cluster_arrive_release();
      cluster_wait_acquire();
    }
  } else {
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t t_row = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int n = row0 + r;
    const bool row_ok = n < p.n_tok;
    // What the epilogue reads from global memory is fetched while the MMAs
    // run, so that no load latency follows the accumulator: this CTA's gamma
    // columns into shared memory (read by every row), the row's ring slot
    // and its RoPE factors (cos, sin per pair) into registers.
    uint4* gamma_s = reinterpret_cast<uint4*>(smem + NST * S::kStageBytes + S::kBarBytes);
    for (int i = threadIdx.x - 64; i < NC / 8; i += 128)
      gamma_s[i] = p.gamma ? __ldg(reinterpret_cast<const uint4*>(p.gamma + c0) + i)
                           : make_uint4(0x3f803f80u, 0x3f803f80u, 0x3f803f80u, 0x3f803f80u);
    const long long f = p.first_frame + n / p.T;
    const long long slot_n = frame_base_slot(f, p.T, p.W, p.S) + n % p.T;
    const long long my_slot =
        row_ok && debug_in_range(slot_n, 0, p.slots, p.status) ? slot_n : -1;
    // does this row start a run of consecutive slots (row n - 1 not in the
    // slot just below)? the tile's first row always does
    bool run_start = my_slot >= 0 && r == 0;
    if (my_slot >= 0 && r > 0) {
      const long long f1 = p.first_frame + (n - 1) / p.T;
      run_start = frame_base_slot(f1, p.T, p.W, p.S) + (n - 1) % p.T != my_slot - 1;
    }
    float2 cs[NK > 0 ? NK / 2 : 1];
    if constexpr (NK > 0) {
      int pa[3] = {0, 0, 0};
      if (row_ok && p.rotate) {
        const int* pp = p.pos + (static_cast<size_t>(b) * p.n_tok + n) * 3;
        pa[0] = __ldg(pp);
        pa[1] = __ldg(pp + 1);
        pa[2] = __ldg(pp + 2);
#pragma unroll
        for (int a = 0; a < 3; ++a)
          if (pa[a] < 0 || pa[a] >= p.rope_len) {
            record_status(p.status, MLA_ERR_RANGE);
            pa[a] = 0;
          }
      }
#pragma unroll
      for (int pr = 0; pr < NK / 2; ++pr) {
        const int ps = pr < p.pairs_t ? pa[0] : (pr < p.pairs_t + p.pairs_h ? pa[1] : pa[2]);
        cs[pr] = p.rotate ? __ldg(p.rope + static_cast<size_t>(ps) * (DR / 2) + pr)
                          : make_float2(1.f, 0.f);
      }
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");  // gamma_s is complete
    const bool have_acc = mbar_wait(acc_full, 0, wc) && !*abort_flag;
    // Each thread stages its finished bf16 row in shared memory (the stage
    // ring is free once the accumulator is complete): c rows dense at
    // stage_c ([128][NC] bf16), k^R rows dense at stage_k ([128][NK]), so that
    // a run of consecutive slots is one contiguous block in shared memory, as
    // it is in the cache. One CTA per tile then hands each run to the
    // bulk-copy engine (one copy for c, one for k^R, one or two runs per
    // tile); a cluster's 64-column slices are written by a coalesced store
    // loop, their rows not being contiguous in the cache.
    uint8_t* stage_c = smem;
    uint8_t* stage_k = smem + kBM * NC * 2;
    long long* slot_of = reinterpret_cast<long long*>(smem + kBM * S::N * 2);  // [128]
    // rows that do not continue a run (run starts and rows past the tokens),
    // one bit per row, one word per warp
    uint32_t* run_breaks = reinterpret_cast<uint32_t*>(slot_of + kBM);  // [4]
    // pass 1: sum of squares of this CTA's c columns (fp32)
    float ss = 0.f;
    if (have_acc) {
      tc_fence_after();
#pragma unroll 1
      for (int cb = 0; cb < NC / 32; ++cb) {
        uint32_t v[32];
        tmem_ld32(t_row + cb * 32, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float f = __uint_as_float(v[i]);
          ss = fmaf(f, f, ss);
        }
      }
    }
    if constexpr (CL > 1) {
      // every CTA pushes its row's partial sum into slot [its rank][row] of
      // every CTA, then all threads of the cluster pass the second barrier
      // phase (release / acquire), on every path, so that no CTA waits for
      // one that left; after it the sums are read locally, in rank order
      const uint32_t local = smem_u32(ss_all + (c0 / 64) * kBM + r);
      for (int q = 0; q < CL; ++q) dsmem_st_f32(dsmem_addr(local, q), ss);
      cluster_arrive_release();
      cluster_wait_acquire();
      ss = 0.f;
      for (int q = 0; q < CL; ++q) ss += ss_all[q * kBM + r];
    }
    const uint32_t breaks = __ballot_sync(0xffffffffu, my_slot < 0 || run_start);
    if (have_acc) {
      slot_of[r] = my_slot;
      if (lane == 0) run_breaks[quarter] = breaks;
      // positional key first, so that its RoPE factors leave the registers
      // before pass 2: RoPE3D at the token's (t, h, w), or unrotated
      if constexpr (NK > 0) {
        uint32_t pk[NK / 2];
#pragma unroll
        for (int cb = 0; cb < NK / 32; ++cb) {
          uint32_t v[32];
          tmem_ld32(t_row + NC + cb * 32, v);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float2 f2 = cs[cb * 16 + i];
            const float x0 = __uint_as_float(v[2 * i]), x1 = __uint_as_float(v[2 * i + 1]);
            pk[cb * 16 + i] = p.rotate ? pack_bf16x2(x0 * f2.x - x1 * f2.y, x0 * f2.y + x1 * f2.x)
                                       : pack_bf16x2(x0, x1);
          }
        }
        stage_row<NK / 8>(stage_k + r * NK * 2, pk, NK == 32 ? (r >> 1) & 3 : r & 7);
      }
      // pass 2: gamma * c / rms -> bf16, one 64-column (128-byte) segment at a time
      const float inv = p.use_rmsnorm ? rsqrtf(ss / DC + p.eps) : 1.f;
      const uint32_t* gamma2 = reinterpret_cast<const uint32_t*>(gamma_s);  // bf16 pairs
#pragma unroll 1
      for (int sg = 0; sg < NC / 64; ++sg) {
        uint32_t va[32], vb[32];
        tmem_ld32(t_row + sg * 64, va);
        tmem_ld32(t_row + sg * 64 + 32, vb);
        tmem_wait_ld();
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const uint32_t ga = gamma2[sg * 32 + i], gb = gamma2[sg * 32 + 16 + i];
          pk[i] = pack_bf16x2(__uint_as_float(va[2 * i]) * inv * bf16_lo(ga),
                              __uint_as_float(va[2 * i + 1]) * inv * bf16_hi(ga));
          pk[16 + i] = pack_bf16x2(__uint_as_float(vb[2 * i]) * inv * bf16_lo(gb),
                                   __uint_as_float(vb[2 * i + 1]) * inv * bf16_hi(gb));
        }
        stage_row<8>(stage_c + r * NC * 2 + sg * 128, pk, r & 7);
      }
    }
    // the staged rows reach the async proxy (the bulk copies), then the four
    // epilogue warps meet; a wait that gave up anywhere shows in abort_flag
    fence_proxy_async_smem();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (have_acc && !*abort_flag) {
      if constexpr (CL == 1) {
        // the thread whose row starts a run of consecutive slots copies the
        // run: c rows to (b * slots + slot) * d_c (+ c0), k^R rows to
        // (b * slots + slot) * d_r, all 16-byte aligned and sized
        if (run_start) {
          int end = kBM;  // the next row that does not continue this run
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            uint32_t m = w < quarter ? 0u : run_breaks[w];
            if (w == quarter) m &= ~((2u << lane) - 1u);  // rows after this one
            if (m != 0u && end == kBM) end = w * 32 + __ffs(static_cast<int>(m)) - 1;
          }
          const int len = end - r;
          const size_t row_id = static_cast<size_t>(b) * p.slots + my_slot;
          if constexpr (NC > 0)
            bulk_store(p.c + row_id * DC + c0, stage_c + r * NC * 2, len * NC * 2);
          if constexpr (NK > 0) bulk_store(p.kr + row_id * DR, stage_k + r * NK * 2, len * NK * 2);
          bulk_commit();
          bulk_wait_read_all();  // the staged rows must outlive the copies' reads
        }
      } else {
        // consecutive threads store consecutive 16-byte pieces of the rows
        constexpr int kChunks = S::N * 2 / 16;  // 16-byte pieces per output row
        constexpr int kChunksC = NC * 2 / 16;
        for (int q = r; q < kBM * kChunks; q += kBM) {
          const int row = q / kChunks, ch = q % kChunks;
          const long long slot = slot_of[row];
          if (slot < 0) continue;
          const size_t row_id = static_cast<size_t>(b) * p.slots + slot;
          if (ch < kChunksC)
            *reinterpret_cast<uint4*>(p.c + row_id * DC + c0 + ch * 8) =
                *reinterpret_cast<const uint4*>(stage_c + row * NC * 2 + ch * 16);
          else
            *reinterpret_cast<uint4*>(p.kr + row_id * DR + (ch - kChunksC) * 8) =
                *reinterpret_cast<const uint4*>(stage_k + row * NK * 2 + (ch - kChunksC) * 16);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, S::kTmemCols);
  }
}

template <int DC, int DR>
__global__ void __launch_bounds__(kThreads, 1)
    mla_append_tc_kernel(const __grid_constant__ CUtensorMap tm_x,
                         const __grid_constant__ CUtensorMap tm_wc,
                         const __grid_constant__ CUtensorMap tm_wk, const AppendKParams p) {
  append_body<DC, DR, DC, DR, 1>(&tm_x, &tm_wc, &tm_wk, p, blockIdx.x, 0);
}

// Grids of more than one wave: two CTAs share each SM (fewer stages each), so
// that one CTA's start-up and epilogue run under the other's K loop.
template <int DC, int DR>
__global__ void __launch_bounds__(kThreads, 2)
    mla_append_tc_kernel_x2(const __grid_constant__ CUtensorMap tm_x,
                            const __grid_constant__ CUtensorMap tm_wc,
                            const __grid_constant__ CUtensorMap tm_wk, const AppendKParams p) {
  append_body<DC, DR, DC, DR, 1, kSmemHalf>(&tm_x, &tm_wc, &tm_wk, p, blockIdx.x, 0);
}

// d_c > 256: blockIdx.z = 0 computes c, 1 computes k^R, for the same tokens
template <int DC, int DR>
__global__ void __launch_bounds__(kThreads, 1)
    mla_append_tc_split_kernel(const __grid_constant__ CUtensorMap tm_x,
                               const __grid_constant__ CUtensorMap tm_wc,
                               const __grid_constant__ CUtensorMap tm_wk, const AppendKParams p) {
  if (blockIdx.z == 0)
    append_body<DC, DR, DC, 0, 1>(&tm_x, &tm_wc, &tm_wk, p, blockIdx.x, 0);
  else
    append_body<DC, DR, 0, DR, 1>(&tm_x, &tm_wc, &tm_wk, p, blockIdx.x, 0);
}

// Small grids: a cluster of d_c/64 CTAs per token tile; rank q computes c
// columns [64q, 64q + 64), the last rank k^R as well.
template <int DC, int DR>
__global__ void __launch_bounds__(kThreads, 1)
    mla_append_tc_cluster_kernel(const __grid_constant__ CUtensorMap tm_x,
                                 const __grid_constant__ CUtensorMap tm_wc,
                                 const __grid_constant__ CUtensorMap tm_wk,
                                 const AppendKParams p) {
  constexpr int CL = DC / 64;
  const int q = static_cast<int>(cluster_ctarank());
  const int tile = blockIdx.x / CL;
  if (q < CL - 1)
    append_body<DC, DR, 64, 0, CL>(&tm_x, &tm_wc, &tm_wk, p, tile, q * 64);
  else
    append_body<DC, DR, 64, DR, CL>(&tm_x, &tm_wc, &tm_wk, p, tile, q * 64);
}

template <int DC, int DR>
int launch_tc(const AppendArgs& a) {
  constexpr bool kSplit = DC > 256;
  constexpr bool kClusterable = DC >= 128 && DC <= 256;
  constexpr int kCl = kClusterable ? DC / 64 : 2;  // cluster size of the small-grid form
  const int tiles = (a.n_tok + kBM - 1) / kBM;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // the cluster form when its CTAs all fit in one wave (e.g. one Wan chunk at
  // batch 1: 37 tiles x 3 = 111 CTAs) and every cluster is resident at once;
  // otherwise one CTA per tile already fills the SMs and streaming the
  // weights once per tile is the cheaper way
  bool cluster = false;
  if constexpr (kClusterable) {
    const long long clusters = static_cast<long long>(tiles) * a.batch;
    if (clusters * kCl <= sms) {
      static int resident = -1;  // co-resident clusters of this shape (per process)
      if (resident < 0) {
        using SC0 = AppendShape<DC, DR, 64, 0, kCl>;
        using SC1 = AppendShape<DC, DR, 64, DR, kCl>;
        constexpr int kSm = SC0::kSmemBytes > SC1::kSmemBytes ? SC0::kSmemBytes : SC1::kSmemBytes;
        auto kc = mla_append_tc_cluster_kernel<DC, DR>;
        int n = 0;
        cudaLaunchConfig_t oc = {};
        oc.gridDim = dim3(kCl * static_cast<unsigned>(clusters), 1, 1);
        oc.blockDim = dim3(kThreads, 1, 1);
        oc.dynamicSmemBytes = kSm;
        cudaLaunchAttribute oa[1];
        oa[0].id = cudaLaunchAttributeClusterDimension;
        oa[0].val.clusterDim.x = kCl;
        oa[0].val.clusterDim.y = 1;
        oa[0].val.clusterDim.z = 1;
        oc.attrs = oa;
        oc.numAttrs = 1;
        if (cudaFuncSetAttribute(kc, cudaFuncAttributeMaxDynamicSharedMemorySize, kSm) !=
                cudaSuccess ||
            cudaOccupancyMaxActiveClusters(&n, kc, &oc) != cudaSuccess) {
          cudaGetLastError();  // a failed query only disables the cluster form
          n = 0;
        }
        resident = n;
      }
      cluster = clusters <= resident;
    }
  }
  // two CTAs per SM when the grid has more than one wave of single CTAs and
  // two stages of the unsplit form fit in half an SM's shared memory
  constexpr int kStageX2 = kBM * kBK * 2 + (DC + DR) * kBK * 2;
  constexpr bool kX2Fits = !kSplit && DC + DR <= 256 &&  // two 256-column TMEM accumulators
                           (kSmemHalf - 1024 - 256 - DC * 2) / kStageX2 >= 2;
  const bool x2 = kX2Fits && !cluster && static_cast<long long>(tiles) * a.batch > sms;
  // shapes of the CTAs each form launches (d_c > 256: the c and k^R halves;
  // the cluster form: a 64-column c slice and k^R; else both parts)
  using S = AppendShape<DC, DR, DC, kSplit ? 0 : DR>;
  using SK = AppendShape<DC, DR, kSplit ? 0 : DC, DR>;
  using SCc = std::conditional_t<kClusterable, AppendShape<DC, DR, 64, 0, kCl>, S>;
  using SCk = std::conditional_t<kClusterable, AppendShape<DC, DR, 64, DR, kCl>, S>;
  constexpr int kSmemPlain = S::kSmemBytes > SK::kSmemBytes ? S::kSmemBytes : SK::kSmemBytes;
  constexpr int kSmemCl = SCc::kSmemBytes > SCk::kSmemBytes ? SCc::kSmemBytes : SCk::kSmemBytes;
  int smem = cluster ? kSmemCl : kSmemPlain;
  if constexpr (kX2Fits)
    if (x2) smem = AppendShape<DC, DR, DC, DR, 1, kSmemHalf>::kSmemBytes;
  CUtensorMap tm_x, tm_wc, tm_wk;
  const unsigned long long H = a.hidden, n_tok = a.n_tok;
  if (!encode_map_3d_bf16(&tm_x, a.x, H, n_tok, a.batch, H * 2, n_tok * H * 2, kBK,
                          kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_wc, a.w_dkv, H, DC, H * 2, kBK, cluster ? 64 : S::kWcBox,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_wk, a.w_kr, H, DR, H * 2, kBK, DR, CU_TENSOR_MAP_SWIZZLE_128B))
    return MLA_ERR_CUDA;
  using KernFn = void (*)(CUtensorMap, CUtensorMap, CUtensorMap, AppendKParams);
  KernFn kern;
  if constexpr (kSplit)
    kern = mla_append_tc_split_kernel<DC, DR>;
  else if constexpr (kClusterable)
    kern = cluster ? mla_append_tc_cluster_kernel<DC, DR> : mla_append_tc_kernel<DC, DR>;
  else
    kern = mla_append_tc_kernel<DC, DR>;
  if constexpr (kX2Fits)
    if (x2) kern = mla_append_tc_kernel_x2<DC, DR>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  AppendKParams kp;
  kp.gamma = static_cast<const __nv_bfloat16*>(a.gamma);
  kp.pos = a.pos;
  kp.rope = reinterpret_cast<const float2*>(a.rope);
  kp.c = static_cast<__nv_bfloat16*>(a.c);
  kp.kr = static_cast<__nv_bfloat16*>(a.kr);
  kp.n_tok = a.n_tok;
  kp.k_blocks = a.hidden / kBK;
  kp.slots = a.slots;
  kp.T = a.tokens_per_frame;
  kp.W = a.window_frames;
  kp.S = a.sink_frames;
  kp.rotate = a.rotate;
  kp.first_frame = a.first_frame;
  kp.rope_len = a.rope_len;
  kp.pairs_t = a.pairs_t;
  kp.pairs_h = a.pairs_h;
  kp.use_rmsnorm = a.use_rmsnorm;
  kp.eps = a.eps;
  kp.status = a.status;
  kp.first_wave = sms * (x2 ? 2 : 1);
  kp.pf_blocks = x2 ? kPrefetchX2 : kPrefetchOne;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cluster ? tiles * kCl : tiles, a.batch, kSplit ? 2 : 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster ? kCl : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_sync
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, kern, tm_x, tm_wc, tm_wk, kp);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace

int launch_append_tc(const AppendArgs& a) {
  if (a.hidden % kBK != 0) return MLA_ERR_UNSUPPORTED;
  if (a.d_r == 32) {
    switch (a.d_c) {
      case 64: return launch_tc<64, 32>(a);
      case 128: return launch_tc<128, 32>(a);
      case 192: return launch_tc<192, 32>(a);
      case 256: return launch_tc<256, 32>(a);
      case 512: return launch_tc<512, 32>(a);
      default: break;
    }
  } else if (a.d_r == 64) {
    switch (a.d_c) {
      case 64: return launch_tc<64, 64>(a);
      case 128: return launch_tc<128, 64>(a);
      case 192: return launch_tc<192, 64>(a);
      case 256: return launch_tc<256, 64>(a);
      case 512: return launch_tc<512, 64>(a);
      default: break;
    }
  }
  return MLA_ERR_UNSUPPORTED;
}

}  // namespace vmla
