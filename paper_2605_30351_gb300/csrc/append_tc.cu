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
//              cache keeps k^R unrotated), bf16, 16-byte stores into the
//              token's slot: (f mod W) * T + k, or with S sink frames f * T + k
//              for f < S and (S + (f - S) mod (W - S)) * T + k after them.
// For d_c = 512 the [128 x (d_c + d_r)] accumulator does not fit the 512
// TMEM columns; the launch then runs two CTAs per token tile (blockIdx.z):
// one accumulates c (two N = 256 MMAs per K step) and applies RMSNorm, the
// other accumulates k^R and applies RoPE. Both stream the same x tile.
#include <cmath>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;

// What one CTA computes: both parts (d_c <= 256), or, for d_c = 512 whose
// [d_c + d_r] accumulator exceeds TMEM, only c or only k^R (the two CTAs of
// a token tile need nothing from each other: RMSNorm runs over c alone).
enum AppendPart { kPartBoth = 0, kPartC = 1, kPartK = 2 };

template <int DC, int DR, int PART = kPartBoth>
struct AppendShape {
  static constexpr int NC = PART == kPartK ? 0 : DC;  // c columns of the accumulator
  static constexpr int NK = PART == kPartC ? 0 : DR;  // k^R columns, after c
  static constexpr int N = NC + NK;
  static constexpr bool kSplitN = N > 256;  // then MMAs of at most 256: c part(s), k part
  static constexpr int kWcBox = DC < 256 ? DC : 256;  // W_dkv rows per TMA box
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = N * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kBarBytes = 256;
  static constexpr int kFit = (232448 - 1024 - kBarBytes) / kStageBytes;
  static constexpr int kStages = kFit > 6 ? 6 : kFit;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kBarBytes;
  static constexpr uint32_t kTmemCols = N <= 32 ? 32 : (N <= 64 ? 64 : (N <= 256 ? 256 : 512));
  // output staging row: N bf16 plus 16 bytes, so rows start on different banks
  static constexpr int kOutStride = N * 2 + 16;
  static_assert(kBM * kOutStride + kBM * 8 <= kStages * kStageBytes, "staging fits in the ring");
  static_assert(DC % 32 == 0 && DR % 32 == 0 && DR <= 64 && (DC <= 256 || DC % 256 == 0),
                "shape");
  static_assert(PART == kPartBoth || DC > 256, "parts are split only when d_c > 256");
  static_assert(N <= 512, "accumulator must fit in TMEM");
  static_assert(kStageBytes % 1024 == 0, "swizzle-atom alignment");
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
};

template <int DC, int DR, int PART>
__device__ __forceinline__ void append_body(const CUtensorMap* tm_x, const CUtensorMap* tm_wc,
                                            const CUtensorMap* tm_wk, const AppendKParams& p) {
  using S = AppendShape<DC, DR, PART>;
  constexpr int NC = S::NC;
  constexpr int NK = S::NK;
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
  const int b = blockIdx.y;
  const int row0 = blockIdx.x * kBM;
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
        mbar_arrive_expect_tx(&full[st], S::kStageBytes);
        tma_load_3d(a, tm_x, &full[st], kb * kBK, row0, b);
        if constexpr (NC > 0)
          for (int h = 0; h < NC / S::kWcBox; ++h)
            tma_load_2d(bm + h * S::kWcBox * 128, tm_wc, &full[st], kb * kBK, h * S::kWcBox);
        if constexpr (NK > 0) tma_load_2d(bm + NC * 128, tm_wk, &full[st], kb * kBK, 0);
        issued = kb + 1;
      }
      if (*abort_flag)
        for (int u = issued > NST ? issued - NST : 0; u < issued; ++u)
          mbar_wait_drain(&full[u % NST], (u / NST) & 1, p.status);
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
  } else {
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t t_row = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int n = row0 + r;
    const bool row_ok = n < p.n_tok;
    const bool have_acc = mbar_wait(acc_full, 0, wc) && !*abort_flag;
    // The finished bf16 rows are staged in shared memory (the stage ring is
    // free once the accumulator is complete) and then written out by all 128
    // threads together, so that consecutive threads store consecutive 16-byte
    // pieces of a row instead of each thread writing its own row.
    uint8_t* stage_out = smem;                                   // [128][kOutStride]
    long long* slot_of = reinterpret_cast<long long*>(smem + kBM * S::kOutStride);  // [128]
    if (have_acc) {
      tc_fence_after();
      // pass 1: mean square of c over d_c (fp32)
      float ss = 0.f;
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
      const float inv = p.use_rmsnorm ? rsqrtf(ss / DC + p.eps) : 1.f;
      const long long f = p.first_frame + n / p.T;
      const long long slot = frame_base_slot(f, p.T, p.W, p.S) + n % p.T;
      slot_of[r] = row_ok && debug_in_range(slot, 0, p.slots, p.status) ? slot : -1;
      uint8_t* srow = stage_out + r * S::kOutStride;
      // pass 2: gamma * c / rms -> bf16
#pragma unroll 1
      for (int cb = 0; cb < NC / 32; ++cb) {
        uint32_t v[32];
        tmem_ld32(t_row + cb * 32, v);
        tmem_wait_ld();
        uint32_t gw[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          uint4 g4 = make_uint4(0x3f803f80u, 0x3f803f80u, 0x3f803f80u, 0x3f803f80u);  // ones
          if (p.gamma) g4 = __ldg(reinterpret_cast<const uint4*>(p.gamma + cb * 32) + i);
          gw[4 * i] = g4.x; gw[4 * i + 1] = g4.y; gw[4 * i + 2] = g4.z; gw[4 * i + 3] = g4.w;
        }
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i)
          pk[i] = pack_bf16x2(__uint_as_float(v[2 * i]) * inv * bf16_lo(gw[i]),
                              __uint_as_float(v[2 * i + 1]) * inv * bf16_hi(gw[i]));
#pragma unroll
        for (int i = 0; i < 4; ++i)
          *reinterpret_cast<uint4*>(srow + cb * 64 + i * 16) =
              make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
      }
      // positional key: RoPE3D at the token's (t, h, w), or unrotated
      int pa[3] = {0, 0, 0};
      if (NK > 0 && row_ok && p.rotate) {
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
#pragma unroll 1
      for (int cb = 0; cb < NK / 32; ++cb) {
        uint32_t v[32];
        tmem_ld32(t_row + NC + cb * 32, v);
        tmem_wait_ld();
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int pr = cb * 16 + i;
          const int ps = pr < p.pairs_t ? pa[0] : (pr < p.pairs_t + p.pairs_h ? pa[1] : pa[2]);
          const float2 cs = __ldg(p.rope + static_cast<size_t>(ps) * (DR / 2) + pr);
          const float x0 = __uint_as_float(v[2 * i]), x1 = __uint_as_float(v[2 * i + 1]);
          pk[i] = p.rotate ? pack_bf16x2(x0 * cs.x - x1 * cs.y, x0 * cs.y + x1 * cs.x)
                           : pack_bf16x2(x0, x1);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
          *reinterpret_cast<uint4*>(srow + NC * 2 + cb * 64 + i * 16) =
              make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
      }
    }
    // the four epilogue warps only
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (have_acc) {
      constexpr int kChunks = S::N * 2 / 16;  // 16-byte pieces per output row
      constexpr int kChunksC = NC * 2 / 16;
      for (int q = r; q < kBM * kChunks; q += kBM) {
        const int row = q / kChunks, ch = q % kChunks;
        const long long slot = slot_of[row];
        if (slot < 0) continue;
        const uint4 v = *reinterpret_cast<const uint4*>(stage_out + row * S::kOutStride + ch * 16);
        if (ch < kChunksC)
          *reinterpret_cast<uint4*>(p.c + (static_cast<size_t>(b) * p.slots + slot) * DC + ch * 8) = v;
        else
          *reinterpret_cast<uint4*>(p.kr + (static_cast<size_t>(b) * p.slots + slot) * DR +
                                    (ch - kChunksC) * 8) = v;
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
  append_body<DC, DR, kPartBoth>(&tm_x, &tm_wc, &tm_wk, p);
}

// d_c > 256: blockIdx.z = 0 computes c, 1 computes k^R, for the same tokens
template <int DC, int DR>
__global__ void __launch_bounds__(kThreads, 1)
    mla_append_tc_split_kernel(const __grid_constant__ CUtensorMap tm_x,
                               const __grid_constant__ CUtensorMap tm_wc,
                               const __grid_constant__ CUtensorMap tm_wk, const AppendKParams p) {
  if (blockIdx.z == 0)
    append_body<DC, DR, kPartC>(&tm_x, &tm_wc, &tm_wk, p);
  else
    append_body<DC, DR, kPartK>(&tm_x, &tm_wc, &tm_wk, p);
}

template <int DC, int DR>
int launch_tc(const AppendArgs& a) {
  constexpr bool kSplit = DC > 256;
  using S = AppendShape<DC, DR, kSplit ? kPartC : kPartBoth>;
  using SK = AppendShape<DC, DR, kSplit ? kPartK : kPartBoth>;
  constexpr int kSmem = S::kSmemBytes > SK::kSmemBytes ? S::kSmemBytes : SK::kSmemBytes;
  CUtensorMap tm_x, tm_wc, tm_wk;
  const unsigned long long H = a.hidden, n_tok = a.n_tok;
  if (!encode_map_3d_bf16(&tm_x, a.x, H, n_tok, a.batch, H * 2, n_tok * H * 2, kBK, kBM,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_wc, a.w_dkv, H, DC, H * 2, kBK, S::kWcBox,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_wk, a.w_kr, H, DR, H * 2, kBK, DR, CU_TENSOR_MAP_SWIZZLE_128B))
    return MLA_ERR_CUDA;
  auto kern = [] {
    if constexpr (kSplit)
      return mla_append_tc_split_kernel<DC, DR>;
    else
      return mla_append_tc_kernel<DC, DR>;
  }();
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
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
  const dim3 grid((a.n_tok + kBM - 1) / kBM, a.batch, kSplit ? 2 : 1);
  kern<<<grid, kThreads, kSmem, a.stream>>>(tm_x, tm_wc, tm_wk, kp);
  e = cudaGetLastError();
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
