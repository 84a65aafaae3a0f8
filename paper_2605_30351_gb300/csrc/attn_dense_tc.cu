// Dense per-head attention on the sm_103a tensor cores: the cache layout
// VideoMLA replaces (every token stores K and V for every head, 2 n_h d_h
// scalars; App. C.1), used as the baseline of the d_c sweep (Table 5a):
//     S = q_h K_h^T / sqrt(d_h),  P = softmax(S),  o_h = P V_h   per head h.
// Same pipeline as the latent kernel: one CTA owns 128 query tokens of one
// head (one TMEM lane each) and walks that head's keys in blocks of 128;
// CTA pairs (consecutive token tiles of the same head) share each key/value
// tile through TMA multicast.
//   warp 0     TMA producer: K_h and V_h tiles [128 keys x d_h] (SW128)
//   warp 1     TMEM allocation; one lane issues S = Q K^T (Q read from TMEM)
//   warp 6     one lane issues O += P V (P read from TMEM, V MN-major)
//   warps 2-5  load Q into TMEM, online softmax, O / l as bf16
// TMEM columns: S [0,128) P [128,192) O [192,192+d_h) Q [192+d_h, +d_h/2).
#include <cmath>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kThreads = 224;
constexpr float kRescaleLog2 = 8.0f;

template <int DH>
struct DenseShape {
  static constexpr int kHalf = kBN * DH * 2;        // one K or V tile
  static constexpr int kTileBytes = 2 * kHalf;      // K then V
  static constexpr int kBarBytes = 256;
  static constexpr int kFit = (232448 - 1024 - kBarBytes) / kTileBytes;
  static constexpr int kStages = kFit > 4 ? 4 : kFit;
  static constexpr int kSmemBytes = 1024 + kTileBytes * kStages + kBarBytes;
  static constexpr int kTmemS = 0, kTmemP = kBN, kTmemO = kBN + kBN / 2, kTmemQ = kTmemO + DH;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kIdescQK = idesc_bf16_f32(kBM, kBN, false, false);
  static constexpr uint32_t kIdescPV = idesc_bf16_f32(kBM, DH, false, true);
  static_assert(DH % 64 == 0 && DH <= 256, "head_dim: multiple of 64 up to 256");
  static_assert(kTmemQ + DH / 2 <= 512, "TMEM budget");
  static_assert(kStages >= 2, "smem");
};

struct DenseKParams {
  const __nv_bfloat16* q;  // [B][Nq][H][DH]
  __nv_bfloat16* o;        // [B][Nq][H][DH]
  int nq, heads, n_valid;
  float scale_log2;
  int* status;
};

template <int DH>
__global__ void __launch_bounds__(kThreads, 1)
    mla_dense_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k,
                             const __grid_constant__ CUtensorMap tm_v, const DenseKParams p) {
  using S = DenseShape<DH>;
  constexpr int NST = S::kStages;
  constexpr uint16_t kPair = 3;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_smem_1024(smem_raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NST * S::kTileBytes);
  uint64_t* q_ready = bars;
  uint64_t* kv_full = bars + 1;
  uint64_t* kv_empty = kv_full + NST;
  uint64_t* s_full = kv_empty + NST;
  uint64_t* s_free = s_full + 1;
  uint64_t* p_full = s_free + 1;
  uint64_t* pv_done = p_full + 1;
  uint64_t* mma_drain = pv_done + 1;  // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_drain + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int h = blockIdx.y, b = blockIdx.z;
  const int bh = b * p.heads + h;  // this head's K/V plane
  const int row0 = blockIdx.x * kBM;
  const int nblk = (p.n_valid + kBN - 1) / kBN;
  const WaitCtx wc{abort_flag, p.status};

  if (threadIdx.x == 0) {
    mbar_init(q_ready, kBM);
    for (int s = 0; s < NST; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 2);  // both CTAs of the pair read every tile
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
  cluster_sync();  // the peer's barriers exist before any multicast lands
  const int crank = static_cast<int>(cluster_ctarank());

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      int issued = 0;
      for (int j = 0; j < nblk; ++j) {
        const int st = j % NST;
        if (j >= NST && !mbar_wait(&kv_empty[st], ((j / NST) - 1) & 1, wc)) break;
        uint8_t* kv = smem + st * S::kTileBytes;
        mbar_arrive_expect_tx(&kv_full[st], S::kTileBytes);
        // 2*DH/64 boxes of [128 keys x 64]: K boxes then V boxes, alternated across the pair
        for (int bx = crank; bx < 2 * (DH / 64); bx += 2) {
          if (bx < DH / 64)
            tma_load_3d_mc(kv + bx * 16384, &tm_k, &kv_full[st], bx * 64, j * kBN, bh, kPair);
          else
            tma_load_3d_mc(kv + S::kHalf + (bx - DH / 64) * 16384, &tm_v, &kv_full[st],
                           (bx - DH / 64) * 64, j * kBN, bh, kPair);
        }
        issued = j + 1;
      }
      for (int st = 0; st < NST && st < nblk && !*abort_flag; ++st)
        mbar_wait(&kv_empty[st], (((nblk - st + NST - 1) / NST) - 1) & 1, wc);
      if (*abort_flag)
        for (int u = issued > NST ? issued - NST : 0; u < issued; ++u)
          mbar_wait_drain(&kv_full[u % NST], (u / NST) & 1, p.status);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(q_ready, 0, wc);
      tc_fence_after();
      for (int j = 0; ok && j < nblk; ++j) {
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
        const uint32_t ka = smem_u32(smem) + st * S::kTileBytes;
#pragma unroll
        for (int cb = 0; cb < DH / 64; ++cb)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_ts(tmem + S::kTmemS, tmem + S::kTmemQ + (cb * 4 + k) * 8,
                    sdesc(ka + cb * 16384 + k * 32, 16, 1024, kSw128), S::kIdescQK,
                    (cb | k) != 0 ? 1u : 0u);
        umma_commit(s_full);
      }
      if (!ok) {
        umma_commit(&mma_drain[0]);
        mbar_wait_drain(&mma_drain[0], 0, p.status);
      }
    }
    __syncwarp();
  } else if (warp == 6) {
    if (lane == 0) {
      bool ok = true;
      for (int i = 0; ok && i < nblk; ++i) {
        if (!mbar_wait(p_full, i & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int st = i % NST;
        const uint32_t va = smem_u32(smem) + st * S::kTileBytes + S::kHalf;
#pragma unroll
        for (int s = 0; s < kBN / 16; ++s)
          umma_ts(tmem + S::kTmemO, tmem + S::kTmemP + s * 8,
                  sdesc(va + s * 2048, 16384, 1024, kSw128), S::kIdescPV,
                  (i > 0 || s > 0) ? 1u : 0u);
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
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t t_lane = static_cast<uint32_t>(quarter * 32) << 16;
    const int n = row0 + r;
    const bool row_ok = n < p.nq;
    const size_t qoff = ((static_cast<size_t>(b) * p.nq + (row_ok ? n : 0)) * p.heads + h) * DH;
    {
      const uint4* qsrc = reinterpret_cast<const uint4*>(p.q + qoff);
#pragma unroll
      for (int c = 0; c < DH / 64; ++c) {
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
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(q_ready);
    }
    float m_run = -INFINITY, l_run = 0.f;
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
      mbar_arrive(s_free);
      float sv[kBN];
#pragma unroll
      for (int c = 0; c < kBN; ++c) sv[c] = __uint_as_float(sr[c]);
      const int valid = p.n_valid - j * kBN;
      if (valid < kBN) {
#pragma unroll
        for (int c = 0; c < kBN; ++c)
          if (c >= valid) sv[c] = -INFINITY;
      }
      // three-input max: two new scores per instruction
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
        if (!mbar_wait(pv_done, (j - 1) & 1, wc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xffffffffu, need)) {
#pragma unroll 1
          for (int c = 0; c < DH / 32; ++c) {
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
    if (ok && mbar_wait(pv_done, (nblk - 1) & 1, wc)) {
      tc_fence_after();
      const float inv_l = 1.f / l_run;
      uint4* dst = reinterpret_cast<uint4*>(p.o + qoff);
#pragma unroll 1
      for (int c = 0; c < DH / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(tmem + t_lane + S::kTmemO + c * 32, ov);
        tmem_wait_ld();
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i)
          pk[i] = pack_bf16x2(__uint_as_float(ov[2 * i]) * inv_l,
                              __uint_as_float(ov[2 * i + 1]) * inv_l);
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < 4; ++i)
            dst[c * 4 + i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
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
  cluster_sync();
}

template <int DH>
int launch_dense(const DenseArgs& a) {
  using S = DenseShape<DH>;
  CUtensorMap tm_k, tm_v;
  const unsigned long long slots = a.slots, planes = static_cast<unsigned long long>(a.batch) * a.heads;
  if (!encode_map_3d_bf16(&tm_k, a.k, DH, a.n_valid, planes, DH * 2ull, slots * DH * 2ull, 64, kBN,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_3d_bf16(&tm_v, a.v, DH, a.n_valid, planes, DH * 2ull, slots * DH * 2ull, 64, kBN,
                          CU_TENSOR_MAP_SWIZZLE_128B))
    return MLA_ERR_CUDA;
  auto kern = mla_dense_attn_tc_kernel<DH>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmemBytes);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  DenseKParams kp;
  kp.q = static_cast<const __nv_bfloat16*>(a.q);
  kp.o = static_cast<__nv_bfloat16*>(a.o);
  kp.nq = a.nq;
  kp.heads = a.heads;
  kp.n_valid = a.n_valid;
  kp.scale_log2 = a.scale_log2;
  kp.status = a.status;
  const int tiles = (a.nq + kBM - 1) / kBM;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((tiles + 1) / 2 * 2, a.heads, a.batch);  // pairs share one head's tiles
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = S::kSmemBytes;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, tm_k, tm_v, kp);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace

int launch_dense_attention_tc(const DenseArgs& a) {
  switch (a.head_dim) {
    case 64: return launch_dense<64>(a);
    case 128: return launch_dense<128>(a);
    default: return MLA_ERR_UNSUPPORTED;
  }
}

}  // namespace vmla
