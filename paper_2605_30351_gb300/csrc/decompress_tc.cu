// Decompression of the latent cache into per-head keys and values: the
// non-absorbed way to attend over it (Sec. 3.1 Eq. reconstruct; App. E is
// what it avoids). For every slot j of batch element b:
//     k[b][h][j] = [W_up,h^K c_j | k_j]      (d_nope + d_r = head_dim)
//     v[b][h][j] =  W_up,h^V c_j             (head_dim)
//
// Weight-stationary tcgen05 GEMM. The output columns are the rows of
// [W_up^K ; W_up^V] (H*d_nope + H*head_dim of them) cut into tiles of BN;
// CTA (t, g) keeps column tile t of the weights in shared memory for its
// whole life and streams the 128-slot tiles g, g + G, g + 2G, ... of c
// through a two-stage TMA ring; a tile never spans two batch elements (each
// element's slots are cut into tiles of their own, the last one ragged).
// Accumulators alternate between two TMEM buffers, so the epilogue of one
// tile overlaps the MMA of the next. The weights leave L2 once per CTA and c
// once per column tile, and every output byte is written once; at the Wan
// window the 201 MB of keys and values written dominate, so the kernel is
// bound by HBM writes.
//   warp 0     TMA producer (weights once, then c tiles)
//   warp 1     TMEM allocation; one lane issues tcgen05.mma (M = 128, N = BN)
//   warps 2-13 epilogue: warps w, w + 4, w + 8 read TMEM lane quarter w % 4
//              (slot rows), each a third of the columns, into shared staging
//              as bf16: one [128 slots x 32 columns] box per 32 columns, in
//              the 64-byte swizzle of the output tensor maps. One thread then
//              writes the tile with a TMA tensor store per box (a box never
//              spans two heads: d_nope and head_dim are multiples of 32; slots
//              past the element's last are clipped by the map). Key tiles
//              also copy each slot's cached positional key behind every head
//              that starts in the tile, with 16-byte stores from registers;
//              those loads are issued before the TMEM reads so their latency
//              hides.
#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kBM = 128;
constexpr int kParts = 3;                // epilogue warps per TMEM lane quarter
constexpr int kEpiWarps = 4 * kParts;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;

template <int DC>
struct DecShape {
  static constexpr int BN = DC <= 192 ? 192 : 96;
  static constexpr int kChunkBytesC = kBM * 128;  // one [128 x 64] bf16 K-chunk, SW128
  static constexpr int kChunkBytesW = BN * 128;   // one [BN x 64] bf16 K-chunk
  static constexpr int kWBytes = (DC / 64) * kChunkBytesW;
  static constexpr int kCBytes = (DC / 64) * kChunkBytesC;
  static constexpr int kBoxBytes = kBM * 64;  // one staged [128 slots x 32 columns] box, SW64
  static constexpr int kStageOff = kWBytes + 2 * kCBytes;
  static constexpr int kBarOff = kStageOff + (BN / 32) * kBoxBytes;
  // per-row output offsets of the positional-key copies
  static constexpr int kRowTabOff = kBarOff + 128;             // long long [2][128]
  static constexpr int kHeadTabOff = kRowTabOff + 2 * kBM * 8;  // long long [BN/8]
  static constexpr int kSmemBytes = 1024 + kHeadTabOff + (BN / 8) * 8;
  static constexpr uint32_t kTmemCols = 2 * BN <= 256 ? 256 : 512;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(kBM, BN, false, false);
  static_assert(DC % 64 == 0 && DC <= 256, "latent width");
  static_assert(BN % 32 == 0 && BN <= 256 && (BN / 32) % kParts == 0 && BN / 32 <= 2 * kParts,
                "tile width: whole 32-column boxes, one or two per epilogue warp");
  static_assert(kChunkBytesW % 1024 == 0 && kStageOff % 1024 == 0, "swizzle-atom alignment");
  static_assert(kSmemBytes <= 232448, "shared memory");
};

struct DecKParams {
  const __nv_bfloat16* kr;  // [M][d_r]
  __nv_bfloat16* k;         // [B][H][slots][head_dim]
  __nv_bfloat16* v;
  int M, tiles_per_b, n_row_tiles, tiles_k, cols_k, cols_v, dn, head_dim, d_r, slots, heads;
  int* status;
};

// All epilogue threads agree on one flag (named barrier 1 with an AND).
__device__ __forceinline__ bool epilogue_all(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.and.pred p, 1, %2, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "n"(kEpiThreads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ void epilogue_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
}

template <int DC>
__global__ void __launch_bounds__(kThreads, 1)
    mla_decompress_tc_kernel(const __grid_constant__ CUtensorMap tm_c,
                             const __grid_constant__ CUtensorMap tm_wk,
                             const __grid_constant__ CUtensorMap tm_wv,
                             const __grid_constant__ CUtensorMap tm_ko,
                             const __grid_constant__ CUtensorMap tm_vo, const DecKParams p) {
  using S = DecShape<DC>;
  constexpr int BN = S::BN;
  constexpr int KC = DC / 64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_smem_1024(smem_raw);
  uint8_t* sW = smem;
  uint8_t* sC = smem + S::kWBytes;
  uint8_t* stage_out = smem + S::kStageOff;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* w_full = bars;
  uint64_t* c_full = bars + 1;     // [2]
  uint64_t* c_empty = bars + 3;    // [2]
  uint64_t* acc_full = bars + 5;   // [2]
  uint64_t* acc_empty = bars + 7;  // [2]
  uint64_t* mma_done = bars + 9;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 10);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  long long* row_base = reinterpret_cast<long long*>(smem + S::kRowTabOff);
  long long* head_off = reinterpret_cast<long long*>(smem + S::kHeadTabOff);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x;  // column tile
  const int g = blockIdx.y, G = gridDim.y;
  const bool is_k = t < p.tiles_k;
  const int col0 = (is_k ? t : t - p.tiles_k) * BN;  // first column within its part
  const int cols = is_k ? p.cols_k : p.cols_v;
  const int n_valid = min(BN, cols - col0);
  const WaitCtx wc{abort_flag, p.status};

  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&c_full[s], 1);
      mbar_init(&c_empty[s], 1);
      mbar_init(&acc_full[s], 1);
      mbar_init(&acc_empty[s], kEpiWarps);  // one arrival per epilogue warp
    }
    mbar_init(mma_done, 1);
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
      const CUtensorMap* tm_w = is_k ? &tm_wk : &tm_wv;
      tma_prefetch_desc(&tm_c);
      tma_prefetch_desc(tm_w);
      mbar_arrive_expect_tx(w_full, S::kWBytes);
      for (int kc = 0; kc < KC; ++kc)
        tma_load_2d(sW + kc * S::kChunkBytesW, tm_w, w_full, kc * 64, col0);
      int issued = 0;
      for (int i = 0, r = g; r < p.n_row_tiles; ++i, r += G) {
        const int s = i & 1;
        if (i >= 2 && !mbar_wait(&c_empty[s], ((i >> 1) - 1) & 1, wc)) break;
        mbar_arrive_expect_tx(&c_full[s], S::kCBytes);
        // slots t*128 .. of batch element bb (rows past its last slot are
        // loaded but never stored)
        const int m0 = (r / p.tiles_per_b) * p.slots + (r % p.tiles_per_b) * kBM;
        for (int kc = 0; kc < KC; ++kc)
          tma_load_2d(sC + s * S::kCBytes + kc * S::kChunkBytesC, &tm_c, &c_full[s], kc * 64, m0);
        issued = i + 1;
      }
      if (*abort_flag) {  // let our own copies land before the CTA exits
        mbar_wait_drain(w_full, 0, p.status);
        for (int u = issued > 2 ? issued - 2 : 0; u < issued; ++u)
          mbar_wait_drain(&c_full[u & 1], (u >> 1) & 1, p.status);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(w_full, 0, wc);
      for (int i = 0, r = g; ok && r < p.n_row_tiles; ++i, r += G) {
        const int s = i & 1;
        if (!mbar_wait(&c_full[s], (i >> 1) & 1, wc) ||
            (i >= 2 && !mbar_wait(&acc_empty[s], ((i >> 1) - 1) & 1, wc))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t ca = smem_u32(sC + s * S::kCBytes);
        const uint32_t wa = smem_u32(sW);
#pragma unroll
        for (int kc = 0; kc < KC; ++kc)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_ss(tmem + s * BN, sdesc(ca + kc * S::kChunkBytesC + k * 32, 16, 1024, kSw128),
                    sdesc(wa + kc * S::kChunkBytesW + k * 32, 16, 1024, kSw128), S::kIdesc,
                    (kc | k) != 0 ? 1u : 0u);
        umma_commit(&c_empty[s]);
        umma_commit(&acc_full[s]);
      }
      umma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, p.status);  // every MMA of this CTA has completed
    }
    __syncwarp();
  } else {
    const int quarter = warp & 3;
    const int part = (warp - 2) >> 2;       // which share of the columns this warp reads
    const int rl = quarter * 32 + lane;     // slot row of the tile this thread reads
    const int et = part * kBM + rl;         // index among the epilogue threads
    const uint32_t t_row = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int seg = is_k ? p.dn : p.head_dim;
    const CUtensorMap* tm_out = is_k ? &tm_ko : &tm_vo;
    __nv_bfloat16* out = is_k ? p.k : p.v;
    const int boxes = n_valid / 32;  // staged 32-column boxes (n_valid is a multiple of 32)
    constexpr int kPhases = BN / 32 / kParts;  // boxes per epilogue warp: 2 (BN = 192) or 1
    // heads whose key rows start in this tile: offsets of their positional part
    int n_heads = 0;
    if (is_k && p.d_r > 0)
      for (int ch = 0; ch < n_valid / 8; ++ch)
        if ((col0 + ch * 8) % seg == 0) {
          if (et == 0)
            head_off[n_heads] =
                static_cast<long long>((col0 + ch * 8) / seg) * p.slots * p.head_dim + p.dn;
          ++n_heads;
        }
    const int kr_chunks = p.d_r / 8;  // 16-byte pieces of one positional key (<= 8)
    for (int i = 0, r = g; r < p.n_row_tiles; ++i, r += G) {
      const int s = i & 1;
      const int bb = r / p.tiles_per_b;
      const int sl0 = (r % p.tiles_per_b) * kBM;  // first slot of the tile
      // positional keys of this tile's slots: piece u = et + 384 k is piece
      // u % kr_chunks of row u / kr_chunks (coalesced), loaded ahead of use
      constexpr int kKr = (kBM * 8 + kEpiThreads - 1) / kEpiThreads;
      uint4 krv[kKr];
      if (n_heads > 0) {
#pragma unroll
        for (int k = 0; k < kKr; ++k) {
          const int u = et + kEpiThreads * k, row = u / kr_chunks;
          if (u < kBM * kr_chunks && sl0 + row < p.slots)
            krv[k] = __ldg(reinterpret_cast<const uint4*>(
                               p.kr + (static_cast<size_t>(bb) * p.slots + sl0 + row) * p.d_r) +
                           u % kr_chunks);
        }
      }
      const bool got = mbar_wait(&acc_full[s], (i >> 1) & 1, wc) && !*abort_flag;
      if (got) tc_fence_after();
      // row rl of box cb, 64-byte swizzle: 16-byte chunk j at j ^ ((rl >> 1) & 3)
      const uint32_t sw = static_cast<uint32_t>((rl >> 1) & 3);
      auto stage_box = [&](int cb) {
        uint32_t v[32];
        tmem_ld32(t_row + s * BN + cb * 32, v);
        tmem_wait_ld();
        uint8_t* brow = stage_out + cb * S::kBoxBytes + rl * 64;
#pragma unroll
        for (int j = 0; j < 4; ++j)
          *reinterpret_cast<uint4*>(brow + ((j ^ sw) << 4)) =
              make_uint4(pack_bf16x2(__uint_as_float(v[8 * j]), __uint_as_float(v[8 * j + 1])),
                         pack_bf16x2(__uint_as_float(v[8 * j + 2]), __uint_as_float(v[8 * j + 3])),
                         pack_bf16x2(__uint_as_float(v[8 * j + 4]), __uint_as_float(v[8 * j + 5])),
                         pack_bf16x2(__uint_as_float(v[8 * j + 6]), __uint_as_float(v[8 * j + 7])));
      };
      // one tensor store per box: columns col .. col + 31 are columns e .. e + 31
      // of head h, slots sl0 .. sl0 + 127 of batch element bb
      auto store_boxes = [&](int bx0, int bx1) {
        for (int bx = bx0; bx < bx1 && bx < boxes; ++bx) {
          const int col = col0 + bx * 32;
          tma_store_3d(tm_out, stage_out + bx * S::kBoxBytes, col % seg, sl0,
                       bb * p.heads + col / seg);
        }
        bulk_commit();
      };
      long long* rbase = row_base + (i & 1) * kBM;  // read by this tile's key copies
      if (part == 0)  // output offset of slot row rl (batch, head 0, slot), -1 past the last slot
        rbase[rl] = sl0 + rl < p.slots
                        ? (static_cast<long long>(bb) * p.heads * p.slots + sl0 + rl) * p.head_dim
                        : -1ll;
      if constexpr (kPhases == 1) {
        if (got) stage_box(part);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[s]);
        fence_proxy_async_smem();       // the staged boxes reach the TMA stores
        if (!epilogue_all(got)) break;  // staged tile complete, or every thread leaves
        if (et == 0) store_boxes(0, BN / 32);
      } else {
        // two phases over the boxes (each part's first box, then its second),
        // so that one phase's stores read shared memory while the other phase
        // is staged
        if (got) stage_box(part);
        fence_proxy_async_smem();
        if (et == 0) bulk_wait_read_all();  // the last tile's second-phase boxes are free
        if (!epilogue_all(got)) break;      // first-phase boxes staged
        if (et == 0) store_boxes(0, kParts);
        if (got) stage_box(part + kParts);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[s]);
        fence_proxy_async_smem();
        if (et == 0) bulk_wait_read_all();  // this tile's first-phase boxes are free again
        epilogue_sync();                    // second-phase boxes staged
        if (et == 0) store_boxes(kParts, 2 * kParts);
      }
      if (n_heads > 0) {
#pragma unroll
        for (int k = 0; k < kKr; ++k) {
          const int u = et + kEpiThreads * k, row = u / kr_chunks;
          if (u < kBM * kr_chunks && rbase[row] >= 0)
            for (int a = 0; a < n_heads; ++a)
              if (debug_in_range(rbase[row] + head_off[a] + 8 * (u % kr_chunks), 0,
                                 static_cast<long long>(p.M) * p.heads * p.head_dim - 7, p.status))
                *reinterpret_cast<uint4*>(out + rbase[row] + head_off[a] + 8 * (u % kr_chunks)) =
                    krv[k];
        }
      }
      if constexpr (kPhases == 1) {
        if (et == 0) bulk_wait_read_all();  // the stores have read the staged boxes
        epilogue_sync();                    // staging free for the next tile
      }
    }
    if (et == 0) bulk_wait_read_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, S::kTmemCols);
  }
}

template <int DC>
int launch_dec(const DecompressArgs& a) {
  using S = DecShape<DC>;
  const int dn = a.head_dim - a.d_r;
  const unsigned long long M = static_cast<unsigned long long>(a.batch) * a.slots;
  const int cols_k = a.heads * dn, cols_v = a.heads * a.head_dim;
  CUtensorMap tm_c, tm_wk, tm_wv, tm_ko, tm_vo;
  // outputs as [batch * heads][slots][head_dim], written in [128 x 32] boxes
  const unsigned long long HD = a.head_dim, SL = a.slots;
  if (!encode_map_2d_bf16(&tm_c, a.c, DC, M, DC * 2ull, 64, kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_wk, a.w_uk, DC, cols_k, DC * 2ull, 64, S::BN,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_2d_bf16(&tm_wv, a.w_uv, DC, cols_v, DC * 2ull, 64, S::BN,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_map_3d_bf16(&tm_ko, a.k, HD, SL, static_cast<unsigned long long>(a.batch) * a.heads,
                          HD * 2, SL * HD * 2, 32, kBM, CU_TENSOR_MAP_SWIZZLE_64B) ||
      !encode_map_3d_bf16(&tm_vo, a.v, HD, SL, static_cast<unsigned long long>(a.batch) * a.heads,
                          HD * 2, SL * HD * 2, 32, kBM, CU_TENSOR_MAP_SWIZZLE_64B))
    return MLA_ERR_CUDA;
  auto kern = mla_decompress_tc_kernel<DC>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmemBytes);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  DecKParams kp;
  kp.kr = static_cast<const __nv_bfloat16*>(a.kr);
  kp.k = static_cast<__nv_bfloat16*>(a.k);
  kp.v = static_cast<__nv_bfloat16*>(a.v);
  kp.M = static_cast<int>(M);
  kp.tiles_per_b = (a.slots + kBM - 1) / kBM;  // a tile never spans two batch elements
  kp.n_row_tiles = kp.tiles_per_b * a.batch;
  kp.tiles_k = (cols_k + S::BN - 1) / S::BN;
  kp.cols_k = cols_k;
  kp.cols_v = cols_v;
  kp.dn = dn;
  kp.head_dim = a.head_dim;
  kp.d_r = a.d_r;
  kp.slots = a.slots;
  kp.heads = a.heads;
  kp.status = a.status;
  const int n_col = kp.tiles_k + (cols_v + S::BN - 1) / S::BN;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // one CTA per SM: as many row groups per column tile as whole waves allow
  int groups = sms / n_col;
  if (groups < 1) groups = 1;
  if (groups > kp.n_row_tiles) groups = kp.n_row_tiles;
  kern<<<dim3(n_col, groups), kThreads, S::kSmemBytes, a.stream>>>(tm_c, tm_wk, tm_wv, tm_ko,
                                                                     tm_vo, kp);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace

int launch_decompress(const DecompressArgs& a) {
  const int dn = a.head_dim - a.d_r;
  // whole 32-column output boxes, none spanning two heads
  if (dn <= 0 || dn % 32 != 0 || a.head_dim % 32 != 0 || a.d_r % 8 != 0)
    return MLA_ERR_UNSUPPORTED;
  if (static_cast<long long>(a.batch) * a.slots >= (1ll << 31)) return MLA_ERR_UNSUPPORTED;
  switch (a.d_c) {
    case 64: return launch_dec<64>(a);
    case 128: return launch_dec<128>(a);
    case 192: return launch_dec<192>(a);
    case 256: return launch_dec<256>(a);
    default: return MLA_ERR_UNSUPPORTED;
  }
}

}  // namespace vmla
