// Window assembly for caches that keep k^R unrotated (App. D.4, D.5).
//
// The long-rollout cache holds S sink frames for good and the newest W - S
// frames in FIFO order. When a chunk attends, the held frames are numbered
// 0, 1, ... in temporal order (sinks first); that number is the temporal
// coordinate of every key of the frame and of the queries of that frame,
// with (h, w) unchanged. This kernel writes the rotated keys of every valid
// slot and the queries' local positions into caller workspace; the
// absorbed-form attention kernel then runs on them unchanged.
//
// One thread per (batch, slot, four complex pairs) reads 16 bytes of k^R and
// writes 16 bytes of RoPE3D(k^R), coalesced along the key; each block first
// tabulates the local time of every frame slot in shared memory. The tail of
// the index range handles one query token each.
#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kThreads = 256;

// Local number of absolute frame f in a window that received fw frames, -1
// if the window does not hold f.
__device__ __forceinline__ long long local_time(long long f, long long fw, int W, int S) {
  if (f < 0 || f >= fw) return -1;
  if (fw <= W || f < S) return f;
  const long long first_local = fw - (W - S);
  return f >= first_local ? S + (f - first_local) : -1;
}

// Newest frame stored in frame slot j (0 <= j < W), -1 if none yet.
__device__ __forceinline__ long long frame_in_slot(int j, long long fw, int W, int S) {
  if (j < S) return j < fw ? j : -1;
  const long long r = j - S, L = W - S, newest = fw - 1 - S;
  if (newest < r) return -1;
  return S + r + L * ((newest - r) / L);
}

__device__ __forceinline__ int checked(int v, int len, int* status) {
  if (v < 0 || v >= len) {
    record_status(status, MLA_ERR_RANGE);
    return 0;
  }
  return v;
}

constexpr int kMaxFrames = 1024;  // window frames whose local times a block tabulates

__global__ void __launch_bounds__(kThreads)
    window_assemble_kernel(const uint4* __restrict__ kr, const int* __restrict__ q_pos,
                           const int2* __restrict__ frame_hw, const float2* __restrict__ rope,
                           uint4* __restrict__ kr_rot, int* __restrict__ q_local, int batch,
                           int nq, int slots, int n_valid, int T, int W, int S, int pairs,
                           long long fw, int rope_len, int pairs_t, int pairs_h, int* status) {
  grid_dep_sync();
  // local time of the frame held in each frame slot (-1: none), once per block
  __shared__ int t_of_slot[kMaxFrames];
  for (int j = threadIdx.x; j < W && j < kMaxFrames; j += kThreads)
    t_of_slot[j] = static_cast<int>(local_time(frame_in_slot(j, fw, W, S), fw, W, S));
  __syncthreads();
  const int J = pairs / 4;  // 16-byte pieces (four complex pairs) per key
  const long long n_key = static_cast<long long>(batch) * n_valid * J;
  const long long n_all = n_key + static_cast<long long>(batch) * nq;
  for (long long i = blockIdx.x * static_cast<long long>(kThreads) + threadIdx.x; i < n_all;
       i += static_cast<long long>(gridDim.x) * kThreads) {
    if (i < n_key) {
      const int c = static_cast<int>(i % J);
      const long long bs = i / J;
      const int s = static_cast<int>(bs % n_valid);
      const int b = static_cast<int>(bs / n_valid);
      const int fslot = s / T, k = s - fslot * T;
      if (!debug_in_range(fslot, 0, W, status)) continue;
      long long t = fslot < kMaxFrames ? t_of_slot[fslot]
                                       : local_time(frame_in_slot(fslot, fw, W, S), fw, W, S);
      if (t < 0) {  // a valid slot always holds a held frame; guard regardless
        record_status(status, MLA_ERR_RANGE);
        t = 0;
      }
      const int ct = checked(static_cast<int>(t), rope_len, status);
      const int2 hw = __ldg(frame_hw + k);
      const int ch = checked(hw.x, rope_len, status), cw = checked(hw.y, rope_len, status);
      const size_t off = (static_cast<size_t>(b) * slots + s) * J + c;
      const uint4 v = __ldg(kr + off);
      const uint32_t in[4] = {v.x, v.y, v.z, v.w};
      uint32_t out[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int pr = 4 * c + q;
        const int coord = pr < pairs_t ? ct : (pr < pairs_t + pairs_h ? ch : cw);
        const float2 cs = __ldg(rope + static_cast<size_t>(coord) * pairs + pr);
        const float x0 = bf16_lo(in[q]), x1 = bf16_hi(in[q]);
        out[q] = pack_bf16x2(x0 * cs.x - x1 * cs.y, x0 * cs.y + x1 * cs.x);
      }
      kr_rot[off] = make_uint4(out[0], out[1], out[2], out[3]);
    } else {
      const long long qi = i - n_key;  // (b, n) flattened
      const int* src = q_pos + qi * 3;
      long long t = local_time(__ldg(src), fw, W, S);
      if (t < 0) {  // the query's frame is not in the window
        record_status(status, MLA_ERR_RANGE);
        t = 0;
      }
      int* dst = q_local + qi * 3;
      dst[0] = static_cast<int>(t);
      dst[1] = __ldg(src + 1);
      dst[2] = __ldg(src + 2);
    }
  }
}

}  // namespace

int launch_window_assemble(const WindowArgs& a) {
  const int pairs = a.d_r / 2;
  if (pairs % 4 != 0) return MLA_ERR_UNSUPPORTED;  // d_r is a multiple of 8 by the config rules
  const long long n_all = static_cast<long long>(a.batch) * a.n_valid * (pairs / 4) +
                          static_cast<long long>(a.batch) * a.nq;
  if (n_all <= 0) return MLA_OK;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long want = (n_all + kThreads - 1) / kThreads;
  const int blocks = static_cast<int>(want < 8ll * sms ? want : 8ll * sms);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(blocks, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_sync
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(
      &cfg, window_assemble_kernel, static_cast<const uint4*>(a.kr), a.q_pos,
      reinterpret_cast<const int2*>(a.frame_hw), reinterpret_cast<const float2*>(a.rope),
      static_cast<uint4*>(a.kr_rot), a.q_pos_local, a.batch, a.nq, a.slots, a.n_valid, a.T, a.W,
      a.S, pairs, a.frames_written, a.rope_len, a.pairs_t, a.pairs_h, a.status);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace vmla
