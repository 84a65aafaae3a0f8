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
// One thread per (batch, slot, complex pair) reads one bf16x2 of k^R and
// writes one bf16x2 of RoPE3D(k^R): 4 bytes in and out, coalesced along the
// pair index. The tail of the index range handles one query token each.
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

__global__ void __launch_bounds__(kThreads)
    window_assemble_kernel(const uint32_t* __restrict__ kr, const int* __restrict__ q_pos,
                           const int* __restrict__ frame_hw, const float2* __restrict__ rope,
                           uint32_t* __restrict__ kr_rot, int* __restrict__ q_local, int batch,
                           int nq, int slots, int n_valid, int T, int W, int S, int pairs,
                           long long fw, int rope_len, int pairs_t, int pairs_h, int* status) {
  const long long n_key = static_cast<long long>(batch) * n_valid * pairs;
  const long long n_all = n_key + static_cast<long long>(batch) * nq;
  for (long long i = blockIdx.x * static_cast<long long>(kThreads) + threadIdx.x; i < n_all;
       i += static_cast<long long>(gridDim.x) * kThreads) {
    if (i < n_key) {
      const int pr = static_cast<int>(i % pairs);
      const long long bs = i / pairs;
      const int s = static_cast<int>(bs % n_valid);
      const int b = static_cast<int>(bs / n_valid);
      const int k = s % T;
      long long t = local_time(frame_in_slot(s / T, fw, W, S), fw, W, S);
      if (t < 0) {  // a valid slot always holds a held frame; guard regardless
        record_status(status, MLA_ERR_RANGE);
        t = 0;
      }
      int coord;
      if (pr < pairs_t)
        coord = checked(static_cast<int>(t), rope_len, status);
      else
        coord = checked(__ldg(frame_hw + 2 * k + (pr < pairs_t + pairs_h ? 0 : 1)), rope_len,
                        status);
      const float2 cs = __ldg(rope + static_cast<size_t>(coord) * pairs + pr);
      const size_t off = (static_cast<size_t>(b) * slots + s) * pairs + pr;
      const uint32_t v = __ldg(kr + off);
      const float x0 = bf16_lo(v), x1 = bf16_hi(v);
      kr_rot[off] = pack_bf16x2(x0 * cs.x - x1 * cs.y, x0 * cs.y + x1 * cs.x);
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
  const long long n_all =
      static_cast<long long>(a.batch) * a.n_valid * pairs + static_cast<long long>(a.batch) * a.nq;
  if (n_all <= 0) return MLA_OK;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long want = (n_all + kThreads - 1) / kThreads;
  const int blocks = static_cast<int>(want < 8ll * sms ? want : 8ll * sms);
  window_assemble_kernel<<<blocks, kThreads, 0, a.stream>>>(
      static_cast<const uint32_t*>(a.kr), a.q_pos, a.frame_hw,
      reinterpret_cast<const float2*>(a.rope), static_cast<uint32_t*>(a.kr_rot), a.q_pos_local,
      a.batch, a.nq, a.slots, a.n_valid, a.T, a.W, a.S, pairs, a.frames_written, a.rope_len,
      a.pairs_t, a.pairs_h, a.status);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace vmla
