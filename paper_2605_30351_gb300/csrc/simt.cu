// Plain SIMT kernels for the same two calls: no tensor cores, no TMA, fp32
// arithmetic throughout. They are the debug reference on the device (selected
// with MLA_FLAG_SIMT) and cover shapes the tcgen05 kernels do not (d_c or d_r
// outside {64, 128, 192, 256, 512} x {32, 64}).
// Same equations as the tensor-core path: Eq. (ckv), App. D.2 RMSNorm,
// Eq. (krope), App. D.4 ring slot; Eq. (score) and App. E latent output.
#include <cmath>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

constexpr int kMaxDK = 640;  // d_c + d_r held per warp in shared memory
constexpr int kMaxDC = 512;

// One block per token: thread n computes output column n of [W_dkv ; W_kr] x.
__global__ void append_simt_kernel(const __nv_bfloat16* __restrict__ x,
                                   const __nv_bfloat16* __restrict__ w_dkv,
                                   const __nv_bfloat16* __restrict__ gamma,
                                   const __nv_bfloat16* __restrict__ w_kr,
                                   const int* __restrict__ pos, const float2* __restrict__ rope,
                                   __nv_bfloat16* c, __nv_bfloat16* kr, int n_tok, int hidden,
                                   int d_c, int d_r, int slots, int T, int W, int S,
                                   long long first_frame, int rope_len, int pairs_t, int pairs_h,
                                   int use_rmsnorm, int rotate, float eps, int* status) {
  extern __shared__ float sh[];  // hidden floats of x, then d_c + d_r outputs
  float* xs = sh;
  float* ys = sh + hidden;
  __shared__ float red[32];
  const int n = blockIdx.x, b = blockIdx.y;
  const __nv_bfloat16* xr = x + (static_cast<size_t>(b) * n_tok + n) * hidden;
  for (int i = threadIdx.x; i < hidden; i += blockDim.x) xs[i] = __bfloat162float(xr[i]);
  __syncthreads();
  const int N = d_c + d_r;
  for (int col = threadIdx.x; col < N; col += blockDim.x) {
    const __nv_bfloat16* wr = col < d_c ? w_dkv + static_cast<size_t>(col) * hidden
                                        : w_kr + static_cast<size_t>(col - d_c) * hidden;
    float acc = 0.f;
    for (int i = 0; i < hidden; ++i) acc = fmaf(xs[i], __bfloat162float(wr[i]), acc);
    ys[col] = acc;
  }
  __syncthreads();
  // mean square over the d_c columns
  float part = 0.f;
  for (int col = threadIdx.x; col < d_c; col += blockDim.x) part = fmaf(ys[col], ys[col], part);
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = use_rmsnorm ? rsqrtf(red[0] / d_c + eps) : 1.f;
  const long long f = first_frame + n / T;
  const long long slot = frame_base_slot(f, T, W, S) + n % T;
  if (!debug_in_range(slot, 0, slots, status)) return;
  __nv_bfloat16* cd = c + (static_cast<size_t>(b) * slots + slot) * d_c;
  for (int col = threadIdx.x; col < d_c; col += blockDim.x) {
    const float g = gamma ? __bfloat162float(gamma[col]) : 1.f;
    cd[col] = __float2bfloat16_rn(ys[col] * inv * g);
  }
  __nv_bfloat16* kd = kr + (static_cast<size_t>(b) * slots + slot) * d_r;
  if (!rotate) {  // the paper's storage: k^R = W_kr x, rotated when the window is assembled
    for (int col = threadIdx.x; col < d_r; col += blockDim.x)
      kd[col] = __float2bfloat16_rn(ys[d_c + col]);
    return;
  }
  const int* pp = pos + (static_cast<size_t>(b) * n_tok + n) * 3;
  int pa[3] = {pp[0], pp[1], pp[2]};
  for (int a = 0; a < 3; ++a)
    if (pa[a] < 0 || pa[a] >= rope_len) {
      if (threadIdx.x == 0) record_status(status, MLA_ERR_RANGE);
      pa[a] = 0;
    }
  for (int pr = threadIdx.x; pr < d_r / 2; pr += blockDim.x) {
    const int ps = pr < pairs_t ? pa[0] : (pr < pairs_t + pairs_h ? pa[1] : pa[2]);
    const float2 cs = rope[static_cast<size_t>(ps) * (d_r / 2) + pr];
    const float x0 = ys[d_c + 2 * pr], x1 = ys[d_c + 2 * pr + 1];
    kd[2 * pr] = __float2bfloat16_rn(x0 * cs.x - x1 * cs.y);
    kd[2 * pr + 1] = __float2bfloat16_rn(x0 * cs.y + x1 * cs.x);
  }
}

// One warp per (token, head) row; online softmax over every valid slot.
__global__ void attn_simt_kernel(const __nv_bfloat16* __restrict__ q_c,
                                 const __nv_bfloat16* __restrict__ q_r,
                                 const int* __restrict__ q_pos, const float2* __restrict__ rope,
                                 const __nv_bfloat16* __restrict__ c,
                                 const __nv_bfloat16* __restrict__ kr, __nv_bfloat16* o, int rows,
                                 int heads, int slots, int n_valid, int d_c, int d_r, int rope_len,
                                 int pairs_t, int pairs_h, float scale_log2, int* status) {
  __shared__ float qs[4][kMaxDK];
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * 4 + wid, b = blockIdx.y;
  if (row >= rows) return;
  float* q = qs[wid];
  const __nv_bfloat16* qc = q_c + (static_cast<size_t>(b) * rows + row) * d_c;
  for (int i = lane; i < d_c; i += 32) q[i] = __bfloat162float(qc[i]);
  const int* pp = q_pos + (static_cast<size_t>(b) * (rows / heads) + row / heads) * 3;
  int pa[3] = {pp[0], pp[1], pp[2]};
  for (int a = 0; a < 3; ++a)
    if (pa[a] < 0 || pa[a] >= rope_len) {
      if (lane == 0) record_status(status, MLA_ERR_RANGE);
      pa[a] = 0;
    }
  const __nv_bfloat16* qr = q_r + (static_cast<size_t>(b) * rows + row) * d_r;
  for (int pr = lane; pr < d_r / 2; pr += 32) {
    const int ps = pr < pairs_t ? pa[0] : (pr < pairs_t + pairs_h ? pa[1] : pa[2]);
    const float2 cs = rope[static_cast<size_t>(ps) * (d_r / 2) + pr];
    const float x0 = __bfloat162float(qr[2 * pr]), x1 = __bfloat162float(qr[2 * pr + 1]);
    // same bf16 rounding of the rotated query as the tensor-core path
    q[d_c + 2 * pr] = __bfloat162float(__float2bfloat16_rn(x0 * cs.x - x1 * cs.y));
    q[d_c + 2 * pr + 1] = __bfloat162float(__float2bfloat16_rn(x0 * cs.y + x1 * cs.x));
  }
  __syncwarp();
  float acc[kMaxDC / 32];
  for (int i = 0; i < kMaxDC / 32; ++i) acc[i] = 0.f;
  float m = -INFINITY, l = 0.f;
  const __nv_bfloat16* cb = c + static_cast<size_t>(b) * slots * d_c;
  const __nv_bfloat16* kb = kr + static_cast<size_t>(b) * slots * d_r;
  for (int j = 0; j < n_valid; ++j) {
    const __nv_bfloat16* cj = cb + static_cast<size_t>(j) * d_c;
    const __nv_bfloat16* kj = kb + static_cast<size_t>(j) * d_r;
    float part = 0.f;
    for (int i = lane; i < d_c; i += 32) part = fmaf(q[i], __bfloat162float(cj[i]), part);
    for (int i = lane; i < d_r; i += 32) part = fmaf(q[d_c + i], __bfloat162float(kj[i]), part);
    for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
    const float s = part * scale_log2;
    const float m_new = fmaxf(m, s);
    const float alpha = exp2f(m - m_new);
    const float pj = exp2f(s - m_new);
    l = l * alpha + pj;
    m = m_new;
    for (int i = 0; i < kMaxDC / 32; ++i) {
      const int d = lane + 32 * i;
      if (d < d_c) acc[i] = acc[i] * alpha + pj * __bfloat162float(cj[d]);
    }
  }
  __nv_bfloat16* od = o + (static_cast<size_t>(b) * rows + row) * d_c;
  for (int i = 0; i < kMaxDC / 32; ++i) {
    const int d = lane + 32 * i;
    if (d < d_c) od[d] = __float2bfloat16_rn(acc[i] / l);
  }
}

}  // namespace

int launch_append_simt(const AppendArgs& a) {
  if (a.d_c + a.d_r > 1024) return MLA_ERR_UNSUPPORTED;
  const size_t smem = static_cast<size_t>(a.hidden + a.d_c + a.d_r) * sizeof(float);
  if (smem > 200 * 1024) return MLA_ERR_UNSUPPORTED;
  cudaError_t e = cudaFuncSetAttribute(append_simt_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  const dim3 grid(a.n_tok, a.batch);
  append_simt_kernel<<<grid, 256, smem, a.stream>>>(
      static_cast<const __nv_bfloat16*>(a.x), static_cast<const __nv_bfloat16*>(a.w_dkv),
      static_cast<const __nv_bfloat16*>(a.gamma), static_cast<const __nv_bfloat16*>(a.w_kr),
      a.pos, reinterpret_cast<const float2*>(a.rope), static_cast<__nv_bfloat16*>(a.c),
      static_cast<__nv_bfloat16*>(a.kr), a.n_tok, a.hidden, a.d_c, a.d_r, a.slots,
      a.tokens_per_frame, a.window_frames, a.sink_frames, a.first_frame, a.rope_len, a.pairs_t,
      a.pairs_h, a.use_rmsnorm, a.rotate, a.eps, a.status);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

int launch_attention_simt(const AttnArgs& a) {
  if (a.d_c > kMaxDC || a.d_c + a.d_r > kMaxDK) return MLA_ERR_UNSUPPORTED;
  const dim3 grid((a.rows + 3) / 4, a.batch);
  attn_simt_kernel<<<grid, 128, 0, a.stream>>>(
      static_cast<const __nv_bfloat16*>(a.q_c), static_cast<const __nv_bfloat16*>(a.q_r),
      a.q_pos, reinterpret_cast<const float2*>(a.rope), static_cast<const __nv_bfloat16*>(a.c),
      static_cast<const __nv_bfloat16*>(a.kr), static_cast<__nv_bfloat16*>(a.o), a.rows, a.heads,
      a.slots, a.n_valid, a.d_c, a.d_r, a.rope_len, a.pairs_t, a.pairs_h, a.scale_log2,
      a.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace vmla
