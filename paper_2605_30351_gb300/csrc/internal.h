// Host-side interface between the C ABI (api.cu) and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "videomla.h"

namespace vmla {

// Column-tile width of the query prologue's first GEMM, which also sets how
// many partial sums of squares per row the workspace holds (ceil(d_q / it)).
constexpr int kQuerySqTile = 192;

// First slot of latent frame f: sink frames (f < S) keep slot f*T for good,
// later frames share the W - S remaining frame slots in FIFO order
// (App. D.4). With S = 0 this is the ring (f mod W)*T.
__host__ __device__ inline long long frame_base_slot(long long f, int T, int W, int S) {
  return (f < S ? f : S + (f - S) % (W - S)) * static_cast<long long>(T);
}

// One attention launch: every (token, head) row of the chunk against the
// valid slots of its batch element's window.
struct AttnArgs {
  const void* q_c;      // bf16 [B][rows][d_c]   rows = Nq * heads
  const void* q_r;      // bf16 [B][rows][d_r]
  const int* q_pos;     // int32 [B][Nq][3]
  const float* rope;    // fp32 [L][d_r/2][2]
  const void* c;        // bf16 [B][slots][d_c]
  const void* kr;       // bf16 [B][slots][d_r]
  void* o;              // bf16 [B][rows][d_c]
  int batch, rows, heads, slots, n_valid;
  int d_c, d_r, rope_len, pairs_t, pairs_h;
  float scale_log2;     // log2(e) / sqrt(head_dim)
  int* status;          // device status word
  cudaStream_t stream;
};

// One append launch: n_tok tokens per batch element into their ring slots.
struct AppendArgs {
  const void* x;        // bf16 [B][n_tok][hidden]
  const void* w_dkv;    // bf16 [d_c][hidden]
  const void* gamma;    // bf16 [d_c] or nullptr
  const void* w_kr;     // bf16 [d_r][hidden]
  const int* pos;       // int32 [B][n_tok][3]
  const float* rope;    // fp32 [L][d_r/2][2]
  void* c;              // bf16 [B][slots][d_c]
  void* kr;             // bf16 [B][slots][d_r]
  int batch, n_tok, hidden, d_c, d_r, slots;
  int tokens_per_frame, window_frames, sink_frames;
  long long first_frame;
  int rope_len, pairs_t, pairs_h;
  int use_rmsnorm;
  int rotate;           // 0: store W_kr x unrotated (pos is not read)
  float eps;
  int* status;
  cudaStream_t stream;
};

// Load-time absorption of the per-head up-projections (App. E).
struct AbsorbArgs {
  const void* w_uq;     // bf16 [H][d_nope][d_q]
  const void* w_uk;     // bf16 [H][d_nope][d_c]
  const void* w_qr;     // bf16 [H][d_r][d_q]
  const void* gamma_q;  // bf16 [d_q] or nullptr
  const void* w_uv;     // bf16 [H][d_h][d_c]
  const void* w_o;      // bf16 [hidden][H*d_h]
  void* w_qcat;         // bf16 [H*(d_c+d_r)][d_q]
  void* w_b;            // bf16 [hidden][H*d_c]
  int hidden, heads, head_dim, d_c, d_r, d_q;
  cudaStream_t stream;
};

// Query prologue: x -> c~ (+ row statistics) -> [q_c | q_r].
struct QueryArgs {
  const void* x;        // bf16 [rows][hidden]
  const void* w_dq;     // bf16 [d_q][hidden]
  const void* w_qcat;   // bf16 [H*(d_c+d_r)][d_q]
  void* c_tilde;        // workspace bf16 [rows][d_q]
  float* sq;            // workspace fp32 [ceil(d_q/256)][rows]
  void* q_c;            // bf16 [rows][H*d_c]
  void* q_r;            // bf16 [rows][H*d_r]
  int rows, hidden, heads, d_c, d_r, d_q;
  float eps;
  int* status;
  cudaStream_t stream;
};

// Output projection y = o_lat W_B^T.
struct OutProjArgs {
  const void* o_lat;    // bf16 [rows][H*d_c]
  const void* w_b;      // bf16 [hidden][H*d_c]
  void* y;              // bf16 [rows][hidden]
  int rows, hidden, heads, d_c;
  int* status;
  cudaStream_t stream;
};

// Dense per-head attention (the baseline cache layout).
struct DenseArgs {
  const void* q;        // bf16 [B][nq][H][head_dim]
  const void* k;        // bf16 [B][H][slots][head_dim]
  const void* v;        // bf16 [B][H][slots][head_dim]
  void* o;              // bf16 [B][nq][H][head_dim]
  int batch, nq, heads, head_dim, slots, n_valid;
  float scale_log2;
  int* status;
  cudaStream_t stream;
};

// Window assembly for rotate-at-use caches (App. D.5): rotated keys of the
// valid slots at window-local times, and local query positions.
struct WindowArgs {
  const void* kr;       // bf16 [B][slots][d_r] unrotated k^R
  const int* q_pos;     // int32 [B][nq][3] absolute (t, h, w)
  const int* frame_hw;  // int32 [T][2]
  const float* rope;    // fp32 [L][d_r/2][2]
  void* kr_rot;         // out bf16 [B][slots][d_r] (first n_valid slots written)
  int* q_pos_local;     // out int32 [B][nq][3]
  int batch, nq, slots, n_valid, T, W, S, d_r;
  long long frames_written;
  int rope_len, pairs_t, pairs_h;
  int* status;
  cudaStream_t stream;
};

// Decompression of the latent cache into per-head keys and values.
struct DecompressArgs {
  const void* c;        // bf16 [B][slots][d_c]
  const void* kr;       // bf16 [B][slots][d_r] rotated positional keys
  const void* w_uk;     // bf16 [H][head_dim - d_r][d_c]
  const void* w_uv;     // bf16 [H][head_dim][d_c]
  void* k;              // out bf16 [B][H][slots][head_dim]
  void* v;              // out bf16 [B][H][slots][head_dim]
  int batch, slots, heads, head_dim, d_c, d_r;
  int* status;
  cudaStream_t stream;
};

// Each launcher returns MLA_OK, MLA_ERR_UNSUPPORTED or MLA_ERR_CUDA.
int launch_attention_tc(const AttnArgs& a);
int launch_attention_simt(const AttnArgs& a);
int launch_append_tc(const AppendArgs& a);
int launch_append_simt(const AppendArgs& a);
int launch_absorb(const AbsorbArgs& a);
int launch_query_prologue(const QueryArgs& a);
int launch_output_projection(const OutProjArgs& a);
int launch_dense_attention_tc(const DenseArgs& a);
int launch_window_assemble(const WindowArgs& a);
int launch_decompress(const DecompressArgs& a);
int launch_wait_selftest(unsigned long long limit_ns, int* status, cudaStream_t stream);
// Device address of the fixed no-allocation scratch on the current device.
int query_scratch_address(void** out);

// Shared by the launchers: cuTensorMapEncodeTiled fetched from the driver.
// Encodes a rank-3 bf16 tiled map over [d2][d1][d0] (d0 contiguous) with
// strides in bytes for dims 1 and 2 and a box of (b0, b1, 1).
bool encode_map_3d_bf16(CUtensorMap* map, const void* base, unsigned long long d0,
                        unsigned long long d1, unsigned long long d2,
                        unsigned long long stride1_bytes, unsigned long long stride2_bytes,
                        unsigned b0, unsigned b1, CUtensorMapSwizzle swizzle);
bool encode_map_2d_bf16(CUtensorMap* map, const void* base, unsigned long long d0,
                        unsigned long long d1, unsigned long long stride1_bytes, unsigned b0,
                        unsigned b1, CUtensorMapSwizzle swizzle);

void set_last_cuda_error(cudaError_t e);

}  // namespace vmla
