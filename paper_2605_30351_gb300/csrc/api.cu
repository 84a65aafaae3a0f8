// C ABI of libvideomla.so: argument checks, the RoPE table, tensor-map
// encoding and dispatch to the kernels. See include/videomla.h.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <initializer_list>
#include <mutex>

#include <cudaTypedefs.h>

#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

// The device status area every kernel receives as `int* status`: the status
// word, a pad, then a 64-bit counter that only debug builds advance (rows of
// the online softmax that rescaled their output; see debug_count_rescale).
struct alignas(8) DeviceStatusArea {
  int status;
  int pad;
  unsigned long long rescales;
};
__device__ DeviceStatusArea g_device_status = {MLA_OK, 0, 0ull};

thread_local int t_last_cuda_error = 0;

constexpr int kMaxDevices = 64;
int* g_status_ptr[kMaxDevices] = {nullptr};
std::mutex g_mu;

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

// Device address of the status word on the current device, looked up once per
// device (the address stays valid until the device's primary context is torn
// down, e.g. by cudaDeviceReset, which the library does not survive). On
// failure returns nullptr with the CUDA error recorded.
int* device_status_ptr() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    t_last_cuda_error = static_cast<int>(e);
    return nullptr;
  }
  if (dev < 0 || dev >= kMaxDevices) {
    t_last_cuda_error = static_cast<int>(cudaErrorInvalidDevice);
    return nullptr;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_device_status);
    if (e != cudaSuccess || !p) {
      t_last_cuda_error = static_cast<int>(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
      return nullptr;
    }
    g_status_ptr[dev] = static_cast<int*>(p);
  }
  return g_status_ptr[dev];
}

// Every buffer handed to a kernel (tensor-map sources included) must be
// device memory of the current device: the kernels' TMA copies, and the
// multicast among the CTAs of a cluster, address this GPU's own memory only.
// Host memory (pageable or pinned), managed memory and another GPU's memory
// are refused with MLA_ERR_ARG before anything is enqueued; null entries
// (optional arguments) are skipped.
int check_resident(std::initializer_list<const void*> ptrs) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    t_last_cuda_error = static_cast<int>(e);
    return MLA_ERR_CUDA;
  }
  for (const void* p : ptrs) {
    if (!p) continue;
    cudaPointerAttributes at{};
    e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) {
      (void)cudaGetLastError();  // not a pointer the runtime knows: clear the sticky error
      return MLA_ERR_ARG;
    }
    if (at.type != cudaMemoryTypeDevice || at.device != dev) return MLA_ERR_ARG;
  }
  return MLA_OK;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  return g_encode;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int pairs_total(const mla_config& c) { return c.rope_pairs_t + c.rope_pairs_h + c.rope_pairs_w; }

int axis_dim(const mla_config& c, int a) {
  const int d = a == 0 ? c.rope_dim_t : (a == 1 ? c.rope_dim_h : c.rope_dim_w);
  const int n = a == 0 ? c.rope_pairs_t : (a == 1 ? c.rope_pairs_h : c.rope_pairs_w);
  return d > 0 ? d : 2 * n;
}

int check_config(const mla_config* c) {
  if (!c) return MLA_ERR_ARG;
  if (c->hidden <= 0 || c->heads <= 0 || c->head_dim <= 0 || c->d_c <= 0 || c->d_r <= 0 ||
      c->tokens_per_frame <= 0 || c->window_frames <= 0 || c->batch <= 0 ||
      c->rope_table_len <= 0 || !(c->rope_theta > 0.0) || !(c->rms_eps >= 0.f))
    return MLA_ERR_ARG;
  if (c->rope_pairs_t < 0 || c->rope_pairs_h < 0 || c->rope_pairs_w < 0) return MLA_ERR_ARG;
  if (2 * pairs_total(*c) != c->d_r) return MLA_ERR_ARG;
  for (int a = 0; a < 3; ++a) {
    const int n = a == 0 ? c->rope_pairs_t : (a == 1 ? c->rope_pairs_h : c->rope_pairs_w);
    if (n > 0 && axis_dim(*c, a) < 2 * n) return MLA_ERR_ARG;
  }
  // every row must be a whole number of 16-byte chunks (vector stores, TMA strides)
  if (c->d_c % 8 != 0 || c->d_r % 8 != 0 || c->hidden % 8 != 0) return MLA_ERR_ARG;
  const long long slots = static_cast<long long>(c->tokens_per_frame) * c->window_frames;
  if (slots > (1ll << 30)) return MLA_ERR_ARG;
  if (c->sink_frames < 0 || c->sink_frames >= c->window_frames) return MLA_ERR_ARG;
  return MLA_OK;
}

int fail_cuda(cudaError_t e);

// Valid slots: the first min(frames_written, W) frame slots (contiguous from
// 0 before the first eviction, all slots after).
long long valid_slots(const mla_cache& cache) {
  const mla_config& c = cache.cfg;
  const long long held = cache.frames_written < c.window_frames ? cache.frames_written
                                                                 : c.window_frames;
  return held * c.tokens_per_frame;
}

bool rotate_at_use(const mla_config& c) { return (c.flags & MLA_FLAG_ROTATE_AT_USE) != 0; }

// Absorbed-form attention over the valid slots, with the given positional
// keys and query positions.
int run_attention(const mla_cache* cache, const void* q_c, const void* q_r, const int* q_pos,
                  int Nq, const void* kr, void* o_lat, cudaStream_t stream) {
  const mla_config& c = cache->cfg;
  const long long n_valid = valid_slots(*cache);
  if (n_valid < 1) return MLA_ERR_ARG;
  const long long rows = static_cast<long long>(Nq) * c.heads;
  if (rows > (1ll << 30)) return MLA_ERR_ARG;
  AttnArgs a;
  a.q_c = q_c;
  a.q_r = q_r;
  a.q_pos = q_pos;
  a.rope = static_cast<const float*>(cache->rope_table);
  a.c = cache->c;
  a.kr = kr;
  a.o = o_lat;
  a.batch = c.batch;
  a.rows = static_cast<int>(rows);
  a.heads = c.heads;
  a.slots = c.tokens_per_frame * c.window_frames;
  a.n_valid = static_cast<int>(n_valid);
  a.d_c = c.d_c;
  a.d_r = c.d_r;
  a.rope_len = c.rope_table_len;
  a.pairs_t = c.rope_pairs_t;
  a.pairs_h = c.rope_pairs_h;
  a.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c.head_dim)));
  a.status = device_status_ptr();
  a.stream = stream;
  if (!a.status) return MLA_ERR_CUDA;
  return (c.flags & MLA_FLAG_SIMT) ? launch_attention_simt(a) : launch_attention_tc(a);
}

unsigned long long round256(unsigned long long v) { return (v + 255) / 256 * 256; }

unsigned long long window_kr_bytes(const mla_config& c) {
  return round256(static_cast<unsigned long long>(c.batch) * c.tokens_per_frame *
                  c.window_frames * c.d_r * 2);
}

int fail_cuda(cudaError_t e) {
  t_last_cuda_error = static_cast<int>(e);
  return MLA_ERR_CUDA;
}

}  // namespace

void set_last_cuda_error(cudaError_t e) { t_last_cuda_error = static_cast<int>(e); }

bool encode_map_3d_bf16(CUtensorMap* map, const void* base, unsigned long long d0,
                        unsigned long long d1, unsigned long long d2,
                        unsigned long long stride1_bytes, unsigned long long stride2_bytes,
                        unsigned b0, unsigned b1, CUtensorMapSwizzle swizzle) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {b0, b1, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_map_2d_bf16(CUtensorMap* map, const void* base, unsigned long long d0,
                        unsigned long long d1, unsigned long long stride1_bytes, unsigned b0,
                        unsigned b1, CUtensorMapSwizzle swizzle) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {d0, d1};
  const cuuint64_t strides[1] = {stride1_bytes};
  const cuuint32_t box[2] = {b0, b1};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace vmla

using namespace vmla;

extern "C" {

int mla_version(void) { return 100; }

int mla_config_check(const mla_config* cfg) { return check_config(cfg); }

unsigned long long mla_rope_table_bytes(const mla_config* cfg) {
  if (check_config(cfg) != MLA_OK) return 0;
  return static_cast<unsigned long long>(cfg->rope_table_len) * (cfg->d_r / 2) * 2 *
         sizeof(float);
}

int mla_rope_table_fill(const mla_config* cfg, float* host_table) {
  if (check_config(cfg) != MLA_OK || !host_table) return MLA_ERR_ARG;
  const int np = cfg->d_r / 2;
  // frequency of each pair: axis blocks t, h, w; band i of axis a -> theta^(-2i/D_a)
  double freq[1024];
  if (np > 1024) return MLA_ERR_ARG;
  int k = 0;
  for (int a = 0; a < 3; ++a) {
    const int n = a == 0 ? cfg->rope_pairs_t : (a == 1 ? cfg->rope_pairs_h : cfg->rope_pairs_w);
    const double D = static_cast<double>(axis_dim(*cfg, a));
    for (int i = 0; i < n; ++i) freq[k++] = std::pow(cfg->rope_theta, -2.0 * i / D);
  }
  for (int pos = 0; pos < cfg->rope_table_len; ++pos)
    for (int i = 0; i < np; ++i) {
      const double ang = static_cast<double>(pos) * freq[i];
      host_table[(static_cast<size_t>(pos) * np + i) * 2 + 0] = static_cast<float>(std::cos(ang));
      host_table[(static_cast<size_t>(pos) * np + i) * 2 + 1] = static_cast<float>(std::sin(ang));
    }
  return MLA_OK;
}

int mla_cache_reset(mla_cache* cache, void* stream) {
  if (!cache) return MLA_ERR_ARG;
  const int rc = check_config(&cache->cfg);
  if (rc != MLA_OK) return rc;
  if (!cache->c || (!cache->kr && cache->cfg.d_r > 0)) return MLA_ERR_ARG;
  const mla_config& c = cache->cfg;
  const int rr = check_resident({cache->c, cache->kr});
  if (rr != MLA_OK) return rr;
  const size_t slots = static_cast<size_t>(c.tokens_per_frame) * c.window_frames;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(cache->c, 0, slots * c.batch * c.d_c * 2, s);
  if (e == cudaSuccess && c.d_r > 0) e = cudaMemsetAsync(cache->kr, 0, slots * c.batch * c.d_r * 2, s);
  if (e != cudaSuccess) return fail_cuda(e);
  cache->frames_written = 0;
  return MLA_OK;
}

int mla_cache_append(mla_cache* cache, const void* x, const void* w_dkv, const void* gamma_kv,
                     const void* w_kr, const int* pos, long long first_frame, int n_frames,
                     void* stream) {
  if (!cache) return MLA_ERR_ARG;
  int rc = check_config(&cache->cfg);
  if (rc != MLA_OK) return rc;
  const mla_config& c = cache->cfg;
  const bool rotate = !rotate_at_use(c);
  if (!cache->c || !cache->kr || !cache->rope_table || !x || !w_dkv || !w_kr || (rotate && !pos))
    return MLA_ERR_ARG;
  if (!aligned16(cache->c) || !aligned16(cache->kr) || !aligned16(x) || !aligned16(w_dkv) ||
      !aligned16(w_kr) || !aligned16(cache->rope_table) || (gamma_kv && !aligned16(gamma_kv)) ||
      (reinterpret_cast<uintptr_t>(pos) & 3u))
    return MLA_ERR_ARG;
  if (n_frames < 1 || n_frames > c.window_frames) return MLA_ERR_RANGE;
  // frames after the sinks share W - S frame slots: two of them in one call
  // would land on the same slots (App. D.4 FIFO), so at most W - S may come
  // at once (with S = 0 this is n_frames <= W)
  {
    const long long sinks_in_call =
        first_frame < c.sink_frames
            ? (c.sink_frames - first_frame < n_frames ? c.sink_frames - first_frame : n_frames)
            : 0;
    if (n_frames - sinks_in_call > c.window_frames - c.sink_frames) return MLA_ERR_RANGE;
  }
  if (first_frame < 0 || first_frame > cache->frames_written ||
      first_frame + n_frames < cache->frames_written)
    return MLA_ERR_ARG;
  rc = check_resident({cache->c, cache->kr, cache->rope_table, x, w_dkv, gamma_kv, w_kr,
                       rotate ? pos : nullptr});
  if (rc != MLA_OK) return rc;
  AppendArgs a;
  a.x = x;
  a.w_dkv = w_dkv;
  a.gamma = gamma_kv;
  a.w_kr = w_kr;
  a.pos = rotate ? pos : nullptr;
  a.rope = static_cast<const float*>(cache->rope_table);
  a.c = cache->c;
  a.kr = cache->kr;
  a.batch = c.batch;
  a.n_tok = n_frames * c.tokens_per_frame;
  a.hidden = c.hidden;
  a.d_c = c.d_c;
  a.d_r = c.d_r;
  a.slots = c.tokens_per_frame * c.window_frames;
  a.tokens_per_frame = c.tokens_per_frame;
  a.window_frames = c.window_frames;
  a.sink_frames = c.sink_frames;
  a.rotate = rotate ? 1 : 0;
  a.first_frame = first_frame;
  a.rope_len = c.rope_table_len;
  a.pairs_t = c.rope_pairs_t;
  a.pairs_h = c.rope_pairs_h;
  a.use_rmsnorm = (c.flags & MLA_FLAG_NO_RMSNORM) ? 0 : 1;
  a.eps = c.rms_eps;
  a.status = device_status_ptr();
  a.stream = static_cast<cudaStream_t>(stream);
  if (!a.status) return MLA_ERR_CUDA;
  rc = (c.flags & MLA_FLAG_SIMT) ? launch_append_simt(a) : launch_append_tc(a);
  if (rc != MLA_OK) return rc;
  cache->frames_written = first_frame + n_frames;
  return MLA_OK;
}

int mla_attention_forward(const mla_cache* cache, const void* q_c, const void* q_r,
                          const int* q_pos, int Nq, void* o_lat, void* stream) {
  if (!cache) return MLA_ERR_ARG;
  int rc = check_config(&cache->cfg);
  if (rc != MLA_OK) return rc;
  const mla_config& c = cache->cfg;
  if (!cache->c || !cache->kr || !cache->rope_table || !q_c || !q_r || !q_pos || !o_lat)
    return MLA_ERR_ARG;
  if (!aligned16(cache->c) || !aligned16(cache->kr) || !aligned16(q_c) || !aligned16(q_r) ||
      !aligned16(o_lat) || !aligned16(cache->rope_table) ||
      (reinterpret_cast<uintptr_t>(q_pos) & 3u))
    return MLA_ERR_ARG;
  if (Nq < 1 || rotate_at_use(c)) return MLA_ERR_ARG;
  rc = check_resident({cache->c, cache->kr, cache->rope_table, q_c, q_r, q_pos, o_lat});
  if (rc != MLA_OK) return rc;
  return run_attention(cache, q_c, q_r, q_pos, Nq, cache->kr, o_lat,
                       static_cast<cudaStream_t>(stream));
}

int mla_decompress_window(const mla_cache* cache, const void* w_uk, const void* w_uv, void* k,
                          void* v, void* stream) {
  if (!cache) return MLA_ERR_ARG;
  const int rc = check_config(&cache->cfg);
  if (rc != MLA_OK) return rc;
  const mla_config& c = cache->cfg;
  if (rotate_at_use(c) || c.head_dim <= c.d_r) return MLA_ERR_ARG;
  if (!cache->c || !cache->kr || !w_uk || !w_uv || !k || !v) return MLA_ERR_ARG;
  if (!aligned16(cache->c) || !aligned16(cache->kr) || !aligned16(w_uk) || !aligned16(w_uv) ||
      !aligned16(k) || !aligned16(v))
    return MLA_ERR_ARG;
  const int rr = check_resident({cache->c, cache->kr, w_uk, w_uv, k, v});
  if (rr != MLA_OK) return rr;
  DecompressArgs a;
  a.c = cache->c;
  a.kr = cache->kr;
  a.w_uk = w_uk;
  a.w_uv = w_uv;
  a.k = k;
  a.v = v;
  a.batch = c.batch;
  a.slots = c.tokens_per_frame * c.window_frames;
  a.heads = c.heads;
  a.head_dim = c.head_dim;
  a.d_c = c.d_c;
  a.d_r = c.d_r;
  a.status = device_status_ptr();
  a.stream = static_cast<cudaStream_t>(stream);
  if (!a.status) return MLA_ERR_CUDA;
  return launch_decompress(a);
}

unsigned long long mla_window_workspace_bytes(const mla_config* cfg, int Nq) {
  if (check_config(cfg) != MLA_OK || Nq < 1) return 0;
  return window_kr_bytes(*cfg) + static_cast<unsigned long long>(cfg->batch) * Nq * 3 * 4;
}

int mla_attention_window_forward(const mla_cache* cache, const void* q_c, const void* q_r,
                                 const int* q_pos, int Nq, const int* frame_hw, void* workspace,
                                 unsigned long long workspace_bytes, void* o_lat, void* stream) {
  if (!cache) return MLA_ERR_ARG;
  int rc = check_config(&cache->cfg);
  if (rc != MLA_OK) return rc;
  const mla_config& c = cache->cfg;
  if (!rotate_at_use(c) || Nq < 1) return MLA_ERR_ARG;
  if (!cache->c || !cache->kr || !cache->rope_table || !q_c || !q_r || !q_pos || !o_lat ||
      !frame_hw || !workspace)
    return MLA_ERR_ARG;
  if (!aligned16(cache->c) || !aligned16(cache->kr) || !aligned16(q_c) || !aligned16(q_r) ||
      !aligned16(o_lat) || !aligned16(cache->rope_table) || !aligned16(workspace) ||
      (reinterpret_cast<uintptr_t>(q_pos) & 3u) || (reinterpret_cast<uintptr_t>(frame_hw) & 7u))
    return MLA_ERR_ARG;
  if (workspace_bytes < mla_window_workspace_bytes(&c, Nq)) return MLA_ERR_ARG;
  const long long n_valid = valid_slots(*cache);
  if (n_valid < 1) return MLA_ERR_ARG;
  rc = check_resident({cache->c, cache->kr, cache->rope_table, q_c, q_r, q_pos, o_lat, frame_hw,
                       workspace});
  if (rc != MLA_OK) return rc;
  WindowArgs w;
  w.kr = cache->kr;
  w.q_pos = q_pos;
  w.frame_hw = frame_hw;
  w.rope = static_cast<const float*>(cache->rope_table);
  w.kr_rot = workspace;
  w.q_pos_local = reinterpret_cast<int*>(static_cast<unsigned char*>(workspace) +
                                         window_kr_bytes(c));
  w.batch = c.batch;
  w.nq = Nq;
  w.slots = c.tokens_per_frame * c.window_frames;
  w.n_valid = static_cast<int>(n_valid);
  w.T = c.tokens_per_frame;
  w.W = c.window_frames;
  w.S = c.sink_frames;
  w.d_r = c.d_r;
  w.frames_written = cache->frames_written;
  w.rope_len = c.rope_table_len;
  w.pairs_t = c.rope_pairs_t;
  w.pairs_h = c.rope_pairs_h;
  w.status = device_status_ptr();
  w.stream = static_cast<cudaStream_t>(stream);
  if (!w.status) return MLA_ERR_CUDA;
  rc = launch_window_assemble(w);
  if (rc != MLA_OK) return rc;
  return run_attention(cache, q_c, q_r, w.q_pos_local, Nq, w.kr_rot, o_lat, w.stream);
}

int mla_absorb_weights(const mla_config* cfg, const void* w_uq, const void* w_uk, const void* w_qr,
                       const void* gamma_q, const void* w_uv, const void* w_o, void* w_qcat,
                       void* w_b, void* stream) {
  const int rc = check_config(cfg);
  if (rc != MLA_OK) return rc;
  if (!w_uq || !w_uk || !w_qr || !w_uv || !w_o || !w_qcat || !w_b) return MLA_ERR_ARG;
  if (cfg->head_dim <= cfg->d_r || cfg->d_q <= 0) return MLA_ERR_ARG;
  const int rr = check_resident({w_uq, w_uk, w_qr, gamma_q, w_uv, w_o, w_qcat, w_b});
  if (rr != MLA_OK) return rr;
  AbsorbArgs a;
  a.w_uq = w_uq;
  a.w_uk = w_uk;
  a.w_qr = w_qr;
  a.gamma_q = gamma_q;
  a.w_uv = w_uv;
  a.w_o = w_o;
  a.w_qcat = w_qcat;
  a.w_b = w_b;
  a.hidden = cfg->hidden;
  a.heads = cfg->heads;
  a.head_dim = cfg->head_dim;
  a.d_c = cfg->d_c;
  a.d_r = cfg->d_r;
  a.d_q = cfg->d_q;
  a.stream = static_cast<cudaStream_t>(stream);
  return launch_absorb(a);
}

unsigned long long mla_query_workspace_bytes(const mla_config* cfg, int Nq) {
  if (check_config(cfg) != MLA_OK || Nq < 1 || cfg->d_q <= 0) return 0;
  const unsigned long long rows = static_cast<unsigned long long>(cfg->batch) * Nq;
  const unsigned long long ct = (rows * cfg->d_q * 2 + 255) / 256 * 256;
  return ct + static_cast<unsigned long long>((cfg->d_q + kQuerySqTile - 1) / kQuerySqTile) *
                  rows * 4;
}

int mla_query_prologue(const mla_config* cfg, const void* x, const void* w_dq, const void* w_qcat,
                       int Nq, void* workspace, unsigned long long workspace_bytes, void* q_c,
                       void* q_r, void* stream) {
  const int rc = check_config(cfg);
  if (rc != MLA_OK) return rc;
  if (!x || !w_dq || !w_qcat || !workspace || !q_c || !q_r || Nq < 1) return MLA_ERR_ARG;
  if (!aligned16(x) || !aligned16(w_dq) || !aligned16(w_qcat) || !aligned16(workspace) ||
      !aligned16(q_c) || !aligned16(q_r))
    return MLA_ERR_ARG;
  if (cfg->d_q <= 0 || cfg->d_q % 64 != 0 || cfg->hidden % 64 != 0) return MLA_ERR_UNSUPPORTED;
  if (workspace_bytes < mla_query_workspace_bytes(cfg, Nq)) return MLA_ERR_ARG;
  const long long rows = static_cast<long long>(cfg->batch) * Nq;
  if (rows > (1ll << 30)) return MLA_ERR_ARG;
  const int rr = check_resident({x, w_dq, w_qcat, workspace, q_c, q_r});
  if (rr != MLA_OK) return rr;
  QueryArgs a;
  a.x = x;
  a.w_dq = w_dq;
  a.w_qcat = w_qcat;
  a.c_tilde = workspace;
  a.sq = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                  (rows * cfg->d_q * 2 + 255) / 256 * 256);
  a.q_c = q_c;
  a.q_r = q_r;
  a.rows = static_cast<int>(rows);
  a.hidden = cfg->hidden;
  a.heads = cfg->heads;
  a.d_c = cfg->d_c;
  a.d_r = cfg->d_r;
  a.d_q = cfg->d_q;
  a.eps = cfg->rms_eps;
  a.status = device_status_ptr();
  a.stream = static_cast<cudaStream_t>(stream);
  if (!a.status) return MLA_ERR_CUDA;
  return launch_query_prologue(a);
}

int mla_query_prologue_noalloc(const mla_config* cfg, const void* x, const void* w_dq,
                               const void* w_qcat, int Nq, void* q_c, void* q_r, void* stream) {
  const int rc = check_config(cfg);
  if (rc != MLA_OK) return rc;
  if (!x || !w_dq || !w_qcat || !q_c || !q_r || Nq < 1) return MLA_ERR_ARG;
  if (!aligned16(x) || !aligned16(w_dq) || !aligned16(w_qcat) || !aligned16(q_c) ||
      !aligned16(q_r))
    return MLA_ERR_ARG;
  if (cfg->d_q <= 0 || cfg->d_q % 64 != 0 || cfg->hidden % 64 != 0) return MLA_ERR_UNSUPPORTED;
  const unsigned long long need = mla_query_workspace_bytes(cfg, Nq);
  if (need == 0) return MLA_ERR_ARG;
  if (need > MLA_NOALLOC_SCRATCH_BYTES) return MLA_ERR_TOO_LARGE;
  const int rr = check_resident({x, w_dq, w_qcat, q_c, q_r});
  if (rr != MLA_OK) return rr;
  void* scratch = nullptr;
  const int sr = query_scratch_address(&scratch);
  if (sr != MLA_OK) return sr;
  const long long rows = static_cast<long long>(cfg->batch) * Nq;
  QueryArgs a;
  a.x = x;
  a.w_dq = w_dq;
  a.w_qcat = w_qcat;
  a.c_tilde = scratch;
  a.sq = reinterpret_cast<float*>(static_cast<char*>(scratch) +
                                  (rows * cfg->d_q * 2 + 255) / 256 * 256);
  a.q_c = q_c;
  a.q_r = q_r;
  a.rows = static_cast<int>(rows);
  a.hidden = cfg->hidden;
  a.heads = cfg->heads;
  a.d_c = cfg->d_c;
  a.d_r = cfg->d_r;
  a.d_q = cfg->d_q;
  a.eps = cfg->rms_eps;
  a.status = device_status_ptr();
  a.stream = static_cast<cudaStream_t>(stream);
  if (!a.status) return MLA_ERR_CUDA;
  return launch_query_prologue(a);
}

int mla_output_projection(const mla_config* cfg, const void* o_lat, const void* w_b, int Nq,
                          void* y, void* stream) {
  const int rc = check_config(cfg);
  if (rc != MLA_OK) return rc;
  if (!o_lat || !w_b || !y || Nq < 1) return MLA_ERR_ARG;
  if (!aligned16(o_lat) || !aligned16(w_b) || !aligned16(y)) return MLA_ERR_ARG;
  if ((cfg->heads * cfg->d_c) % 64 != 0) return MLA_ERR_UNSUPPORTED;
  const long long rows = static_cast<long long>(cfg->batch) * Nq;
  if (rows > (1ll << 30)) return MLA_ERR_ARG;
  const int rr = check_resident({o_lat, w_b, y});
  if (rr != MLA_OK) return rr;
  OutProjArgs a;
  a.o_lat = o_lat;
  a.w_b = w_b;
  a.y = y;
  a.rows = static_cast<int>(rows);
  a.hidden = cfg->hidden;
  a.heads = cfg->heads;
  a.d_c = cfg->d_c;
  a.status = device_status_ptr();
  a.stream = static_cast<cudaStream_t>(stream);
  if (!a.status) return MLA_ERR_CUDA;
  return launch_output_projection(a);
}

int mla_dense_attention_forward(const mla_config* cfg, const void* q, const void* k,
                                const void* v, int slots, int n_valid, int Nq, void* o,
                                void* stream) {
  const int rc = check_config(cfg);
  if (rc != MLA_OK) return rc;
  if (!q || !k || !v || !o || Nq < 1 || slots < 1 || n_valid < 1 || n_valid > slots)
    return MLA_ERR_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o)) return MLA_ERR_ARG;
  const int rr = check_resident({q, k, v, o});
  if (rr != MLA_OK) return rr;
  DenseArgs a;
  a.q = q;
  a.k = k;
  a.v = v;
  a.o = o;
  a.batch = cfg->batch;
  a.nq = Nq;
  a.heads = cfg->heads;
  a.head_dim = cfg->head_dim;
  a.slots = slots;
  a.n_valid = n_valid;
  a.scale_log2 =
      static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(cfg->head_dim)));
  a.status = device_status_ptr();
  a.stream = static_cast<cudaStream_t>(stream);
  if (!a.status) return MLA_ERR_CUDA;
  return launch_dense_attention_tc(a);
}

int mla_selftest_bounded_wait(unsigned long long limit_ns, void* stream) {
  if (limit_ns == 0 || limit_ns > 2000000000ull) return MLA_ERR_ARG;
  int* st = device_status_ptr();
  if (!st) return MLA_ERR_CUDA;
  return launch_wait_selftest(limit_ns, st, static_cast<cudaStream_t>(stream));
}

const char* mla_status_string(int status) {
  switch (status) {
    case MLA_OK: return "ok";
    case MLA_ERR_ARG: return "invalid argument";
    case MLA_ERR_UNSUPPORTED: return "shape not supported by this kernel";
    case MLA_ERR_RANGE: return "frame count or position out of range";
    case MLA_ERR_CUDA: return "CUDA error";
    case MLA_ERR_TIMEOUT: return "device wait timed out";
    case MLA_ERR_TOO_LARGE: return "request exceeds the fixed no-allocation scratch";
    default: return "unknown status";
  }
}

int mla_last_cuda_error(void) { return t_last_cuda_error; }

int mla_debug_rescale_count(unsigned long long* count, int clear) {
  if (!count) return MLA_ERR_ARG;
#if VMLA_DEBUG_CHECKS
  int* p = device_status_ptr();
  if (!p) return MLA_ERR_CUDA;
  unsigned long long* ctr = reinterpret_cast<unsigned long long*>(p + 2);
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(count, ctr, sizeof(*count), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && clear) {
    const unsigned long long zero = 0;
    e = cudaMemcpy(ctr, &zero, sizeof(zero), cudaMemcpyHostToDevice);
  }
  return e == cudaSuccess ? MLA_OK : fail_cuda(e);
#else
  (void)clear;
  *count = 0;
  return MLA_ERR_UNSUPPORTED;
#endif
}

int mla_device_status(int* status, int clear) {
  if (!status) return MLA_ERR_ARG;
  int* p = device_status_ptr();
  if (!p) return MLA_ERR_CUDA;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(status, p, sizeof(int), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && clear) {
    const int zero = MLA_OK;
    e = cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice);
  }
  return e == cudaSuccess ? MLA_OK : fail_cuda(e);
}

}  // extern "C"
