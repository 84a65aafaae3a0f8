/*
 * videomla.h -- C ABI of libvideomla.so: the latent KV cache and the
 * absorbed-form Multi-Head Latent Attention of VideoMLA (arXiv 2605.30351)
 * on one GB300 (sm_103a).
 *
 * Conventions for every entry point
 *  - All tensors are caller-owned device memory (for example torch tensors
 *    passed by data_ptr()). The library allocates no device memory, keeps no
 *    per-cache state of its own and never synchronises the stream.
 *  - Every buffer must be device memory (cudaMalloc or a pool built on it)
 *    of the CURRENT device: host memory, pinned or not, managed memory and
 *    another GPU's memory are refused with MLA_ERR_ARG before any launch.
 *    The kernels copy tiles with TMA, and the attention kernels share key
 *    tiles among the CTAs of a cluster by multicast, which addresses this
 *    GPU's own memory only.
 *  - The library caches, per device, the device addresses of its two
 *    file-scope arrays (the status word and the no-allocation scratch). It
 *    does not survive cudaDeviceReset (or any other teardown of the
 *    device's primary context) within the process.
 *  - Calls are asynchronous on `stream` (a cudaStream_t passed as void*;
 *    NULL is the legacy default stream).
 *  - bf16 = IEEE bfloat16 stored as 2 bytes. All arrays are dense, row-major,
 *    with the last dimension contiguous, and start on a 16-byte boundary.
 *  - Return 0 (MLA_OK) or a negative MLA_ERR_* code. Host-side validation
 *    runs before any launch, so an error return means nothing was enqueued.
 *    Faults the host cannot see (a position outside the RoPE table, a device
 *    wait that ran out) are recorded in a device status word that
 *    mla_device_status() reads; the kernel skips the offending work instead
 *    of trapping.
 */
#ifndef VIDEOMLA_H_
#define VIDEOMLA_H_

#ifdef __cplusplus
extern "C" {
#endif

#define MLA_OK 0
#define MLA_ERR_ARG (-1)         /* null pointer, misaligned pointer, bad shape */
#define MLA_ERR_UNSUPPORTED (-2) /* no kernel instance for this shape */
#define MLA_ERR_RANGE (-3)       /* frame count or position outside the window/table */
#define MLA_ERR_CUDA (-4)        /* launch or runtime error (see mla_last_cuda_error) */
#define MLA_ERR_TIMEOUT (-5)     /* a bounded device-side wait ran out */
#define MLA_ERR_TOO_LARGE (-6)   /* request does not fit the library's fixed scratch */

/* Size of the fixed device scratch used by mla_query_prologue_noalloc. */
#define MLA_NOALLOC_SCRATCH_BYTES (8u * 1024u * 1024u)

/* cfg.flags */
#define MLA_FLAG_NO_RMSNORM 1u   /* store c^KV = W_dkv x without RMSNorm (App. D.2 off) */
#define MLA_FLAG_SIMT 2u         /* use the plain SIMT debug kernels (no tensor cores) */
#define MLA_FLAG_ROTATE_AT_USE 4u /* cache k^R unrotated; attend with
                                     mla_attention_window_forward (App. D.5) */

/*
 * Shape of one VideoMLA attention layer (Sec. 3; App. D.2-D.4).
 *  hidden          d, the model width (1536 for Wan2.1-1.3B)
 *  heads           n_h (12)
 *  head_dim        d_h = d_nope + d_rope (128); the score is divided by
 *                  sqrt(head_dim) (Eq. score)
 *  d_c             width of the shared KV latent c^KV (192)   (Eq. ckv)
 *  d_r             width of the shared positional key k^R (32) (Eq. krope);
 *                  positive (the decoupled key always exists on this path)
 *  d_q             width of the query latent c^Q (768), used by the query prologue
 *  rope_pairs_*    complex pairs per axis; 2*(t+h+w) must equal d_r (App. D.3)
 *  rope_dim_*      band width D_a of each axis: pair i of axis a rotates with
 *                  theta^(-2i/D_a), i.e. the highest-frequency bands of the
 *                  backbone's per-axis split (44/42/42 for a 128-wide head);
 *                  0 means D_a = 2 * rope_pairs_a
 *  rope_theta      RoPE base (10000)
 *  rope_table_len  positions per axis the table covers (1024, App. C.1)
 *  tokens_per_frame T, tokens of one latent frame (30*52 = 1560, App. D.1)
 *  window_frames   W, latent frames the cache holds (21, Sec. 1 / App. D.4;
 *                  7 = 1 sink + 6 local for long rollouts, App. D.4)
 *  batch           B, independent sequences, each with its own ring
 *  rms_eps         RMSNorm epsilon (1e-6)
 *  flags           MLA_FLAG_*
 *  sink_frames     S, leading latent frames that are never evicted (0 for the
 *                  plain 21-frame ring, 1 for the long-rollout window of
 *                  App. D.4); 0 <= S < W
 */
typedef struct mla_config {
  int hidden;
  int heads;
  int head_dim;
  int d_c;
  int d_r;
  int d_q;
  int rope_pairs_t, rope_pairs_h, rope_pairs_w;
  int rope_dim_t, rope_dim_h, rope_dim_w;
  double rope_theta;
  int rope_table_len;
  int tokens_per_frame;
  int window_frames;
  int batch;
  float rms_eps;
  unsigned flags;
  int sink_frames;
} mla_config;

/*
 * The sliding-window latent cache (App. D.4). Caller-owned device buffers:
 *  c          bf16 [batch][window_frames*tokens_per_frame][d_c]   latent c^KV
 *  kr         bf16 [batch][window_frames*tokens_per_frame][d_r]   k^R, rotated
 *             at append, or unrotated with MLA_FLAG_ROTATE_AT_USE
 *  rope_table fp32 [rope_table_len][d_r/2][2] = (cos, sin) of position p
 *             times the pair's frequency; fill it with mla_rope_table_fill()
 *             and copy it to the device.
 *  frames_written  number of latent frames appended so far (advanced by
 *             mla_cache_append on the host; reset by mla_cache_reset).
 * Token k of latent frame f lives in slot f*T + k if f < S (a sink frame),
 * else in slot (S + (f - S) mod (W - S))*T + k: the frames after the sinks
 * share W - S frame slots in FIFO order (App. D.4). With S = 0 this is the
 * ring (f mod W)*T + k. Slots of frames that were never written are not read.
 */
typedef struct mla_cache {
  void* c;
  void* kr;
  const void* rope_table;
  long long frames_written;
  mla_config cfg;
} mla_cache;

/* Bytes of the host buffer mla_rope_table_fill writes (0 on a bad config). */
unsigned long long mla_rope_table_bytes(const mla_config* cfg);

/*
 * Fill host_table (fp32 [rope_table_len][d_r/2][2]) with cos/sin of
 * p * theta^(-2i/D_a) for every position p and pair (axis a, band i),
 * computed in double and rounded once (Sec. 3.2, App. D.3).
 * Returns MLA_ERR_ARG on a null pointer or an inconsistent config.
 */
int mla_rope_table_fill(const mla_config* cfg, float* host_table);

/* Check a configuration without launching anything. */
int mla_config_check(const mla_config* cfg);

/*
 * Zero both cache buffers and set frames_written = 0 (asynchronous memset
 * on `stream`).
 */
int mla_cache_reset(mla_cache* cache, void* stream);

/*
 * Append n_frames latent frames (first_frame .. first_frame+n_frames-1) of
 * token activations to the cache (Eqs. ckv and krope; App. D.2, D.4):
 *     c = RMSNorm_gamma(W_dkv x)        -> cache.c  at the frame's slots
 *     k = RoPE3D(W_kr x, pos)           -> cache.kr at the frame's slots
 *  x        bf16 [batch][n_frames*T][hidden]
 *  w_dkv    bf16 [d_c][hidden]        joint KV down-projection
 *  gamma_kv bf16 [d_c] RMSNorm weight, or NULL for ones
 *  w_kr     bf16 [d_r][hidden]        decoupled RoPE key projection
 *  pos      int32 [batch][n_frames*T][3]  (t, h, w) of every token; each
 *           coordinate must lie in [0, rope_table_len) (device-checked).
 *           Not read (may be NULL) with MLA_FLAG_ROTATE_AT_USE.
 * The positional key is rotated here with the absolute positions given;
 * for a contiguous window the scores only depend on position differences,
 * so this matches rotating at use with window-relative coordinates
 * (Sec. 3.2, App. D.5). With MLA_FLAG_ROTATE_AT_USE the cache keeps
 * k = W_kr x unrotated, the paper's own storage (App. D.5).
 * Rules: 1 <= n_frames <= window_frames, and at most W - S of the frames
 * are past the sinks (frames >= S share W - S frame slots, so two of them in
 * one call would land on the same slots): n_frames - max(0, min(n_frames,
 * S - first_frame)) <= W - S (else MLA_ERR_RANGE; with S = 0 both rules are
 * n_frames <= W);
 * 0 <= first_frame <= frames_written <= first_frame + n_frames (no gap, and
 * the range reaches the newest frame: extend the window or rewrite the
 * current chunk, as each denoising step does). Afterwards
 * frames_written = first_frame + n_frames.
 * Tensor-core kernel for d_c in {64, 128, 192, 256, 512} and d_r in {32, 64}
 * with hidden a multiple of 64 (at d_c = 512 the c and k^R halves run in
 * separate CTAs); other shapes return MLA_ERR_UNSUPPORTED unless
 * MLA_FLAG_SIMT selects the SIMT kernel.
 */
int mla_cache_append(mla_cache* cache, const void* x, const void* w_dkv,
                     const void* gamma_kv, const void* w_kr, const int* pos,
                     long long first_frame, int n_frames, void* stream);

/*
 * Absorbed-form attention of a query chunk against every valid slot of the
 * window (Eq. score; App. E, Eqs. absorb-q and absorb-v):
 *     s_hj  = (q_c,h . c_j + RoPE3D(q_r,h, q_pos) . k_j) / sqrt(head_dim)
 *     o_h   = sum_j softmax_j(s_hj) c_j            (latent output, d_c wide)
 *  q_c   bf16 [batch][Nq][heads][d_c]  absorbed content queries A_h^T c^Q
 *  q_r   bf16 [batch][Nq][heads][d_r]  unrotated positional queries
 *  q_pos int32 [batch][Nq][3]          query positions (device-checked)
 *  o_lat bf16 [batch][Nq][heads][d_c]  output; the caller applies
 *        B_h = W_O,h W_up,h^V to mix heads (Eq. absorb-v)
 * Valid slots: the first min(frames_written, W)*T slots before the ring
 * first wraps, all slots after. The query chunk is taken to be the newest
 * chunk, so the chunk-causal mask (App. D.4) keeps every valid slot.
 * MLA_ERR_ARG if no slot is valid, Nq < 1, or the cache keeps k^R unrotated
 * (MLA_FLAG_ROTATE_AT_USE: use mla_attention_window_forward).
 * Tensor-core kernel for d_c in {64, 128, 192, 256, 512} and d_r in {32, 64}
 * (at d_c = 512 two CTAs share each 128-row tile, 256 output columns each);
 * other shapes return MLA_ERR_UNSUPPORTED unless MLA_FLAG_SIMT is set.
 */
int mla_attention_forward(const mla_cache* cache, const void* q_c,
                          const void* q_r, const int* q_pos, int Nq,
                          void* o_lat, void* stream);

/* Bytes of caller-owned device workspace mla_attention_window_forward needs
 * for Nq query tokens per batch element (0 on a bad config). */
unsigned long long mla_window_workspace_bytes(const mla_config* cfg, int Nq);

/*
 * Attention over the assembled window of a cache that keeps k^R unrotated
 * (MLA_FLAG_ROTATE_AT_USE), with window-relative RoPE (App. D.4, D.5):
 *  1. the held frames (the S sinks, then the newest frames in temporal
 *     order) are numbered 0, 1, ...; that number is the temporal coordinate
 *     of every key of the frame, which is rotated by RoPE3D at
 *     (local t, h, w) into the workspace;
 *  2. each query's absolute frame q_pos[.][0] is mapped to the local number
 *     of that frame (the frame must be held: the current chunk is appended
 *     first), (h, w) unchanged;
 *  3. the same absorbed-form attention as mla_attention_forward runs over
 *     the valid slots with the rotated window keys.
 * Before any eviction local and absolute times agree. Arguments as for
 * mla_attention_forward, plus:
 *  frame_hw  int32 [tokens_per_frame][2], 8-byte aligned: (h, w) of token k
 *            of every latent frame (the latent grid is the same for all
 *            frames); each must lie in [0, rope_table_len) (device-checked)
 *  workspace device memory of at least mla_window_workspace_bytes(cfg, Nq)
 *            bytes, 16-byte aligned, owned by the caller (scratch)
 * A query frame the window does not hold is recorded as MLA_ERR_RANGE in
 * the device status (its rows use local time 0). MLA_ERR_ARG unless the
 * cache has MLA_FLAG_ROTATE_AT_USE.
 */
int mla_attention_window_forward(const mla_cache* cache, const void* q_c, const void* q_r,
                                 const int* q_pos, int Nq, const int* frame_hw,
                                 void* workspace, unsigned long long workspace_bytes,
                                 void* o_lat, void* stream);

/*
 * Load-time weight absorption (App. E, Eqs. absorb-q and absorb-v), computed
 * on the device with fp32 accumulation and rounded once to bf16:
 *   w_qcat bf16 [H*(d_c+d_r)][d_q]: rows (h, c), c < d_c, hold
 *          A_h[:, c] * gamma_q = sum_e W_up,h^Q[e][:] W_up,h^K[e][c] * gamma_q,
 *          rows H*d_c + (h, j) hold W_R,h^Q[j][:] * gamma_q (Eq. qrope);
 *   w_b    bf16 [hidden][H*d_c]: B_h = W_O,h W_up,h^V side by side.
 * Inputs (bf16): w_uq [H][d_nope][d_q], w_uk [H][d_nope][d_c],
 * w_qr [H][d_r][d_q], gamma_q [d_q] or NULL (ones), w_uv [H][d_h][d_c],
 * w_o [hidden][H*d_h]; d_nope = head_dim - d_r. Asynchronous on `stream`.
 */
int mla_absorb_weights(const mla_config* cfg, const void* w_uq, const void* w_uk,
                       const void* w_qr, const void* gamma_q, const void* w_uv,
                       const void* w_o, void* w_qcat, void* w_b, void* stream);

/* Bytes of caller-owned device workspace mla_query_prologue needs for Nq
 * query tokens per batch element (0 on a bad config). */
unsigned long long mla_query_workspace_bytes(const mla_config* cfg, int Nq);

/*
 * Query path of a chunk (Eqs. cq, qnope, qrope; App. D.2 RMSNorm; App. E):
 *     c~        = W_dn^Q x                       (bf16 in the workspace)
 *     [q_c|q_r] = [W_qc ; W_qr] diag(gamma_q) c~ / rms(c~)
 * The RMSNorm statistics come from the fp32 accumulator of the first GEMM;
 * the per-row scale is applied in the second GEMM's epilogue (it commutes
 * with the linear map). Outputs are exactly mla_attention_forward's inputs:
 *  x       bf16 [batch][Nq][hidden]
 *  w_dq    bf16 [d_q][hidden]
 *  w_qcat  bf16 [H*(d_c+d_r)][d_q] from mla_absorb_weights
 *  workspace  device memory of at least mla_query_workspace_bytes(cfg, Nq)
 *             bytes, 16-byte aligned, owned by the caller; its contents are
 *             scratch between the two GEMMs of this call
 *  q_c     bf16 [batch][Nq][H][d_c];  q_r bf16 [batch][Nq][H][d_r] (unrotated)
 * MLA_ERR_UNSUPPORTED unless d_q and hidden are multiples of 64 and
 * batch * Nq <= 8,388,352 (65,534 tiles of 128 query tokens).
 */
int mla_query_prologue(const mla_config* cfg, const void* x, const void* w_dq,
                       const void* w_qcat, int Nq, void* workspace,
                       unsigned long long workspace_bytes, void* q_c, void* q_r,
                       void* stream);

/*
 * mla_query_prologue without a caller workspace: the same computation and
 * outputs, but the intermediate c~ and its row statistics live in a fixed
 * array inside the library. The paper has no counterpart of this entry point;
 * it exists for callers that cannot allocate device memory at the point of
 * the call, e.g. code running inside another framework's memory pool or a
 * real-time loop where any cudaMalloc/cudaFree would stall or be forbidden.
 *  - Nothing is allocated: no cudaMalloc, cudaFree or allocating library call.
 *  - The array holds MLA_NOALLOC_SCRATCH_BYTES bytes on every GPU that loads
 *    the library, for the life of the process. Requests whose
 *    mla_query_workspace_bytes(cfg, Nq) exceed it return MLA_ERR_TOO_LARGE
 *    before anything is enqueued (the Wan-1.3B chunk of 4680 tokens at batch 1
 *    needs about 7.2 MB and fits).
 *  - The first call on each device looks up the array's device address with
 *    cudaGetSymbolAddress; make that first call before any stream capture.
 *  - All calls share the one array, and it keeps the previous call's
 *    contents (nothing in it needs to start at zero: every call overwrites
 *    what it reads). Calls whose work overlaps on the GPU, e.g. on two
 *    streams at once, race on it; serialise them.
 * Arguments and outputs as for mla_query_prologue.
 */
int mla_query_prologue_noalloc(const mla_config* cfg, const void* x, const void* w_dq,
                               const void* w_qcat, int Nq, void* q_c, void* q_r,
                               void* stream);

/*
 * Output projection of the latent attention output (Eq. absorb-v):
 *     y = sum_h B_h o_lat,h = o_lat W_B^T
 *  o_lat bf16 [batch][Nq][H][d_c], w_b bf16 [hidden][H*d_c],
 *  y bf16 [batch][Nq][hidden]. MLA_ERR_UNSUPPORTED unless H*d_c % 64 == 0 and
 *  batch * Nq <= 8,388,352 (65,534 tiles of 128 tokens).
 */
int mla_output_projection(const mla_config* cfg, const void* o_lat, const void* w_b, int Nq,
                          void* y, void* stream);

/*
 * Dense per-head attention: the baseline VideoMLA replaces, where every token
 * caches K and V for every head, 2*n_h*d_h scalars (App. C.1; the dense rows
 * of Table 1). Used for the d_c sweep's comparison (Table 5a); same window
 * and query chunk as mla_attention_forward:
 *     o_h = softmax_j(q_h . k_{h,j} / sqrt(head_dim)) v_{h,j}
 *  q bf16 [batch][Nq][heads][head_dim] (RoPE already applied)
 *  k, v bf16 [batch][heads][slots][head_dim] (k rotated); the first n_valid
 *       slots of each head are read
 *  o bf16 [batch][Nq][heads][head_dim]
 * MLA_ERR_UNSUPPORTED unless head_dim is 64 or 128.
 */
int mla_dense_attention_forward(const mla_config* cfg, const void* q, const void* k,
                                const void* v, int slots, int n_valid, int Nq, void* o,
                                void* stream);

/*
 * Decompress-then-dense: the non-absorbed way to run attention on the latent
 * cache (Sec. 3.1 Eq. reconstruct; App. E is what it avoids). Expands every
 * slot of the cache into per-head keys and values,
 *     k[b][h][j] = [ W_up,h^K c_j | k_j ]     (d_nope + d_r = head_dim columns)
 *     v[b][h][j] =   W_up,h^V c_j             (head_dim columns)
 * so that mla_dense_attention_forward can run on them with per-head queries
 * [q^nope_h | RoPE3D(q^R_h)] (Eq. score). All W*T slots are written.
 *  w_uk  bf16 [heads][head_dim - d_r][d_c]    W_up^K
 *  w_uv  bf16 [heads][head_dim][d_c]          W_up^V
 *  k, v  bf16 [batch][heads][W*T][head_dim]   outputs (caller-owned)
 * MLA_ERR_ARG for a cache with MLA_FLAG_ROTATE_AT_USE (its k is unrotated);
 * MLA_ERR_UNSUPPORTED unless d_c is a multiple of 64 and head_dim and
 * head_dim - d_r are multiples of 32.
 */
int mla_decompress_window(const mla_cache* cache, const void* w_uk, const void* w_uv, void* k,
                          void* v, void* stream);

/*
 * Self-test of the bounded device waits that guard every mbarrier wait in the
 * tensor-core kernels (a device wait never hangs: after its limit it records
 * MLA_ERR_TIMEOUT in the device status word and the kernel returns). Launches
 * one thread that waits, through the same code, on a barrier nothing arrives
 * on, for limit_ns nanoseconds (1 ns .. 2 s); afterwards mla_device_status
 * reports MLA_ERR_TIMEOUT and the context remains usable. MLA_ERR_ARG for a
 * limit outside that range.
 */
int mla_selftest_bounded_wait(unsigned long long limit_ns, void* stream);

/* Human-readable name of a status code. */
const char* mla_status_string(int status);

/* The cudaError_t of the last MLA_ERR_CUDA return (0 if none). */
int mla_last_cuda_error(void);

/*
 * Read (and, if clear != 0, reset) the device status word that kernels set
 * when they skip work: MLA_OK, MLA_ERR_RANGE or MLA_ERR_TIMEOUT. The first
 * error recorded wins. Synchronises the device.
 */
int mla_device_status(int* status, int clear);

/*
 * Debug builds only (libvideomla_debug.so, built with VMLA_DEBUG_CHECKS=1):
 * read (and, if clear != 0, reset) the number of query rows whose online
 * softmax rescaled its running output because the running maximum of the
 * scores grew by more than 2^8 (in log2 units) from one key block to a later
 * one (Eq. score; the softmax over the window, Sec. 3.3). Counted by the
 * tensor-core attention kernels, absorbed and dense, once per (row, block)
 * that rescales. Synchronises the device. A release build sets *count = 0
 * and returns MLA_ERR_UNSUPPORTED; MLA_ERR_ARG for a null pointer.
 */
int mla_debug_rescale_count(unsigned long long* count, int clear);

/* Library version, e.g. 100 for 0.1.0. */
int mla_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VIDEOMLA_H_ */
