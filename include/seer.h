/*
 * libseer -- C ABI of the Seer hot path on one GB300 (sm_103a).
 *
 * Seer (arXiv 2607.14557) detects, at denoising step 0, where the valid text
 * response of a diffusion multimodal LLM ends (Sec. 3.2-3.3), truncates the
 * padded suffix once, and runs every later layer and step over the ragged
 * sequences [visual prefix + prompt + truncated response] (Sec. 3.4-3.6).
 *
 * Conventions shared by every entry point:
 *  - Pointers marked "device" are CUDA device pointers owned by the caller.
 *    The library never allocates, frees or synchronises device memory except
 *    where an entry point says so (seer_check_device, seer_profile_read).
 *  - `stream` is a cudaStream_t passed as void*; all work is enqueued on it.
 *  - Matrices are row-major.  Weight matrices use the nn.Linear layout
 *    [out_features, in_features] (K-major for the tensor cores).
 *  - Argument checks that need only host values run before any launch and
 *    return SEER_ERR_INVALID_ARG / SEER_ERR_UNSUPPORTED with a message in
 *    seer_last_error().  Values that live on the device (row counts,
 *    cu_seqlens) are checked by the kernels, which record a code that
 *    seer_check_device() reports; a kernel never traps.
 *  - 16-bit work (bf16 / f16) runs on hand-written tcgen05/TMEM/TMA kernels
 *    and needs d_model % 256 == 0, d_ff % 128 == 0, head_dim == 128 and
 *    16-byte aligned pointers.  fp32 work (small shapes) runs on CUDA-core
 *    kernels and needs d_model % 8 == 0, head_dim <= 128, head_dim % 4 == 0.
 *  - Precision of a bf16 layer: its input x and output y are bf16, but its
 *    weights and every intermediate tensor are f16 (same tensor-core rate,
 *    three more mantissa bits) with fp32 accumulation.  A layer that stored
 *    its intermediates in bf16 misses |err| <= 1e-2 + 1e-2|ref| against the
 *    exact result on a few percent of outputs at d = 4096, F = 12288; with
 *    f16 intermediates it meets it.  Values must stay within the f16 range
 *    (|v| <= 65504): every 16-bit store of the GEMM, attention and RMSNorm
 *    kernels passes a range guard, and a value that overflowed to infinity
 *    (or is NaN) records device error code 6, which seer_check_device reports.
 *  - There is no CPU fallback: without a usable GPU every call fails with
 *    SEER_ERR_CUDA.
 */
#ifndef SEER_H
#define SEER_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SEER_OK = 0,
  SEER_ERR_INVALID_ARG = 1,   /* a host-side argument is out of range or null */
  SEER_ERR_UNSUPPORTED = 2,   /* shape/alignment the kernels do not handle */
  SEER_ERR_WORKSPACE = 3,     /* workspace missing or smaller than required */
  SEER_ERR_CUDA = 4,          /* a CUDA runtime call failed (see seer_last_error) */
  SEER_ERR_TIMEOUT = 5,       /* seer_poll_ctrl gave up waiting */
  SEER_ERR_DEVICE = 6         /* a kernel recorded a device-side error */
} seer_status;

typedef enum { SEER_F32 = 0, SEER_BF16 = 1, SEER_F16 = 2 } seer_dtype;

/* Layer geometry.  A pre-norm block: RMSNorm -> QKV -> bidirectional MHA ->
 * O projection + residual -> RMSNorm -> SwiGLU MLP + residual.  The paper
 * does not spell out the block (it evaluates LLaDA-style backbones); this
 * LLaMA-style reading uses no biases.  The paper names no positional scheme:
 * rope_theta > 0 turns on a rotary embedding of q and k (half-split pairs
 * (i, i + dh/2) rotated by pos * rope_theta^(-2i/dh), pos = the row's index
 * in its sequence, restarting at 0 in every segment); 0 leaves it off. */
typedef struct {
  int d_model;
  int n_heads;
  int head_dim;      /* d_model == n_heads * head_dim */
  int d_ff;          /* SwiGLU intermediate width F */
  float rms_eps;     /* 1e-5 */
  float rope_theta;  /* 0 = no rotation; > 0 = rotary base (e.g. 10000) */
} seer_dims;

/* Detector and routing parameters (Sec. 3.3-3.4; defaults in brackets). */
typedef struct {
  float act_eps;         /* |a| < act_eps counts as a near-zero activation; the paper
                            uses an absolute threshold whose value it does not print */
  double tau_jump;       /* minimum sparsity jump [0.03] */
  double gamma;          /* plateau tolerance: noise <= gamma * jump [0.6] */
  int window;            /* look-ahead window size w [3] */
  double tau_pad;        /* padding waste threshold for the static path [0.2] */
  int eager_max_bucket;  /* buckets <= this go to the eager path [4] */
  int bucket_min;        /* smallest micro-bucket; the set doubles from it up to N [8] */
} seer_params;

/* Device pointers of one block's weights: f16 for a bf16 or f16 layer (make
 * them once with seer_convert), fp32 for an fp32 layer.
 * w_qkv [3*d, d] = rows of Wq, then Wk, then Wv;  w_o [d, d];
 * w_gate, w_up [F, d];  w_down [d, F];  g_attn, g_mlp [d] RMSNorm gains. */
typedef struct {
  const void* w_qkv;
  const void* w_o;
  const void* w_gate;
  const void* w_up;
  const void* w_down;
  const void* g_attn;
  const void* g_mlp;
} seer_layer_weights;

/* Execution paths of the hybrid router (Sec. 3.4). */
enum { SEER_PATH_STATIC = 0, SEER_PATH_VARLEN = 1, SEER_PATH_EAGER = 2 };

/* Control word written by seer_pack_ragged to pinned host memory (Sec. 3.5:
 * the CPU polls a small signal instead of waiting for the tensors).
 * int32 words:
 *   [0] epoch (written last; equals the `epoch` argument once ready)
 *   [1] total packed rows            [2] longest segment (rows)
 *   [3] graph capacity (rows): the smallest m * 2^e >= total, m in 8..15
 *   [4] number of groups              [5] bit mask of the paths in use
 *   [6] rows of bucket padding added by static groups   [7] reserved
 *   then per group g < SEER_MAX_GROUPS, 4 words at 8 + 4g:
 *   bucket, member count, path, rho in parts per million (rounded down). */
#define SEER_MAX_GROUPS 32
#define SEER_CTRL_WORDS (8 + 4 * SEER_MAX_GROUPS)

/* ---------------------------------------------------------------------------
 * Step-0 boundary detector (Sec. 3.2-3.3).
 *
 * For each sequence b the response rows x[resp_start[b] + t], t < N, go
 * through the SwiGLU MLP a = SiLU(x Wg^T) * (x Wu^T) on the tensor cores; the
 * epilogue counts |a| < act_eps per row (never storing a), giving
 * counts_out[b*N + t] (the sparsity s_t = counts/F).  The SNR scan then finds
 * the first 0-based i in [1, N-w] with jump = min(s_i..s_{i+w-1}) - s_{i-1}
 * >= tau_jump and max(..) - min(..) <= gamma * jump, evaluated in fp64 in that
 * order; L* = i* + 1, or L* = N and i* = -1 when nothing passes.
 *
 * x          device [T_rows, d] rows of the full windows (dtype dt)
 * resp_start device int32 [B]: first response row of each sequence; every
 *            resp_start[b] + N must be <= T_rows (checked on the device)
 * w_gate, w_up  device [F, d], same dtype as x (bf16 operands feed the
 *            tensor cores directly; the counts need no intermediate storage)
 * counts_out device int32 [B*N] (overwritten)
 * L_star_out, i_star_out  device int32 [B] (i_star_out may be NULL)
 * Requires B >= 1, N >= 1.  No workspace.
 * ------------------------------------------------------------------------- */
seer_status seer_detect_boundary(const void* x, seer_dtype dt, int T_rows, const int32_t* resp_start,
                                 int B, int N, const void* w_gate, const void* w_up,
                                 const seer_dims* dims, const seer_params* params,
                                 int32_t* counts_out, int32_t* L_star_out, int32_t* i_star_out,
                                 void* stream);

/* The sparsity counts alone (Sec. 3.2; S1 of seer_detect_boundary): for each
 * response row t of each sequence, the number of |a_j| < act_eps over the F
 * SwiGLU activations of that row with the given gate/up weights.  With
 * accumulate != 0 the counts are added to counts_inout instead of replacing
 * it, so several layers' gate/up weights can be tapped (a multi-layer
 * sparsity signal, Sec. 4.5 / Table 12): the sum is then a count out of
 * k * F for seer_snr_scan.  Arguments as for seer_detect_boundary. */
seer_status seer_sparsity_counts(const void* x, seer_dtype dt, int T_rows, const int32_t* resp_start, int B, int N,
                                 const void* w_gate, const void* w_up, const seer_dims* dims, float act_eps,
                                 int accumulate, int32_t* counts_inout, void* stream);

/* The SNR scan alone (Sec. 3.3) over precomputed counts: counts device int32
 * [B*N] of near-zero activations out of F; writes L_star_out (and i_star_out
 * when not NULL), device int32 [B].  Same fp64 evaluation as above.  Any
 * look-ahead window 1 <= window <= N - 1 (params->window). */
seer_status seer_snr_scan(const int32_t* counts, int B, int N, int F, const seer_params* params,
                          int32_t* L_star_out, int32_t* i_star_out, void* stream);

/* ---------------------------------------------------------------------------
 * Routing + device-resident compaction (Sec. 3.4-3.5), one fused kernel.
 *
 * Groups the sequences by micro-bucket (smallest of {m, 2m, 4m, ..., <N} U {N}
 * that holds L*_b, m = params->bucket_min, 8 in the paper), computes each group's padding waste ratio (Eq. 4) and path:
 * eager if bucket <= eager_max_bucket or the group has one member, else
 * static if rho <= tau_pad, else varlen.  Static members keep ctx_b + bucket
 * rows (the rows past ctx_b + L*_b are padding, masked as keys), the others
 * keep ctx_b + L*_b rows.  Rows are copied from the full-window layout into
 * x_packed back to back with 16-byte vector copies.
 *
 * x_full        device [cu_full[B], d] full-window rows (ctx_b + N per sequence)
 * cu_full       device int32 [B+1]
 * ctx_len       device int32 [B]: visual + prompt rows of each sequence
 * L_star        device int32 [B] (1 <= L* <= N; checked on the device)
 * N             generation window (for the bucket set)
 * T_capacity    rows available in x_packed; the packed total must fit
 * x_packed      device [T_capacity, d] (rows past the total are untouched)
 * cu_out        device int32 [B+1] segment offsets;  kv_len_out device int32 [B]
 * meta_out      device int32 [SEER_CTRL_WORDS]: the same words as the control word
 * host_ctrl     pinned, device-mapped host memory of SEER_CTRL_WORDS int32, or
 *               NULL; receives the control word with word 0 = epoch written last
 * ------------------------------------------------------------------------- */
seer_status seer_pack_ragged(const void* x_full, seer_dtype dt, const int32_t* cu_full,
                             const int32_t* ctx_len, const int32_t* L_star, int B, int d, int N,
                             int T_capacity, const seer_params* params, void* x_packed,
                             int32_t* cu_out, int32_t* kv_len_out, int32_t* meta_out,
                             int32_t* host_ctrl, int32_t epoch, void* stream);

/* Spin on the host control word until word 0 equals `epoch` (acquire), then
 * copy SEER_CTRL_WORDS words to ctrl_copy.  Never touches the GPU.  Returns
 * SEER_ERR_TIMEOUT after timeout_us microseconds. */
seer_status seer_poll_ctrl(const int32_t* host_ctrl, int32_t epoch, int timeout_us, int32_t* ctrl_copy);

/* ---------------------------------------------------------------------------
 * One truncated denoising layer over packed ragged sequences (Sec. 3.1 Eq. 2,
 * Sec. 3.6 Eqs. 9-10): every segment attends bidirectionally to its own first
 * kv_len[b] rows only.
 *
 *   xn = RMSNorm(x); [q k v] = xn Wqkv^T; o = MHA(q, k, v); h = x + o Wo^T;
 *   hn = RMSNorm(h); a = SiLU(hn Wg^T) * (hn Wu^T); y = h + a Wd^T
 * x and y have the layer dtype dt; every tensor between ops is f16 for a
 * 16-bit layer and fp32 for an fp32 layer (see the precision note above).
 *
 * x, y          device [T_capacity, d]; y must not alias x
 * cu_seqlens    device int32 [B+1]; total rows cu_seqlens[B] <= T_capacity is
 *               read on the device, so one captured CUDA graph serves any
 *               total up to the capacity
 * kv_len        device int32 [B] valid keys per segment, or NULL (= segment length)
 * count_resp_start  optional device int32 [B] (NULL disables): packed row of
 *               each sequence's first response token; the SwiGLU epilogue then
 *               adds |a| < act_eps counts of rows [start, start+N) (inside the
 *               segment) into counts_out[b*N + t] (device int32 [B*N], zeroed
 *               by this call) -- the step-0 detection layer hook
 * ws, ws_bytes  device workspace of at least seer_layer_workspace_size() bytes
 * ------------------------------------------------------------------------- */
seer_status seer_layer_forward(const seer_layer_weights* w, const seer_dims* dims, seer_dtype dt,
                               const void* x, void* y, const int32_t* cu_seqlens,
                               const int32_t* kv_len, int B, int T_capacity,
                               const int32_t* count_resp_start, int N, float act_eps,
                               int32_t* counts_out, void* ws, size_t ws_bytes, void* stream);

seer_status seer_layer_workspace_size(const seer_dims* dims, seer_dtype dt, int T_capacity, int B,
                                      size_t* bytes);

/* ---------------------------------------------------------------------------
 * The layer's steps one at a time (same kernels as seer_layer_forward).
 * Row counts: M_dev (device int32, may be NULL) overrides M_cap when set.
 * ------------------------------------------------------------------------- */

/* y[M, d] = x * rsqrt(mean(x^2) + eps) * g, fp32 arithmetic.  g has y's
 * dtype.  Type pairs: bf16->f16, bf16->bf16, f16->f16, f32->f32; d % 8 == 0. */
seer_status seer_rmsnorm(const void* x, seer_dtype x_dt, const void* g, void* y, seer_dtype y_dt, int M_cap,
                         const int32_t* M_dev, int d, float eps, void* stream);

/* c[M, N] = a[M, K] w[N, K]^T (+ r[M, N] when r != NULL), fp32 accumulation.
 * a and w share op_dt; with 16-bit operands r and c may each be bf16 or f16
 * (N % 256 == 0, K % 64 == 0); with fp32 operands everything is fp32. */
seer_status seer_linear(const void* a, const void* w, seer_dtype op_dt, const void* r, seer_dtype r_dt, void* c,
                        seer_dtype c_dt, int M_cap, const int32_t* M_dev, int N, int K, void* stream);

/* In-place rotary embedding of the q and k heads of qkv [T, 3*H*dh]
 * (q | k | v column blocks, any dtype), as seer_layer_forward applies it when
 * rope_theta > 0 (there fused into the QKV projection's epilogue for 16-bit
 * layers): pair (i, i + dh/2) of a head turns by pos * theta^(-2i/dh), pos =
 * row - cu_seqlens[b] for the segment b holding the row.  Rows past
 * cu_seqlens[B] (device) are untouched.  theta > 0, head_dim even and <= 128.
 * Not from the paper (which names no positional scheme). */
seer_status seer_rope(void* qkv, seer_dtype dt, const int32_t* cu_seqlens, int B, int T_capacity, int n_heads,
                      int head_dim, float theta, void* stream);

/* act[M, F] = SiLU(a w_gate^T) * (a w_up^T) (F % 128 == 0 for 16-bit
 * operands); near-zero counts as in seer_layer_forward. */
seer_status seer_swiglu(const void* a, const void* w_gate, const void* w_up, seer_dtype op_dt, void* act,
                        seer_dtype act_dt, int M_cap, const int32_t* M_dev, int F, int K, const int32_t* cu_seqlens,
                        int B, const int32_t* count_resp_start, int N, float act_eps, int32_t* counts_out,
                        void* stream);

/* seer_attention for callers that cannot allocate device memory, such as code
 * whose device memory is owned by another allocator (an engine's pool, a
 * plugin without cudaMalloc) or that must not allocate on its hot path.  The
 * paper has no counterpart; this is a service of the library.
 * Same arguments and results as seer_attention, minus the workspace: the
 * schedule lives in a fixed 1 MiB __device__ array compiled into libseer,
 * held by every GPU that loads the library until the process exits.
 * For 16-bit attention n_heads * (ceil(T_capacity/128) + B) must stay
 * <= 65520 (the work units whose schedule fits the array), else the call
 * returns SEER_ERR_WORKSPACE; fp32 attention uses no schedule and has no such
 * limit.  The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current, so make it before any
 * stream capture; the address is kept for the process, so resetting the
 * device (cudaDeviceReset) while libseer is loaded is not supported.
 * Allocates nothing.  Every call reuses the same array: calls whose kernels
 * overlap on the GPU race and must not be issued (nothing in the array needs
 * to start at zero). */
seer_status seer_attention_noalloc(const void* qkv, void* o, seer_dtype dt, const int32_t* cu_seqlens,
                                   const int32_t* kv_len, int B, int T_capacity, int n_heads, int head_dim,
                                   void* stream);

/* dst[i] = src[i] converted (round to nearest even) for i < n; n % 8 == 0.
 * bf16 -> f16 is exact for |v| >= 2^-14 and below 65504 (f16's normal range);
 * a 16-bit result that is infinite or NaN records device error code 6.
 * Used once per model to make the f16 weight copies of bf16 layers. */
seer_status seer_convert(const void* src, seer_dtype src_dt, void* dst, seer_dtype dst_dt, size_t n, void* stream);

/* o[T, H*dh]: per segment b and head h, softmax(q k^T / sqrt(dh)) v over the
 * segment's first kv_len[b] keys (Eqs. 6-7, no causal mask).  qkv [T, 3*H*dh]
 * holds q | k | v.  ws as for seer_layer_forward (only the scheduling part:
 * the work units, their count and the counter from which the attention
 * kernel's persistent CTAs take units; all rewritten by every call, so calls
 * that share a workspace must not overlap on the GPU). */
seer_status seer_attention(const void* qkv, void* o, seer_dtype dt, const int32_t* cu_seqlens,
                           const int32_t* kv_len, int B, int T_capacity, int n_heads, int head_dim,
                           void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Prefix key/value caching combined with truncation (the paper reports that
 * Seer composes with KV caching of the visual + prompt prefix, Table 7).
 * A K/V cache of one layer is a [T_kv_cap, 2*H*dh] matrix (K | V per row, the
 * layer's intermediate type: f16 for 16-bit layers, f32 for f32 ones) laid
 * out like the packed truncated sequences: segment b owns rows
 * [cu_kv[b], cu_kv[b+1]), its first ctx_len[b] rows hold the prefix's keys
 * and values (seer_kv_prefill) and the rest the response rows' own, which
 * seer_layer_forward_cached writes on every call.  cu_kv is the cu_seqlens of
 * seer_pack_ragged.  Rotary embeddings are not supported on this path.
 * ------------------------------------------------------------------------- */

/* Fills the prefix part of a layer's K/V cache: for each segment b, the rows
 * [cu_x[b], cu_x[b] + ctx_len[b]) of x (the layer's input hidden states, any
 * row layout, dtype dt) are normalised and projected with the K and V rows of
 * w->w_qkv, and the results stored at cache rows [cu_kv[b], cu_kv[b] +
 * ctx_len[b]).  ws: seer_layer_workspace_size(dims, dt, T_x_cap, B) bytes.
 * Row counts are read on the device; segments that would fall outside x or
 * the cache are skipped and recorded (seer_check_device). */
seer_status seer_kv_prefill(const seer_layer_weights* w, const seer_dims* dims, seer_dtype dt, const void* x,
                            const int32_t* cu_x, const int32_t* ctx_len, int B, int T_x_cap, void* kv_cache,
                            const int32_t* cu_kv, int T_kv_cap, void* ws, size_t ws_bytes, void* stream);

/* The block over the response rows only (packed by cu_resp, dtype dt in and
 * out, as from seer_gather_response): queries are the response rows, keys and
 * values the segment's cached prefix rows followed by its response rows (the
 * first kv_len[b] rows of the segment in all, kv_len as from
 * seer_pack_ragged; NULL = the whole segment).  Writes the response rows'
 * K and V into the cache first.  y_resp must not alias x_resp.  ws:
 * seer_layer_workspace_size(dims, dt, T_resp_cap, B) bytes. */
seer_status seer_layer_forward_cached(const seer_layer_weights* w, const seer_dims* dims, seer_dtype dt,
                                      const void* x_resp, void* y_resp, const int32_t* cu_resp, const int32_t* ctx_len,
                                      int B, int T_resp_cap, void* kv_cache, const int32_t* cu_kv,
                                      const int32_t* kv_len, int T_kv_cap, void* ws, size_t ws_bytes, void* stream);

/* Response rows of packed sequences: cu_resp_out[b] = cu[b] - (ctx_len[0] +
 * ... + ctx_len[b-1]) (device int32 [B+1]) and x_resp rows [cu_resp_out[b],
 * cu_resp_out[b+1]) = x_packed rows [cu[b] + ctx_len[b], cu[b+1]).  d * size
 * of dt must be a multiple of 16 bytes. */
seer_status seer_gather_response(const void* x_packed, seer_dtype dt, const int32_t* cu, const int32_t* ctx_len, int B,
                                 int d, int T_cap, void* x_resp, int32_t* cu_resp_out, void* stream);

/* ---------------------------------------------------------------------------
 * Diagnostics.
 * ------------------------------------------------------------------------- */
/* Thread-local message describing the last failure of this thread. */
const char* seer_last_error(void);

/* Synchronises the current device, then reports (and clears) the first
 * device-side error recorded by any kernel: SEER_OK or SEER_ERR_DEVICE with
 * code_out set (1 bad row count, 2 bad sequence layout, 3 pipeline wait timed
 * out, 4 boundary out of range, 5 capacity exceeded, 6 a stored 16-bit value
 * is infinite or NaN: an f16 intermediate overflowed +-65504, or the input
 * held a non-finite value). */
seer_status seer_check_device(int* code_out);

/* Failure-detection self-test: enqueues a kernel whose pipeline wait can
 * never complete (an mbarrier that no thread arrives on).  Like every wait
 * in the library's kernels it gives up after a time limit, here limit_us
 * (1 .. 1e7), records the timeout code (3) in the device error word and
 * returns, so the context stays usable; seer_check_device then reports
 * SEER_ERR_DEVICE with code 3.  Enqueues only; never waits. */
seer_status seer_selftest_wait_timeout(int limit_us, void* stream);

/* Launch overlap (programmatic dependent launch).  When on (the default),
 * each kernel of the library is launched as a programmatic dependent of the
 * previous kernel in its stream: the GPU may place its blocks while that
 * kernel finishes, which hides most of the launch gap between consecutive
 * kernels.  Every kernel waits at entry until the kernels before it have
 * completed and their writes are visible, so results are the same with the
 * setting on or off.  Process-wide; returns the previous setting (1 or 0). */
int seer_set_launch_overlap(int on);

/* Per-phase timing with CUDA events recorded on the call's stream.
 * Phases: 0 detect GEMM, 1 SNR scan, 2 pack, 3 norm1, 4 QKV, 5 attention,
 * 6 O proj, 7 norm2, 8 gate/up, 9 down, 10 K/V cache copies and prefix
 * projections.  seer_profile_read synchronises on the recorded events and
 * returns accumulated milliseconds and launch counts since the last reset. */
#define SEER_N_PHASES 11
seer_status seer_profile_enable(int on);
/* Restricts recording to the phases whose bit is set in phase_mask (bit i =
 * phase i; default all).  Each recorded phase adds two events to its stream,
 * which also keeps launch overlap from spanning that phase's boundaries. */
seer_status seer_profile_select(uint32_t phase_mask);
seer_status seer_profile_reset(void);
seer_status seer_profile_read(float* ms_out, int32_t* launches_out);

/* Number of SMs of the current device (used to size persistent grids). */
int seer_num_sms(void);

const char* seer_version(void);

#ifdef __cplusplus
}
#endif
#endif /* SEER_H */
