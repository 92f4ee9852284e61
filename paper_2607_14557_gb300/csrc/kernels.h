// Internal launch interface between the C-ABI layer (seer_api.cu) and the
// kernel translation units.  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace seer {

// Epilogue variants of the GEMM kernels.
enum GemmMode : int {
  kGemmStore = 0,     // C = A B^T
  kGemmResidual = 1,  // C = A B^T + R
  kGemmSwiglu = 2,    // act = SiLU(A Bg^T) * (A Bu^T), optional near-zero counts
  kGemmCount = 3,     // counts only (detector): A rows gathered per sequence window
  kGemmRope = 4,      // C = A B^T, then columns < rope_cols rotated per head (rotary embedding)
};

struct GemmParams {
  int M_cap;              // rows available in A / C
  const int* M_dev;       // optional device row count (<= M_cap)
  int N;                  // output columns (Swiglu/Count: F)
  int K;
  void* C;                // output [M, ldc]
  int ldc;
  const void* R;          // residual [M, ldr]
  int ldr;
  int* counts;            // [B * Nw] near-zero counts (Swiglu hook / Count)
  float act_eps;
  const int* cu;          // segment offsets [B+1] for the Swiglu count hook
  int B;
  const int* resp_start;  // first response row per sequence
  int Nw;                 // response window
  int* err;               // device error word
  uint32_t idesc;         // tcgen05 instruction descriptor (operand type f16 or bf16)
  int out_type;           // ElemType of C (kBF16 / kF16; kF32 on the CUDA-core path)
  int res_type;           // ElemType of R
  int group_m;            // raster: m-tiles per group (see tc_gemm.cu)
  float rope_theta;       // Rope: frequency base (> 0)
  int rope_cols;          // Rope: leading output columns that are rotated (the q|k columns)
};

struct AttnParams {
  const int* cu;          // [B+1] query segment offsets (rows of the q source)
  const int* kv_len;      // [B] keys per segment, or null (= the K/V segment length)
  const int* cu_kv;       // [B+1] K/V segment offsets, or null (= cu: q, k, v share rows)
  const void* kv;         // K/V rows (fp32 path), or null (= the qkv buffer)
  int ld_kv;              // elements per K/V row
  int xk0, xv0;           // column of head 0's K and V inside a K/V row
  int B;
  int T_cap;
  int n_heads;
  int head_dim;
  void* out;              // [T, H*dh]
  int ldo;                // elements
  const int4* work;       // schedule: (b, h, first q-tile, q-tiles)
  const int* work_count;  // units in `work`
  int* work_next;         // next unit to hand out (zeroed by the schedule kernel)
  int* err;
};

// tcgen05 / TMA kernels (16-bit operands).  Tensor maps are encoded on the host.
int tc_gemm_smem_bytes();
// L2 raster of the persistent GEMM (GemmParams::group_m) for a B operand of
// b_bytes and an A row-tile of a_tile_bytes.
int tc_gemm_group_m(long b_bytes, long a_tile_bytes);
// mC: the 16-bit output C (Store, Residual, Rope) or act (Swiglu) with 32 x 32
// boxes and no swizzle, for the epilogue's TMA stores (unused by Count).
cudaError_t launch_tc_gemm(int mode, const CUtensorMap& mA, const CUtensorMap& mB0, const CUtensorMap& mB1,
                           const CUtensorMap& mC, const GemmParams& p, int num_sms, cudaStream_t st);
int tc_attn_smem_bytes();
// grid: persistent CTAs (at most one per SM); they take the units of the
// schedule from p.work_next until *p.work_count are done
cudaError_t launch_tc_attn(const CUtensorMap& mQ, const CUtensorMap& mKV, const AttnParams& p, int grid, bool f16,
                           cudaStream_t st);
// Bytes of schedule workspace the 16-bit attention kernels need for a launch
// sized for T_cap rows, B segments and H heads: H * (ceil(T_cap/128) + B) work
// units of 16 bytes, rounded up to 256 bytes, plus 256 bytes for the unit
// count and the persistent kernel's unit counter.
size_t attn_sched_bytes(int T_cap, int B, int H);
// writes the units to work, their number to work_count[0] and zeroes
// work_count[1] (the attention kernel's unit counter)
cudaError_t launch_attn_schedule(const int* cu, const int* cu_kv, const int* kv_len, int B, int n_heads, int T_cap,
                                 int4* work, int* work_count, int max_units, int* err, cudaStream_t st);

// CUDA-core kernels (fp32 storage; small shapes).
cudaError_t launch_simt_gemm(int mode, const float* A, const float* B0, const float* B1, const GemmParams& p,
                             cudaStream_t st);
cudaError_t launch_simt_attn(const float* qkv, const AttnParams& p, cudaStream_t st);

// Element-wise / scan kernels (both storage types).
cudaError_t launch_rmsnorm(const void* x, int in_type, const void* g, void* y, int out_type, int M_cap,
                           const int* M_dev, int d, float eps, int* err, cudaStream_t st);
cudaError_t launch_rope(void* qkv, int type, const int* cu, int B, int T_cap, int n_heads, int head_dim, float theta,
                        int* err, int num_sms, cudaStream_t st);
// Per-segment row copies (see aux_kernels.cu): rows of segment b go from src
// rows src_start[b] (+ src_add[b]) to dst rows dst_start[b] (+ dst_add[b]);
// n = (len ? len[b] : src_start[b+1] - src_start[b]) (- len_sub[b]).
// Offsets and sizes in bytes; max_rows bounds any segment's n (grid size).
cudaError_t launch_rows_copy(const void* src, long src_ld, int src_c0, void* dst, long dst_ld, int dst_c0, int row_bytes,
                             const int* src_start, const int* src_add, const int* len, const int* len_sub,
                             const int* dst_start, const int* dst_add, int B, int src_rows, int dst_rows, int max_rows,
                             int* err, cudaStream_t st);
// cu_ctx = exclusive sums of ctx; cu_resp[b] = cu[b] - cu_ctx[b] (either output may be null).
cudaError_t launch_resp_layout(const int* cu, const int* ctx, int B, int* cu_resp, int* cu_ctx, int* err,
                               cudaStream_t st);
// A bounded wait on a barrier that never completes (records kErrTimeout).
cudaError_t launch_wait_selftest(uint64_t limit_ns, int* err, cudaStream_t st);
cudaError_t launch_convert(const void* src, int in_type, void* dst, int out_type, size_t n, int* err, cudaStream_t st);
cudaError_t launch_snr_scan(const int* counts, int B, int N, int F, double tau_jump, double gamma, int window,
                            int* L_star, int* i_star, cudaStream_t st);
cudaError_t launch_pack_route(const void* x_full, int elem_bytes, const int* cu_full, const int* ctx_len,
                              const int* L_star, int B, int d, int N, int T_cap, double tau_pad,
                              int eager_max_bucket, int bucket_min, void* x_packed, int* cu_out, int* kv_out,
                              int* meta_out,
                              int* host_ctrl_dev, int epoch, int* err, int num_sms, cudaStream_t st);

// Sets the message returned by seer_last_error() on this thread.
void set_last_error(const char* msg);

constexpr int kCtrlMaxGroups = 32;
constexpr int kCtrlWords = 8 + 4 * kCtrlMaxGroups;

}  // namespace seer
