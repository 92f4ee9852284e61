// C ABI of libseer (declared in include/seer.h).  Host-side argument checks,
// TMA descriptor encoding, workspace layout and kernel sequencing; all
// arithmetic runs in the kernels of tc_gemm.cu, tc_attn.cu, simt.cu and
// aux_kernels.cu.
#include <cudaTypedefs.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include "../../include/seer.h"
#include "common.cuh"
#include "kernels.h"

using namespace seer;

static_assert(SEER_CTRL_WORDS == seer::kCtrlWords, "control word layout mismatch");
static_assert(SEER_MAX_GROUPS == seer::kCtrlMaxGroups, "control word layout mismatch");
static_assert(static_cast<int>(SEER_F32) == kF32 && static_cast<int>(SEER_BF16) == kBF16 &&
                  static_cast<int>(SEER_F16) == kF16,
              "dtype codes must match the kernels' element types");

namespace {

thread_local std::string g_msg;

seer_status fail(seer_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_msg = buf;
  return st;
}

seer_status cuda_fail(cudaError_t e, const char* where) {
  return fail(SEER_ERR_CUDA, "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
}

#define SEER_CUDA(call, where)                          \
  do {                                                  \
    cudaError_t e_ = (call);                            \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

#define SEER_TRY(expr)                 \
  do {                                 \
    seer_status s_ = (expr);           \
    if (s_ != SEER_OK) return s_;      \
  } while (0)

__device__ int g_dev_err;

struct DeviceInfo {
  int* err = nullptr;
  int num_sms = 0;
};

std::mutex g_dev_mu;
DeviceInfo g_dev[64];

seer_status device_info(DeviceInfo** out) {
  int dev = 0;
  SEER_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(SEER_ERR_CUDA, "device index %d out of range", dev);
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DeviceInfo& di = g_dev[dev];
  if (di.err == nullptr) {
    void* p = nullptr;
    SEER_CUDA(cudaGetSymbolAddress(&p, g_dev_err), "cudaGetSymbolAddress");
    SEER_CUDA(cudaDeviceGetAttribute(&di.num_sms, cudaDevAttrMultiProcessorCount, dev), "cudaDeviceGetAttribute");
    di.err = static_cast<int*>(p);
  }
  *out = &di;
  return SEER_OK;
}

bool valid_dt(seer_dtype dt) { return dt == SEER_F32 || dt == SEER_BF16 || dt == SEER_F16; }
bool is16(seer_dtype dt) { return dt == SEER_BF16 || dt == SEER_F16; }
size_t esize(seer_dtype dt) { return dt == SEER_F32 ? 4 : 2; }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ------------------------------------------------------------ TMA descriptors
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

// Row-major [rows, cols] 16-bit matrix with leading dimension ld elements, in
// boxes of box_cols columns x box_rows rows: 128-byte swizzle for operand
// tiles (64 columns = 128 bytes), none for the GEMM epilogue's store chunks.
seer_status make_map16(CUtensorMap* m, const void* base, seer_dtype dt, uint64_t rows, uint64_t cols, uint64_t ld,
                       uint32_t box_rows, uint32_t box_cols = 64, bool swizzle128 = true) {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (g_encode == nullptr) return fail(SEER_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {cols, rows > 0 ? rows : 1};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapDataType ty = dt == SEER_F16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUresult r = g_encode(m, ty, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SEER_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return SEER_OK;
}

// ------------------------------------------------------------ profiling
struct Profiler {
  std::mutex mu;
  bool on = false;
  uint32_t mask = 0xffffffffu;       // phases recorded while on
  std::vector<cudaEvent_t> pool;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending[SEER_N_PHASES];
  double ms[SEER_N_PHASES] = {};
  int launches[SEER_N_PHASES] = {};
  cudaEvent_t get() {
    if (!pool.empty()) {
      cudaEvent_t e = pool.back();
      pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
  }
};
Profiler g_prof;

// NVTX range names of the phases (same order as seer_profile_read).
const char* const kPhaseNames[SEER_N_PHASES] = {"seer:detect_gemm", "seer:snr_scan", "seer:pack",  "seer:norm1",
                                                 "seer:qkv",         "seer:attention", "seer:o_proj", "seer:norm2",
                                                 "seer:gate_up",     "seer:down",      "seer:kv_cache"};

// Marks one kernel launch: an NVTX range on the host timeline (a no-op unless
// a tool such as nsys or ncu --nvtx is attached), and, when profiling is on,
// a pair of CUDA events on the launch's stream.
class Phase {
 public:
  Phase(int ph, cudaStream_t st) : ph_(ph), st_(st) {
    nvtxRangePushA(kPhaseNames[ph]);
    std::lock_guard<std::mutex> lk(g_prof.mu);
    if (!g_prof.on || ((g_prof.mask >> ph) & 1u) == 0) return;
    a_ = g_prof.get();
    b_ = g_prof.get();
    if (a_ && b_) cudaEventRecord(a_, st_);
  }
  ~Phase() {
    nvtxRangePop();
    if (!a_ || !b_) return;
    cudaEventRecord(b_, st_);
    std::lock_guard<std::mutex> lk(g_prof.mu);
    g_prof.pending[ph_].push_back({a_, b_});
  }

 private:
  int ph_;
  cudaStream_t st_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
};

enum { PH_DETECT = 0, PH_SCAN, PH_PACK, PH_NORM1, PH_QKV, PH_ATTN, PH_OPROJ, PH_NORM2, PH_GATEUP, PH_DOWN, PH_KV };

// ------------------------------------------------------------ workspace
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct LayerWs {
  size_t off_xn, off_qkv, off_h, off_act, off_sched, total;
};


// Intermediates of one layer: fp32 for an fp32 layer, fp16 otherwise.
LayerWs layer_ws(const seer_dims& d, seer_dtype dt, int T_cap, int B) {
  const size_t es = dt == SEER_F32 ? 4 : 2;
  const size_t T = static_cast<size_t>(T_cap);
  LayerWs w;
  size_t o = 0;
  w.off_xn = o; o = align256(o + T * d.d_model * es);
  w.off_qkv = o; o = align256(o + T * 3 * d.d_model * es);
  w.off_h = o; o = align256(o + T * d.d_model * es);
  w.off_act = o; o = align256(o + T * d.d_ff * es);
  w.off_sched = o; o = align256(o + attn_sched_bytes(T_cap, B, d.n_heads));
  w.total = o;
  return w;
}

seer_status check_dims(const seer_dims* dims, seer_dtype dt) {
  if (!dims) return fail(SEER_ERR_INVALID_ARG, "dims is null");
  const seer_dims& d = *dims;
  if (d.d_model <= 0 || d.n_heads <= 0 || d.head_dim <= 0 || d.d_ff <= 0)
    return fail(SEER_ERR_INVALID_ARG, "dims must be positive");
  if (d.n_heads * d.head_dim != d.d_model)
    return fail(SEER_ERR_INVALID_ARG, "n_heads * head_dim (%d) != d_model (%d)", d.n_heads * d.head_dim, d.d_model);
  if (!(d.rope_theta >= 0.f) || !std::isfinite(d.rope_theta))
    return fail(SEER_ERR_INVALID_ARG, "rope_theta must be 0 (off) or a finite positive base");
  if (!(d.rms_eps >= 0.f)) return fail(SEER_ERR_INVALID_ARG, "rms_eps must be >= 0");
  if (is16(dt)) {
    if (d.d_model % 256 != 0) return fail(SEER_ERR_UNSUPPORTED, "16-bit layers need d_model %% 256 == 0 (got %d)", d.d_model);
    if (d.d_ff % 128 != 0) return fail(SEER_ERR_UNSUPPORTED, "16-bit layers need d_ff %% 128 == 0 (got %d)", d.d_ff);
    if (d.head_dim != 128) return fail(SEER_ERR_UNSUPPORTED, "16-bit attention needs head_dim == 128 (got %d)", d.head_dim);
  } else if (dt == SEER_F32) {
    if (d.d_model % 8 != 0 || d.head_dim % 4 != 0 || d.head_dim > 128)
      return fail(SEER_ERR_UNSUPPORTED, "fp32 layers need d_model %% 8 == 0, head_dim %% 4 == 0 and head_dim <= 128");
  } else {
    return fail(SEER_ERR_INVALID_ARG, "unknown dtype %d", static_cast<int>(dt));
  }
  return SEER_OK;
}

// ------------------------------------------------------------ op launchers
// Rotation of the q|k output columns (rotary embedding), applied by do_linear
// when theta > 0: positions come from the segment offsets cu[0..B].
struct RopeArgs {
  float theta = 0.f;
  const int32_t* cu = nullptr;
  int B = 0;
  int n_heads = 0;
  int head_dim = 0;
};

seer_status do_linear(const void* a, const void* w, seer_dtype op_dt, const void* r, seer_dtype r_dt, void* c,
                      seer_dtype c_dt, int M_cap, const int32_t* M_dev, int N, int K, cudaStream_t st, int phase,
                      const RopeArgs& rope = RopeArgs()) {
  if (M_cap < 0 || N <= 0 || K <= 0) return fail(SEER_ERR_INVALID_ARG, "linear: bad sizes M=%d N=%d K=%d", M_cap, N, K);
  if (!a || !w || !c) return fail(SEER_ERR_INVALID_ARG, "linear: null pointer");
  if (!valid_dt(op_dt) || !valid_dt(c_dt) || (r && !valid_dt(r_dt))) return fail(SEER_ERR_INVALID_ARG, "linear: unknown dtype");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  GemmParams p{};
  p.M_cap = M_cap;
  p.M_dev = M_dev;
  p.N = N;
  p.K = K;
  p.C = c;
  p.ldc = N;
  p.R = r;
  p.ldr = N;
  p.err = di->err;
  p.out_type = c_dt;
  p.res_type = r ? r_dt : c_dt;
  const bool rot = rope.theta > 0.f;
  if (rot && (r || !rope.cu || rope.B <= 0 || N != 3 * rope.n_heads * rope.head_dim))
    return fail(SEER_ERR_INVALID_ARG, "linear: the rotary epilogue needs a q|k|v output, cu_seqlens and no residual");
  const int mode = r ? kGemmResidual : (rot ? kGemmRope : kGemmStore);
  if (rot) {
    p.rope_theta = rope.theta;
    p.rope_cols = 2 * rope.n_heads * rope.head_dim;
    p.cu = rope.cu;
    p.B = rope.B;
  }
  if (is16(op_dt)) {
    if (rot && rope.head_dim != 128) return fail(SEER_ERR_UNSUPPORTED, "16-bit rotary epilogue needs head_dim == 128");
    if (!is16(c_dt) || (r && !is16(r_dt))) return fail(SEER_ERR_UNSUPPORTED, "16-bit linear needs 16-bit output and residual");
    if (N % 256 != 0 || K % 64 != 0)
      return fail(SEER_ERR_UNSUPPORTED, "16-bit linear needs N %% 256 == 0 and K %% 64 == 0 (N=%d K=%d)", N, K);
    if (!aligned16(a) || !aligned16(w) || !aligned16(c) || (r && !aligned16(r)))
      return fail(SEER_ERR_UNSUPPORTED, "16-bit linear needs 16-byte aligned pointers");
    if (M_cap == 0) return SEER_OK;
    p.idesc = make_idesc(128, 256, 0, op_dt == SEER_F16);
    p.group_m = tc_gemm_group_m(2l * N * K, 2l * 128 * K);
    CUtensorMap mA, mB, mC;
    SEER_TRY(make_map16(&mA, a, op_dt, M_cap, K, K, 128));
    SEER_TRY(make_map16(&mB, w, op_dt, N, K, K, 128));
    SEER_TRY(make_map16(&mC, c, c_dt, M_cap, N, N, 32, 32, false));
    Phase ph(phase, st);
    SEER_CUDA(launch_tc_gemm(mode, mA, mB, mB, mC, p, di->num_sms, st), "tc_gemm launch");
  } else {
    if (c_dt != SEER_F32 || (r && r_dt != SEER_F32)) return fail(SEER_ERR_UNSUPPORTED, "fp32 linear needs fp32 output");
    if (M_cap == 0) return SEER_OK;
    Phase ph(phase, st);
    SEER_CUDA(launch_simt_gemm(rot ? kGemmStore : mode, static_cast<const float*>(a), static_cast<const float*>(w),
                               nullptr, p, st),
              "simt_gemm launch");
    if (rot)
      SEER_CUDA(launch_rope(c, kF32, rope.cu, rope.B, M_cap, rope.n_heads, rope.head_dim, rope.theta, di->err,
                            di->num_sms, st),
                "rope launch");
  }
  return SEER_OK;
}

seer_status do_swiglu(const void* a, const void* wg, const void* wu, seer_dtype op_dt, void* act, seer_dtype act_dt,
                      int M_cap, const int32_t* M_dev, int F, int K, const int32_t* cu, int B, const int32_t* resp_start,
                      int N, float act_eps, int32_t* counts, cudaStream_t st, int mode, int phase,
                      bool accumulate = false) {
  if (M_cap < 0 || F <= 0 || K <= 0) return fail(SEER_ERR_INVALID_ARG, "swiglu: bad sizes");
  if (!a || !wg || !wu) return fail(SEER_ERR_INVALID_ARG, "swiglu: null pointer");
  if (!valid_dt(op_dt) || (mode == kGemmSwiglu && !valid_dt(act_dt))) return fail(SEER_ERR_INVALID_ARG, "swiglu: unknown dtype");
  if (mode == kGemmSwiglu && !act) return fail(SEER_ERR_INVALID_ARG, "swiglu: null output");
  if (counts && (B <= 0 || N <= 0 || !resp_start || (mode == kGemmSwiglu && !cu)))
    return fail(SEER_ERR_INVALID_ARG, "swiglu: counting needs B, N, resp_start and cu_seqlens");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  GemmParams p{};
  p.M_cap = M_cap;
  p.M_dev = M_dev;
  p.N = F;
  p.K = K;
  p.C = act;
  p.ldc = F;
  p.counts = counts;
  p.act_eps = act_eps;
  p.cu = cu;
  p.B = B;
  p.resp_start = resp_start;
  p.Nw = N;
  p.err = di->err;
  p.out_type = act_dt;
  p.res_type = act_dt;
  if (is16(op_dt)) {
    if (mode == kGemmSwiglu && !is16(act_dt)) return fail(SEER_ERR_UNSUPPORTED, "16-bit swiglu needs a 16-bit output");
    if (F % 128 != 0 || K % 64 != 0)
      return fail(SEER_ERR_UNSUPPORTED, "16-bit swiglu needs F %% 128 == 0 and K %% 64 == 0 (F=%d K=%d)", F, K);
    if (!aligned16(a) || !aligned16(wg) || !aligned16(wu) || (act && !aligned16(act)))
      return fail(SEER_ERR_UNSUPPORTED, "16-bit swiglu needs 16-byte aligned pointers");
  } else if (mode == kGemmSwiglu && act_dt != SEER_F32) {
    return fail(SEER_ERR_UNSUPPORTED, "fp32 swiglu needs an fp32 output");
  }
  if (counts && !accumulate)
    SEER_CUDA(cudaMemsetAsync(counts, 0, sizeof(int32_t) * static_cast<size_t>(B) * N, st), "memset counts");
  if (M_cap == 0) return SEER_OK;
  if (is16(op_dt)) {
    p.idesc = make_idesc(128, 256, 0, op_dt == SEER_F16);
    p.group_m = tc_gemm_group_m(2l * 2 * F * K, 2l * 128 * K);
    CUtensorMap mA, mG, mU, mC;
    SEER_TRY(make_map16(&mA, a, op_dt, M_cap, K, K, 128));
    SEER_TRY(make_map16(&mG, wg, op_dt, F, K, K, 128));
    SEER_TRY(make_map16(&mU, wu, op_dt, F, K, K, 128));
    if (mode == kGemmSwiglu) SEER_TRY(make_map16(&mC, act, act_dt, M_cap, F, F, 32, 32, false));
    else mC = mA;                                  // Count stores nothing
    Phase ph(phase, st);
    SEER_CUDA(launch_tc_gemm(mode, mA, mG, mU, mC, p, di->num_sms, st), "tc_gemm launch");
  } else {
    Phase ph(phase, st);
    SEER_CUDA(launch_simt_gemm(mode, static_cast<const float*>(a), static_cast<const float*>(wg),
                               static_cast<const float*>(wu), p, st),
              "simt_gemm launch");
  }
  return SEER_OK;
}

seer_status do_rmsnorm(const void* x, seer_dtype x_dt, const void* g, void* y, seer_dtype y_dt, int M_cap,
                       const int32_t* M_dev, int d, float eps, cudaStream_t st, int phase) {
  if (!x || !g || !y) return fail(SEER_ERR_INVALID_ARG, "rmsnorm: null pointer");
  if (M_cap < 0 || d <= 0) return fail(SEER_ERR_INVALID_ARG, "rmsnorm: bad sizes");
  if (!valid_dt(x_dt) || !valid_dt(y_dt)) return fail(SEER_ERR_INVALID_ARG, "rmsnorm: unknown dtype");
  if (d % 8 != 0) return fail(SEER_ERR_UNSUPPORTED, "rmsnorm needs d %% 8 == 0");
  if (!aligned16(x) || !aligned16(g) || !aligned16(y)) return fail(SEER_ERR_UNSUPPORTED, "rmsnorm needs 16-byte aligned pointers");
  const bool ok = (x_dt == SEER_BF16 && (y_dt == SEER_F16 || y_dt == SEER_BF16)) || (x_dt == SEER_F16 && y_dt == SEER_F16) ||
                  (x_dt == SEER_F32 && y_dt == SEER_F32);
  if (!ok) return fail(SEER_ERR_UNSUPPORTED, "rmsnorm: unsupported type pair %d -> %d", x_dt, y_dt);
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  Phase ph(phase, st);
  SEER_CUDA(launch_rmsnorm(x, x_dt, g, y, y_dt, M_cap, M_dev, d, eps, di->err, st), "rmsnorm launch");
  return SEER_OK;
}

// Where an attention call finds its keys and values (default: the K and V
// column blocks of the qkv buffer itself, rows shared with the queries).
struct KvSource {
  const void* kv = nullptr;      // [T_kv_cap, ld] rows holding K | V
  int ld = 0;                    // elements per row
  int xk0 = 0, xv0 = 0;          // columns of head 0's K and V
  const int32_t* cu_kv = nullptr;
  int T_kv_cap = 0;
};

seer_status do_attention(const void* qkv, void* o, seer_dtype dt, const int32_t* cu, const int32_t* kv_len, int B,
                         int T_cap, int H, int dh, void* sched, size_t sched_bytes, cudaStream_t st,
                         const KvSource& kvs = KvSource()) {
  if (!qkv || !o || !cu) return fail(SEER_ERR_INVALID_ARG, "attention: null pointer");
  if (kvs.kv && (!kvs.cu_kv || kvs.T_kv_cap < 0 || kvs.ld < 2 * H * dh))
    return fail(SEER_ERR_INVALID_ARG, "attention: a separate K/V source needs cu_kv, a capacity and rows of >= 2*H*dh");
  if (B <= 0 || T_cap < 0 || H <= 0 || dh <= 0) return fail(SEER_ERR_INVALID_ARG, "attention: bad sizes");
  if (!valid_dt(dt)) return fail(SEER_ERR_INVALID_ARG, "attention: unknown dtype");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  AttnParams p{};
  p.cu = cu;
  p.kv_len = kv_len;
  p.B = B;
  p.T_cap = T_cap;
  p.n_heads = H;
  p.head_dim = dh;
  p.out = o;
  p.ldo = H * dh;
  p.err = di->err;
  p.kv = kvs.kv;
  p.cu_kv = kvs.kv ? kvs.cu_kv : nullptr;
  p.ld_kv = kvs.kv ? kvs.ld : 3 * H * dh;
  p.xk0 = kvs.kv ? kvs.xk0 : H * dh;
  p.xv0 = kvs.kv ? kvs.xv0 : 2 * H * dh;
  if (is16(dt)) {
    if (dh != 128) return fail(SEER_ERR_UNSUPPORTED, "16-bit attention needs head_dim == 128");
    if (kvs.kv && (!aligned16(kvs.kv) || (static_cast<long>(kvs.ld) * 2) % 16 != 0 || kvs.xk0 % 64 != 0 || kvs.xv0 % 64 != 0))
      return fail(SEER_ERR_UNSUPPORTED, "attention: K/V rows must be 16-byte aligned with 64-element column offsets");
    const size_t need = attn_sched_bytes(T_cap, B, H);
    if (!sched || sched_bytes < need)
      return fail(SEER_ERR_WORKSPACE, "attention needs %zu bytes of schedule workspace", need);
    if (!aligned16(qkv) || !aligned16(o) || !aligned16(sched))
      return fail(SEER_ERR_UNSUPPORTED, "attention needs 16-byte aligned pointers");
    if (T_cap == 0) return SEER_OK;
    const int max_units = static_cast<int>(static_cast<size_t>(H) * ((T_cap + 127) / 128 + B));
    int4* work = static_cast<int4*>(sched);
    int* count = reinterpret_cast<int*>(static_cast<uint8_t*>(sched) + align256(static_cast<size_t>(max_units) * sizeof(int4)));
    p.work = work;
    p.work_count = count;
    p.work_next = count + 1;
    CUtensorMap m, mkv;
    SEER_TRY(make_map16(&m, qkv, dt, T_cap, 3 * H * dh, 3 * H * dh, 128));
    if (kvs.kv) SEER_TRY(make_map16(&mkv, kvs.kv, dt, kvs.T_kv_cap > 0 ? kvs.T_kv_cap : 1, kvs.ld, kvs.ld, 128));
    SEER_CUDA(launch_attn_schedule(cu, p.cu_kv, kv_len, B, H, T_cap, work, count, max_units, di->err, st),
              "attn schedule");
    // the attention phase brackets the attention kernel alone (the one-block
    // schedule kernel before it takes a few microseconds)
    Phase ph(PH_ATTN, st);
    // persistent: one CTA per SM (at most one per unit)
    SEER_CUDA(launch_tc_attn(m, kvs.kv ? mkv : m, p, std::min(max_units, di->num_sms), dt == SEER_F16, st),
              "tc_attn launch");
  } else {
    if (dh > 128 || dh % 4 != 0) return fail(SEER_ERR_UNSUPPORTED, "fp32 attention needs head_dim <= 128, %% 4 == 0");
    if (T_cap == 0) return SEER_OK;
    Phase ph(PH_ATTN, st);
    SEER_CUDA(launch_simt_attn(static_cast<const float*>(qkv), p, st), "simt_attn launch");
  }
  return SEER_OK;
}

}  // namespace

namespace {
std::atomic<int> g_launch_overlap{1};
}  // namespace

namespace seer {
size_t attn_sched_bytes(int T_cap, int B, int H) {
  const size_t units = static_cast<size_t>(H) * (static_cast<size_t>((T_cap + 127) / 128) + static_cast<size_t>(B));
  return ((units * sizeof(int4) + 255) & ~size_t(255)) + 256;
}

// Lets other translation units of the library report a message through
// seer_last_error().
void set_last_error(const char* msg) { g_msg = msg; }
bool launch_overlap_enabled() { return g_launch_overlap.load(std::memory_order_relaxed) != 0; }
}  // namespace seer

extern "C" {

const char* seer_last_error(void) { return g_msg.c_str(); }

const char* seer_version(void) { return "libseer 0.2 (sm_103a)"; }

int seer_set_launch_overlap(int on) { return g_launch_overlap.exchange(on ? 1 : 0); }

int seer_num_sms(void) {
  DeviceInfo* di;
  if (device_info(&di) != SEER_OK) return -1;
  return di->num_sms;
}

seer_status seer_check_device(int* code_out) {
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  SEER_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
  int code = 0, zero = 0;
  SEER_CUDA(cudaMemcpyFromSymbol(&code, g_dev_err, sizeof(int)), "read device error");
  SEER_CUDA(cudaMemcpyToSymbol(g_dev_err, &zero, sizeof(int)), "clear device error");
  if (code_out) *code_out = code;
  if (code != 0) return fail(SEER_ERR_DEVICE, "device-side error code %d", code);
  return SEER_OK;
}

seer_status seer_selftest_wait_timeout(int limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 10000000) return fail(SEER_ERR_INVALID_ARG, "selftest: limit_us must be in [1, 1e7]");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  SEER_CUDA(launch_wait_selftest(static_cast<uint64_t>(limit_us) * 1000ull, di->err, static_cast<cudaStream_t>(stream)),
            "wait selftest launch");
  return SEER_OK;
}

seer_status seer_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  g_prof.on = on != 0;
  return SEER_OK;
}

seer_status seer_profile_select(uint32_t phase_mask) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  g_prof.mask = phase_mask;
  return SEER_OK;
}

seer_status seer_profile_reset(void) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  for (int i = 0; i < SEER_N_PHASES; ++i) {
    for (auto& pr : g_prof.pending[i]) {
      cudaEventSynchronize(pr.second);
      g_prof.pool.push_back(pr.first);
      g_prof.pool.push_back(pr.second);
    }
    g_prof.pending[i].clear();
    g_prof.ms[i] = 0;
    g_prof.launches[i] = 0;
  }
  return SEER_OK;
}

seer_status seer_profile_read(float* ms_out, int32_t* launches_out) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  for (int i = 0; i < SEER_N_PHASES; ++i) {
    for (auto& pr : g_prof.pending[i]) {
      cudaError_t e = cudaEventSynchronize(pr.second);
      if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
      float ms = 0.f;
      e = cudaEventElapsedTime(&ms, pr.first, pr.second);
      if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
      g_prof.ms[i] += ms;
      g_prof.launches[i] += 1;
      g_prof.pool.push_back(pr.first);
      g_prof.pool.push_back(pr.second);
    }
    g_prof.pending[i].clear();
    if (ms_out) ms_out[i] = static_cast<float>(g_prof.ms[i]);
    if (launches_out) launches_out[i] = g_prof.launches[i];
  }
  return SEER_OK;
}

seer_status seer_convert(const void* src, seer_dtype src_dt, void* dst, seer_dtype dst_dt, size_t n, void* stream) {
  if (!src || !dst) return fail(SEER_ERR_INVALID_ARG, "convert: null pointer");
  if (!valid_dt(src_dt) || !valid_dt(dst_dt) || src_dt == dst_dt) return fail(SEER_ERR_INVALID_ARG, "convert: bad dtypes");
  if (n % 8 != 0) return fail(SEER_ERR_UNSUPPORTED, "convert: n must be a multiple of 8");
  if (!aligned16(src) || !aligned16(dst)) return fail(SEER_ERR_UNSUPPORTED, "convert: 16-byte aligned pointers required");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  SEER_CUDA(launch_convert(src, src_dt, dst, dst_dt, n, di->err, static_cast<cudaStream_t>(stream)), "convert launch");
  return SEER_OK;
}

seer_status seer_rmsnorm(const void* x, seer_dtype x_dt, const void* g, void* y, seer_dtype y_dt, int M_cap,
                         const int32_t* M_dev, int d, float eps, void* stream) {
  return do_rmsnorm(x, x_dt, g, y, y_dt, M_cap, M_dev, d, eps, static_cast<cudaStream_t>(stream), PH_NORM1);
}

seer_status seer_linear(const void* a, const void* w, seer_dtype op_dt, const void* r, seer_dtype r_dt, void* c,
                        seer_dtype c_dt, int M_cap, const int32_t* M_dev, int N, int K, void* stream) {
  return do_linear(a, w, op_dt, r, r_dt, c, c_dt, M_cap, M_dev, N, K, static_cast<cudaStream_t>(stream),
                   r ? PH_OPROJ : PH_QKV);
}

seer_status seer_rope(void* qkv, seer_dtype dt, const int32_t* cu_seqlens, int B, int T_capacity, int n_heads,
                      int head_dim, float theta, void* stream) {
  if (!valid_dt(dt)) return fail(SEER_ERR_INVALID_ARG, "rope: unknown dtype");
  if (!qkv || !cu_seqlens) return fail(SEER_ERR_INVALID_ARG, "rope: null pointer");
  if (B <= 0 || T_capacity < 0 || n_heads <= 0 || head_dim <= 0) return fail(SEER_ERR_INVALID_ARG, "rope: bad sizes");
  if (!(theta > 0.f) || !std::isfinite(theta)) return fail(SEER_ERR_INVALID_ARG, "rope: theta must be finite and > 0");
  if (head_dim % 2 != 0 || head_dim > 128) return fail(SEER_ERR_UNSUPPORTED, "rope: head_dim must be even and <= 128");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Phase ph(PH_QKV, st);
  SEER_CUDA(launch_rope(qkv, dt, cu_seqlens, B, T_capacity, n_heads, head_dim, theta, di->err, di->num_sms, st),
            "rope launch");
  return SEER_OK;
}

seer_status seer_swiglu(const void* a, const void* w_gate, const void* w_up, seer_dtype op_dt, void* act,
                        seer_dtype act_dt, int M_cap, const int32_t* M_dev, int F, int K, const int32_t* cu_seqlens,
                        int B, const int32_t* count_resp_start, int N, float act_eps, int32_t* counts_out,
                        void* stream) {
  if (count_resp_start && !counts_out) return fail(SEER_ERR_INVALID_ARG, "swiglu: counts_out is null");
  return do_swiglu(a, w_gate, w_up, op_dt, act, act_dt, M_cap, M_dev, F, K, cu_seqlens, B, count_resp_start, N,
                   act_eps, count_resp_start ? counts_out : nullptr, static_cast<cudaStream_t>(stream), kGemmSwiglu,
                   PH_GATEUP);
}

seer_status seer_attention(const void* qkv, void* o, seer_dtype dt, const int32_t* cu_seqlens, const int32_t* kv_len,
                           int B, int T_capacity, int n_heads, int head_dim, void* ws, size_t ws_bytes, void* stream) {
  return do_attention(qkv, o, dt, cu_seqlens, kv_len, B, T_capacity, n_heads, head_dim, ws, ws_bytes,
                      static_cast<cudaStream_t>(stream));
}

seer_status seer_detect_boundary(const void* x, seer_dtype dt, int T_rows, const int32_t* resp_start, int B, int N,
                                 const void* w_gate, const void* w_up, const seer_dims* dims, const seer_params* params,
                                 int32_t* counts_out, int32_t* L_star_out, int32_t* i_star_out, void* stream) {
  SEER_TRY(check_dims(dims, dt));
  if (!params) return fail(SEER_ERR_INVALID_ARG, "params is null");
  if (!x || !resp_start || !w_gate || !w_up || !counts_out || !L_star_out)
    return fail(SEER_ERR_INVALID_ARG, "detect: null pointer");
  if (B <= 0 || N <= 0 || T_rows < N) return fail(SEER_ERR_INVALID_ARG, "detect: need B >= 1, N >= 1, T_rows >= N");
  if (params->window < 1) return fail(SEER_ERR_INVALID_ARG, "window must be >= 1");
  if (!(params->gamma >= 0.0) || !(params->tau_jump >= 0.0)) return fail(SEER_ERR_INVALID_ARG, "tau_jump and gamma must be >= 0");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  SEER_TRY(do_swiglu(x, w_gate, w_up, dt, nullptr, dt, T_rows, nullptr, dims->d_ff, dims->d_model, nullptr, B,
                     resp_start, N, params->act_eps, counts_out, st, kGemmCount, PH_DETECT));
  Phase ph(PH_SCAN, st);
  SEER_CUDA(launch_snr_scan(counts_out, B, N, dims->d_ff, params->tau_jump, params->gamma, params->window, L_star_out,
                            i_star_out, st),
            "snr scan launch");
  return SEER_OK;
}

seer_status seer_sparsity_counts(const void* x, seer_dtype dt, int T_rows, const int32_t* resp_start, int B, int N,
                                 const void* w_gate, const void* w_up, const seer_dims* dims, float act_eps,
                                 int accumulate, int32_t* counts_inout, void* stream) {
  SEER_TRY(check_dims(dims, dt));
  if (!x || !resp_start || !w_gate || !w_up || !counts_inout) return fail(SEER_ERR_INVALID_ARG, "counts: null pointer");
  if (B <= 0 || N <= 0 || T_rows < N) return fail(SEER_ERR_INVALID_ARG, "counts: need B >= 1, N >= 1, T_rows >= N");
  return do_swiglu(x, w_gate, w_up, dt, nullptr, dt, T_rows, nullptr, dims->d_ff, dims->d_model, nullptr, B, resp_start,
                   N, act_eps, counts_inout, static_cast<cudaStream_t>(stream), kGemmCount, PH_DETECT, accumulate != 0);
}

seer_status seer_snr_scan(const int32_t* counts, int B, int N, int F, const seer_params* params, int32_t* L_star_out,
                          int32_t* i_star_out, void* stream) {
  if (!counts || !params || !L_star_out) return fail(SEER_ERR_INVALID_ARG, "scan: null pointer");
  if (B <= 0 || N <= 0 || F <= 0 || params->window < 1) return fail(SEER_ERR_INVALID_ARG, "scan: bad sizes");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Phase ph(PH_SCAN, st);
  SEER_CUDA(launch_snr_scan(counts, B, N, F, params->tau_jump, params->gamma, params->window, L_star_out, i_star_out, st),
            "snr scan launch");
  return SEER_OK;
}

seer_status seer_pack_ragged(const void* x_full, seer_dtype dt, const int32_t* cu_full, const int32_t* ctx_len,
                             const int32_t* L_star, int B, int d, int N, int T_capacity, const seer_params* params,
                             void* x_packed, int32_t* cu_out, int32_t* kv_len_out, int32_t* meta_out,
                             int32_t* host_ctrl, int32_t epoch, void* stream) {
  if (!valid_dt(dt)) return fail(SEER_ERR_INVALID_ARG, "unknown dtype");
  if (!params) return fail(SEER_ERR_INVALID_ARG, "params is null");
  if (!x_full || !cu_full || !ctx_len || !L_star || !x_packed || !cu_out || !kv_len_out || !meta_out)
    return fail(SEER_ERR_INVALID_ARG, "pack: null pointer");
  if (B <= 0 || d <= 0 || N <= 0 || T_capacity < 0) return fail(SEER_ERR_INVALID_ARG, "pack: bad sizes");
  if (params->bucket_min < 1) return fail(SEER_ERR_INVALID_ARG, "pack: bucket_min must be >= 1");
  const int es = static_cast<int>(esize(dt));
  if ((static_cast<long>(d) * es) % 16 != 0) return fail(SEER_ERR_UNSUPPORTED, "pack: rows must be a multiple of 16 bytes");
  if (!aligned16(x_full) || !aligned16(x_packed)) return fail(SEER_ERR_UNSUPPORTED, "pack: 16-byte aligned pointers required");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  int* hc_dev = nullptr;
  if (host_ctrl) {
    void* dp = nullptr;
    cudaError_t e = cudaHostGetDevicePointer(&dp, host_ctrl, 0);
    if (e != cudaSuccess)
      return fail(SEER_ERR_INVALID_ARG, "host_ctrl is not pinned, device-mapped memory (%s)", cudaGetErrorName(e));
    hc_dev = static_cast<int*>(dp);
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Phase ph(PH_PACK, st);
  SEER_CUDA(launch_pack_route(x_full, es, cu_full, ctx_len, L_star, B, d, N, T_capacity, params->tau_pad,
                              params->eager_max_bucket, params->bucket_min, x_packed, cu_out, kv_len_out, meta_out,
                              hc_dev, epoch, di->err,
                              di->num_sms, st),
            "pack launch");
  return SEER_OK;
}

seer_status seer_poll_ctrl(const int32_t* host_ctrl, int32_t epoch, int timeout_us, int32_t* ctrl_copy) {
  if (!host_ctrl) return fail(SEER_ERR_INVALID_ARG, "host_ctrl is null");
  const volatile int32_t* w = host_ctrl;
  const auto t0 = std::chrono::steady_clock::now();
  long spins = 0;
  while (w[0] != epoch) {
    if ((++spins & 1023) == 0) {
      const auto us = std::chrono::duration_cast<std::chrono::microseconds>(std::chrono::steady_clock::now() - t0).count();
      if (us > timeout_us) return fail(SEER_ERR_TIMEOUT, "control word not ready after %d us", timeout_us);
      std::this_thread::yield();
    }
  }
  std::atomic_thread_fence(std::memory_order_acquire);
  if (ctrl_copy)
    for (int i = 0; i < SEER_CTRL_WORDS; ++i) ctrl_copy[i] = w[i];
  return SEER_OK;
}

seer_status seer_layer_workspace_size(const seer_dims* dims, seer_dtype dt, int T_capacity, int B, size_t* bytes) {
  SEER_TRY(check_dims(dims, dt));
  if (T_capacity < 0 || B <= 0 || !bytes) return fail(SEER_ERR_INVALID_ARG, "workspace: bad arguments");
  *bytes = layer_ws(*dims, dt, T_capacity, B).total;
  return SEER_OK;
}

seer_status seer_layer_forward(const seer_layer_weights* w, const seer_dims* dims, seer_dtype dt, const void* x, void* y,
                               const int32_t* cu_seqlens, const int32_t* kv_len, int B, int T_capacity,
                               const int32_t* count_resp_start, int N, float act_eps, int32_t* counts_out, void* ws,
                               size_t ws_bytes, void* stream) {
  SEER_TRY(check_dims(dims, dt));
  if (!w || !w->w_qkv || !w->w_o || !w->w_gate || !w->w_up || !w->w_down || !w->g_attn || !w->g_mlp)
    return fail(SEER_ERR_INVALID_ARG, "layer: null weight pointer");
  if (!x || !y || !cu_seqlens) return fail(SEER_ERR_INVALID_ARG, "layer: null pointer");
  if (x == y) return fail(SEER_ERR_INVALID_ARG, "layer: y must not alias x");
  if (B <= 0 || T_capacity < 0) return fail(SEER_ERR_INVALID_ARG, "layer: bad sizes");
  if (count_resp_start && (!counts_out || N <= 0)) return fail(SEER_ERR_INVALID_ARG, "layer: counting needs counts_out and N");
  const LayerWs L = layer_ws(*dims, dt, T_capacity, B);
  if (!ws || ws_bytes < L.total) return fail(SEER_ERR_WORKSPACE, "layer needs %zu bytes of workspace", L.total);
  if (!aligned16(ws) || !aligned16(x) || !aligned16(y)) return fail(SEER_ERR_UNSUPPORTED, "layer needs 16-byte aligned pointers");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int d = dims->d_model, F = dims->d_ff, H = dims->n_heads, dh = dims->head_dim;
  // x and y keep the layer dtype; weights and every intermediate are f16 for
  // a 16-bit layer (f32 for an f32 layer).
  const seer_dtype it = dt == SEER_F32 ? SEER_F32 : SEER_F16;
  uint8_t* base = static_cast<uint8_t*>(ws);
  void* xn = base + L.off_xn;
  void* qkv = base + L.off_qkv;
  void* h = base + L.off_h;
  void* act = base + L.off_act;
  void* sched = base + L.off_sched;
  const int32_t* M_dev = cu_seqlens + B;   // device total rows
  const float eps = dims->rms_eps;

  SEER_TRY(do_rmsnorm(x, dt, w->g_attn, xn, it, T_capacity, M_dev, d, eps, st, PH_NORM1));
  RopeArgs rope;
  rope.theta = dims->rope_theta;
  rope.cu = cu_seqlens;
  rope.B = B;
  rope.n_heads = H;
  rope.head_dim = dh;
  SEER_TRY(do_linear(xn, w->w_qkv, it, nullptr, it, qkv, it, T_capacity, M_dev, 3 * d, d, st, PH_QKV, rope));
  SEER_TRY(do_attention(qkv, xn, it, cu_seqlens, kv_len, B, T_capacity, H, dh, sched, L.total - L.off_sched, st));
  SEER_TRY(do_linear(xn, w->w_o, it, x, dt, h, it, T_capacity, M_dev, d, d, st, PH_OPROJ));
  SEER_TRY(do_rmsnorm(h, it, w->g_mlp, xn, it, T_capacity, M_dev, d, eps, st, PH_NORM2));
  SEER_TRY(do_swiglu(xn, w->w_gate, w->w_up, it, act, it, T_capacity, M_dev, F, d, cu_seqlens, B, count_resp_start, N,
                     act_eps, count_resp_start ? counts_out : nullptr, st, kGemmSwiglu, PH_GATEUP));
  SEER_TRY(do_linear(act, w->w_down, it, h, it, y, dt, T_capacity, M_dev, d, F, st, PH_DOWN));
  return SEER_OK;
}


seer_status seer_gather_response(const void* x_packed, seer_dtype dt, const int32_t* cu, const int32_t* ctx_len, int B,
                                 int d, int T_cap, void* x_resp, int32_t* cu_resp_out, void* stream) {
  if (!valid_dt(dt)) return fail(SEER_ERR_INVALID_ARG, "gather: unknown dtype");
  if (!x_packed || !cu || !ctx_len || !x_resp || !cu_resp_out) return fail(SEER_ERR_INVALID_ARG, "gather: null pointer");
  if (B <= 0 || d <= 0 || T_cap < 0) return fail(SEER_ERR_INVALID_ARG, "gather: bad sizes");
  const long row = static_cast<long>(d) * static_cast<long>(esize(dt));
  if (row % 16 != 0 || !aligned16(x_packed) || !aligned16(x_resp))
    return fail(SEER_ERR_UNSUPPORTED, "gather: 16-byte aligned rows required");
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Phase ph(PH_KV, st);
  SEER_CUDA(launch_resp_layout(cu, ctx_len, B, cu_resp_out, nullptr, di->err, st), "response layout");
  SEER_CUDA(launch_rows_copy(x_packed, row, 0, x_resp, row, 0, static_cast<int>(row), cu, ctx_len, nullptr, ctx_len,
                             cu_resp_out, nullptr, B, T_cap, T_cap, T_cap, di->err, st),
            "response gather");
  return SEER_OK;
}

seer_status seer_kv_prefill(const seer_layer_weights* w, const seer_dims* dims, seer_dtype dt, const void* x,
                            const int32_t* cu_x, const int32_t* ctx_len, int B, int T_x_cap, void* kv_cache,
                            const int32_t* cu_kv, int T_kv_cap, void* ws, size_t ws_bytes, void* stream) {
  SEER_TRY(check_dims(dims, dt));
  if (!w || !w->w_qkv || !w->g_attn) return fail(SEER_ERR_INVALID_ARG, "prefill: null weight pointer");
  if (!x || !cu_x || !ctx_len || !kv_cache || !cu_kv) return fail(SEER_ERR_INVALID_ARG, "prefill: null pointer");
  if (B <= 0 || T_x_cap < 0 || T_kv_cap < 0) return fail(SEER_ERR_INVALID_ARG, "prefill: bad sizes");
  if (dims->rope_theta != 0.f) return fail(SEER_ERR_UNSUPPORTED, "the K/V cache path has no rotary embedding");
  const LayerWs L = layer_ws(*dims, dt, T_x_cap, B);
  if (!ws || ws_bytes < L.total) return fail(SEER_ERR_WORKSPACE, "prefill needs %zu bytes of workspace", L.total);
  if (!aligned16(ws) || !aligned16(x) || !aligned16(kv_cache)) return fail(SEER_ERR_UNSUPPORTED, "prefill needs 16-byte aligned pointers");
  if (T_x_cap == 0) return SEER_OK;
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int d = dims->d_model, D2 = 2 * dims->n_heads * dims->head_dim;
  const seer_dtype it = dt == SEER_F32 ? SEER_F32 : SEER_F16;
  const long xrow = static_cast<long>(d) * esize(dt), irow = static_cast<long>(d) * esize(it);
  const long kvrow = static_cast<long>(D2) * esize(it);
  uint8_t* base = static_cast<uint8_t*>(ws);
  void* xp = base + L.off_h;                     // prefix rows, packed  [sum ctx, d]
  void* xn = base + L.off_xn;                    // normalised           [sum ctx, d]
  void* kvp = base + L.off_qkv;                  // their K | V          [sum ctx, 2D]
  int32_t* cu_ctx = reinterpret_cast<int32_t*>(base + L.off_sched);   // [B+1], before the (unused) schedule
  {
    Phase ph(PH_KV, st);
    SEER_CUDA(launch_resp_layout(nullptr, ctx_len, B, nullptr, cu_ctx, di->err, st), "prefix layout");
    SEER_CUDA(launch_rows_copy(x, xrow, 0, xp, xrow, 0, static_cast<int>(xrow), cu_x, nullptr, ctx_len, nullptr, cu_ctx,
                               nullptr, B, T_x_cap, T_x_cap, T_x_cap, di->err, st),
              "prefix gather");
  }
  SEER_TRY(do_rmsnorm(xp, dt, w->g_attn, xn, it, T_x_cap, cu_ctx + B, d, dims->rms_eps, st, PH_KV));
  const void* w_kv = static_cast<const uint8_t*>(w->w_qkv) + static_cast<size_t>(D2 / 2) * d * esize(it);
  SEER_TRY(do_linear(xn, w_kv, it, nullptr, it, kvp, it, T_x_cap, cu_ctx + B, D2, d, st, PH_KV));
  Phase ph(PH_KV, st);
  SEER_CUDA(launch_rows_copy(kvp, kvrow, 0, kv_cache, kvrow, 0, static_cast<int>(kvrow), cu_ctx, nullptr, nullptr, nullptr,
                             cu_kv, nullptr, B, T_x_cap, T_kv_cap, T_x_cap, di->err, st),
            "prefix K/V scatter");
  return SEER_OK;
}

seer_status seer_layer_forward_cached(const seer_layer_weights* w, const seer_dims* dims, seer_dtype dt,
                                      const void* x_resp, void* y_resp, const int32_t* cu_resp, const int32_t* ctx_len,
                                      int B, int T_resp_cap, void* kv_cache, const int32_t* cu_kv,
                                      const int32_t* kv_len, int T_kv_cap, void* ws, size_t ws_bytes, void* stream) {
  SEER_TRY(check_dims(dims, dt));
  if (!w || !w->w_qkv || !w->w_o || !w->w_gate || !w->w_up || !w->w_down || !w->g_attn || !w->g_mlp)
    return fail(SEER_ERR_INVALID_ARG, "cached layer: null weight pointer");
  if (!x_resp || !y_resp || !cu_resp || !ctx_len || !kv_cache || !cu_kv)
    return fail(SEER_ERR_INVALID_ARG, "cached layer: null pointer");
  if (x_resp == y_resp) return fail(SEER_ERR_INVALID_ARG, "cached layer: y must not alias x");
  if (B <= 0 || T_resp_cap < 0 || T_kv_cap < 0) return fail(SEER_ERR_INVALID_ARG, "cached layer: bad sizes");
  if (dims->rope_theta != 0.f) return fail(SEER_ERR_UNSUPPORTED, "the K/V cache path has no rotary embedding");
  const LayerWs L = layer_ws(*dims, dt, T_resp_cap, B);
  if (!ws || ws_bytes < L.total) return fail(SEER_ERR_WORKSPACE, "cached layer needs %zu bytes of workspace", L.total);
  if (!aligned16(ws) || !aligned16(x_resp) || !aligned16(y_resp) || !aligned16(kv_cache))
    return fail(SEER_ERR_UNSUPPORTED, "cached layer needs 16-byte aligned pointers");
  if (T_resp_cap == 0) return SEER_OK;
  DeviceInfo* di;
  SEER_TRY(device_info(&di));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int d = dims->d_model, F = dims->d_ff, H = dims->n_heads, dh = dims->head_dim, D = H * dh;
  const seer_dtype it = dt == SEER_F32 ? SEER_F32 : SEER_F16;
  const long es = static_cast<long>(esize(it));
  uint8_t* base = static_cast<uint8_t*>(ws);
  void* xn = base + L.off_xn;
  void* qkv = base + L.off_qkv;
  void* h = base + L.off_h;
  void* act = base + L.off_act;
  void* sched = base + L.off_sched;
  const int32_t* M_dev = cu_resp + B;
  const float eps = dims->rms_eps;

  SEER_TRY(do_rmsnorm(x_resp, dt, w->g_attn, xn, it, T_resp_cap, M_dev, d, eps, st, PH_NORM1));
  SEER_TRY(do_linear(xn, w->w_qkv, it, nullptr, it, qkv, it, T_resp_cap, M_dev, 3 * d, d, st, PH_QKV));
  {
    // the response rows' K | V into the cache, after each segment's prefix
    Phase ph(PH_KV, st);
    SEER_CUDA(launch_rows_copy(qkv, 3 * D * es, static_cast<int>(D * es), kv_cache, 2 * D * es, 0,
                               static_cast<int>(2 * D * es), cu_resp, nullptr, nullptr, nullptr, cu_kv, ctx_len, B,
                               T_resp_cap, T_kv_cap, T_resp_cap, di->err, st),
              "response K/V scatter");
  }
  KvSource kvs;
  kvs.kv = kv_cache;
  kvs.ld = 2 * D;
  kvs.xk0 = 0;
  kvs.xv0 = D;
  kvs.cu_kv = cu_kv;
  kvs.T_kv_cap = T_kv_cap;
  SEER_TRY(do_attention(qkv, xn, it, cu_resp, kv_len, B, T_resp_cap, H, dh, sched, L.total - L.off_sched, st, kvs));
  SEER_TRY(do_linear(xn, w->w_o, it, x_resp, dt, h, it, T_resp_cap, M_dev, d, d, st, PH_OPROJ));
  SEER_TRY(do_rmsnorm(h, it, w->g_mlp, xn, it, T_resp_cap, M_dev, d, eps, st, PH_NORM2));
  SEER_TRY(do_swiglu(xn, w->w_gate, w->w_up, it, act, it, T_resp_cap, M_dev, F, d, cu_resp, B, nullptr, 0, 0.f, nullptr,
                     st, kGemmSwiglu, PH_GATEUP));
  SEER_TRY(do_linear(act, w->w_down, it, h, it, y_resp, dt, T_resp_cap, M_dev, d, F, st, PH_DOWN));
  return SEER_OK;
}

}  // extern "C"
