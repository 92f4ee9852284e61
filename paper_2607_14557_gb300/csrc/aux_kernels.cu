// Memory- and latency-bound kernels of the hot path:
//   rmsnorm          pre-attention / pre-MLP normalisation (one warp per row;
//                    16-bit rows up to 4096 wide held in registers, else two passes)
//   snr_scan         Seer Sec. 3.3 boundary criterion, one warp per sequence
//   pack_route       Seer Sec. 3.4-3.5: micro-bucket routing (Eq. 4) fused
//                    with device-resident compaction and the pinned control word
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace seer {
namespace {

// ------------------------------------------------------------------ RMSNorm
template <int T>
__device__ __forceinline__ void load8(const void* base, size_t i8, float (&v)[8]) {
  if (T == kF32) {
    const float4* p = reinterpret_cast<const float4*>(base) + 2 * i8;
    const float4 a = p[0], b = p[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  } else {
    const uint4 q = reinterpret_cast<const uint4*>(base)[i8];
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      v[2 * i] = lo16(w[i], T == kF16);
      v[2 * i + 1] = hi16(w[i], T == kF16);
    }
  }
}
// Stores 8 values; for 16-bit storage returns the range-guard terms of the
// stored words (nonfinite_term), 0 for fp32.
template <int T>
__device__ __forceinline__ uint32_t store8(void* base, size_t i8, const float (&v)[8]) {
  if (T == kF32) {
    float4* p = reinterpret_cast<float4*>(base) + 2 * i8;
    p[0] = make_float4(v[0], v[1], v[2], v[3]);
    p[1] = make_float4(v[4], v[5], v[6], v[7]);
    return 0u;
  } else {
    uint32_t o[4];
    uint32_t nf = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      o[k] = pack2(v[2 * k], v[2 * k + 1], T == kF16);
      nf |= nonfinite_term(o[k], T == kF16);
    }
    reinterpret_cast<uint4*>(base)[i8] = make_uint4(o[0], o[1], o[2], o[3]);
    return nf;
  }
}

// y = x * rsqrt(mean(x^2) + eps) * g, one warp per row; input type IN, output
// (and gain) type OUT; fp32 arithmetic.
template <int IN, int OUT>
__global__ void __launch_bounds__(256) rmsnorm_kernel(const void* __restrict__ x, const void* __restrict__ g,
                                                      void* __restrict__ y, int M_cap, const int* M_dev, int d,
                                                      float eps, int* err) {
  pdl_enter();
  int M = M_cap;
  if (M_dev != nullptr) {
    const int md = *M_dev;
    if (md < 0 || md > M_cap) {
      if (blockIdx.x == 0 && threadIdx.x == 0) record_error(err, kErrRows);
      M = md < 0 ? 0 : M_cap;
    } else {
      M = md;
    }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = gridDim.x * 8;
  const int d8 = d / 8;
  uint32_t nonfinite = 0;
  for (int row = blockIdx.x * 8 + warp; row < M; row += nwarps) {
    const size_t base8 = static_cast<size_t>(row) * d8;
    float ss = 0.f;
    for (int v = lane; v < d8; v += 32) {
      float e[8];
      load8<IN>(x, base8 + v, e);
#pragma unroll
      for (int i = 0; i < 8; ++i) ss = fmaf(e[i], e[i], ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const float inv = rsqrtf(ss / static_cast<float>(d) + eps);
    for (int v = lane; v < d8; v += 32) {
      float e[8], gg[8];
      load8<IN>(x, base8 + v, e);
      load8<OUT>(g, v, gg);
#pragma unroll
      for (int i = 0; i < 8; ++i) e[i] = e[i] * inv * gg[i];
      nonfinite |= store8<OUT>(y, base8 + v, e);
    }
  }
  if (OUT != kF32) report_range(nonfinite, err);
}

// 16-bit rows of up to 256 * VPL elements: the row is read once into
// registers (VPL 16-byte vectors per lane, all loads in flight together), the
// sum of squares reduced across the warp, and the row scaled from registers.
// Two blocks per SM (at most 128 registers): 16 resident warps keep enough
// loads in flight (35194 x 4096 rows: 6.36 TB/s, against 5.4 for the
// two-pass streaming kernel and 4.9 at one block per SM).  The gain vector g,
// the same for every row, is staged once per block in shared memory (8 KB at
// d = 4096); read from global memory per row, its loads were hoisted beside
// the row's 64 registers and spilled.
template <int IN, int OUT, int VPL>
__global__ void __launch_bounds__(256, 2) rmsnorm_rows_kernel(const void* __restrict__ x, const void* __restrict__ g,
                                                           void* __restrict__ y, int M_cap, const int* M_dev, int d,
                                                           float eps, int* err) {
  pdl_enter();
  int M = M_cap;
  if (M_dev != nullptr) {
    const int md = *M_dev;
    if (md < 0 || md > M_cap) {
      if (blockIdx.x == 0 && threadIdx.x == 0) record_error(err, kErrRows);
      M = md < 0 ? 0 : M_cap;
    } else {
      M = md;
    }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = gridDim.x * 8;
  const int d8 = d / 8;
  const uint4* xv = reinterpret_cast<const uint4*>(x);
  __shared__ uint4 g_sh[32 * VPL];
  for (int v = threadIdx.x; v < d8; v += blockDim.x) g_sh[v] = __ldg(reinterpret_cast<const uint4*>(g) + v);
  __syncthreads();
  uint4* yv = reinterpret_cast<uint4*>(y);
  uint32_t nonfinite = 0;
  for (int row = blockIdx.x * 8 + warp; row < M; row += nwarps) {
    const size_t base8 = static_cast<size_t>(row) * d8;
    uint4 raw[VPL];
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      raw[i] = v < d8 ? __ldg(xv + base8 + v) : make_uint4(0, 0, 0, 0);
    }
    // the sum of squares unpacks through an opaque copy of each word, so the
    // scaling below unpacks again instead of keeping 8 floats per vector live
    // from here (that reuse needed 128 float registers and spilled)
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const uint32_t w[4] = {raw[i].x, raw[i].y, raw[i].z, raw[i].w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        uint32_t wc;
        asm volatile("mov.b32 %0, %1;" : "=r"(wc) : "r"(w[k]));
        const float a = lo16(wc, IN == kF16), b = hi16(wc, IN == kF16);
        ss = fmaf(a, a, ss);
        ss = fmaf(b, b, ss);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const float inv = rsqrtf(ss / static_cast<float>(d) + eps);
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      if (v < d8) {
        const uint4 gq = g_sh[v];
        const uint32_t w[4] = {raw[i].x, raw[i].y, raw[i].z, raw[i].w};
        const uint32_t gw[4] = {gq.x, gq.y, gq.z, gq.w};
        uint32_t o[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          o[k] = pack2(lo16(w[k], IN == kF16) * inv * lo16(gw[k], OUT == kF16),
                       hi16(w[k], IN == kF16) * inv * hi16(gw[k], OUT == kF16), OUT == kF16);
          nonfinite |= nonfinite_term(o[k], OUT == kF16);
        }
        yv[base8 + v] = make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
  }
  report_range(nonfinite, err);
}

// Element-wise storage conversion (used once per model for f16 weight copies);
// a 16-bit result that is infinite or NaN (a bf16 weight beyond the f16
// range) records kErrRange.
template <int IN, int OUT>
__global__ void convert_kernel(const void* __restrict__ src, void* __restrict__ dst, size_t n8, int* err) {
  pdl_enter();
  uint32_t nonfinite = 0;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n8;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    float e[8];
    load8<IN>(src, i, e);
    nonfinite |= store8<OUT>(dst, i, e);
  }
  if (OUT != kF32) report_range(nonfinite, err);
}

// ------------------------------------------------------------------ rotary embedding
template <int T>
__device__ __forceinline__ float ld1(const void* base, size_t i) {
  if (T == kF32) return reinterpret_cast<const float*>(base)[i];
  const uint16_t v = reinterpret_cast<const uint16_t*>(base)[i];
  return T == kF16 ? f16_lo(v) : bf16_lo(v);
}
template <int T>
__device__ __forceinline__ void st1(void* base, size_t i, float x) {
  if (T == kF32) {
    reinterpret_cast<float*>(base)[i] = x;
  } else {
    reinterpret_cast<uint16_t*>(base)[i] = static_cast<uint16_t>(pack2(x, 0.f, T == kF16) & 0xFFFFu);
  }
}

// In-place rotation of the q and k heads of qkv [T, 3*H*dh] (q | k | v column
// blocks): pair (i, i + dh/2) of every head turns by pos * theta^(-2i/dh),
// pos = the row's position in its segment.  One block per row at a time.
template <int T>
__global__ void __launch_bounds__(256) rope_kernel(void* __restrict__ qkv, const int* __restrict__ cu, int B, int T_cap,
                                                   int H, int dh, float theta, int* err) {
  pdl_enter();
  __shared__ float2 tab[64];
  const int half = dh / 2;
  for (int i = threadIdx.x; i < half; i += blockDim.x) tab[i] = rope_inv_freq(i, dh, theta);
  __syncthreads();
  int M = cu[B];
  if (M < 0 || M > T_cap) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(err, kErrRows);
    M = M < 0 ? 0 : T_cap;
  }
  const size_t ld = static_cast<size_t>(3) * H * dh;
  const int pairs = H * dh;                       // 2H heads (q and k) x dh/2 pairs
  for (int row = blockIdx.x; row < M; row += gridDim.x) {
    const float pos = static_cast<float>(row_position(cu, B, row));
    for (int j = threadIdx.x; j < pairs; j += blockDim.x) {
      const int hh = j / half, i = j - hh * half;
      const size_t a = row * ld + static_cast<size_t>(hh) * dh + i, b = a + half;
      float c, sn;
      rope_cos_sin(pos, tab[i], c, sn);
      const float x0 = ld1<T>(qkv, a), x1 = ld1<T>(qkv, b);
      st1<T>(qkv, a, fmaf(x0, c, -x1 * sn));
      st1<T>(qkv, b, fmaf(x1, c, x0 * sn));
    }
  }
}

// ------------------------------------------------------------------ segment row copies
// For each segment b: n rows starting at src row s0 (columns [src_c0, src_c0 +
// row) in bytes) go to dst rows starting at d0, with
//   s0 = src_start[b] (+ src_add[b]),  d0 = dst_start[b] (+ dst_add[b]),
//   n  = (len ? len[b] : src_start[b+1] - src_start[b]) (- len_sub[b]).
// A warp per row, 16-byte vectors; segments whose rows fall outside either
// buffer are skipped and recorded.
struct RowsCopyArgs {
  const uint8_t* src;
  long src_ld;                 // bytes per source row
  int src_c0;                  // byte offset of the copied columns in a source row
  uint8_t* dst;
  long dst_ld;
  int dst_c0;
  int row;                     // bytes copied per row (multiple of 16)
  const int* src_start;
  const int* src_add;
  const int* len;
  const int* len_sub;
  const int* dst_start;
  const int* dst_add;
  int B, src_rows, dst_rows;
  int* err;
};

__global__ void __launch_bounds__(256) rows_copy_kernel(const RowsCopyArgs a) {
  pdl_enter();
  const int b = blockIdx.y;
  const int s0 = a.src_start[b] + (a.src_add ? a.src_add[b] : 0);
  const int d0 = a.dst_start[b] + (a.dst_add ? a.dst_add[b] : 0);
  const int n = (a.len ? a.len[b] : a.src_start[b + 1] - a.src_start[b]) - (a.len_sub ? a.len_sub[b] : 0);
  if (n <= 0) return;
  if (s0 < 0 || d0 < 0 || s0 + n > a.src_rows || d0 + n > a.dst_rows) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(a.err, kErrLayout);
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int v16 = a.row / 16;
  for (int i = blockIdx.x * 8 + warp; i < n; i += gridDim.x * 8) {
    const uint4* sp = reinterpret_cast<const uint4*>(a.src + static_cast<size_t>(s0 + i) * a.src_ld + a.src_c0);
    uint4* dp = reinterpret_cast<uint4*>(a.dst + static_cast<size_t>(d0 + i) * a.dst_ld + a.dst_c0);
    for (int v = lane; v < v16; v += 32) dp[v] = sp[v];
  }
}

// cu_ctx = exclusive prefix sums of ctx (B+1 entries); cu_resp[b] = cu[b] -
// cu_ctx[b]: the offsets of the rows past each segment's first ctx[b] rows.
__global__ void resp_layout_kernel(const int* cu, const int* ctx, int B, int* cu_resp, int* cu_ctx, int* err) {
  pdl_enter();
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  int acc = 0;
  for (int b = 0; b <= B; ++b) {
    if (cu_ctx) cu_ctx[b] = acc;
    if (cu_resp && cu) {
      const int r = cu[b] - acc;
      if (r < 0 || (b > 0 && ctx[b - 1] > cu[b] - cu[b - 1])) record_error(err, kErrLayout);
      cu_resp[b] = r < 0 ? 0 : r;
    }
    if (b < B) acc += ctx[b];
  }
}

// ------------------------------------------------------------------ wait self-test
// A pipeline wait that can never complete (an mbarrier nothing arrives on),
// bounded by limit_ns: the same give-up path every tcgen05 kernel's waits
// take, recording kErrTimeout instead of hanging.
__global__ void wait_selftest_kernel(uint64_t limit_ns, int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  abort_flag = 0;
  fence_barrier_init();
  mbar_wait_for(&bar, 0, &abort_flag, err, limit_ns);
}

// ------------------------------------------------------------------ SNR scan
constexpr int kScanSmemInts = 12288;   // 48 KB of staged counts per sequence at most
// Sec. 3.3: first 0-based i in [1, N-w] with
//   jump  = min(s_i .. s_{i+w-1}) - s_{i-1} >= tau_jump
//   noise = max(s_i .. s_{i+w-1}) - min(..)  <= gamma * jump,   s = c / F,
// evaluated in IEEE fp64 with explicit round-to-nearest operations (no FMA
// contraction) so the decision is exactly reproducible.  L* = i* + 1, or N.
__global__ void __launch_bounds__(32) snr_scan_kernel(const int* __restrict__ counts, int N, int F, double tau_jump,
                                                      double gamma, int window, int* __restrict__ L_star,
                                                      int* __restrict__ i_star) {
  pdl_enter();
  const int b = blockIdx.x;
  const int lane = threadIdx.x;
  const int* c = counts + static_cast<size_t>(b) * N;
  // the sequence's counts staged in shared memory by one coalesced pass (all
  // loads in flight at once) when they fit; the scan then reads them there
  extern __shared__ int staged[];
  if (N <= kScanSmemInts) {
    for (int i = lane; i < N; i += 32) staged[i] = c[i];
    __syncwarp();
    c = staged;
  }
  const double Fd = static_cast<double>(F);
  int found = -1;
  const int last = N - window;   // inclusive
  for (int base = 1; base <= last; base += 32) {
    const int i = base + lane;
    bool hit = false;
    if (i <= last) {
      int lo = c[i], hi = c[i];
      for (int k = 1; k < window; ++k) {
        const int v = c[i + k];
        lo = min(lo, v);
        hi = max(hi, v);
      }
      const double s_lo = __ddiv_rn(static_cast<double>(lo), Fd);
      const double s_hi = __ddiv_rn(static_cast<double>(hi), Fd);
      const double s_prev = __ddiv_rn(static_cast<double>(c[i - 1]), Fd);
      const double jump = __dsub_rn(s_lo, s_prev);
      const double noise = __dsub_rn(s_hi, s_lo);
      hit = (jump >= tau_jump) && (noise <= __dmul_rn(gamma, jump));
    }
    const unsigned mask = __ballot_sync(0xffffffffu, hit);
    if (mask) {
      found = base + __ffs(mask) - 1;
      break;
    }
  }
  if (lane == 0) {
    L_star[b] = found >= 0 ? found + 1 : N;
    if (i_star) i_star[b] = found;
  }
}

// ------------------------------------------------------------------ route + pack
struct RouteSmem {
  int n_buckets;
  int bucket[kCtrlMaxGroups];
  int count[kCtrlMaxGroups];
  long long sum[kCtrlMaxGroups];
  int path[kCtrlMaxGroups];
  int rho_ppm[kCtrlMaxGroups];
  int total, max_seg, pad_rows, path_mask, n_groups;
};

__device__ __forceinline__ int graph_capacity(int total) {
  // smallest m * 2^e >= total with m in [8, 15]
  if (total <= 8) return 8;
  int e = 0;
  while ((15 << e) < total) ++e;
  const int m = (total + (1 << e) - 1) >> e;
  return m << e;
}

// Every block recomputes the (tiny) routing decision in shared memory, block 0
// publishes it, then all blocks copy rows.  Dynamic smem: seg/cu/bucket-index
// arrays of B+1 ints each.
__global__ void __launch_bounds__(256, 4) pack_route_kernel(const uint8_t* __restrict__ x_full, int row_bytes,
                                                         const int* __restrict__ cu_full,
                                                         const int* __restrict__ ctx_len,
                                                         const int* __restrict__ L_star, int B, int N, int T_cap,
                                                         double tau_pad, int eager_max_bucket, int bucket_min,
                                                         uint8_t* __restrict__ x_packed, int* cu_out, int* kv_out,
                                                         int* meta_out, int* host_ctrl, int epoch, int* err) {
  pdl_enter();
  extern __shared__ int dyn[];
  int* seg = dyn;              // [B]
  int* cus = dyn + B;          // [B+1]
  int* bidx = dyn + 2 * B + 1; // [B]
  __shared__ RouteSmem rs;

  if (threadIdx.x == 0) {
    int nb = 0;
    for (int b = bucket_min; b < N && nb < kCtrlMaxGroups - 1; b *= 2) rs.bucket[nb++] = b;
    rs.bucket[nb++] = N;
    rs.n_buckets = nb;
    for (int k = 0; k < nb; ++k) { rs.count[k] = 0; rs.sum[k] = 0; }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    int Ls = L_star[i];
    if (Ls < 1 || Ls > N) {
      if (blockIdx.x == 0) record_error(err, kErrBoundary);
      Ls = Ls < 1 ? 1 : N;
    }
    int k = 0;
    while (k < rs.n_buckets - 1 && Ls > rs.bucket[k]) ++k;
    bidx[i] = k;
    atomicAdd(&rs.count[k], 1);
    atomicAdd(reinterpret_cast<unsigned long long*>(&rs.sum[k]), static_cast<unsigned long long>(Ls));
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int mask = 0, ng = 0;
    for (int k = 0; k < rs.n_buckets; ++k) {
      if (rs.count[k] == 0) { rs.path[k] = -1; continue; }
      // Eq. 4, in fp64 exactly as written
      const double rho = 1.0 - static_cast<double>(rs.sum[k]) / static_cast<double>(static_cast<long long>(rs.count[k]) * rs.bucket[k]);
      int path;
      if (rs.bucket[k] <= eager_max_bucket || rs.count[k] == 1) path = 2;
      else if (rho <= tau_pad) path = 0;
      else path = 1;
      rs.path[k] = path;
      rs.rho_ppm[k] = static_cast<int>(floor(rho * 1e6));
      mask |= 1 << path;
      ++ng;
    }
    rs.path_mask = mask;
    rs.n_groups = ng;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    int Ls = L_star[i];
    Ls = Ls < 1 ? 1 : (Ls > N ? N : Ls);
    const int k = bidx[i];
    const int keep = rs.path[k] == 0 ? rs.bucket[k] : Ls;
    const int ctx = ctx_len[i];
    const int avail = cu_full[i + 1] - cu_full[i];
    if (ctx < 0 || ctx + N > avail) {
      if (blockIdx.x == 0) record_error(err, kErrLayout);
    }
    seg[i] = max(0, min(ctx + keep, avail));
    if (blockIdx.x == 0) kv_out[i] = max(0, min(ctx + Ls, avail));
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0, mx = 0, pad = 0;
    for (int i = 0; i < B; ++i) {
      cus[i] = acc;
      acc += seg[i];
      mx = max(mx, seg[i]);
      int Ls = L_star[i];
      Ls = Ls < 1 ? 1 : (Ls > N ? N : Ls);
      if (rs.path[bidx[i]] == 0) pad += rs.bucket[bidx[i]] - Ls;
    }
    cus[B] = acc;
    rs.total = acc;
    rs.max_seg = mx;
    rs.pad_rows = pad;
    if (acc > T_cap && blockIdx.x == 0) record_error(err, kErrCapacity);
  }
  __syncthreads();

  if (blockIdx.x == 0) {
    for (int i = threadIdx.x; i <= B; i += blockDim.x) cu_out[i] = cus[i];
    if (threadIdx.x == 0) {
      // the control word is assembled in place in meta_out (a local array of
      // kCtrlWords ints would live on the stack and cost registers in every block)
      for (int i = 0; i < kCtrlWords; ++i) meta_out[i] = 0;
      meta_out[1] = rs.total;
      meta_out[2] = rs.max_seg;
      meta_out[3] = graph_capacity(rs.total);
      meta_out[4] = rs.n_groups;
      meta_out[5] = rs.path_mask;
      meta_out[6] = rs.pad_rows;
      int g = 0;
      for (int k = 0; k < rs.n_buckets && g < kCtrlMaxGroups; ++k) {
        if (rs.count[k] == 0) continue;
        meta_out[8 + 4 * g + 0] = rs.bucket[k];
        meta_out[8 + 4 * g + 1] = rs.count[k];
        meta_out[8 + 4 * g + 2] = rs.path[k];
        meta_out[8 + 4 * g + 3] = rs.rho_ppm[k];
        ++g;
      }
      meta_out[0] = epoch;
      if (host_ctrl != nullptr) {
        volatile int* hc = host_ctrl;
        for (int i = 1; i < kCtrlWords; ++i) hc[i] = meta_out[i];
        __threadfence_system();
        hc[0] = epoch;
        __threadfence_system();
      }
    }
  }

  // ---- copy rows, one warp per row, 16-byte vectors; four loads in flight
  // per lane before their stores
  const int total = min(rs.total, T_cap);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int vec = row_bytes / 16;
  for (int r = blockIdx.x * 8 + warp; r < total; r += gridDim.x * 8) {
    int lo = 0, hi = B;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (cus[mid] <= r) lo = mid; else hi = mid;
    }
    const int src = cu_full[lo] + (r - cus[lo]);
    const uint4* s = reinterpret_cast<const uint4*>(x_full + static_cast<size_t>(src) * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>(x_packed + static_cast<size_t>(r) * row_bytes);
    int v = lane;
    for (; v + 96 < vec; v += 128) {
      const uint4 a0 = s[v], a1 = s[v + 32], a2 = s[v + 64], a3 = s[v + 96];
      dst[v] = a0;
      dst[v + 32] = a1;
      dst[v + 64] = a2;
      dst[v + 96] = a3;
    }
    for (; v < vec; v += 32) dst[v] = s[v];
  }
}

}  // namespace

cudaError_t launch_rmsnorm(const void* x, int in_type, const void* g, void* y, int out_type, int M_cap,
                           const int* M_dev, int d, float eps, int* err, cudaStream_t st) {
  if (M_cap <= 0) return cudaSuccess;
  int blocks = (M_cap + 7) / 8;
  if (blocks > 65535 * 4) blocks = 65535 * 4;
  // 16-bit rows up to 4096 wide: register-resident variant sized to the row
  const int vpl = (d / 8 + 31) / 32;
#define SEER_NORM_ROWS(I, O, V)                                                                                   \
  if (in_type == I && out_type == O && vpl <= V)                                                                 \
    return launch_kernel(rmsnorm_rows_kernel<I, O, V>, dim3(blocks), dim3(256), 0, st, x, g, y, M_cap, M_dev, d, \
                         eps, err);
#define SEER_NORM_16(I, O) SEER_NORM_ROWS(I, O, 4) SEER_NORM_ROWS(I, O, 8) SEER_NORM_ROWS(I, O, 16)
  SEER_NORM_16(kBF16, kF16)
  SEER_NORM_16(kF16, kF16)
  SEER_NORM_16(kBF16, kBF16)
#undef SEER_NORM_16
#undef SEER_NORM_ROWS
#define SEER_NORM(I, O) \
  if (in_type == I && out_type == O) return launch_kernel(rmsnorm_kernel<I, O>, dim3(blocks), dim3(256), 0, st, x, g, y, M_cap, M_dev, d, eps, err);
  SEER_NORM(kBF16, kF16)
  SEER_NORM(kF16, kF16)
  SEER_NORM(kBF16, kBF16)
  SEER_NORM(kF32, kF32)
#undef SEER_NORM
  return cudaErrorInvalidValue;
}

cudaError_t launch_convert(const void* src, int in_type, void* dst, int out_type, size_t n, int* err, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  if (n % 8 != 0) return cudaErrorInvalidValue;
  const size_t n8 = n / 8;
  const int blocks = static_cast<int>(n8 / 256 + 1 < 4096 ? n8 / 256 + 1 : 4096);
#define SEER_CONV(I, O) \
  if (in_type == I && out_type == O) return launch_kernel(convert_kernel<I, O>, dim3(blocks), dim3(256), 0, st, src, dst, n8, err);
  SEER_CONV(kBF16, kF16)
  SEER_CONV(kF16, kBF16)
  SEER_CONV(kBF16, kF32)
  SEER_CONV(kF16, kF32)
  SEER_CONV(kF32, kBF16)
  SEER_CONV(kF32, kF16)
#undef SEER_CONV
  return cudaErrorInvalidValue;
}

cudaError_t launch_rope(void* qkv, int type, const int* cu, int B, int T_cap, int n_heads, int head_dim, float theta,
                        int* err, int num_sms, cudaStream_t st) {
  if (T_cap <= 0) return cudaSuccess;
  if (head_dim % 2 != 0 || head_dim > 128) return cudaErrorInvalidValue;
  const int blocks = T_cap < 8 * num_sms ? T_cap : 8 * num_sms;
  switch (type) {
    case kF32: return launch_kernel(rope_kernel<kF32>, dim3(blocks), dim3(256), 0, st, qkv, cu, B, T_cap, n_heads, head_dim, theta, err);
    case kF16: return launch_kernel(rope_kernel<kF16>, dim3(blocks), dim3(256), 0, st, qkv, cu, B, T_cap, n_heads, head_dim, theta, err);
    case kBF16: return launch_kernel(rope_kernel<kBF16>, dim3(blocks), dim3(256), 0, st, qkv, cu, B, T_cap, n_heads, head_dim, theta, err);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_rows_copy(const void* src, long src_ld, int src_c0, void* dst, long dst_ld, int dst_c0, int row_bytes,
                             const int* src_start, const int* src_add, const int* len, const int* len_sub,
                             const int* dst_start, const int* dst_add, int B, int src_rows, int dst_rows, int max_rows,
                             int* err, cudaStream_t st) {
  if (B <= 0 || row_bytes <= 0 || max_rows <= 0) return cudaSuccess;
  if (row_bytes % 16 != 0 || src_c0 % 16 != 0 || dst_c0 % 16 != 0 || src_ld % 16 != 0 || dst_ld % 16 != 0 ||
      (reinterpret_cast<uintptr_t>(src) & 15u) != 0 || (reinterpret_cast<uintptr_t>(dst) & 15u) != 0)
    return cudaErrorInvalidValue;
  RowsCopyArgs a{static_cast<const uint8_t*>(src), src_ld, src_c0, static_cast<uint8_t*>(dst), dst_ld, dst_c0, row_bytes,
                 src_start, src_add, len, len_sub, dst_start, dst_add, B, src_rows, dst_rows, err};
  const int gx = (max_rows + 7) / 8 < 64 ? (max_rows + 7) / 8 : 64;
  return launch_kernel(rows_copy_kernel, dim3(gx, B), dim3(256), 0, st, a);
}

cudaError_t launch_resp_layout(const int* cu, const int* ctx, int B, int* cu_resp, int* cu_ctx, int* err,
                               cudaStream_t st) {
  return launch_kernel(resp_layout_kernel, dim3(1), dim3(32), 0, st, cu, ctx, B, cu_resp, cu_ctx, err);
}

cudaError_t launch_wait_selftest(uint64_t limit_ns, int* err, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(limit_ns, err);
  return cudaGetLastError();
}

cudaError_t launch_snr_scan(const int* counts, int B, int N, int F, double tau_jump, double gamma, int window,
                            int* L_star, int* i_star, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  const size_t sm = N <= kScanSmemInts ? static_cast<size_t>(N) * sizeof(int) : 0;
  return launch_kernel(snr_scan_kernel, dim3(B), dim3(32), sm, st, counts, N, F, tau_jump, gamma, window, L_star, i_star);
}

cudaError_t launch_pack_route(const void* x_full, int elem_bytes, const int* cu_full, const int* ctx_len,
                              const int* L_star, int B, int d, int N, int T_cap, double tau_pad,
                              int eager_max_bucket, int bucket_min, void* x_packed, int* cu_out, int* kv_out,
                              int* meta_out, int* host_ctrl_dev, int epoch, int* err, int num_sms, cudaStream_t st) {
  const size_t sm = static_cast<size_t>(3 * B + 1) * sizeof(int);
  if (sm > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(pack_route_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(sm));
    if (e != cudaSuccess) return e;
  }
  // four 256-thread blocks per SM are resident (64 registers): one wave, the warps
  // looping over the rows
  int blocks = (T_cap + 7) / 8;
  const int cap = num_sms * 4;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return launch_kernel(pack_route_kernel, dim3(blocks), dim3(256), sm, st, reinterpret_cast<const uint8_t*>(x_full),
                       d * elem_bytes, cu_full, ctx_len, L_star, B, N, T_cap, tau_pad, eager_max_bucket, bucket_min,
                       reinterpret_cast<uint8_t*>(x_packed), cu_out, kv_out, meta_out, host_ctrl_dev, epoch, err);
}

}  // namespace seer
