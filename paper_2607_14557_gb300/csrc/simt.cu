// CUDA-core kernels for fp32 storage (the small fp32 workload).  The tensor
// cores have no fp32-input mode, so fp32 layers run here with fp32 FMAs.
// Same epilogues and count hooks as the tcgen05 GEMM (tc_gemm.cu), and the
// same attention definition as tc_attn.cu (Sec. 3.6 Eqs. 6-7, 9-10).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace seer {
namespace {

constexpr int TB = 64;   // output tile (rows and columns)
constexpr int TK = 32;
constexpr int LPT = TB * TK / 256;   // elements of each operand tile a thread loads per k-step

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + __expf(-g)); }

// C tile 64x64, 256 threads, 4x4 outputs per thread.  For Swiglu/Count the
// block computes matching gate and up tiles of the same F columns.
template <int MODE>
__global__ void __launch_bounds__(256) simt_gemm_kernel(const float* __restrict__ A, const float* __restrict__ B0,
                                                        const float* __restrict__ B1, const GemmParams p) {
  pdl_enter();
  __shared__ float As[TK][TB + 1];
  __shared__ float Bs0[TK][TB + 1];
  __shared__ float Bs1[TK][TB + 1];
  constexpr bool TWO = (MODE == kGemmSwiglu || MODE == kGemmCount);

  int M = p.M_cap;
  int tiles_per_seq = 1;
  if (MODE == kGemmCount) {
    tiles_per_seq = (p.Nw + TB - 1) / TB;
  } else if (p.M_dev != nullptr) {
    const int md = *p.M_dev;
    if (md < 0 || md > p.M_cap) {
      if (threadIdx.x == 0 && blockIdx.x == 0 && blockIdx.y == 0) record_error(p.err, kErrRows);
      M = md < 0 ? 0 : p.M_cap;
    } else {
      M = md;
    }
  }
  const int mt = blockIdx.y, nt = blockIdx.x;
  int row_base, rows_here, seq = 0;
  if (MODE == kGemmCount) {
    seq = mt / tiles_per_seq;
    if (seq >= p.B) return;
    const int j = mt - seq * tiles_per_seq;
    const int rs = p.resp_start[seq];
    if (rs < 0 || rs + p.Nw > p.M_cap) {
      if (threadIdx.x == 0) record_error(p.err, kErrLayout);
      return;
    }
    row_base = rs + j * TB;
    rows_here = min(TB, p.Nw - j * TB);
  } else {
    row_base = mt * TB;
    if (row_base >= M) return;
    rows_here = min(TB, M - row_base);
  }
  const int col_base = nt * TB;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc0[4][4] = {}, acc1[4][4] = {};

  // the next k-step's operands are loaded into registers while the current
  // one is multiplied out of shared memory
  float ra[LPT], rb0[LPT], rb1[LPT];
  auto load = [&](int k0) {
#pragma unroll
    for (int e = 0; e < LPT; ++e) {
      const int i = threadIdx.x + 256 * e;
      const int r = i / TK, kk = k0 + i % TK;
      ra[e] = (r < rows_here && kk < p.K) ? A[static_cast<size_t>(row_base + r) * p.K + kk] : 0.f;
      const int c = col_base + r;
      rb0[e] = (c < p.N && kk < p.K) ? B0[static_cast<size_t>(c) * p.K + kk] : 0.f;
      if (TWO) rb1[e] = (c < p.N && kk < p.K) ? B1[static_cast<size_t>(c) * p.K + kk] : 0.f;
    }
  };
  load(0);
  for (int k0 = 0; k0 < p.K; k0 += TK) {
#pragma unroll
    for (int e = 0; e < LPT; ++e) {
      const int i = threadIdx.x + 256 * e;
      const int r = i / TK, k = i % TK;
      As[k][r] = ra[e];
      Bs0[k][r] = rb0[e];
      if (TWO) Bs1[k][r] = rb1[e];
    }
    __syncthreads();
    if (k0 + TK < p.K) load(k0 + TK);
#pragma unroll
    for (int k = 0; k < TK; ++k) {
      float a[4], b0[4], b1[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[k][ty * 4 + i];
        b0[i] = Bs0[k][tx * 4 + i];
        if (TWO) b1[i] = Bs1[k][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          acc0[i][jj] = fmaf(a[i], b0[jj], acc0[i][jj]);
          if (TWO) acc1[i][jj] = fmaf(a[i], b1[jj], acc1[i][jj]);
        }
    }
    __syncthreads();
  }

  float* C = reinterpret_cast<float*>(p.C);
  const float* R = reinterpret_cast<const float*>(p.R);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int lr = ty * 4 + i;
    if (lr >= rows_here) continue;
    const int row = row_base + lr;
    int cnt = 0;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int col = col_base + tx * 4 + jj;
      if (col >= p.N) continue;
      if (MODE == kGemmStore) {
        C[static_cast<size_t>(row) * p.ldc + col] = acc0[i][jj];
      } else if (MODE == kGemmResidual) {
        C[static_cast<size_t>(row) * p.ldc + col] = acc0[i][jj] + R[static_cast<size_t>(row) * p.ldr + col];
      } else {
        const float a = silu_f(acc0[i][jj]) * acc1[i][jj];
        cnt += fabsf(a) < p.act_eps ? 1 : 0;
        if (MODE == kGemmSwiglu) C[static_cast<size_t>(row) * p.ldc + col] = a;
      }
    }
    if (TWO && p.counts != nullptr && cnt > 0) {
      int idx = -1;
      if (MODE == kGemmCount) {
        idx = seq * p.Nw + (mt - seq * tiles_per_seq) * TB + lr;
      } else {
        int lo = 0, hi = p.B;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (p.cu[mid] <= row) lo = mid; else hi = mid;
        }
        const int tl = row - p.resp_start[lo];
        if (tl >= 0 && tl < p.Nw && row < p.cu[lo + 1]) idx = lo * p.Nw + tl;
      }
      if (idx >= 0) atomicAdd(&p.counts[idx], cnt);
    }
  }
}

// One warp per (query row, head): lanes split the head dimension, keys are
// visited in order with an online softmax (fp32).
__global__ void __launch_bounds__(256) simt_attn_kernel(const float* __restrict__ qkv, const AttnParams p) {
  pdl_enter();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long task = static_cast<long>(blockIdx.x) * 8 + warp;
  const int H = p.n_heads, dh = p.head_dim, D = H * dh;
  const int total = p.cu[p.B];
  if (total < 0 || total > p.T_cap) {
    if (task == 0 && lane == 0) record_error(p.err, kErrRows);
    return;
  }
  if (task >= static_cast<long>(total) * H) return;
  const int row = static_cast<int>(task / H), h = static_cast<int>(task % H);
  int lo = 0, hi = p.B;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.cu[mid] <= row) lo = mid; else hi = mid;
  }
  const int seq0 = p.cu[lo];
  const int kv0 = p.cu_kv ? p.cu_kv[lo] : seq0;
  const int Lkv = p.cu_kv ? p.cu_kv[lo + 1] - kv0 : p.cu[lo + 1] - seq0;
  const int kvL = p.kv_len ? p.kv_len[lo] : Lkv;
  if (kvL <= 0 || kvL > Lkv) {
    if (lane == 0) record_error(p.err, kErrLayout);
    return;
  }
  const float* kvsrc = p.kv ? static_cast<const float*>(p.kv) : qkv;
  const int per = (dh + 31) / 32;   // <= 4
  float q[4], o[4];
  const float* qrow = qkv + static_cast<size_t>(row) * 3 * D + h * dh;
  for (int i = 0; i < 4; ++i) {
    const int c = lane + 32 * i;
    q[i] = (i < per && c < dh) ? qrow[c] : 0.f;
    o[i] = 0.f;
  }
  const float scale = 1.0f / sqrtf(static_cast<float>(dh));
  float m = -INFINITY, l = 0.f;
  // keys in chunks of KC: the chunk's loads are all in flight together and its
  // KC warp reductions are independent, then one online-softmax update
  constexpr int KC = 8;
  for (int k0 = 0; k0 < kvL; k0 += KC) {
    float kv_k[KC][4], kv_v[KC][4], sc[KC];
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      const bool valid = k0 + j < kvL;
      const float* kvrow = kvsrc + static_cast<size_t>(kv0 + (valid ? k0 + j : 0)) * p.ld_kv;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int c = lane + 32 * i;
        const bool in = valid && i < per && c < dh;
        kv_k[j][i] = in ? kvrow[p.xk0 + h * dh + c] : 0.f;
        kv_v[j][i] = in ? kvrow[p.xv0 + h * dh + c] : 0.f;
      }
    }
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      float part = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) part = fmaf(q[i], kv_k[j][i], part);
      sc[j] = part;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
#pragma unroll
      for (int j = 0; j < KC; ++j) sc[j] += __shfl_xor_sync(0xffffffffu, sc[j], off);
    float m_new = m;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      sc[j] = k0 + j < kvL ? sc[j] * scale : -INFINITY;
      m_new = fmaxf(m_new, sc[j]);
    }
    const float alpha = expf(m - m_new);
    l *= alpha;
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] *= alpha;
#pragma unroll
    for (int j = 0; j < KC; ++j) {
      const float pr = expf(sc[j] - m_new);
      l += pr;
#pragma unroll
      for (int i = 0; i < 4; ++i) o[i] = fmaf(pr, kv_v[j][i], o[i]);
    }
    m = m_new;
  }
  float* out = reinterpret_cast<float*>(p.out) + static_cast<size_t>(row) * p.ldo + h * dh;
  for (int i = 0; i < per; ++i) {
    const int c = lane + 32 * i;
    if (c < dh) out[c] = o[i] / l;
  }
}

}  // namespace

cudaError_t launch_simt_gemm(int mode, const float* A, const float* B0, const float* B1, const GemmParams& p,
                             cudaStream_t st) {
  int mtiles;
  if (mode == kGemmCount) mtiles = p.B * ((p.Nw + TB - 1) / TB);
  else mtiles = (p.M_cap + TB - 1) / TB;
  const int ntiles = (p.N + TB - 1) / TB;
  if (mtiles <= 0 || ntiles <= 0) return cudaSuccess;
  if (mtiles > 65535) return cudaErrorInvalidValue;
  dim3 grid(ntiles, mtiles);
  switch (mode) {
    case kGemmStore: return launch_kernel(simt_gemm_kernel<kGemmStore>, grid, dim3(256), 0, st, A, B0, B1, p);
    case kGemmResidual: return launch_kernel(simt_gemm_kernel<kGemmResidual>, grid, dim3(256), 0, st, A, B0, B1, p);
    case kGemmSwiglu: return launch_kernel(simt_gemm_kernel<kGemmSwiglu>, grid, dim3(256), 0, st, A, B0, B1, p);
    case kGemmCount: return launch_kernel(simt_gemm_kernel<kGemmCount>, grid, dim3(256), 0, st, A, B0, B1, p);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_simt_attn(const float* qkv, const AttnParams& p, cudaStream_t st) {
  const long tasks = static_cast<long>(p.T_cap) * p.n_heads;
  if (tasks <= 0) return cudaSuccess;
  const long blocks = (tasks + 7) / 8;
  if (blocks > 0x7fffffffL) return cudaErrorInvalidValue;
  return launch_kernel(simt_attn_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, qkv, p);
}

}  // namespace seer
