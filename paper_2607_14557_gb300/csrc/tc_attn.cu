// Varlen bidirectional attention on tcgen05 for sm_103a (head_dim 128; q, k,
// v, the probabilities P and the output all f16, or all bf16).
//
// Seer Sec. 3.6 Eqs. 6-7 and 9-10: every query row of a segment attends to
// the first kv_len[b] rows of the same segment, with no causal mask; rows
// beyond kv_len (bucket padding of the static path) are never keys.
//
// One CTA per (segment, head, 128-query tile); 64 + 128 * NGRP threads:
//   warp 0     TMA producer: Q tile once, then K_j and V_j (128 keys x 128
//              dims, 128-byte swizzle) into a 2-deep ring;
//   warp 1     TMEM allocator + MMA issuer: S_j = Q K_j^T (M=N=128, K=16 x 8)
//              into one of two S buffers, then O += P_j V_j (V as an MN-major
//              operand) into the O accumulator;
//   warps 2.. softmax, NGRP groups of four warps: a query row (one TMEM
//              lane) is shared by one thread of each group, which owns
//              128 / NGRP of the key columns (and of the output dims); the
//              parts of a row exchange their maxima through shared memory
//              once per key tile (an mbarrier, so every wait is bounded).
//              Online softmax in the log2 domain with lazy rescaling: O is
//              rescaled in TMEM only when the running max grows by more than
//              2^8.  P_j goes to shared memory in the swizzled K-major layout
//              the tensor core reads.
// The QK^T MMA of tile j+1 overlaps the softmax of tile j.
// The schedule kernel orders work units longest segment first.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace seer {
namespace {

constexpr int BQ = 128;
constexpr int BKV = 128;
constexpr int DH = 128;
constexpr int NGRP = 2;                     // softmax column groups (4 warps each)
constexpr int COLS = BKV / NGRP;            // key columns / output dims per softmax thread
constexpr int SOFTMAX_WARPS = 4 * NGRP;
constexpr int THREADS = 64 + 32 * SOFTMAX_WARPS;
constexpr int TILE_BYTES = 128 * DH * 2;   // 32 KB: 128 rows x 128 16-bit values as two 16 KB swizzle panels
constexpr int PANEL = 16384;
constexpr int OFF_Q = 0;
constexpr int OFF_K = TILE_BYTES;           // 2 buffers
constexpr int OFF_V = 3 * TILE_BYTES;       // 2 buffers
constexpr int OFF_P = 5 * TILE_BYTES;
constexpr int OFF_BAR = 6 * TILE_BYTES;
constexpr int OFF_RED = OFF_BAR + 256;      // float max[2 tiles][NGRP][128] + float sum[NGRP][128]
constexpr int SMEM_BYTES = OFF_RED + (2 * NGRP * 128 + NGRP * 128) * 4 + 1024;
constexpr uint32_t TMEM_COLS = 512;         // S0 [0,128), S1 [128,256), O [256,384)
constexpr float RESCALE_THRESHOLD = 8.0f;   // log2 units

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <bool F16>
__global__ void __launch_bounds__(THREADS, 1)
    tc_attn_kernel(const __grid_constant__ CUtensorMap mQKV, const AttnParams p) {
  const int u = blockIdx.x;
  if (u >= *p.work_count) return;
  const int4 wk = p.work[u];
  const int b = wk.x, h = wk.y, qt = wk.z;
  const int seq0 = p.cu[b];
  const int L = p.cu[b + 1] - seq0;
  const int kvL = p.kv_len ? p.kv_len[b] : L;
  const int q0 = seq0 + qt * BQ;
  const int nkv = (kvL + BKV - 1) / BKV;
  const int D = p.n_heads * DH;
  const int xq = h * DH, xk = D + h * DH, xv = 2 * D + h * DH;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* k_full = bars + 1;     // [2]
  uint64_t* k_empty = bars + 3;    // [2]
  uint64_t* v_full = bars + 5;     // [2]
  uint64_t* v_empty = bars + 7;    // [2]
  uint64_t* s_full = bars + 9;     // [2]
  uint64_t* s_empty = bars + 11;   // [2]
  uint64_t* p_full = bars + 13;
  uint64_t* pv_done = bars + 14;
  uint64_t* max_ready = bars + 15; // [2] row-max exchange, one per tile parity
  uint64_t* sum_ready = bars + 17;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* red_max = reinterpret_cast<float*>(smem + OFF_RED);   // [2 tiles][NGRP][128] partial row maxima
  float* red_sum = red_max + 2 * NGRP * 128;                   // [NGRP][128] partial row sums

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], SOFTMAX_WARPS);
      mbar_init(&max_ready[i], SOFTMAX_WARPS);
    }
    mbar_init(p_full, SOFTMAX_WARPS);
    mbar_init(pv_done, 1);
    mbar_init(sum_ready, SOFTMAX_WARPS);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      tma_prefetch_desc(&mQKV);
      int issued_k = 0, issued_v = 0;
      mbar_arrive_expect_tx(q_full, TILE_BYTES);
      tma_load_2d(smem + OFF_Q, &mQKV, q_full, xq, q0);
      tma_load_2d(smem + OFF_Q + PANEL, &mQKV, q_full, xq + 64, q0);
      for (int j = 0; j < nkv; ++j) {
        const int sb = j & 1, use = j >> 1;
        const int row = seq0 + j * BKV;
        if (use > 0 && !mbar_wait(&k_empty[sb], (use - 1) & 1, abort_flag, p.err)) break;
        uint8_t* kd = smem + OFF_K + sb * TILE_BYTES;
        mbar_arrive_expect_tx(&k_full[sb], TILE_BYTES);
        tma_load_2d(kd, &mQKV, &k_full[sb], xk, row);
        tma_load_2d(kd + PANEL, &mQKV, &k_full[sb], xk + 64, row);
        ++issued_k;
        if (use > 0 && !mbar_wait(&v_empty[sb], (use - 1) & 1, abort_flag, p.err)) break;
        uint8_t* vd = smem + OFF_V + sb * TILE_BYTES;
        mbar_arrive_expect_tx(&v_full[sb], TILE_BYTES);
        tma_load_2d(vd, &mQKV, &v_full[sb], xv, row);
        tma_load_2d(vd + PANEL, &mQKV, &v_full[sb], xv + 64, row);
        ++issued_v;
      }
      if (*abort_flag) {
        mbar_wait_drain(q_full, 0, 200000000ull);
        for (int j = issued_k > 2 ? issued_k - 2 : 0; j < issued_k; ++j)
          mbar_wait_drain(&k_full[j & 1], (j >> 1) & 1, 200000000ull);
        for (int j = issued_v > 2 ? issued_v - 2 : 0; j < issued_v; ++j)
          mbar_wait_drain(&v_full[j & 1], (j >> 1) & 1, 200000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t idesc_qk = make_idesc(BQ, BKV, 0, F16);
      constexpr uint32_t idesc_pv = make_idesc(BQ, DH, 1, F16);
      const uint32_t sq = smem_u32(smem + OFF_Q);
      const uint32_t sp = smem_u32(smem + OFF_P);
      auto issue_pv = [&](int i) -> bool {
        const int sb = i & 1, use = i >> 1;
        if (!mbar_wait(&v_full[sb], use & 1, abort_flag, p.err)) return false;
        if (!mbar_wait(p_full, i & 1, abort_flag, p.err)) return false;
        tc_fence_after();
        const uint32_t sv = smem_u32(smem + OFF_V + sb * TILE_BYTES);
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k) {
          const uint64_t ad = make_sdesc_sw128(sp + (k >> 2) * PANEL + (k & 3) * 32, 16, 1024);
          // V is [keys, dims] with dims contiguous: MN-major B operand; the two
          // 64-dim panels are PANEL bytes apart (LBO), 8-key groups 1 KB apart (SBO)
          const uint64_t bd = make_sdesc_sw128(sv + k * 16 * 128, PANEL, 1024);
          tc_mma_f16(tmem + 256, ad, bd, idesc_pv, (i > 0 || k > 0) ? 1u : 0u);
        }
        tc_commit(&v_empty[sb]);
        tc_commit(pv_done);
        return true;
      };
      bool ok = mbar_wait(q_full, 0, abort_flag, p.err);
      for (int j = 0; ok && j < nkv; ++j) {
        const int sb = j & 1, use = j >> 1;
        if (!mbar_wait(&k_full[sb], use & 1, abort_flag, p.err)) { ok = false; break; }
        if (use > 0 && !mbar_wait(&s_empty[sb], (use - 1) & 1, abort_flag, p.err)) { ok = false; break; }
        tc_fence_after();
        const uint32_t sk = smem_u32(smem + OFF_K + sb * TILE_BYTES);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint32_t off = (k >> 2) * PANEL + (k & 3) * 32;
          tc_mma_f16(tmem + sb * 128, make_sdesc_sw128(sq + off, 16, 1024), make_sdesc_sw128(sk + off, 16, 1024),
                     idesc_qk, k > 0 ? 1u : 0u);
        }
        tc_commit(&k_empty[sb]);
        tc_commit(&s_full[sb]);
        if (j > 0 && !issue_pv(j - 1)) { ok = false; break; }
      }
      if (ok && nkv > 0) issue_pv(nkv - 1);
    }
  } else {
    // -------------------------------------------------- softmax warps 2..
    const int grp = (warp - 2) >> 2;              // column group: keys / output dims [COLS grp, COLS grp + COLS)
    const int qw = warp & 3;
    const int r = qw * 32 + lane;                 // query row inside the tile == TMEM lane
    const int col0 = grp * COLS;
    const uint32_t lane_off = static_cast<uint32_t>(qw * 32) << 16;
    const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));
    // P row r, keys [col0, col0 + COLS): 16-byte chunks (col0 % 64) / 8 + c of
    // panel col0 / 64 in the swizzled K-major layout (chunk k of row r sits at
    // (r / 8) * 1024 + (r % 8) * 128 + ((k ^ (r % 8)) * 16))
    uint8_t* sProw = smem + OFF_P + (col0 / 64) * PANEL + (r >> 3) * 1024 + (r & 7) * 128;
    const int chunk0 = (col0 % 64) / 8;
    float m_ref = -INFINITY;                      // running max, log2 units
    float l = 0.f;                                // partial row sum over this thread's columns
    bool ok = true;
    for (int j = 0; j < nkv; ++j) {
      const int sb = j & 1, use = j >> 1;
      if (!mbar_wait(&s_full[sb], use & 1, abort_flag, p.err)) { ok = false; break; }
      tc_fence_after();
      float s[COLS];
      {
        uint32_t ra[COLS / 32][32];
#pragma unroll
        for (int c = 0; c < COLS / 32; ++c) tmem_ld32(tmem + lane_off + sb * 128 + col0 + 32 * c, ra[c]);
        tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < COLS / 32; ++c)
#pragma unroll
          for (int i = 0; i < 32; ++i) s[32 * c + i] = __uint_as_float(ra[c][i]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[sb]);

      const int valid_all = kvL - j * BKV;        // keys of this tile, >= 1
      const int valid = valid_all - col0;         // keys of this group (may be <= 0 or >= COLS)
      if (valid < COLS) {
#pragma unroll
        for (int c = 0; c < COLS; ++c) s[c] = c < valid ? s[c] : -INFINITY;
      }
      // tree-shaped max over this group's columns, then exchange with the
      // other groups of the row (double-buffered by tile parity, bounded wait)
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = s[i];
#pragma unroll
      for (int c = 8; c < COLS; c += 8) {
#pragma unroll
        for (int i = 0; i < 8; ++i) mx[i] = fmaxf(mx[i], s[c + i]);
      }
      const float mloc = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                               fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      float* rm = red_max + (j & 1) * (NGRP * 128);
      rm[grp * 128 + r] = mloc;
      __syncwarp();
      if (lane == 0) mbar_arrive(&max_ready[j & 1]);
      if (!mbar_wait(&max_ready[j & 1], use & 1, abort_flag, p.err)) { ok = false; break; }
      float mall = rm[r];
#pragma unroll
      for (int g = 1; g < NGRP; ++g) mall = fmaxf(mall, rm[g * 128 + r]);
      const float mt = mall * scale_log2;
      const float m_new = fmaxf(m_ref, mt);
      const bool need = (j == 0) || (m_new > m_ref + RESCALE_THRESHOLD);
      float alpha = 1.f;
      if (need) {
        alpha = (j == 0) ? 0.f : ex2(m_ref - m_new);
        m_ref = m_new;
      }
      const float neg = -m_ref;
      float rs[4] = {0.f, 0.f, 0.f, 0.f};
      uint32_t pk[COLS / 2];
#pragma unroll
      for (int c = 0; c < COLS; c += 2) {
        const float p0 = ex2(fmaf(s[c], scale_log2, neg));
        const float p1 = ex2(fmaf(s[c + 1], scale_log2, neg));
        rs[(c >> 1) & 3] += p0 + p1;
        pk[c >> 1] = pack2(p0, p1, F16);
      }
      l = l * alpha + ((rs[0] + rs[1]) + (rs[2] + rs[3]));

      if (valid_all < BKV && grp < 2) {
        // last, partial key tile: groups 0 and 1 clear value panels 0 and 1
        // of the rows past kv_len so stale (possibly non-finite) data cannot
        // meet the zero probabilities
        if (!mbar_wait(&v_full[sb], use & 1, abort_flag, p.err)) { ok = false; break; }
        if (r >= valid_all) {
          uint4* v = reinterpret_cast<uint4*>(smem + OFF_V + sb * TILE_BYTES + grp * PANEL + r * 128);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] = make_uint4(0, 0, 0, 0);
        }
      }
      if (j > 0) {
        if (!mbar_wait(pv_done, (j - 1) & 1, abort_flag, p.err)) { ok = false; break; }
        tc_fence_after();
        if (__any_sync(0xffffffffu, need)) {
#pragma unroll 1
          for (int c = 0; c < COLS / 32; ++c) {
            uint32_t rr[32];
            const uint32_t ta = tmem + lane_off + 256 + col0 + 32 * c;
            tmem_ld32(ta, rr);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) rr[i] = __float_as_uint(__uint_as_float(rr[i]) * alpha);
            tmem_st32(ta, rr);
          }
          tmem_st_wait();
        }
      }
#pragma unroll
      for (int c = 0; c < COLS / 8; ++c) {
        uint4* dst = reinterpret_cast<uint4*>(sProw + (((chunk0 + c) ^ (r & 7)) * 16));
        *dst = make_uint4(pk[4 * c + 0], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    if (ok && nkv > 0) {
      red_sum[grp * 128 + r] = l;
      __syncwarp();
      if (lane == 0) mbar_arrive(sum_ready);
      ok = mbar_wait(sum_ready, 0, abort_flag, p.err) && mbar_wait(pv_done, (nkv - 1) & 1, abort_flag, p.err);
    }
    if (ok && nkv > 0) {
      tc_fence_after();
      float lsum = 0.f;
#pragma unroll
      for (int g = 0; g < NGRP; ++g) lsum += red_sum[g * 128 + r];
      const float inv_l = 1.f / lsum;
      const int row = q0 + r;
      const bool valid_row = (qt * BQ + r) < L;
      uint16_t* orow =
          reinterpret_cast<uint16_t*>(p.out) + static_cast<size_t>(valid_row ? row : 0) * p.ldo + h * DH + col0;
#pragma unroll 1
      for (int c = 0; c < COLS / 32; ++c) {
        uint32_t rr[32];
        tmem_ld32(tmem + lane_off + 256 + col0 + 32 * c, rr);
        tmem_ld_wait();
        if (valid_row) {
          uint4* dst = reinterpret_cast<uint4*>(orow + 32 * c);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            dst[i] = make_uint4(pack2(__uint_as_float(rr[8 * i + 0]) * inv_l, __uint_as_float(rr[8 * i + 1]) * inv_l, F16),
                                pack2(__uint_as_float(rr[8 * i + 2]) * inv_l, __uint_as_float(rr[8 * i + 3]) * inv_l, F16),
                                pack2(__uint_as_float(rr[8 * i + 4]) * inv_l, __uint_as_float(rr[8 * i + 5]) * inv_l, F16),
                                pack2(__uint_as_float(rr[8 * i + 6]) * inv_l, __uint_as_float(rr[8 * i + 7]) * inv_l, F16));
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// One block: per-segment key counts -> work units (b, h, q-tile) ordered by
// descending kv length so the longest segments start first.
__global__ void attn_schedule_kernel(const int* cu, const int* kv_len, int B, int H, int T_cap, int4* work,
                                     int* work_count, int max_units, int* err) {
  extern __shared__ int sh[];
  int* ntile = sh;           // [B]
  int* kvs = sh + B;         // [B]
  int* off = sh + 2 * B;     // [B]
  int* rank = sh + 3 * B;    // [B]
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    const int L = cu[i + 1] - cu[i];
    int kv = kv_len ? kv_len[i] : L;
    if (L < 0 || cu[i] < 0 || cu[i + 1] > T_cap || kv > L || (L > 0 && kv <= 0)) {
      record_error(err, kErrLayout);
      kv = 0;
    }
    ntile[i] = (kv > 0) ? (L + BQ - 1) / BQ : 0;
    kvs[i] = kv;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    int rk = 0;
    for (int k = 0; k < B; ++k) rk += (kvs[k] > kvs[i]) || (kvs[k] == kvs[i] && k < i);
    rank[i] = rk;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // walk segments in rank order accumulating offsets
    int acc = 0;
    for (int rk = 0; rk < B; ++rk) {
      for (int i = 0; i < B; ++i) {
        if (rank[i] == rk) {
          off[i] = acc;
          acc += H * ntile[i];
          break;
        }
      }
    }
    if (acc > max_units) {
      record_error(err, kErrCapacity);
      acc = max_units;
    }
    *work_count = acc;
  }
  __syncthreads();
  for (int i = 0; i < B; ++i) {
    const int n = H * ntile[i];
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
      const int idx = off[i] + k;
      if (idx < max_units) work[idx] = make_int4(i, k / ntile[i], k % ntile[i], 0);
    }
  }
}

template <bool F16>
cudaError_t launch_typed(const CUtensorMap& mQKV, const AttnParams& p, int grid, cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(tc_attn_kernel<F16>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  if (grid <= 0) return cudaSuccess;
  tc_attn_kernel<F16><<<grid, THREADS, SMEM_BYTES, st>>>(mQKV, p);
  return cudaGetLastError();
}

}  // namespace

int tc_attn_smem_bytes() { return SMEM_BYTES; }

cudaError_t launch_tc_attn(const CUtensorMap& mQKV, const AttnParams& p, int grid, bool f16, cudaStream_t st) {
  return f16 ? launch_typed<true>(mQKV, p, grid, st) : launch_typed<false>(mQKV, p, grid, st);
}

cudaError_t launch_attn_schedule(const int* cu, const int* kv_len, int B, int n_heads, int T_cap, int4* work,
                                 int* work_count, int max_units, int* err, cudaStream_t st) {
  const size_t sm = static_cast<size_t>(4) * B * sizeof(int);
  if (sm > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(attn_schedule_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(sm));
    if (e != cudaSuccess) return e;
  }
  attn_schedule_kernel<<<1, 256, sm, st>>>(cu, kv_len, B, n_heads, T_cap, work, work_count, max_units, err);
  return cudaGetLastError();
}

}  // namespace seer
