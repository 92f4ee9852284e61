// Varlen bidirectional attention on tcgen05 for sm_103a (head_dim 128; q, k,
// v, the probabilities P and the output all f16, or all bf16).
//
// Seer Sec. 3.6 Eqs. 6-7 and 9-10: every query row of a segment attends to
// the first kv_len[b] rows of the same segment, with no causal mask; rows
// beyond kv_len (bucket padding of the static path) are never keys.
//
// One CTA per (segment, head, 128-query tile); 64 + 128 * NGRP threads:
//   warp 0     TMA producers: Q once, then K_j (lane 0) and V_j (lane 1),
//              128 keys x 128 dims with 128-byte swizzle, each in a 3-deep
//              ring (key tiles take ~2000 cycles to land under load);
//   warp 1     TMEM allocator + MMA issuer: S_j = Q K_j^T (M=N=128, K=16 x 8)
//              into one of two S buffers, then O += P_j V_j (V as an MN-major
//              operand) into the O accumulator.  Q and P are A operands read
//              from tensor memory, so each MMA streams only its B operand
//              from shared memory (shared-memory bandwidth bounds an
//              all-shared-memory version);
//   warps 2.. softmax, NGRP groups of four warps: a query row (one TMEM
//              lane) is shared by one thread of each group, which owns
//              128 / NGRP of the key columns (and of the output dims); the
//              parts of a row exchange their maxima through shared memory
//              once per key tile (an mbarrier, so every wait is bounded).
//              Online softmax in the log2 domain with lazy rescaling: O is
//              rescaled in TMEM only when the running max grows by more than
//              2^8.  The softmax warps stage Q into tensor memory once and
//              write each P_j there (tcgen05.st).
// The QK^T MMAs run up to two key tiles ahead of the softmax.
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
// Six 32 KB slots: Q in slot 0 (free again once Q sits in tensor memory),
// K stages 0, 1, 2 in slots 1, 2, 0 and V stages 0, 1, 2 in slots 3, 4, 5.
constexpr int KV_STAGES = 3;
constexpr int OFF_Q = 0;
__host__ __device__ constexpr int k_slot(int st) { return (st == 2 ? 0 : st + 1) * TILE_BYTES; }
__host__ __device__ constexpr int v_slot(int st) { return (3 + st) * TILE_BYTES; }
constexpr int OFF_BAR = 6 * TILE_BYTES;
constexpr int OFF_RED = OFF_BAR + 256;      // float max[2 tiles][NGRP][128] + float sum[NGRP][128]
constexpr int SMEM_BYTES = OFF_RED + (2 * NGRP * 128 + NGRP * 128) * 4 + 1024;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t TM_O = 256;              // TMEM columns: S0 [0,128), S1 [128,256), O [256,384),
constexpr uint32_t TM_Q = 384;              //   Q [384,448) and P [448,512) as packed 16-bit pairs
constexpr uint32_t TM_P = 448;
static_assert(NGRP == 2, "the TMEM staging of Q and P assumes two 64-column groups");
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
  uint64_t* k_full = bars + 1;     // [KV_STAGES]
  uint64_t* k_empty = bars + 4;    // [KV_STAGES]
  uint64_t* v_full = bars + 7;     // [KV_STAGES]
  uint64_t* v_empty = bars + 10;   // [KV_STAGES]
  uint64_t* s_full = bars + 13;    // [2]
  uint64_t* s_empty = bars + 15;   // [2]
  uint64_t* p_full = bars + 17;
  uint64_t* pv_done = bars + 18;
  uint64_t* max_ready = bars + 19; // [2] row-max exchange, one per tile parity
  uint64_t* sum_ready = bars + 21;
  uint64_t* q_staged = bars + 22;  // Q copied from shared to tensor memory
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 23);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* red_max = reinterpret_cast<float*>(smem + OFF_RED);   // [2 tiles][NGRP][128] partial row maxima
  float* red_sum = red_max + 2 * NGRP * 128;                   // [NGRP][128] partial row sums

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < KV_STAGES; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], SOFTMAX_WARPS);
      mbar_init(&max_ready[i], SOFTMAX_WARPS);
    }
    mbar_init(p_full, SOFTMAX_WARPS);
    mbar_init(pv_done, 1);
    mbar_init(sum_ready, SOFTMAX_WARPS);
    mbar_init(q_staged, SOFTMAX_WARPS);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // -------------------------------------------------- TMA producer
    // lane 0 loads Q and the K tiles, lane 1 the V tiles, so waiting for a V
    // buffer (freed by PV) never delays the next K (needed by QK^T).
    if (lane == 0) {
      tma_prefetch_desc(&mQKV);
      mbar_arrive_expect_tx(q_full, TILE_BYTES);
      tma_load_2d(smem + OFF_Q, &mQKV, q_full, xq, q0);
      tma_load_2d(smem + OFF_Q + PANEL, &mQKV, q_full, xq + 64, q0);
    }
    if (lane < 2) {
      const bool is_k = lane == 0;
      uint64_t* full = is_k ? k_full : v_full;
      uint64_t* empty = is_k ? k_empty : v_empty;
      const int x = is_k ? xk : xv;
      int issued = 0;
      for (int j = 0; j < nkv; ++j) {
        const int st = j % KV_STAGES, use = j / KV_STAGES;
        if (use > 0 && !mbar_wait(&empty[st], (use - 1) & 1, abort_flag, p.err)) break;
        // K stage 2 reuses Q's slot: wait until Q has been staged in tensor memory
        if (is_k && j == 2 && !mbar_wait(q_staged, 0, abort_flag, p.err)) break;
        uint8_t* dst = smem + (is_k ? k_slot(st) : v_slot(st));
        mbar_arrive_expect_tx(&full[st], TILE_BYTES);
        tma_load_2d(dst, &mQKV, &full[st], x, seq0 + j * BKV);
        tma_load_2d(dst + PANEL, &mQKV, &full[st], x + 64, seq0 + j * BKV);
        ++issued;
      }
      if (*abort_flag) {
        if (is_k) mbar_wait_drain(q_full, 0, 200000000ull);
        for (int j = issued > KV_STAGES ? issued - KV_STAGES : 0; j < issued; ++j)
          mbar_wait_drain(&full[j % KV_STAGES], (j / KV_STAGES) & 1, 200000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      // Issues QK^T for tile js as soon as K_js has landed and its S buffer is
      // free (up to two tiles ahead of the softmax), and PV for tile jp as soon
      // as P_jp is ready; both conditions are polled, never blocked on, so a
      // slow softmax never holds back the next QK^T.
      constexpr uint32_t idesc_qk = make_idesc(BQ, BKV, 0, F16);
      constexpr uint32_t idesc_pv = make_idesc(BQ, DH, 1, F16);
      bool ok = mbar_wait(q_staged, 0, abort_flag, p.err);
      int js = 0, jp = 0;
      uint64_t t_idle = 0;
      uint32_t spins = 0;
      while (ok && jp < nkv) {
        bool progressed = false;
        if (js < nkv) {
          const int sb = js & 1, use = js >> 1;
          const int kst = js % KV_STAGES, kuse = js / KV_STAGES;
          if (mbar_test_wait(&k_full[kst], kuse & 1) && (use == 0 || mbar_test_wait(&s_empty[sb], (use - 1) & 1))) {
            tc_fence_after();
            const uint32_t sk = smem_u32(smem + k_slot(kst));
#pragma unroll
            for (int k = 0; k < DH / 16; ++k) {
              // A = Q from tensor memory, B = K_js (K-major, 128-byte swizzle)
              const uint32_t off = (k >> 2) * PANEL + (k & 3) * 32;
              tc_mma_f16_tmem_a(tmem + sb * 128, tmem + TM_Q + 8 * k, make_sdesc_sw128(sk + off, 16, 1024), idesc_qk,
                                k > 0 ? 1u : 0u);
            }
            tc_commit(&k_empty[kst]);
            tc_commit(&s_full[sb]);
            ++js;
            progressed = true;
          }
        }
        if (jp < js) {
          const int vst = jp % KV_STAGES, vuse = jp / KV_STAGES;
          if (mbar_test_wait(&v_full[vst], vuse & 1) && mbar_test_wait(p_full, jp & 1)) {
            tc_fence_after();
            const uint32_t sv = smem_u32(smem + v_slot(vst));
#pragma unroll
            for (int k = 0; k < BKV / 16; ++k) {
              // A = P from tensor memory (8 columns per 16 keys); B = V, which is
              // [keys, dims] with dims contiguous: an MN-major operand whose two
              // 64-dim panels are PANEL bytes apart (LBO), 8-key groups 1 KB apart (SBO)
              const uint64_t bd = make_sdesc_sw128(sv + k * 16 * 128, PANEL, 1024);
              tc_mma_f16_tmem_a(tmem + TM_O, tmem + TM_P + 8 * k, bd, idesc_pv, (jp > 0 || k > 0) ? 1u : 0u);
            }
            tc_commit(&v_empty[vst]);
            tc_commit(pv_done);
            ++jp;
            progressed = true;
          }
        }
        if (progressed) {
          spins = 0;
        } else if ((++spins & 255u) == 0) {
          // bounded: give up (and let every role unwind) after the wait limit
          const uint64_t now = globaltimer_ns();
          if (t_idle == 0) t_idle = now;
          if (*abort_flag) break;
          if (now - t_idle > kWaitLimitNs) {
            *abort_flag = 1;
            record_error(p.err, kErrTimeout);
            break;
          }
        }
        if (progressed) t_idle = 0;
      }
    }
  } else {
    // -------------------------------------------------- softmax warps 2..
    const int grp = (warp - 2) >> 2;              // column group: keys / output dims [COLS grp, COLS grp + COLS)
    const int qw = warp & 3;
    const int r = qw * 32 + lane;                 // query row inside the tile == TMEM lane
    const int col0 = grp * COLS;
    const uint32_t lane_off = static_cast<uint32_t>(qw * 32) << 16;
    const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));
    float m_ref = -INFINITY;                      // running max, log2 units
    float l = 0.f;                                // partial row sum over this thread's columns
    bool ok = mbar_wait(q_full, 0, abort_flag, p.err);
    if (ok) {
      // stage Q row r, dims [col0, col0 + 64) (swizzle panel grp) into tensor
      // memory: 16-byte chunk c of the row sits at (r / 8) * 1024 + (r % 8) * 128
      // + ((c ^ (r % 8)) * 16) of the panel
      const uint8_t* qrow = smem + OFF_Q + grp * PANEL + (r >> 3) * 1024 + (r & 7) * 128;
      uint32_t qv[32];
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        const uint4 v = *reinterpret_cast<const uint4*>(qrow + ((c ^ (r & 7)) * 16));
        qv[4 * c + 0] = v.x; qv[4 * c + 1] = v.y; qv[4 * c + 2] = v.z; qv[4 * c + 3] = v.w;
      }
      tmem_st32(tmem + lane_off + TM_Q + 32 * grp, qv);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_staged);
    }
    for (int j = 0; ok && j < nkv; ++j) {
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
      // pairwise max tree over this group's columns, then exchange with the
      // other groups of the row (double-buffered by tile parity, bounded wait)
      float mx[COLS / 2];
#pragma unroll
      for (int i = 0; i < COLS / 2; ++i) mx[i] = fmaxf(s[2 * i], s[2 * i + 1]);
#pragma unroll
      for (int w = COLS / 4; w >= 1; w >>= 1) {
#pragma unroll
        for (int i = 0; i < w; ++i) mx[i] = fmaxf(mx[i], mx[i + w]);
      }
      const float mloc = mx[0];
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
        const int vst = j % KV_STAGES;
        if (!mbar_wait(&v_full[vst], (j / KV_STAGES) & 1, abort_flag, p.err)) { ok = false; break; }
        if (r >= valid_all) {
          uint4* v = reinterpret_cast<uint4*>(smem + v_slot(vst) + grp * PANEL + r * 128);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
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
      // this thread's keys of row r -> P in tensor memory (packed pairs)
      tmem_st32(tmem + lane_off + TM_P + 32 * grp, pk);
      tmem_st_wait();
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
