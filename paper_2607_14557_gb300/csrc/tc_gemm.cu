// Persistent tcgen05 GEMM for sm_103a: C[M, N] = A[M, K] * B[N, K]^T with
// 16-bit operands (both f16 or both bf16, chosen by the instruction
// descriptor) and fp32 accumulation in tensor memory (TMEM); C and the
// residual R are f16 or bf16 independently.
//
// One CTA per SM, 192 threads, warp-specialised:
//   warp 0      TMA producer: 128x64 A tile + two 128x64 B tiles per stage
//               (128-byte swizzle), 4-stage ring of 48 KB stages;
//   warp 1      TMEM allocator + MMA issuer: 4 x tcgen05.mma (M=128, N=256,
//               K=16) per stage into one of two 256-column fp32
//               accumulators (double buffered, 512 columns);
//               producer and issuer are whole warps in lockstep, one elected
//               lane issuing;
//   warps 2-5   epilogue: tcgen05.ld of the accumulator (each warp owns one
//               32-lane quarter of TMEM = 32 output rows), fused epilogue,
//               32 x 32 output chunks staged in shared memory and written by
//               TMA stores marked L2 evict-first (a tile whose rows run past
//               the device row count stores its valid rows lane by lane).
// The epilogue of tile t overlaps the main loop of tile t+1.  Every CTA waits
// for the previous kernel of the stream at entry (griddepcontrol.wait) and
// lets the next kernel launch once its last MMAs are issued.
//
// Epilogues (Sec. 3.1 Eq. 2 projections; Sec. 3.2 sparsity hook):
//   Store     C = A B^T                                    (QKV projection)
//   Residual  C = A B^T + R                                (O / down projection)
//   Swiglu    B = [Wg tile ; Wu tile] -> act = SiLU(g) * u  (gate/up), plus the
//             per-row count of |act| < eps on response rows (step-0 hook)
//   Count     detector: A rows gathered per sequence window, counts only
//   Rope      Store, then the q|k columns rotated per 128-wide head by the
//             rotary embedding at each row's position in its sequence
// Every stored 16-bit value passes a range guard: an infinite or NaN result
// (an f16 intermediate that overflowed +-65504) records kErrRange in the
// device error word, which seer_check_device reports.
#include "common.cuh"
#include "kernels.h"

namespace seer {
namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;
constexpr int STAGES = 4;
constexpr int A_TILE_BYTES = BM * BK * 2;            // 16 KB
constexpr int B_HALF_BYTES = 128 * BK * 2;           // 16 KB
constexpr int STAGE_BYTES = A_TILE_BYTES + 2 * B_HALF_BYTES;  // 48 KB
constexpr int THREADS = 192;
constexpr int ACC_COLS = 256;
constexpr int TMEM_COLS = 512;
constexpr int BAR_BYTES = 256;
constexpr int ROPE_HEAD = 128;                       // head width of the Rope epilogue
constexpr int ROPE_BYTES = ROPE_HEAD / 2 * 8;        // (hi, lo) inverse frequency per pair
constexpr int EPI_CHUNK = 32 * 32 * 2;              // a warp's 32 rows x 32 columns, 16-bit
constexpr int EPI_BYTES = 4 * 2 * EPI_CHUNK;         // 4 epilogue warps x 2 staging buffers
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + BAR_BYTES + ROPE_BYTES + EPI_BYTES + 1024;

// Raster: groups of `group_m` m-tiles; inside a group m varies fastest and
// the group sweeps every n-tile.  group_m = 1 keeps the whole B operand hot in
// L2 while A streams once; a large group_m keeps a slab of A hot while B
// streams once per group (chosen on the host from the operand sizes).
__device__ __forceinline__ void tile_coords(int t, int num_m, int num_n, int group_m, int& m, int& n) {
  const int per_group = group_m * num_n;
  const int g = t / per_group;
  const int r = t - g * per_group;
  const int m0 = g * group_m;
  const int gm = min(group_m, num_m - m0);
  m = m0 + r % gm;
  n = r / gm;
}

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + __expf(-g)); }

template <int MODE>
__global__ void __launch_bounds__(THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB0,
                   const __grid_constant__ CUtensorMap mB1, const __grid_constant__ CUtensorMap mC, const GemmParams p) {
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float2* rope_tab = reinterpret_cast<float2*>(smem + STAGES * STAGE_BYTES + BAR_BYTES);
  uint8_t* epi_stage = smem + STAGES * STAGE_BYTES + BAR_BYTES + ROPE_BYTES;   // [4 warps][2][EPI_CHUNK]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- problem size (device row counts are clamped, never trusted blindly)
  int M = p.M_cap;
  int num_m, tiles_per_seq = 1;
  if (MODE == kGemmCount) {
    tiles_per_seq = (p.Nw + BM - 1) / BM;
    num_m = p.B * tiles_per_seq;
  } else {
    if (p.M_dev != nullptr) {
      const int md = *p.M_dev;
      if (md < 0 || md > p.M_cap) {
        if (threadIdx.x == 0 && blockIdx.x == 0) record_error(p.err, kErrRows);
        M = md < 0 ? 0 : p.M_cap;
      } else {
        M = md;
      }
    }
    num_m = (M + BM - 1) / BM;
  }
  const bool halfN = (MODE == kGemmSwiglu || MODE == kGemmCount);
  const int num_n = halfN ? p.N / 128 : p.N / BN;
  const int num_tiles = num_m * num_n;
  const int KB = p.K / BK;
  const int group_m = p.group_m > 0 ? p.group_m : 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    // Producer and issuer run as whole warps in lockstep (every wait by all
    // lanes, with a warp-uniform outcome); the elected lane issues the copies
    // and MMAs.  A lone lane in a divergent branch loses issue slots to the
    // FMA-heavy epilogue warp on its SM sub-partition.
    const bool leader = elect_one();
    if (leader) {
      tma_prefetch_desc(&mA);
      tma_prefetch_desc(&mB0);
      tma_prefetch_desc(&mB1);
    }
    int s = 0;
    uint32_t ph = 0;
    long issued = 0;
    for (int t = blockIdx.x; t < num_tiles && !__any_sync(0xffffffffu, *abort_flag != 0); t += gridDim.x) {
      int m, n;
      tile_coords(t, num_m, num_n, group_m, m, n);
      int a_row;
      if (MODE == kGemmCount) {
        const int b = m / tiles_per_seq;
        const int j = m - b * tiles_per_seq;
        const int rs = p.resp_start[b];
        if (leader && (rs < 0 || rs + p.Nw > p.M_cap)) record_error(p.err, kErrLayout);
        a_row = rs + j * BM;
      } else {
        a_row = m * BM;
      }
      const int b_row0 = halfN ? n * 128 : n * BN;
      const int b_row1 = halfN ? n * 128 : n * BN + 128;
      bool ok = true;
      for (int kb = 0; kb < KB; ++kb) {
        if (!warp_wait(&empty[s], ph ^ 1u, abort_flag, p.err)) { ok = false; break; }
        if (leader) {
          uint8_t* sa = smem + s * STAGE_BYTES;
          mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
          tma_load_2d(sa, &mA, &full[s], kb * BK, a_row);
          tma_load_2d(sa + A_TILE_BYTES, &mB0, &full[s], kb * BK, b_row0);
          tma_load_2d(sa + A_TILE_BYTES + B_HALF_BYTES, &mB1, &full[s], kb * BK, b_row1);
        }
        __syncwarp();
        ++issued;
        if (++s == STAGES) { s = 0; ph ^= 1u; }
      }
      if (!ok) break;
    }
    if (*abort_flag && leader) {
      // let copies still in flight land before the CTA's shared memory is released
      const long first = issued > STAGES ? issued - STAGES : 0;
      for (long i = first; i < issued; ++i)
        mbar_wait_drain(&full[i % STAGES], static_cast<uint32_t>((i / STAGES) & 1), 200000000ull);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    const bool leader = elect_one();
    const uint32_t idesc = p.idesc;
    int s = 0;
    uint32_t ph = 0;
    int acc = 0;
    uint32_t acc_ph = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
      if (!warp_wait(&acc_empty[acc], acc_ph ^ 1u, abort_flag, p.err)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * ACC_COLS);
      bool ok = true;
      for (int kb = 0; kb < KB; ++kb) {
        if (!warp_wait(&full[s], ph, abort_flag, p.err)) { ok = false; break; }
        tc_fence_after();
        if (leader) {
          const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
          const uint64_t adesc = make_sdesc_sw128(sa, 16, 1024);
          const uint64_t bdesc = make_sdesc_sw128(sa + A_TILE_BYTES, 16, 1024);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // +32 bytes along K inside the 128-byte swizzle atom = +2 in the address field
            tc_mma_f16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb | k) != 0 ? 1u : 0u);
          }
          tc_commit(&empty[s]);
        }
        __syncwarp();
        if (++s == STAGES) { s = 0; ph ^= 1u; }
      }
      if (!ok) break;
      if (leader) tc_commit(&acc_full[acc]);
      __syncwarp();
      if (++acc == 2) { acc = 0; acc_ph ^= 1u; }
    }
    if (leader) pdl_trigger();                   // last MMAs issued: the next kernel may launch
  } else {
    // -------------------------------------------------- epilogue warps 2..5
    const int q = warp & 3;                    // TMEM lane quarter owned by this warp
    const int row_in_tile = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    uint8_t* my_stage = epi_stage + q * 2 * EPI_CHUNK;
    // outputs stream through L2 marked evict-first, so they do not push the
    // operand slabs the raster keeps resident out of the cache
    const uint64_t out_policy = l2_policy_evict_first();
    int n_chunks = 0;                            // bulk stores issued by this warp (staging buffer = n & 1)
    // one staged 32 x 32 chunk of this warp's rows -> a TMA store at (x, y); the
    // buffer used two chunks ago is reused only once its store has read it
    auto store_chunk = [&](const uint32_t (&w)[16], int x, int y) {
      uint8_t* buf = my_stage + (n_chunks & 1) * EPI_CHUNK;
      if (lane == 0 && n_chunks >= 2) bulk_wait_read_1();
      __syncwarp();
      uint4* d = reinterpret_cast<uint4*>(buf + lane * 64);
#pragma unroll
      for (int i = 0; i < 4; ++i) d[i] = make_uint4(w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d_hint(&mC, buf, x, y, out_policy);
        bulk_commit();
      }
      ++n_chunks;
    };
    if (MODE == kGemmRope) {
      const int et = threadIdx.x - 64;                 // 0..127 over the epilogue warps
      if (et < ROPE_HEAD / 2) rope_tab[et] = rope_inv_freq(et, ROPE_HEAD, p.rope_theta);
      asm volatile("bar.sync 1, 128;" ::: "memory");
    }
    int acc = 0;
    uint32_t acc_ph = 0;
    uint32_t nonfinite = 0;                      // range guard over this thread's stores
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
      int m, n;
      tile_coords(t, num_m, num_n, group_m, m, n);
      // warp-uniform outcome: the TMEM loads below are warp-collective, and
      // after an abort the lanes of a warp could otherwise decide differently
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[acc], acc_ph, abort_flag, p.err))) break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + lane_off + static_cast<uint32_t>(acc * ACC_COLS);
      if (MODE == kGemmRope) {
        // the tile holds two heads; pair (c, c + 64) of a head rotates by pos * f_c
        const int row = m * BM + row_in_tile;
        const bool valid = row < M;
        const bool rotate = n * BN < p.rope_cols;       // tile-uniform (rope_cols % BN == 0)
        const bool of16 = p.out_type == kF16;
        uint16_t* crow = reinterpret_cast<uint16_t*>(p.C) + static_cast<size_t>(valid ? row : 0) * p.ldc + n * BN;
        const float pos = (valid && rotate) ? static_cast<float>(row_position(p.cu, p.B, row)) : 0.f;
#pragma unroll 1
        for (int c = 0; c < ROPE_HEAD / 64; ++c) {
          float cs[32], sn[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            if (rotate) rope_cos_sin(pos, rope_tab[c * 32 + e], cs[e], sn[e]);
            else { cs[e] = 1.f; sn[e] = 0.f; }
          }
#pragma unroll 1
          for (int hh = 0; hh < BN / ROPE_HEAD; ++hh) {
            const int c0 = hh * ROPE_HEAD + c * 32, c1 = c0 + ROPE_HEAD / 2;
            uint32_t r0[32], r1[32];
            tmem_ld32(tacc + c0, r0);
            tmem_ld32(tacc + c1, r1);
            tmem_ld_wait();
            if (valid) {
              float v0[32], v1[32];
#pragma unroll
              for (int e = 0; e < 32; ++e) {
                const float x0 = __uint_as_float(r0[e]), x1 = __uint_as_float(r1[e]);
                v0[e] = fmaf(x0, cs[e], -x1 * sn[e]);
                v1[e] = fmaf(x1, cs[e], x0 * sn[e]);
              }
#pragma unroll
              for (int i = 0; i < 2; ++i) {
                uint32_t q0[8], q1[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                  q0[e] = pack2(v0[16 * i + 2 * e], v0[16 * i + 2 * e + 1], of16);
                  q1[e] = pack2(v1[16 * i + 2 * e], v1[16 * i + 2 * e + 1], of16);
                  nonfinite |= nonfinite_term(q0[e], of16) | nonfinite_term(q1[e], of16);
                }
                st_global_v8(crow + c0 + 16 * i, q0[0], q0[1], q0[2], q0[3], q0[4], q0[5], q0[6], q0[7]);
                st_global_v8(crow + c1 + 16 * i, q1[0], q1[1], q1[2], q1[3], q1[4], q1[5], q1[6], q1[7]);
              }
            }
          }
        }
      } else if (MODE == kGemmStore || MODE == kGemmResidual) {
        const int row = m * BM + row_in_tile;
        const bool valid = row < M;
        const bool slab_full = m * BM + q * 32 + 32 <= M;      // this warp's 32 rows all valid: TMA store
        const bool of16 = p.out_type == kF16, rf16 = p.res_type == kF16;
        uint16_t* crow = reinterpret_cast<uint16_t*>(p.C) + static_cast<size_t>(valid ? row : 0) * p.ldc + n * BN;
        const uint16_t* rrow =
            MODE == kGemmResidual ? reinterpret_cast<const uint16_t*>(p.R) + static_cast<size_t>(valid ? row : 0) * p.ldr + n * BN
                                  : nullptr;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tacc + c * 32, r);
          tmem_ld_wait();
          if (slab_full || valid) {
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
            if (MODE == kGemmResidual) {
              const uint4* rp = reinterpret_cast<const uint4*>(rrow + c * 32);
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const uint4 rv = rp[i];
                v[8 * i + 0] += lo16(rv.x, rf16); v[8 * i + 1] += hi16(rv.x, rf16);
                v[8 * i + 2] += lo16(rv.y, rf16); v[8 * i + 3] += hi16(rv.y, rf16);
                v[8 * i + 4] += lo16(rv.z, rf16); v[8 * i + 5] += hi16(rv.z, rf16);
                v[8 * i + 6] += lo16(rv.w, rf16); v[8 * i + 7] += hi16(rv.w, rf16);
              }
            }
            uint32_t w[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              w[i] = pack2(v[2 * i], v[2 * i + 1], of16);
              nonfinite |= nonfinite_term(w[i], of16);
            }
            if (slab_full) {
              store_chunk(w, n * BN + c * 32, m * BM + q * 32);
            } else {
              // a lane owns one row: 64 contiguous bytes as two full 32-byte sectors
              st_global_v8(crow + c * 32, w[0], w[1], w[2], w[3], w[4], w[5], w[6], w[7]);
              st_global_v8(crow + c * 32 + 16, w[8], w[9], w[10], w[11], w[12], w[13], w[14], w[15]);
            }
          }
        }
      } else {
        // gate columns 0..127, up columns 128..255 of the accumulator
        int row, cnt_idx = -1;
        bool store = false;
        if (MODE == kGemmCount) {
          const int b = m / tiles_per_seq;
          const int tl = (m - b * tiles_per_seq) * BM + row_in_tile;
          row = -1;
          if (tl < p.Nw) cnt_idx = b * p.Nw + tl;
        } else {
          row = m * BM + row_in_tile;
          store = row < M;
          if (store && p.counts != nullptr) {
            // segment of this row (binary search in cu), then its window offset
            int lo = 0, hi = p.B;
            while (hi - lo > 1) {
              const int mid = (lo + hi) >> 1;
              if (p.cu[mid] <= row) lo = mid; else hi = mid;
            }
            const int tl = row - p.resp_start[lo];
            if (tl >= 0 && tl < p.Nw && row < p.cu[lo + 1]) cnt_idx = lo * p.Nw + tl;
          }
        }
        int cnt = 0;
        const bool of16 = p.out_type == kF16;
        uint16_t* arow =
            MODE == kGemmSwiglu ? reinterpret_cast<uint16_t*>(p.C) + static_cast<size_t>(store ? row : 0) * p.ldc + n * 128
                                : nullptr;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t g[32], u[32];
          tmem_ld32(tacc + c * 32, g);
          tmem_ld32(tacc + 128 + c * 32, u);
          tmem_ld_wait();
          float a[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            a[i] = silu_f(__uint_as_float(g[i])) * __uint_as_float(u[i]);
            cnt += fabsf(a[i]) < p.act_eps ? 1 : 0;
          }
          if (MODE == kGemmSwiglu) {
            const bool slab_full = m * BM + q * 32 + 32 <= M;
            if (slab_full || store) {
              uint32_t w[16];
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                w[i] = pack2(a[2 * i], a[2 * i + 1], of16);
                nonfinite |= nonfinite_term(w[i], of16);
              }
              if (slab_full) {
                store_chunk(w, n * 128 + c * 32, m * BM + q * 32);
              } else {
                st_global_v8(arow + c * 32, w[0], w[1], w[2], w[3], w[4], w[5], w[6], w[7]);
                st_global_v8(arow + c * 32 + 16, w[8], w[9], w[10], w[11], w[12], w[13], w[14], w[15]);
              }
            }
          }
        }
        if (cnt_idx >= 0 && p.counts != nullptr) atomicAdd(&p.counts[cnt_idx], cnt);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);
      if (++acc == 2) { acc = 0; acc_ph ^= 1u; }
    }
    report_range(nonfinite, p.err);              // a stored value overflowed the 16-bit type (or was NaN)
    if (lane == 0) bulk_wait_all();              // outputs written before the CTA exits
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

template <int MODE>
cudaError_t launch_mode(const CUtensorMap& mA, const CUtensorMap& mB0, const CUtensorMap& mB1, const CUtensorMap& mC,
                        const GemmParams& p, int num_sms, cudaStream_t st) {
  static bool attr_set[64] = {};
  cudaError_t e = set_smem_limit_once(tc_gemm_kernel<MODE>, SMEM_BYTES, attr_set);
  if (e != cudaSuccess) return e;
  long num_m;
  if (MODE == kGemmCount) num_m = static_cast<long>(p.B) * ((p.Nw + BM - 1) / BM);
  else num_m = (p.M_cap + BM - 1) / BM;
  const long num_n = (MODE == kGemmSwiglu || MODE == kGemmCount) ? p.N / 128 : p.N / BN;
  long tiles = num_m * num_n;
  if (tiles <= 0) return cudaSuccess;
  const int grid = static_cast<int>(tiles < num_sms ? tiles : num_sms);
  // Overlapping the launch with the previous kernel pays off for short GEMMs,
  // where the launch gap is a visible share of the run.  Long GEMMs launched
  // that way measured 5-8% slower on GB300 (cause not isolated; their blocks
  // are then placed in the order the previous kernel's blocks retire), so
  // they launch normally.
  constexpr long kOverlapMaxSteps = 320;     // k-blocks per CTA (about five 64-deep tiles)
  const long steps = (tiles * (p.K / BK) + grid - 1) / grid;
  const bool overlap = launch_overlap_enabled() && steps <= kOverlapMaxSteps;
  return launch_kernel_overlap(overlap, tc_gemm_kernel<MODE>, dim3(grid), dim3(THREADS), SMEM_BYTES, st, mA, mB0, mB1,
                               mC, p);
}

}  // namespace

int tc_gemm_smem_bytes() { return SMEM_BYTES; }

// L2 raster of the tcgen05 GEMM: keep the whole weight operand resident when
// it is at most 40 MB (group_m = 1, n varies fastest), otherwise keep about
// 48 MB of 128-row slabs of A resident while the weights stream past them.
// Both budgets come from sweeps on GB300 at the 8B layer shapes (35194 rows,
// burst clocks, a cool-down before every point): the O projection (33.5 MB
// of weights) is fastest with its weights resident; with 48 MB of slabs the
// down projection (3 MB slabs, group 16) runs 1618 -> 1676 TFLOP/s and the
// 4096-deep GEMMs (1 MB slabs, group 48) stay within 1% of 24 MB.
int tc_gemm_group_m(long b_bytes, long a_tile_bytes) {
  constexpr long kResident = 40l << 20;
  constexpr long kBudget = 48l << 20;
  if (b_bytes <= kResident) return 1;
  const long g = kBudget / (a_tile_bytes > 0 ? a_tile_bytes : 1);
  return static_cast<int>(g < 1 ? 1 : (g > 4096 ? 4096 : g));
}

cudaError_t launch_tc_gemm(int mode, const CUtensorMap& mA, const CUtensorMap& mB0, const CUtensorMap& mB1,
                           const CUtensorMap& mC, const GemmParams& p, int num_sms, cudaStream_t st) {
  switch (mode) {
    case kGemmStore: return launch_mode<kGemmStore>(mA, mB0, mB1, mC, p, num_sms, st);
    case kGemmResidual: return launch_mode<kGemmResidual>(mA, mB0, mB1, mC, p, num_sms, st);
    case kGemmSwiglu: return launch_mode<kGemmSwiglu>(mA, mB0, mB1, mC, p, num_sms, st);
    case kGemmCount: return launch_mode<kGemmCount>(mA, mB0, mB1, mC, p, num_sms, st);
    case kGemmRope: return launch_mode<kGemmRope>(mA, mB0, mB1, mC, p, num_sms, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace seer
