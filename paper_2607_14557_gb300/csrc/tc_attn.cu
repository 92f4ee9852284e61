// Varlen bidirectional attention on tcgen05 for sm_103a (head_dim 128; q, k,
// v, the probabilities P and the output all f16, or all bf16).
//
// Seer Sec. 3.6 Eqs. 6-7 and 9-10: every query row of a segment attends to
// the first kv_len[b] rows of the same segment, with no causal mask; rows
// beyond kv_len (bucket padding of the static path) are never keys.
//
// Work unit = (segment, head, pair of 128-query tiles).  Persistent CTAs, one
// per SM (384 threads), take units from a global counter in schedule order
// (longest segment first) until none are left; every ring and barrier phase
// runs on across units, so a unit's Q / K loads and first QK^T overlap the
// previous unit's last PV and epilogue (a CTA per unit paid ~3.4 us of
// setup and teardown per unit, the persistent loop ~0.3 us).
//   warp 0     TMA producer: takes the next unit (atomic counter) and
//              publishes its index in a 4-entry shared ring, loads the unit's
//              Q tiles once both issuers are done with the previous ones,
//              then K_j and V_j in turn (two 2-deep rings); 128 keys x 128
//              dims with 128-byte swizzle;
//   warps 1-2  TMEM allocator (warp 1) and one MMA issuer per query tile t:
//              O_t += P_t,j-1 V_j-1 (P from tensor memory, V an MN-major
//              shared operand), then S_t,j = Q_t K_j^T (both from shared
//              memory).  The tensor pipe executes one thread's MMAs in issue
//              order, so S_t,j may overwrite the columns that held P_t,j-1.
//              Two issuers keep one tile's barrier waits off the other
//              tile's MMA stream (the pipe's issue queue is shallow); a turn
//              token passed between them keeps the rounds in ping-pong order
//              (tile 0's PV + QK^T, then tile 1's), so the two softmax groups
//              work in alternation instead of in lock step.  The issuer sits
//              on each round's critical path (softmax -> P -> next MMAs), so
//              its steady-state loop carries no per-round conditions: the
//              first (QK^T only) and last (PV only) rounds are peeled, and
//              ring positions are unsigned counters (stage = c % 2, phase =
//              c / 2 % 2).  A tile idle in a unit (odd tile count) only
//              releases the Q, K and V stages it would have used;
//              producer and issuers are whole warps running their loops in
//              lockstep, one elected lane issuing (a lone lane in a divergent
//              branch lost issue slots to the FMA-heavy softmax warps of its
//              SM sub-partition, and the tensor pipe then ran at its pace:
//              7-9% slower overall).  A round's PV goes out in two halves of
//              64 keys as the softmax warps release the halves of P_t, so the
//              first half's MMAs overlap the second half's exponentials
//              (5-8% faster);
//   warps 4-7  softmax of query tile 0, warps 8-11 of tile 1: one thread per
//              query row holds the row's 128 scores, so no exchange between
//              threads is needed.  While one group exponentiates its tile,
//              the tensor pipe multiplies the other tile (ping-pong).
// Online softmax in the log2 domain with lazy rescaling: O_t is rescaled in
// tensor memory only when the running max grows by more than 2^8.
// Tensor memory (512 columns): S_0 | S_1 | O_0 | O_1, P_t packed into the
// first 64 columns of S_t; a unit's first PV waits until the softmax warps
// have read the previous unit's O_t out.
//
// Measured alternative, not adopted: 64-key sub-tiles with two 64-column score
// buffers per tile, so the next QK^T runs during the softmax, were 11-16%
// slower on GB300.  A QK^T of N = 64 reads its Q operand from shared memory at
// the cost of one of N = 128 (the tensor core's shared-memory operand path
// moves ~128 B/clk: M128 N64 K16 runs at 60% of the MMA rate alone, a 64-key
// sub-tile's QK^T + PV at 82%), and beside the softmax's tensor-memory
// traffic those MMAs ran at about half their isolated rate.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace seer {
namespace {

constexpr int BQ = 128;
constexpr int BKV = 128;
constexpr int DH = 128;
constexpr int NT = 2;                       // query tiles per CTA
constexpr int THREADS = 128 + 128 * NT;    // warps 0-3 producer/issuers, 4 warps per tile
constexpr int TILE_BYTES = 128 * DH * 2;    // 32 KB: 128 rows x 128 16-bit values as two 16 KB swizzle panels
constexpr int PANEL = 16384;
constexpr int K_STAGES = 2;                 // 3 measured 1% slower
constexpr int V_STAGES = 2;
static_assert(K_STAGES == 2 && V_STAGES == 2, "the MMA issuer takes ring stage = count & 1, phase = count >> 1 & 1");
constexpr int OFF_Q = 0;                                   // Q tiles 0, 1
constexpr int OFF_K = NT * TILE_BYTES;
constexpr int OFF_V = OFF_K + K_STAGES * TILE_BYTES;
constexpr int OFF_BAR = OFF_V + V_STAGES * TILE_BYTES;
constexpr int BAR_BYTES = 512;
constexpr int SMEM_BYTES = OFF_BAR + BAR_BYTES + 1024;
static_assert(SMEM_BYTES <= 232448, "shared memory per CTA");
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t TM_S = 0;                // S_t at TM_S + 128 t
constexpr uint32_t TM_O = 256;              // O_t at TM_O + 128 t
constexpr float RESCALE_THRESHOLD = 8.0f;   // log2 units
constexpr int U_SLOTS = 4;                  // unit indices published ahead
constexpr int U_READERS = NT + 4 * NT;       // NT issuers, 4 softmax warps per tile
// barriers (8 bytes each), the unit ring, the TMEM base and the abort flag
static_assert(8 * (2 + 2 * K_STAGES + 2 * V_STAGES + 6 * NT + 2 * U_SLOTS) + 4 * U_SLOTS + 8 <= BAR_BYTES,
              "barrier block");

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float y;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
  return y;
}

// 2^x of two packed f16 values in one MUFU operation.
__device__ __forceinline__ uint32_t ex2_h2(uint32_t x) {
  uint32_t y;
  asm("ex2.approx.f16x2 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
// acc + (f16 half of v), in fp32 (mixed-precision add).
__device__ __forceinline__ float add_f16_lo(uint32_t v, float acc) {
  float d;
  asm("{\n\t.reg .b16 l, h;\n\tmov.b32 {l, h}, %1;\n\tadd.rn.f32.f16 %0, l, %2;\n\t}" : "=f"(d) : "r"(v), "f"(acc));
  return d;
}
__device__ __forceinline__ float add_f16_hi(uint32_t v, float acc) {
  float d;
  asm("{\n\t.reg .b16 l, h;\n\tmov.b32 {l, h}, %1;\n\tadd.rn.f32.f16 %0, h, %2;\n\t}" : "=f"(d) : "r"(v), "f"(acc));
  return d;
}


// Two fp32 fused multiply-adds in one instruction (packed f32x2, sm_100+).
__device__ __forceinline__ void ffma2(float a0, float a1, float b0, float b1, float c0, float c1, float& d0, float& d1) {
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\t"
      "mov.b64 rb, {%4, %5};\n\t"
      "mov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\t"
      "mov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d0), "=f"(d1) : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}

// Packed probabilities of keys 32c .. 32c+31 of one row: p = 2^(s * scale - m),
// accumulated into the row sum.  f16: the exponents x of a pair come from one
// packed f32x2 FMA, are rounded to f16, and two probabilities come from one
// MUFU operation (ex2.approx.f16x2); P is stored in f16 anyway.  bf16: one
// fp32 ex2 per probability.  Either way the row sum adds the stored (rounded)
// probabilities.  The softmax of a tile sits on its tile's critical chain, so
// its instruction count matters: the packed FMA is 2.5% faster on GB300, while
// moving a quarter of the exponentials to a polynomial on the FMA pipes was 9%
// slower (more instructions, no MUFU relief).
template <bool F16>
__device__ __forceinline__ void row_probs(const float* s, float scale_log2, float neg, float (&rs)[4],
                                          uint32_t (&pk)[16]) {
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    if (F16) {
      float x0, x1;
      ffma2(s[2 * i], s[2 * i + 1], scale_log2, scale_log2, neg, neg, x0, x1);
      const uint32_t ph = ex2_h2(pack_f16x2(x0, x1));
      rs[(2 * i) & 3] = add_f16_lo(ph, rs[(2 * i) & 3]);
      rs[(2 * i + 1) & 3] = add_f16_hi(ph, rs[(2 * i + 1) & 3]);
      pk[i] = ph;
    } else {
      const float x0 = fmaf(s[2 * i], scale_log2, neg), x1 = fmaf(s[2 * i + 1], scale_log2, neg);
      // the row sum adds the rounded probabilities the PV product reads, so
      // numerator and normaliser carry the same rounding
      const uint32_t ph = pack_bf16x2(ex2(x0), ex2(x1));
      rs[i & 3] += bf16_lo(ph) + bf16_hi(ph);
      pk[i] = ph;
    }
  }
}

struct Unit {
  int b, h, qt0, nt, seq0, L, kv0, kvL, q0, nkv, xq, xk, xv;
};

__device__ __forceinline__ Unit decode_unit(const AttnParams& p, int u) {
  Unit d;
  const int4 wk = p.work[u];
  d.b = wk.x;
  d.h = wk.y;
  d.qt0 = wk.z;
  d.nt = wk.w;
  d.seq0 = p.cu[d.b];
  d.L = p.cu[d.b + 1] - d.seq0;
  d.kv0 = p.cu_kv ? p.cu_kv[d.b] : d.seq0;
  d.kvL = p.kv_len ? p.kv_len[d.b] : (p.cu_kv ? p.cu_kv[d.b + 1] - d.kv0 : d.L);
  d.q0 = d.seq0 + d.qt0 * BQ;
  d.nkv = (d.kvL + BKV - 1) / BKV;
  d.xq = d.h * DH;
  d.xk = p.xk0 + d.h * DH;
  d.xv = p.xv0 + d.h * DH;
  return d;
}

// Unit index of this CTA's i-th unit, read from the shared ring (-1: no more
// units or an abort); `arrive` releases the slot for this reader.
__device__ __forceinline__ int read_unit(uint64_t* u_full, uint64_t* u_empty, const int* unit_slot, int i,
                                         volatile int* abort, int* err, bool arrive) {
  const int s = i % U_SLOTS;
  if (!mbar_wait(&u_full[s], (i / U_SLOTS) & 1, abort, err)) return -1;
  const int u = unit_slot[s];
  if (arrive) mbar_arrive(&u_empty[s]);
  return u;
}

template <bool F16>
__global__ void __launch_bounds__(THREADS, 1)
    tc_attn_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mKV, const AttnParams p) {
  pdl_enter();
  const int count = *p.work_count;
  if (static_cast<int>(blockIdx.x) >= count) return;
  const int G = gridDim.x;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* q_empty = bars + 1;              // both issuers are done with the Q tiles of a unit
  uint64_t* k_full = bars + 2;               // [K_STAGES]
  uint64_t* k_empty = k_full + K_STAGES;     // [K_STAGES]
  uint64_t* v_full = k_empty + K_STAGES;     // [V_STAGES]
  uint64_t* v_empty = v_full + V_STAGES;     // [V_STAGES]
  uint64_t* s_full = v_empty + V_STAGES;     // [NT] S_t,j written (and O_t += P_t,j-1 V done)
  uint64_t* p_full = s_full + NT;            // [NT] P_t,j of keys 0..63 in tensor memory (O_t rescaled)
  uint64_t* p_full2 = p_full + NT;           // [NT] P_t,j of keys 64..127 in tensor memory
  uint64_t* o_done = p_full2 + NT;           // [NT] last PV of tile t of a unit complete
  uint64_t* o_free = o_done + NT;            // [NT] O_t of a unit read out by the softmax warps
  uint64_t* turn = o_free + NT;              // [NT] issuer t may enqueue its next round
  uint64_t* u_full = turn + NT;              // [U_SLOTS] unit index published
  uint64_t* u_empty = u_full + U_SLOTS;      // [U_SLOTS] unit index read by every role
  int* unit_slot = reinterpret_cast<int*>(u_empty + U_SLOTS);   // [U_SLOTS]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(unit_slot + U_SLOTS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, NT);
    for (int i = 0; i < K_STAGES; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], NT);      // one commit (or, for an idle tile, one arrive) per issuer
    }
    for (int i = 0; i < V_STAGES; ++i) {
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], NT);
    }
    for (int t = 0; t < NT; ++t) {
      mbar_init(&s_full[t], 1);
      mbar_init(&p_full[t], 4);
      mbar_init(&p_full2[t], 4);
      mbar_init(&o_done[t], 1);
      mbar_init(&o_free[t], 4);
      mbar_init(&turn[t], 1);
    }
    for (int i = 0; i < U_SLOTS; ++i) {
      mbar_init(&u_full[i], 1);
      mbar_init(&u_empty[i], U_READERS);
    }
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
    // The whole warp runs the loop in lockstep (every wait by all lanes, with
    // a warp-uniform outcome) and the elected lane issues: it takes the units
    // from the global counter and publishes them in the shared ring, loads
    // each unit's Q tiles (once the previous unit's QK^T are done with them),
    // then its K_j and V_j in turn.  K_j needs the stage QK^T of round j-2
    // released and V_j the stage PV of round j-2 (issued in round j-1)
    // released, so one stream for both rings waits for nothing extra.  Both
    // rings run on across the units of this CTA.
    const bool leader = elect_one();
    const int leader_lane = __ffs(__ballot_sync(0xffffffffu, leader)) - 1;
    if (leader) {
      tma_prefetch_desc(&mQ);
      tma_prefetch_desc(&mKV);
      unit_slot[0] = blockIdx.x;
      mbar_arrive(&u_full[0]);
    }
    __syncwarp();
    int q_issued = 0, k_issued = 0, v_issued = 0;
    bool ok = true;
    int u = blockIdx.x;
    for (int i = 0; ok && u >= 0; ++i) {
      const Unit d = decode_unit(p, u);
      if (i > 0 && !warp_wait(q_empty, (i - 1) & 1, abort_flag, p.err)) break;
      if (leader) {
        mbar_arrive_expect_tx(q_full, d.nt * TILE_BYTES);
        for (int t = 0; t < d.nt; ++t) {
          tma_load_2d(smem + OFF_Q + t * TILE_BYTES, &mQ, q_full, d.xq, d.q0 + t * BQ);
          tma_load_2d(smem + OFF_Q + t * TILE_BYTES + PANEL, &mQ, q_full, d.xq + 64, d.q0 + t * BQ);
        }
      }
      __syncwarp();
      ++q_issued;
      // publish unit i+1 now, so the other roles can look ahead
      const int n = i + 1, sl = n % U_SLOTS;
      if (n >= U_SLOTS && !warp_wait(&u_empty[sl], (n / U_SLOTS - 1) & 1, abort_flag, p.err)) break;
      int un = 0;
      if (leader) {
        un = G + atomicAdd(p.work_next, 1);
        if (un >= count) un = -1;
        unit_slot[sl] = un;
        mbar_arrive(&u_full[sl]);
      }
      un = __shfl_sync(0xffffffffu, un, leader_lane);
      for (int j = 0; j < d.nkv; ++j) {
        const int ks = k_issued % K_STAGES, ku = k_issued / K_STAGES;
        if (ku > 0 && !warp_wait(&k_empty[ks], (ku - 1) & 1, abort_flag, p.err)) { ok = false; break; }
        if (leader) {
          uint8_t* dst = smem + OFF_K + ks * TILE_BYTES;
          mbar_arrive_expect_tx(&k_full[ks], TILE_BYTES);
          tma_load_2d(dst, &mKV, &k_full[ks], d.xk, d.kv0 + j * BKV);
          tma_load_2d(dst + PANEL, &mKV, &k_full[ks], d.xk + 64, d.kv0 + j * BKV);
        }
        __syncwarp();
        ++k_issued;
        const int vs = v_issued % V_STAGES, vu = v_issued / V_STAGES;
        if (vu > 0 && !warp_wait(&v_empty[vs], (vu - 1) & 1, abort_flag, p.err)) { ok = false; break; }
        if (leader) {
          uint8_t* dst = smem + OFF_V + vs * TILE_BYTES;
          mbar_arrive_expect_tx(&v_full[vs], TILE_BYTES);
          tma_load_2d(dst, &mKV, &v_full[vs], d.xv, d.kv0 + j * BKV);
          tma_load_2d(dst + PANEL, &mKV, &v_full[vs], d.xv + 64, d.kv0 + j * BKV);
        }
        __syncwarp();
        ++v_issued;
      }
      u = un;
    }
    if (*abort_flag && leader) {
      // let copies still in flight land before the CTA's shared memory is released
      if (q_issued > 0) mbar_wait_drain(q_full, (q_issued - 1) & 1, 200000000ull);
      for (int j = k_issued > K_STAGES ? k_issued - K_STAGES : 0; j < k_issued; ++j)
        mbar_wait_drain(&k_full[j % K_STAGES], (j / K_STAGES) & 1, 200000000ull);
      for (int j = v_issued > V_STAGES ? v_issued - V_STAGES : 0; j < v_issued; ++j)
        mbar_wait_drain(&v_full[j % V_STAGES], (j / V_STAGES) & 1, 200000000ull);
    }
  } else if (warp == 1 || warp == 2) {
    // -------------------------------------------------- MMA issuer of tile t
    // The whole warp runs the issue loop in lockstep (every wait by all lanes,
    // with a warp-uniform outcome); the elected lane issues the MMAs, commits
    // and arrivals.  A lone issuing lane in a divergent branch lost issue
    // slots to the FMA-heavy softmax warps on its sub-partition, and the
    // tensor pipe ran at its pace (84-94 cycles per 64-cycle MMA).
    const int t = warp - 1;
    const bool leader = elect_one();
    constexpr uint32_t idesc_qk = make_idesc(BQ, BKV, 0, F16);
    constexpr uint32_t idesc_pv = make_idesc(BQ, DH, 1, F16);
    // descriptors built once; a K=16 step adds a constant to the
    // start-address field (stage s of a ring: + s * TILE_BYTES / 16)
    const uint64_t dq = make_sdesc_sw128(smem_u32(smem + OFF_Q + t * TILE_BYTES), 16, 1024);
    const uint64_t dk0 = make_sdesc_sw128(smem_u32(smem + OFF_K), 16, 1024);
    const uint64_t dv0 = make_sdesc_sw128(smem_u32(smem + OFF_V), PANEL, 1024);
    const uint32_t dS = tmem + TM_S + 128 * t, dO = tmem + TM_O + 128 * t;
    // ring positions run on across units: stage = count % 2, phase = count / 2 % 2
    unsigned kc = 0, vc = 0;       // K / V tiles consumed
    unsigned pc = 0, tc = 0;       // P tiles consumed, turn waits
    unsigned oc = 0;               // units of this tile finished
    bool paired_before = false;    // a unit with both tiles active was seen
    bool ok = true;
    // S_t = Q_t K^T for the K tile at ring position kc (both K-major, 128-byte swizzle)
    auto qk = [&](unsigned c) {
      if (leader) {
        const uint64_t dk = dk0 + static_cast<uint64_t>((c & 1u) * (TILE_BYTES >> 4));
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint64_t off = static_cast<uint64_t>(((k >> 2) * PANEL + (k & 3) * 32) >> 4);
          tc_mma_f16(dS, dq + off, dk + off, idesc_qk, k > 0 ? 1u : 0u);
        }
        tc_commit(&s_full[t]);
        tc_commit(&k_empty[c & 1u]);
      }
      __syncwarp();
    };
    // O_t (+)= P_t V for the V tile at ring position c: A = P from tensor
    // memory (8 columns per 16 keys), B = V [keys, dims] with dims
    // contiguous, an MN-major operand whose 64-dim panels are PANEL bytes
    // apart (LBO) and 8-key groups 1 KB apart (SBO)
    // (vt: the V tile's index in the unit; tile 0 starts a fresh O_t).
    // Issued in two halves of 64 keys, each once the softmax warps have
    // released that half of P_t.
    auto pv = [&](unsigned c, int vt, int half) {
      if (leader) {
        const uint64_t dv = dv0 + static_cast<uint64_t>((c & 1u) * (TILE_BYTES >> 4));
#pragma unroll
        for (int kk = 0; kk < BKV / 32; ++kk) {
          const int k = half * (BKV / 32) + kk;
          tc_mma_f16_tmem_a(dO, dS + 8 * k, dv + static_cast<uint64_t>(k * 128), idesc_pv, (vt > 0 || k > 0) ? 1u : 0u);
        }
        if (half == 1) tc_commit(&v_empty[c & 1u]);
      }
      __syncwarp();
    };
    auto arrive = [&](uint64_t* bar) {
      if (leader) mbar_arrive(bar);
      __syncwarp();
    };
    for (int i = 0; ok; ++i) {
      const int u = __shfl_sync(0xffffffffu, read_unit(u_full, u_empty, unit_slot, i, abort_flag, p.err, lane == 0), 0);
      if (u < 0) break;
      const Unit d = decode_unit(p, u);
      if (!warp_wait(q_full, i & 1, abort_flag, p.err)) break;
      if (t >= d.nt) {
        // idle this unit: release Q and every K / V stage as they pass
        arrive(q_empty);
        for (int j = 0; j < d.nkv; ++j, ++kc, ++vc) {
          if (!warp_wait(&k_full[kc & 1u], (kc >> 1) & 1u, abort_flag, p.err) ||
              !warp_wait(&v_full[vc & 1u], (vc >> 1) & 1u, abort_flag, p.err)) {
            ok = false;
            break;
          }
          arrive(&k_empty[kc & 1u]);
          arrive(&v_empty[vc & 1u]);
        }
        continue;
      }
      const bool pair = d.nt > 1;
      const int nkv = d.nkv;
      // rounds: 0 = QK^T of K_0; j = 1 .. nkv-1: PV of V_j-1, then QK^T of
      // K_j; nkv = PV of V_nkv-1.  Round j of tile 1 follows round j of tile
      // 0, which follows round j-1 of tile 1 (the turn token); tile 0's
      // round 0 follows tile 1's last round of the previous paired unit.
      if (!warp_wait(&k_full[kc & 1u], (kc >> 1) & 1u, abort_flag, p.err)) break;
      if (pair && (t == 1 || paired_before)) {
        if (!warp_wait(&turn[t], tc & 1u, abort_flag, p.err)) break;
        ++tc;
      }
      tc_fence_after();
      qk(kc);
      ++kc;
      if (nkv == 1 && leader) tc_commit(q_empty);
      if (pair) arrive(&turn[t ^ 1]);
      // the first PV overwrites O_t: the previous unit's O_t must be read out
      if (oc > 0 && !warp_wait(&o_free[t], (oc - 1) & 1u, abort_flag, p.err)) break;
      for (int j = 1; j < nkv; ++j) {
        // operands first (usually landed long before), then this tile's P,
        // then the turn: after P arrives only the turn is left to check
        if (!warp_wait(&v_full[vc & 1u], (vc >> 1) & 1u, abort_flag, p.err) ||
            !warp_wait(&k_full[kc & 1u], (kc >> 1) & 1u, abort_flag, p.err) ||
            !warp_wait(&p_full[t], pc & 1u, abort_flag, p.err) ||
            (pair && !warp_wait(&turn[t], tc & 1u, abort_flag, p.err))) {
          ok = false;
          break;
        }
        tc += pair ? 1u : 0u;
        tc_fence_after();
        pv(vc, j - 1, 0);
        if (!warp_wait(&p_full2[t], pc & 1u, abort_flag, p.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        pv(vc, j - 1, 1);
        qk(kc);
        ++vc;
        ++pc;
        ++kc;
        if (pair) arrive(&turn[t ^ 1]);
      }
      if (!ok) break;
      if (nkv > 1 && leader) tc_commit(q_empty);
      if (!warp_wait(&v_full[vc & 1u], (vc >> 1) & 1u, abort_flag, p.err) ||
          !warp_wait(&p_full[t], pc & 1u, abort_flag, p.err) ||
          (pair && !warp_wait(&turn[t], tc & 1u, abort_flag, p.err)))
        break;
      tc += pair ? 1u : 0u;
      tc_fence_after();
      pv(vc, nkv - 1, 0);
      if (!warp_wait(&p_full2[t], pc & 1u, abort_flag, p.err)) break;
      tc_fence_after();
      pv(vc, nkv - 1, 1);
      if (leader) tc_commit(&o_done[t]);
      __syncwarp();
      ++vc;
      ++pc;
      if (pair) arrive(&turn[t ^ 1]);
      if (pair) paired_before = true;
      ++oc;
    }
  } else if (warp >= 4) {
    // -------------------------------------------------- softmax warps 4..11
    const int t = (warp - 4) >> 2;                // query tile of this group
    const int qw = warp & 3;                      // TMEM lane quarter
    const int r = qw * 32 + lane;                 // query row inside the tile == TMEM lane
    const uint32_t lane_off = static_cast<uint32_t>(qw * 32) << 16;
    const uint32_t tS = tmem + lane_off + TM_S + 128 * t;
    const uint32_t tO = tmem + lane_off + TM_O + 128 * t;
    const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));
    int cs = 0, co = 0, cv = 0;                   // S tiles seen, units done (this tile), V tiles before the unit
    uint32_t nonfinite = 0;                       // range guard over this thread's output stores
    bool ok = true;
    for (int i = 0; ok; ++i) {
      const int u = __shfl_sync(0xffffffffu, read_unit(u_full, u_empty, unit_slot, i, abort_flag, p.err, lane == 0), 0);
      if (u < 0) break;
      const Unit d = decode_unit(p, u);
      if (t >= d.nt) {
        cv += d.nkv;
        continue;
      }
      float m_ref = -INFINITY;                    // running max, log2 units
      float l = 0.f;                              // row sum
      for (int j = 0; ok && j < d.nkv; ++j) {
        // warp-uniform outcomes: the TMEM accesses that follow are warp-collective
        if (!__all_sync(0xffffffffu, mbar_wait(&s_full[t], cs & 1, abort_flag, p.err))) { ok = false; break; }
        ++cs;
        tc_fence_after();
        float s[BKV];
        {
          uint32_t ra[BKV / 32][32];
#pragma unroll
          for (int cc = 0; cc < BKV / 32; ++cc) tmem_ld32(tS + 32 * cc, ra[cc]);
          tmem_ld_wait();
#pragma unroll
          for (int cc = 0; cc < BKV / 32; ++cc)
#pragma unroll
            for (int e = 0; e < 32; ++e) s[32 * cc + e] = __uint_as_float(ra[cc][e]);
        }
        const int valid = d.kvL - j * BKV;        // keys of this tile, >= 1
        if (valid < BKV) {
#pragma unroll
          for (int cc = 0; cc < BKV; ++cc) s[cc] = cc < valid ? s[cc] : -INFINITY;
        }
        // row max: eight independent chains, then a tree
        float mx[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx[e] = fmaxf(s[e], s[e + 8]);
#pragma unroll
        for (int cc = 16; cc < BKV; cc += 16)
#pragma unroll
          for (int e = 0; e < 8; ++e) mx[e] = max3(mx[e], s[cc + e], s[cc + 8 + e]);
#pragma unroll
        for (int w = 4; w >= 1; w >>= 1)
#pragma unroll
          for (int e = 0; e < w; ++e) mx[e] = fmaxf(mx[e], mx[e + w]);
        const float m_new = fmaxf(m_ref, mx[0] * scale_log2);
        const bool need = (j == 0) || (m_new > m_ref + RESCALE_THRESHOLD);
        const bool any_need = __any_sync(0xffffffffu, need);
        float alpha = 1.f;
        if (need) {
          alpha = (j == 0) ? 0.f : ex2(m_ref - m_new);
          m_ref = m_new;
        }
        // P_t,j: keys 32c .. 32c+31 -> 16 packed columns 16c .. 16c+15 of S_t
        // (the scores were all read above; O_t += P_t,j-1 V_j-1 has completed),
        // released to the PV MMAs in two halves of 64 keys, so the first
        // half's MMAs run while the second half is exponentiated
        const float neg = -m_ref;
        float rs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
#pragma unroll
          for (int cc = 2 * hf; cc < 2 * hf + 2; ++cc) {
            uint32_t pk[16];
            row_probs<F16>(s + 32 * cc, scale_log2, neg, rs, pk);
            tmem_st16(tS + 16 * cc, pk);
          }
          if (hf == 0) {
            // before the first half is released: rescale O_t in tensor memory
            // if the reference max moved ...
            if (j > 0 && any_need) {
#pragma unroll 1
              for (int cc = 0; cc < DH / 32; ++cc) {
                uint32_t rr[32];
                tmem_ld32(tO + 32 * cc, rr);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 32; ++e) rr[e] = __float_as_uint(__uint_as_float(rr[e]) * alpha);
                tmem_st32(tO + 32 * cc, rr);
              }
            }
            // ... and, on the last, partial key tile, clear the value rows past
            // kv_len so stale (possibly non-finite) data cannot meet the zero
            // probabilities (both groups write the same zeros: each must see
            // them before its PV)
            if (valid < BKV) {
              const int vsi = cv + j, vst = vsi % V_STAGES;
              if (!__all_sync(0xffffffffu, mbar_wait(&v_full[vst], (vsi / V_STAGES) & 1, abort_flag, p.err))) {
                ok = false;
                break;
              }
              if (r >= valid) {
#pragma unroll
                for (int pn = 0; pn < 2; ++pn) {
                  uint4* v = reinterpret_cast<uint4*>(smem + OFF_V + vst * TILE_BYTES + pn * PANEL + r * 128);
#pragma unroll
                  for (int e = 0; e < 8; ++e) v[e] = make_uint4(0, 0, 0, 0);
                }
              }
              fence_proxy_async_smem();
            }
          }
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(hf == 0 ? &p_full[t] : &p_full2[t]);
        }
        if (!ok) break;
        l = l * alpha + ((rs[0] + rs[1]) + (rs[2] + rs[3]));
      }
      if (!ok) break;
      if (!__all_sync(0xffffffffu, mbar_wait(&o_done[t], co & 1, abort_flag, p.err))) break;
      tc_fence_after();
      const float inv_l = 1.f / l;
      const int qrow = (d.qt0 + t) * BQ + r;      // row inside the segment
      const bool valid_row = qrow < d.L;
      uint16_t* orow =
          reinterpret_cast<uint16_t*>(p.out) + static_cast<size_t>(valid_row ? d.seq0 + qrow : 0) * p.ldo + d.h * DH;
#pragma unroll 1
      for (int cc = 0; cc < DH / 32; ++cc) {
        uint32_t rr[32];
        tmem_ld32(tO + 32 * cc, rr);
        tmem_ld_wait();
        if (valid_row) {
          uint4* dst = reinterpret_cast<uint4*>(orow + 32 * cc);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            uint32_t q[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              q[k] = pack2(__uint_as_float(rr[8 * e + 2 * k]) * inv_l, __uint_as_float(rr[8 * e + 2 * k + 1]) * inv_l, F16);
              nonfinite |= nonfinite_term(q[k], F16);
            }
            dst[e] = make_uint4(q[0], q[1], q[2], q[3]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&o_free[t]);
      ++co;
      cv += d.nkv;
    }
    report_range(nonfinite, p.err);               // an output value was infinite or NaN
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// One block: per-segment key counts -> work units (b, h, first q-tile, tiles)
// of up to NT query tiles, ordered by descending kv length so the longest
// segments start first.
__global__ void attn_schedule_kernel(const int* cu, const int* cu_kv, const int* kv_len, int B, int H, int T_cap,
                                     int4* work, int* work_count, int max_units, int* err) {
  pdl_enter();
  extern __shared__ int sh[];
  int* ntile = sh;           // [B]
  int* kvs = sh + B;         // [B]
  int* off = sh + 2 * B;     // [B]
  int* rank = sh + 3 * B;    // [B]
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    const int L = cu[i + 1] - cu[i];
    const int Lkv = cu_kv ? cu_kv[i + 1] - cu_kv[i] : L;   // rows of the segment's K/V
    int kv = kv_len ? kv_len[i] : Lkv;
    if (L < 0 || cu[i] < 0 || cu[i + 1] > T_cap || kv > Lkv || (L > 0 && kv <= 0)) {
      record_error(err, kErrLayout);
      kv = 0;
    }
    ntile[i] = (kv > 0) ? (L + BQ * NT - 1) / (BQ * NT) : 0;   // work units (tile groups) per head
    kvs[i] = kv;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    int rk = 0;
    for (int k = 0; k < B; ++k) rk += (kvs[k] > kvs[i]) || (kvs[k] == kvs[i] && k < i);
    rank[i] = rk;
  }
  __syncthreads();
  // offsets in rank order: a segment's units follow those of every segment
  // ranked before it (the ranks are a permutation of 0..B-1)
  for (int i = threadIdx.x; i < B; i += blockDim.x) {
    int before = 0;
    for (int k = 0; k < B; ++k) before += rank[k] < rank[i] ? ntile[k] : 0;
    off[i] = H * before;
  }
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int i = 0; i < B; ++i) acc += H * ntile[i];
    if (acc > max_units) {
      record_error(err, kErrCapacity);
      acc = max_units;
    }
    work_count[0] = acc;
    work_count[1] = 0;            // next unit handed out by the attention kernel
  }
  __syncthreads();
  for (int i = 0; i < B; ++i) {
    const int n = H * ntile[i];
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
      const int idx = off[i] + k;
      if (idx < max_units) {
        const int g = k % ntile[i];
        const int tiles = (cu[i + 1] - cu[i] + BQ - 1) / BQ;
        work[idx] = make_int4(i, k / ntile[i], g * NT, min(NT, tiles - g * NT));
      }
    }
  }
}

template <bool F16>
cudaError_t launch_typed(const CUtensorMap& mQ, const CUtensorMap& mKV, const AttnParams& p, int grid, cudaStream_t st) {
  static bool attr_set[64] = {};
  cudaError_t e = set_smem_limit_once(tc_attn_kernel<F16>, SMEM_BYTES, attr_set);
  if (e != cudaSuccess) return e;
  if (grid <= 0) return cudaSuccess;
  return launch_kernel(tc_attn_kernel<F16>, dim3(grid), dim3(THREADS), SMEM_BYTES, st, mQ, mKV, p);
}

}  // namespace

int tc_attn_smem_bytes() { return SMEM_BYTES; }

cudaError_t launch_tc_attn(const CUtensorMap& mQ, const CUtensorMap& mKV, const AttnParams& p, int grid, bool f16,
                           cudaStream_t st) {
  return f16 ? launch_typed<true>(mQ, mKV, p, grid, st) : launch_typed<false>(mQ, mKV, p, grid, st);
}

cudaError_t launch_attn_schedule(const int* cu, const int* cu_kv, const int* kv_len, int B, int n_heads, int T_cap,
                                 int4* work, int* work_count, int max_units, int* err, cudaStream_t st) {
  const size_t sm = static_cast<size_t>(4) * B * sizeof(int);
  if (sm > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(attn_schedule_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(sm));
    if (e != cudaSuccess) return e;
  }
  return launch_kernel(attn_schedule_kernel, dim3(1), dim3(256), sm, st, cu, cu_kv, kv_len, B, n_heads, T_cap, work,
                       work_count, max_units, err);
}

}  // namespace seer
