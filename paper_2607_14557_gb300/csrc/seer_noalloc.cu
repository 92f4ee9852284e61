// seer_attention_noalloc: the varlen attention entry point for callers that
// must not allocate device memory.
//
// seer_attention needs a small scratch buffer for its work schedule, which the
// caller normally passes in.  Some callers cannot provide one: code that runs
// where the device memory is entirely owned by another allocator (a serving
// engine's memory pool, a plugin with no access to cudaMalloc), or that must
// not allocate at all on its hot path.  For them this entry point uses a
// fixed scratch array compiled into the library instead.
//
// The array is a file-scope __device__ variable of kScratchBytes (1 MiB), so
// every GPU that loads libseer holds it until the process exits.  Host code
// only sees a host-side stand-in for it; the device address is looked up once
// per device with cudaGetSymbolAddress on the first call made while that
// device is current.  That first call therefore performs set-up and should
// come before any CUDA stream capture.  No call allocates or frees memory.
// The cached address belongs to the device's current context: resetting the
// device (cudaDeviceReset) while libseer is loaded is not supported.
//
// All calls share the one array and leave their schedule in it.  Nothing in
// it has to start at zero: the schedule kernel rewrites the entries and the
// count it uses on every call.  Calls whose kernels overlap on the GPU (for
// example on two streams at once) race on the array and must not be issued.
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdio>
#include <mutex>

#include "../../include/seer.h"
#include "kernels.h"

namespace {

constexpr size_t kScratchBytes = size_t(1) << 20;

static __device__ __align__(256) unsigned char g_attn_scratch[kScratchBytes];

// Largest number of work units, n_heads * (ceil(T_capacity/128) + B), whose
// schedule fits the array: units * 16 bytes rounded up to 256, plus 256 bytes
// for the unit count and counter (65520 for 1 MiB).
constexpr size_t kMaxUnits = (kScratchBytes - 256) / 16 / 16 * 16;
static_assert(((kMaxUnits * 16 + 255) & ~size_t(255)) + 256 <= kScratchBytes, "limit must fit the array");
static_assert((((kMaxUnits + 1) * 16 + 255) & ~size_t(255)) + 256 > kScratchBytes, "limit must be the largest");

std::mutex g_mu;
void* g_scratch_addr[64] = {};

}  // namespace

extern "C" seer_status seer_attention_noalloc(const void* qkv, void* o, seer_dtype dt, const int32_t* cu_seqlens,
                                              const int32_t* kv_len, int B, int T_capacity, int n_heads, int head_dim,
                                              void* stream) {
  if (B <= 0 || T_capacity < 0 || n_heads <= 0) {
    seer::set_last_error("seer_attention_noalloc: bad sizes");
    return SEER_ERR_INVALID_ARG;
  }
  // fp32 attention runs on CUDA cores without a schedule: nothing to hold
  if (dt == SEER_F32)
    return seer_attention(qkv, o, dt, cu_seqlens, kv_len, B, T_capacity, n_heads, head_dim, nullptr, 0, stream);
  const size_t need = seer::attn_sched_bytes(T_capacity, B, n_heads);
  if (need > kScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "seer_attention_noalloc: this batch needs a larger schedule than the built-in scratch of 1 MiB holds "
             "(n_heads * (ceil(T_capacity/128) + B) must stay <= %zu); use seer_attention with a caller-provided "
             "workspace",
             kMaxUnits);
    seer::set_last_error(msg);
    return SEER_ERR_WORKSPACE;
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64) {
    seer::set_last_error("seer_attention_noalloc: no usable current device");
    return SEER_ERR_CUDA;
  }
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_scratch_addr[dev] == nullptr) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_attn_scratch);
      if (e != cudaSuccess) {
        seer::set_last_error("seer_attention_noalloc: cudaGetSymbolAddress of the scratch array failed");
        return SEER_ERR_CUDA;
      }
      g_scratch_addr[dev] = p;
    }
    scratch = g_scratch_addr[dev];
  }
  return seer_attention(qkv, o, dt, cu_seqlens, kv_len, B, T_capacity, n_heads, head_dim, scratch, kScratchBytes,
                        stream);
}
