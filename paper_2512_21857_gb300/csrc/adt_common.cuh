// Shared host and device helpers of libadt (internal, not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "adt.h"
#include <nvtx3/nvToolsExt.h>

namespace adt {

// An NVTX range named after the library call, for profilers' timelines
// (header-only NVTX: without a tool attached a push and a pop cost a few
// nanoseconds).
struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};

// ---------------------------------------------------------------- host side

struct DeviceInfo {
  int device;
  int sm_count;
  int max_smem_optin;     // bytes of shared memory a block may opt into
  unsigned* error_word;   // device address of this device's error word
};

// Cached per device; thread-safe.  Returns ADT_ERR_CUDA when the runtime fails.
adt_status device_info(DeviceInfo* out);

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

#define ADT_REQUIRE(cond)                 \
  do {                                    \
    if (!(cond)) return ADT_ERR_INVALID_ARG; \
  } while (0)

#define ADT_CUDA_TRY(expr)                  \
  do {                                      \
    cudaError_t adt_e_ = (expr);            \
    if (adt_e_ != cudaSuccess) return ADT_ERR_CUDA; \
  } while (0)

// Launch attribute that allows a kernel to overlap the tail of the previous
// one (its device code executes griddepcontrol.wait before touching memory).
inline cudaLaunchAttribute pdl_attribute() {
  cudaLaunchAttribute a;
  a.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  a.val.programmaticStreamSerializationAllowed = 1;
  return a;
}

inline adt_status launch_status() {
  return cudaGetLastError() == cudaSuccess ? ADT_OK : ADT_ERR_CUDA;
}

// ---------------------------------------------------------------- device side

constexpr unsigned kFullMask = 0xffffffffu;

// Programmatic dependent launch: wait until the previous kernel in the
// stream has completed and its memory is visible (immediate when this launch
// does not overlap one), then let the next kernel begin launching.  Called
// before the kernel's first global-memory access.
// Atomic add at device scope with acquire-release order: writes made
// visible to the calling thread before it (e.g. through a block barrier)
// are published with it, and what other threads published with their own
// add is visible after it.  Returns the old value.
__device__ __forceinline__ unsigned atomic_add_acq_rel_gpu(unsigned* addr, unsigned v) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;\n" : "=r"(old) : "l"(addr), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ void pdl_wait_then_release() {
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

__device__ __forceinline__ void raise_error(unsigned* word, unsigned bits) {
  if (word) atomicOr(word, bits);
}

// Classifier-free guidance on one logit: u + s (c - u), each operation
// rounded to fp32 as written (no contraction), so that the selections made
// on the result match a reference that rounds the same way.
__device__ __forceinline__ float cfg_combine(float c, float u, float s) {
  return __fadd_rn(u, __fmul_rn(s, __fsub_rn(c, u)));
}

// Order-preserving map of a finite float to uint32 (larger float -> larger
// key); -0.0 and +0.0 map to the same key.
__device__ __forceinline__ uint32_t float_order_key(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u << 1) == 0) u = 0;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float float_from_order_key(uint32_t k) {
  uint32_t u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
  return __uint_as_float(u);
}

// 64-bit selection key: value order in the high word, and within equal values
// the lower index ranks higher.  Keys of distinct indices are distinct and
// never 0, so 0 can pad an array.
__device__ __forceinline__ uint64_t select_key(float value, uint32_t index) {
  return (static_cast<uint64_t>(float_order_key(value)) << 32) | (0xffffffffu - index);
}
__device__ __forceinline__ uint32_t select_key_index(uint64_t key) {
  return 0xffffffffu - static_cast<uint32_t>(key);
}
__device__ __forceinline__ float select_key_value(uint64_t key) {
  return float_from_order_key(static_cast<uint32_t>(key >> 32));
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFullMask, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFullMask, v, o));
  return v;
}

// Block-wide reductions; `scratch` holds >= 32 elements of T.  Every thread
// receives the result.  Must be called by all threads of the block.
template <int THREADS, typename T>
__device__ T block_sum(T v, T* scratch) {
  static_assert(THREADS % 32 == 0, "");
  constexpr int W = THREADS / 32;
  v = warp_sum(v);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  T r = (lane < W) ? scratch[lane] : T(0);
  r = warp_sum(r);
  return r;
}

template <int THREADS>
__device__ float block_max(float v, float* scratch) {
  constexpr int W = THREADS / 32;
  v = warp_max(v);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  float r = (lane < W) ? scratch[lane] : -INFINITY;
  return warp_max(r);
}

// Shared memory used by block_topk_threshold.
struct RadixScratch {
  uint32_t hist[256];
  uint32_t bcast[4];
};

// Finds T such that exactly k of the n (distinct, non-zero) keys are >= T,
// by most-significant-digit radix selection with 8-bit digits.  key_at(i)
// returns key i (i < n); keys that should not compete can be returned as 0
// as long as at least k keys are non-zero.  1 <= k <= n.  All threads of the
// block must call it; every thread receives T.
template <int THREADS, class KeyAt>
__device__ uint64_t block_topk_threshold(KeyAt key_at, int n, int k, RadixScratch* rs) {
  uint64_t prefix = 0, mask = 0;
  uint32_t need = static_cast<uint32_t>(k);
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += THREADS) rs->hist[i] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += THREADS) {
      const uint64_t x = key_at(i);
      if ((x & mask) == prefix) atomicAdd(&rs->hist[(x >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      const int lane = threadIdx.x;
      uint32_t c[8];
      uint32_t tot = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = rs->hist[lane * 8 + j];
        tot += c[j];
      }
      uint32_t suf = tot;  // sum over lanes >= lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_down_sync(kFullMask, suf, o);
        if (lane + o < 32) suf += y;
      }
      uint32_t acc = suf - tot;  // keys in bins above this lane's bins
#pragma unroll
      for (int j = 7; j >= 0; --j) {
        if (acc < need && need <= acc + c[j]) {
          rs->bcast[0] = static_cast<uint32_t>(lane * 8 + j);
          rs->bcast[1] = need - acc;
          rs->bcast[2] = c[j];
        }
        acc += c[j];
      }
    }
    __syncthreads();
    const uint64_t d = rs->bcast[0];
    need = rs->bcast[1];
    const uint32_t cnt = rs->bcast[2];
    prefix |= d << shift;
    mask |= static_cast<uint64_t>(255) << shift;
    __syncthreads();  // bcast is rewritten in the next round
    if (cnt == need) break;  // every key with this prefix is selected
  }
  return prefix;
}

// Sorts `size` (a power of two) keys in shared memory in descending order.
template <int THREADS>
__device__ void block_bitonic_sort_desc(uint64_t* a, int size) {
  for (int k2 = 2; k2 <= size; k2 <<= 1) {
    for (int j = k2 >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < size; i += THREADS) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const bool desc = (i & k2) == 0;
          const uint64_t x = a[i], y = a[ixj];
          if (desc ? (x < y) : (x > y)) {
            a[i] = y;
            a[ixj] = x;
          }
        }
      }
      __syncthreads();
    }
  }
}

__host__ __device__ constexpr int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

}  // namespace adt
