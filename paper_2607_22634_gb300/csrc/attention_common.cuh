// Pieces shared by the two tree-attention schedules (tree_attention.cu for short KV
// runs, tree_attention_pair.cu for long ones): tile constants, packed fp32x2
// arithmetic for the softmax, and the TMA tensor maps of the operands.
#pragma once

#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include "common.cuh"

namespace presto {
namespace attn {

constexpr int kBM = 128;             // query rows per tile (TMEM lanes)
constexpr int kBN = 128;             // keys per KV tile
constexpr int kRowBytes = 128;       // one 128-byte-swizzled row: 64 bf16
constexpr float kRescaleLog2 = 8.f;  // move the running max only when it grows by > 2^8
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr uint32_t kTmemCols = 512;
constexpr int kWidePartialKeys = 1024;  // prefixes shorter than this merge float32 partials
constexpr int kMaxSplits = 16;          // KV splits of a row block (long runs: the CTAs of its cluster)

// Packed fp32 pairs (f32x2 arithmetic issues one instruction per two values) and
// the three-input max.
__device__ __forceinline__ uint64_t pack2(float x, float y) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
  return r;
}
__device__ __forceinline__ void unpack2(uint64_t r, float& x, float& y) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(r));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// 32 scores of a row -> their maximum, as four independent three-input-max chains.
__device__ __forceinline__ float row_max32(const float* v) {
  float q[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float* w = v + 8 * i;
    q[i] = fmaxf(max3(max3(max3(w[0], w[1], w[2]), w[3], w[4]), w[5], w[6]), w[7]);
  }
  return max3(q[0], q[1], fmaxf(q[2], q[3]));
}

inline PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

// 3-D bf16 tensor map with a 128-byte-swizzled box (64 x b1 x b2 elements).
inline bool make_map(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
              uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b1, uint32_t b2) {
  auto fn = encoder();
  if (!fn) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {64, b1, b2};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace attn
}  // namespace presto
