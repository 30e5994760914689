// synth.cu -- device side of the seeded synthetic input generator
// (libkvev_synth.so).  Produces exactly the bits of the host generator in
// paper_2606_15157_gb300/inputs.py: integer hashing, exact int->fp32
// conversion, correctly rounded fp32 multiply/add (no contraction), and
// round-to-nearest-even to bf16.  Holds none of the eviction arithmetic.
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kvev_synth.h"

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kM1 = 0xBF58476D1CE4E5B9ull;
constexpr uint64_t kM2 = 0x94D049BB133111EBull;
constexpr uint32_t kIH4ScaleBits = 0x37ddb3d8u;  // fp32(1 / 37837.226)

__device__ __forceinline__ uint64_t hash64(uint64_t key, uint64_t i) {
  uint64_t z = key + (i + 1) * kGamma;
  z = (z ^ (z >> 30)) * kM1;
  z = (z ^ (z >> 27)) * kM2;
  return z ^ (z >> 31);
}

__device__ __forceinline__ float gauss_f32(uint64_t key, uint64_t i) {
  const uint64_t h = hash64(key, i);
  const int64_t s = static_cast<int64_t>((h & 0xFFFF) + ((h >> 16) & 0xFFFF) +
                                         ((h >> 32) & 0xFFFF) + (h >> 48));
  const float c = __int2float_rn(static_cast<int>(s - 131070));
  return __fmul_rn(c, __uint_as_float(kIH4ScaleBits));
}

__device__ __forceinline__ uint16_t bf16_rne(float x) {
  const uint32_t u = __float_as_uint(x);
  const uint32_t bias = 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>((u + bias) >> 16);
}

__device__ __forceinline__ uint16_t value_bits(uint64_t key, uint64_t i) {
  uint16_t b = static_cast<uint16_t>(hash64(key, i) & 0xFFFF);
  if ((b & 0x7F80) == 0x7F80) b &= 0xFF7F;
  return b;
}

__device__ __forceinline__ void store8(uint16_t* dst, uint64_t i, const uint16_t (&v)[8]) {
  uint4 w;
  w.x = v[0] | (static_cast<uint32_t>(v[1]) << 16);
  w.y = v[2] | (static_cast<uint32_t>(v[3]) << 16);
  w.z = v[4] | (static_cast<uint32_t>(v[5]) << 16);
  w.w = v[6] | (static_cast<uint32_t>(v[7]) << 16);
  *reinterpret_cast<uint4*>(dst + i) = w;
}

__global__ void k_kernel(uint16_t* dst, uint64_t count, int H_kv, int S_cap, int d, uint64_t key,
                         int sink_tokens, float sink_scale, int plant_lo, int plant_hi,
                         float gamma, const float* u) {
  const uint64_t n8 = count / 8;
  for (uint64_t v = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; v < n8;
       v += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint64_t i0 = v * 8;
    const uint64_t row = i0 / d;
    const int j0 = static_cast<int>(i0 - row * d);
    const int pos = static_cast<int>(row % S_cap);
    const int h = static_cast<int>((row / S_cap) % H_kv);
    uint16_t out[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float x = gauss_f32(key, i0 + e);
      if (pos < sink_tokens) x = __fmul_rn(x, sink_scale);
      if (u != nullptr && pos >= plant_lo && pos < plant_hi)
        x = __fadd_rn(x, __fmul_rn(gamma, u[h * d + j0 + e]));
      out[e] = bf16_rne(x);
    }
    store8(dst, i0, out);
  }
}

__global__ void q_kernel(uint16_t* dst, uint64_t count, int H_q, int W, int d, int G, uint64_t key,
                         float alpha, const float* u) {
  const uint64_t n8 = count / 8;
  for (uint64_t v = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; v < n8;
       v += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint64_t i0 = v * 8;
    const uint64_t row = i0 / d;
    const int j0 = static_cast<int>(i0 - row * d);
    const int hq = static_cast<int>((row / W) % H_q);
    uint16_t out[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float x = gauss_f32(key, i0 + e);
      if (u != nullptr)
        x = __fadd_rn(__fmul_rn(alpha, u[(hq / G) * d + j0 + e]), __fmul_rn(0.1f, x));
      out[e] = bf16_rne(x);
    }
    store8(dst, i0, out);
  }
}

__global__ void gauss_kernel(uint16_t* dst, uint64_t count, uint64_t key, uint64_t base) {
  for (uint64_t i = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; i < count;
       i += static_cast<uint64_t>(gridDim.x) * blockDim.x)
    dst[i] = bf16_rne(gauss_f32(key, base + i));
}

__global__ void bits_kernel(uint16_t* dst, uint64_t count, uint64_t key, uint64_t base) {
  for (uint64_t i = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; i < count;
       i += static_cast<uint64_t>(gridDim.x) * blockDim.x)
    dst[i] = value_bits(key, base + i);
}

int grid_for(uint64_t work) {
  uint64_t g = (work + 255) / 256;
  if (g > 152ull * 64) g = 152ull * 64;
  return static_cast<int>(g < 1 ? 1 : g);
}

}  // namespace

extern "C" int kvev_synth_k(uint16_t* dst, int B, int H_kv, int S_cap, int d, uint64_t key,
                            int sink_tokens, float sink_scale, int plant_lo, int plant_hi,
                            float gamma, const float* u, void* stream) {
  if (d % 8 != 0) return static_cast<int>(cudaErrorInvalidValue);
  const uint64_t count = static_cast<uint64_t>(B) * H_kv * S_cap * d;
  k_kernel<<<grid_for(count / 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      dst, count, H_kv, S_cap, d, key, sink_tokens, sink_scale, plant_lo, plant_hi, gamma, u);
  return static_cast<int>(cudaGetLastError());
}

extern "C" int kvev_synth_q(uint16_t* dst, int B, int H_q, int W, int d, int G, uint64_t key,
                            float alpha, const float* u, void* stream) {
  if (d % 8 != 0) return static_cast<int>(cudaErrorInvalidValue);
  const uint64_t count = static_cast<uint64_t>(B) * H_q * W * d;
  q_kernel<<<grid_for(count / 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      dst, count, H_q, W, d, G, key, alpha, u);
  return static_cast<int>(cudaGetLastError());
}

extern "C" int kvev_synth_gauss(uint16_t* dst, uint64_t count, uint64_t key, uint64_t index_base,
                                void* stream) {
  gauss_kernel<<<grid_for(count), 256, 0, static_cast<cudaStream_t>(stream)>>>(dst, count, key,
                                                                                 index_base);
  return static_cast<int>(cudaGetLastError());
}

extern "C" int kvev_synth_bits(uint16_t* dst, uint64_t count, uint64_t key, uint64_t index_base,
                               void* stream) {
  bits_kernel<<<grid_for(count), 256, 0, static_cast<cudaStream_t>(stream)>>>(dst, count, key,
                                                                                index_base);
  return static_cast<int>(cudaGetLastError());
}
