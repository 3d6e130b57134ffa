// Checks the integer-only conversions of sjd_device.cuh against CUDA's own
// casts, element by element, on edge values (powers of two and their
// neighbours, exact ties at every rounding position, the largest values)
// and on seeded random ones. Prints the number of mismatches of each; the
// test that builds it (test_gpu_conversions.py) wants zeros.

#include <cstdio>
#include <cstdint>
#include <cuda_runtime.h>

#include "sjd_device.cuh"

__device__ unsigned long long mix64(unsigned long long x) {  // splitmix64 finaliser
  x += 0x9E3779B97F4A7C15ull;
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

// The i-th test value: edge values for i < 64 * 64, seeded random ones after.
__device__ unsigned long long value(unsigned long long i) {
  if (i < 64ull * 64ull) {
    const int k = static_cast<int>(i / 64), v = static_cast<int>(i % 64);
    const unsigned long long p = 1ull << k;
    switch (v % 8) {
      case 0: return p;
      case 1: return p - 1;
      case 2: return p + 1;
      case 3: return k >= 25 ? p + (1ull << (k - 24)) : p + 3;       // a tie at 24 bits
      case 4: return k >= 54 ? p + (1ull << (k - 53)) : p + 5;       // a tie at 53 bits
      case 5: return k >= 25 ? p + (3ull << (k - 24)) : p + 7;       // the next tie at 24 bits
      case 6: return ~0ull - static_cast<unsigned long long>(v);     // the largest values
      default: return mix64(i) >> (i % 64);
    }
  }
  const unsigned long long r = mix64(i);
  return r >> (r & 63);  // every magnitude
}

__global__ void check(unsigned long long n, unsigned int* bad) {
  for (unsigned long long i = blockIdx.x * static_cast<unsigned long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<unsigned long long>(gridDim.x) * blockDim.x) {
    const unsigned long long x = value(i);
    if (x != 0ull) {
      if (__float_as_uint(sjd::u64_to_f32_rn(x)) != __float_as_uint(__ull2float_rn(x))) atomicAdd(bad + 0, 1u);
      if (__double_as_longlong(sjd::u64_to_f64_rn(x)) != __double_as_longlong(__ull2double_rn(x)))
        atomicAdd(bad + 1, 1u);
      const unsigned long long z = x >> 1;  // a weight total (below 2^63)
      if (__float_as_uint(sjd::fix_to_f32(z)) !=
          __float_as_uint(__double2float_rn(__dmul_rn(__ull2double_rn(z), 0x1p-47))))
        atomicAdd(bad + 2, 1u);
    }
    // every finite float bit pattern class: the low 32 bits as a float
    const uint32_t b = static_cast<uint32_t>(x) & 0x7FFFFFFFu;
    if ((b >> 23) != 0xFFu) {
      const float f = __uint_as_float(b);
      if (__double_as_longlong(sjd::f32_to_f64(f)) != __double_as_longlong(static_cast<double>(f)))
        atomicAdd(bad + 3, 1u);
    }
  }
}

int main() {
  unsigned int* bad;
  unsigned int h[4] = {0, 0, 0, 0};
  if (cudaMalloc(&bad, sizeof(h)) != cudaSuccess) return 2;
  cudaMemset(bad, 0, sizeof(h));
  const unsigned long long n = 1ull << 26;
  check<<<1024, 256>>>(n, bad);
  if (cudaMemcpy(h, bad, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return 3;
  std::printf("values %llu mismatches u64_to_f32_rn %u u64_to_f64_rn %u fix_to_f32 %u f32_to_f64 %u\n", n, h[0],
              h[1], h[2], h[3]);
  return (h[0] | h[1] | h[2] | h[3]) ? 1 : 0;
}
