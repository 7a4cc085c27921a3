// Throughput of the MUFU exp2 on sm_103a: independent chains of ex2.approx.ftz.f32 (each
// followed by one FMA that keeps the argument in (-0.75, -0.25)), and of the packed
// ex2.approx.f16x2, with 4 to 32 warps per SM.  Prints exponentials per clock per SM
// sub-partition.
//
//   mufu_rate
#include <cuda_fp16.h>
#include <stdint.h>

#include <cstdio>
#include <vector>

namespace {

template <bool PACKED>
__global__ void __launch_bounds__(1024, 1) mufu_kernel(int iters, long long* cycles, float* sink) {
  constexpr int CH = 16;   // independent chains per thread
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float x[CH];
  uint32_t h[CH];
  for (int k = 0; k < CH; ++k) {
    x[k] = -0.01f * (k + lane);
    __half2 v = __floats2half2_rn(x[k], x[k] - 0.5f);
    h[k] = *reinterpret_cast<uint32_t*>(&v);
  }
  __syncthreads();
  const long long t0 = clock64();
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int k = 0; k < CH; ++k) {
      if (!PACKED) {
        float y;
        asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x[k]));
        x[k] = fmaf(y, -0.5f, -0.25f);
      } else {
        uint32_t y;
        asm volatile("ex2.approx.f16x2 %0, %1;" : "=r"(y) : "r"(h[k]));
        __half2 t = *reinterpret_cast<__half2*>(&y);
        t = __hfma2(t, __floats2half2_rn(-0.5f, -0.5f), __floats2half2_rn(-0.25f, -0.25f));
        h[k] = *reinterpret_cast<uint32_t*>(&t);
      }
    }
  }
  const long long t1 = clock64();
  if (lane == 0) cycles[blockIdx.x * 32 + warp] = t1 - t0;
  float s = 0;
  for (int k = 0; k < CH; ++k) s += x[k] + __half2float(reinterpret_cast<__half2*>(&h[k])->x);
  if (s == 1234.5f) sink[0] = s;
}

}  // namespace

int main() {
  int nsm = 0;
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, 0);
  long long* d_cycles = nullptr;
  float* d_sink = nullptr;
  cudaMalloc(&d_cycles, nsm * 32 * sizeof(long long));
  cudaMalloc(&d_sink, sizeof(float));
  const int iters = 512;
  printf("%-20s %10s %22s\n", "instruction", "warps/SM", "exps/clk/sub-partition");
  for (int packed = 0; packed < 2; ++packed)
    for (int w : {4, 8, 16, 32}) {
      void (*k)(int, long long*, float*) = packed ? mufu_kernel<true> : mufu_kernel<false>;
      k<<<nsm, w * 32>>>(iters, d_cycles, d_sink);   // warm-up
      k<<<nsm, w * 32>>>(iters, d_cycles, d_sink);
      const cudaError_t e = cudaDeviceSynchronize();
      if (e != cudaSuccess) {
        printf("CUDA error %s\n", cudaGetErrorString(e));
        return 1;
      }
      std::vector<long long> c(nsm * 32);
      cudaMemcpy(c.data(), d_cycles, c.size() * sizeof(long long), cudaMemcpyDeviceToHost);
      double avg = 0;
      for (int b = 0; b < nsm; ++b)
        for (int i = 0; i < w; ++i) avg += static_cast<double>(c[b * 32 + i]);
      avg /= static_cast<double>(nsm) * w;
      const double exps = static_cast<double>(iters) * 16 * 32 * (w / 4) * (packed ? 2 : 1);   // per sub-partition
      printf("%-20s %10d %22.2f\n", packed ? "ex2.approx.f16x2" : "ex2.approx.ftz.f32", w, exps / avg);
    }
  return 0;
}
