// For every k in [1, 2^24]: x = -2 ln(k 2^-24) with the fill's own ln, and
// the fill's radius square root against the IEEE square root (__fsqrt_rn),
// bit for bit.  Prints the number of differing inputs; exit status 0 when
// there are none.  Built and run by tests/test_gpu_parity.py.
#include <cstdio>
#include <cuda_runtime.h>
#include "fill_math.cuh"
#include "ln_table.h"

__global__ void check(unsigned long long *bad, unsigned int *first) {
  // the ln table as the fill keeps it: kLnCopies copies of each row side by side
  __shared__ float4 tab[ASMV_LN_TABLE_ROWS * asmv::kLnCopies];
  for (int i = threadIdx.x; i < ASMV_LN_TABLE_ROWS * (int)asmv::kLnCopies; i += blockDim.x)
    tab[i] = kLnTableInit[i / asmv::kLnCopies];
  __syncthreads();
  const unsigned int k = blockIdx.x * blockDim.x + threadIdx.x + 1u;   // 1 .. 2^24
  if (k > (1u << 24)) return;
  const uint32_t row0 = (uint32_t)__cvta_generic_to_shared(tab) + 16u * (threadIdx.x % asmv::kLnCopies);
  const float x = __fmul_rn(-2.0f, asmv::ln_u24(k, row0));
  if (__float_as_uint(__fsqrt_rn(x)) != __float_as_uint(asmv::sqrt_radius(x))) {
    atomicAdd(bad, 1ull);
    atomicMin(first, k);
  }
}

int main() {
  unsigned long long *bad = nullptr;
  unsigned int *first = nullptr;
  if (cudaMalloc(&bad, 8) != cudaSuccess || cudaMalloc(&first, 4) != cudaSuccess) return 2;
  cudaMemset(bad, 0, 8);
  cudaMemset(first, 0xFF, 4);
  const int threads = 256, blocks = (1 << 24) / threads;             // exactly 2^24 threads
  check<<<blocks, threads>>>(bad, first);
  unsigned long long hb = 0;
  unsigned int hf = 0;
  const cudaError_t e = cudaMemcpy(&hb, bad, 8, cudaMemcpyDeviceToHost);
  cudaMemcpy(&hf, first, 4, cudaMemcpyDeviceToHost);
  printf("cuda %d differing %llu first_k %u\n", (int)e, hb, hf);
  cudaFree(bad);
  cudaFree(first);
  return (e == cudaSuccess && hb == 0) ? 0 : 1;
}
