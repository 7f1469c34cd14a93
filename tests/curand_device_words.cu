// Prints Philox4x32-10 words from cuRAND's device API (a library run on the
// GPU) for a few (seed, subsequence, offset) triples, one line per triple:
//   seed subsequence offset w0 w1 w2 w3 w4 w5 w6 w7
// Used by tests/test_gpu_curand_pin.py to pin the oracle's Philox counter
// words 2 and 3 (the subsequence) and, through offsets beyond 4 * 2^32,
// word 1 independently of this repository's code.
#include <cstdio>
#include <cstdint>
#include <curand_kernel.h>

__global__ void words(const unsigned long long *args, int n, unsigned int *out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  curandStatePhilox4_32_10_t st;
  curand_init(args[3 * i], args[3 * i + 1], args[3 * i + 2], &st);
  for (int k = 0; k < 8; ++k) out[8 * i + k] = curand(&st);
}

int main() {
  const unsigned long long cases[][3] = {
      {0ull, 0ull, 0ull},         {0x123456789ABCDEF0ull, 5ull, 0ull},
      {42ull, 1ull << 32, 0ull},  {42ull, (3ull << 32) | 17ull, 0ull},
      {7ull, (1ull << 33) + 1234, 4ull * 1000},  {2ull, 0xFFFFFFFF00000003ull, 8ull},
      // offsets past 4 * 2^32 carry into counter word 1; these reach the
      // auxiliary streams' word 1 = (purpose << 24) | sub
      {5ull, 9ull, 4ull * ((1ull << 32) * ((1ull << 24) | 3ull) + 100ull)},
      {11ull, (4ull << 32) | 2ull, 4ull * ((1ull << 32) * ((4ull << 24) | 77ull) + 7ull)},
      {13ull, 3ull, 4ull * ((1ull << 32) * ((5ull << 24) | 0xFFFFFFull))}};
  const int n = sizeof(cases) / sizeof(cases[0]);
  unsigned long long *d_args;
  unsigned int *d_out;
  if (cudaMalloc(&d_args, sizeof(cases)) != cudaSuccess) return 1;
  if (cudaMalloc(&d_out, n * 8 * sizeof(unsigned int)) != cudaSuccess) return 1;
  cudaMemcpy(d_args, cases, sizeof(cases), cudaMemcpyHostToDevice);
  words<<<1, 32>>>(d_args, n, d_out);
  unsigned int out[8 * 16];
  if (cudaMemcpy(out, d_out, n * 8 * sizeof(unsigned int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return 1;
  for (int i = 0; i < n; ++i) {
    printf("%llu %llu %llu", cases[i][0], cases[i][1], cases[i][2]);
    for (int k = 0; k < 8; ++k) printf(" %u", out[8 * i + k]);
    printf("\n");
  }
  cudaFree(d_args);
  cudaFree(d_out);
  return 0;
}
