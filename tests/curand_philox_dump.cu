// Test helper: prints Philox4x32-10 blocks computed on the GPU by cuRAND's
// device generator (curandStatePhilox4_32_10_t), an implementation independent
// of the oracle. Reads lines "seed subsequence block" (decimal uint64, block
// < 2^62) from stdin; for each, one thread calls curand_init(seed, subsequence,
// 4 * block) and curand4, i.e. the block at counter (block_lo, block_hi,
// subsequence_lo, subsequence_hi) under key (seed_lo, seed_hi). Writes the
// four 32-bit outputs of each block per line.
#include <cuda_runtime.h>
#include <curand_kernel.h>

#include <cstdio>
#include <vector>

__global__ void dump(const unsigned long long* seed, const unsigned long long* sub,
                     const unsigned long long* block, int n, uint4* out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  curandStatePhilox4_32_10_t st;
  curand_init(seed[i], sub[i], 4ull * block[i], &st);
  out[i] = curand4(&st);
}

static int check(cudaError_t err, const char* what) {
  if (err != cudaSuccess) {
    std::fprintf(stderr, "%s: %s\n", what, cudaGetErrorString(err));
    return 1;
  }
  return 0;
}

int main() {
  std::vector<unsigned long long> seed, sub, block;
  unsigned long long s, q, b;
  while (std::scanf("%llu %llu %llu", &s, &q, &b) == 3) {
    if (b >= (1ull << 62)) {
      std::fprintf(stderr, "block %llu >= 2^62\n", b);
      return 2;
    }
    seed.push_back(s);
    sub.push_back(q);
    block.push_back(b);
  }
  const int n = static_cast<int>(seed.size());
  if (n == 0) return 0;
  const size_t bytes = sizeof(unsigned long long) * n;
  unsigned long long *d_seed = nullptr, *d_sub = nullptr, *d_block = nullptr;
  uint4* d_out = nullptr;
  if (check(cudaMalloc(&d_seed, bytes), "cudaMalloc") || check(cudaMalloc(&d_sub, bytes), "cudaMalloc") ||
      check(cudaMalloc(&d_block, bytes), "cudaMalloc") ||
      check(cudaMalloc(&d_out, sizeof(uint4) * n), "cudaMalloc"))
    return 1;
  if (check(cudaMemcpy(d_seed, seed.data(), bytes, cudaMemcpyHostToDevice), "copy") ||
      check(cudaMemcpy(d_sub, sub.data(), bytes, cudaMemcpyHostToDevice), "copy") ||
      check(cudaMemcpy(d_block, block.data(), bytes, cudaMemcpyHostToDevice), "copy"))
    return 1;
  dump<<<(n + 127) / 128, 128>>>(d_seed, d_sub, d_block, n, d_out);
  if (check(cudaGetLastError(), "launch") || check(cudaDeviceSynchronize(), "kernel")) return 1;
  std::vector<uint4> out(n);
  if (check(cudaMemcpy(out.data(), d_out, sizeof(uint4) * n, cudaMemcpyDeviceToHost), "copy back"))
    return 1;
  for (const uint4& w : out) std::printf("%u %u %u %u\n", w.x, w.y, w.z, w.w);
  cudaFree(d_seed);
  cudaFree(d_sub);
  cudaFree(d_block);
  cudaFree(d_out);
  return 0;
}
