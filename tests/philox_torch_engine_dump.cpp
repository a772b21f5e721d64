// Test helper: prints Philox4x32-10 blocks computed by PyTorch's host Philox
// engine (ATen/core/PhiloxRNGEngine.h), an implementation independent of the
// oracle. Reads lines "seed subsequence offset" (decimal uint64) from stdin and
// writes the four 32-bit outputs of that block per line.
#include <ATen/core/PhiloxRNGEngine.h>

#include <cinttypes>
#include <cstdio>

int main() {
  unsigned long long seed, subsequence, offset;
  while (std::scanf("%llu %llu %llu", &seed, &subsequence, &offset) == 3) {
    at::Philox4_32 engine(seed, subsequence, offset);
    uint32_t w0 = engine(), w1 = engine(), w2 = engine(), w3 = engine();
    std::printf("%u %u %u %u\n", w0, w1, w2, w3);
  }
  return 0;
}
