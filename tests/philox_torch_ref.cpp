// Independent Philox4x32-10 reference for pinning the oracle: PyTorch's
// header-only at::philox_engine (ATen/core/PhiloxRNGEngine.h).
// Reads lines "seed step quad" (decimal uint64) on stdin; prints the four
// 32-bit output words of the block with key = seed, counter =
// (lo(quad), hi(quad), lo(step), hi(step)) as decimal numbers.
#include <ATen/core/PhiloxRNGEngine.h>
#include <cinttypes>
#include <cstdio>

int main() {
  unsigned long long seed, step, quad;
  while (std::scanf("%llu %llu %llu", &seed, &step, &quad) == 3) {
    // subsequence fills counter words 2..3, offset fills words 0..1
    at::philox_engine eng(seed, step, quad);
    uint32_t w0 = eng(), w1 = eng(), w2 = eng(), w3 = eng();
    std::printf("%u %u %u %u\n", w0, w1, w2, w3);
  }
  return 0;
}
