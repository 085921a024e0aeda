// Black-box driver for PyTorch's header-only Philox4x32-10 engine
// (ATen/core/PhiloxRNGEngine.h), used only as an independent pin of the
// oracle's Philox.  Reads "seed subsequence offset" triples from stdin and
// prints the four 32-bit words of that block.  The engine puts
// (offset lo, offset hi, subsequence lo, subsequence hi) in the counter and
// (seed lo, seed hi) in the key.
#include <ATen/core/PhiloxRNGEngine.h>
#include <cstdio>

int main() {
  unsigned long long seed, sub, off;
  while (std::scanf("%llu %llu %llu", &seed, &sub, &off) == 3) {
    at::Philox4_32 eng(seed, sub, off);
    unsigned a = eng(), b = eng(), c = eng(), d = eng();
    std::printf("%u %u %u %u\n", a, b, c, d);
  }
  return 0;
}
