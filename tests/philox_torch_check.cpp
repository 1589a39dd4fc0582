// Independent cross-check for the oracle's Philox4x32-10: runs PyTorch's
// installed, source-level Philox engine header on counters read from stdin
// and prints the four output words of each block.
// Input lines: seed subsequence offset (decimal); output: four hex words.
#include <ATen/core/PhiloxRNGEngine.h>
#include <cstdio>
#include <cinttypes>

int main() {
  unsigned long long seed, subseq, offset;
  while (std::scanf("%llu %llu %llu", &seed, &subseq, &offset) == 3) {
    at::philox_engine eng(seed, subseq, offset);
    unsigned int w[4];
    for (int i = 0; i < 4; ++i) w[i] = eng();
    std::printf("%08x %08x %08x %08x\n", w[0], w[1], w[2], w[3]);
  }
  return 0;
}
