// Host build of the CUDA path's Philox4x32-10 forms (csrc/copes_internal.h, compiled here
// by a plain C++ compiler): for each line of (key, counter, tag) read from stdin it prints
// the words of the plain form (philox4x32_10), of the precomputed-round-key form
// (philox4x32_10_rk) and, for counters below 2^32, of the folded form the update uses
// (philox4x32_10_folded with philox_folded_keys), for tests/test_philox_forms.py to check
// against the oracle's independent implementation.
#include <cinttypes>
#include <cstdio>

#include "../paper_2608_02391_gb300/csrc/copes_internal.h"

int main() {
  unsigned long long key, ctr;
  unsigned tag;
  while (std::scanf("%llu %llu %u", &key, &ctr, &tag) == 3) {
    const uint32_t k0 = (uint32_t)key, k1 = (uint32_t)(key >> 32);
    const uint32_t c0 = (uint32_t)ctr, c1 = (uint32_t)(ctr >> 32);
    uint32_t plain[4], viark[4], folded[4] = {0, 0, 0, 0}, rk[20], fk[20];
    copes::philox4x32_10(c0, c1, 0u, tag, k0, k1, plain);
    copes::philox_round_keys(k0, k1, rk);
    copes::philox4x32_10_rk(c0, c1, 0u, tag, rk, viark);
    int has_folded = 0;
    if (c1 == 0) {
      copes::philox_folded_keys(rk, tag, fk);
      const uint64_t m = (uint64_t)copes::kPhiloxM0 * c0;
      copes::philox4x32_10_folded((uint32_t)m, (uint32_t)(m >> 32), fk, folded);
      has_folded = 1;
    }
    std::printf("%u %u %u %u | %u %u %u %u | %d %u %u %u %u\n", plain[0], plain[1], plain[2], plain[3],
                viark[0], viark[1], viark[2], viark[3], has_folded, folded[0], folded[1], folded[2],
                folded[3]);
  }
  return 0;
}
