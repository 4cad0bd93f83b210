// Checks the multiply-based division of the tensor-core kernel's epilogue
// against integer division: every divisor up to 4096 and sampled larger
// ones, each with small dividends, dividends around multiples of the
// divisor and sampled dividends up to 2^31 - 1.
#include <cstdint>
#include <cstdio>

#include "fastdiv.h"

static uint64_t state = 0x9e3779b97f4a7c15ull;
static uint32_t rnd31() {   // xorshift64*
  state ^= state >> 12;
  state ^= state << 25;
  state ^= state >> 27;
  return (uint32_t)((state * 0x2545f4914f6cdd1dull) >> 33);
}

static int check(int64_t d) {
  uint32_t m, s;
  dirigo::fast_div_make(d, &m, &s);
  auto one = [&](uint32_t x) {
    if (x >= (1u << 31)) return 0;
    const uint32_t want = (uint32_t)(x / (uint64_t)d), got = dirigo::fast_div(x, m, s);
    if (want != got) {
      std::printf("FAIL d=%lld x=%u want=%u got=%u\n", (long long)d, x, want, got);
      return 1;
    }
    return 0;
  };
  int bad = 0;
  for (uint32_t x = 0; x < 2048; ++x) bad |= one(x);
  bad |= one((1u << 31) - 1);
  for (int k = 0; k < 64; ++k) {
    const uint64_t q = rnd31() % ((1ull << 31) / (uint64_t)d + 1);
    const uint64_t x = q * (uint64_t)d;
    if (x >= 1) bad |= one((uint32_t)(x - 1));
    if (x < (1ull << 31)) bad |= one((uint32_t)x);
    if (x + 1 < (1ull << 31)) bad |= one((uint32_t)(x + 1));
  }
  for (int k = 0; k < 256; ++k) bad |= one(rnd31());
  return bad;
}

int main() {
  int bad = 0;
  for (int64_t d = 1; d <= 4096; ++d) bad |= check(d);
  for (int k = 0; k < 4096; ++k) bad |= check((int64_t)(rnd31() % ((1u << 31) - 1)) + 1);
  const int64_t edges[] = {(1ll << 16) - 1, 1ll << 16, (1ll << 16) + 1, (1ll << 30) + 1,
                           (1ll << 31) - 1, 1ll << 31};
  for (int64_t d : edges) bad |= check(d);
  std::printf(bad ? "FAIL\n" : "ok\n");
  return bad;
}
