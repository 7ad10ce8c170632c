// Host check of the register sorting networks used by the bulk append: for
// random sets of 128 distinct 32-bit keys (and adversarial patterns), the full
// sort and the top-64 selection must equal std::sort's decreasing order.
// Prints "ok <trials>" and exits 0, or prints the first mismatch and exits 1.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <functional>
#include <random>
#include <vector>

#include "sortnet.cuh"

static uint32_t g_one = 1;

static int check(const std::vector<uint32_t>& keys, const char* what) {
  uint32_t full[128], top[128];
  for (int i = 0; i < 128; ++i) full[i] = top[i] = keys[i];
  swan::sortnet::sort128_desc_full(full, g_one);
  swan::sortnet::top64_of128_desc(top, g_one);
  std::vector<uint32_t> want(keys);
  std::sort(want.begin(), want.end(), std::greater<uint32_t>());
  for (int i = 0; i < 128; ++i) {
    if (full[i] != want[i]) {
      std::printf("%s: full sort differs at rank %d\n", what, i);
      return 1;
    }
    if (i < 64 && top[i] != want[i]) {
      std::printf("%s: top-64 differs at rank %d\n", what, i);
      return 1;
    }
  }
  return 0;
}

int main(int argc, char** argv) {
  const int trials = argc > 1 ? std::atoi(argv[1]) : 20000;
  if (argc > 2) g_one = (uint32_t)std::atoi(argv[2]);  // the run-time 1 of the multiply-adds
  std::mt19937_64 gen(20251124);
  std::vector<uint32_t> keys(128);
  // structured cases: sorted, reversed, one large key at each position
  for (int i = 0; i < 128; ++i) keys[i] = 1000u + (uint32_t)i;
  if (check(keys, "increasing")) return 1;
  std::reverse(keys.begin(), keys.end());
  if (check(keys, "decreasing")) return 1;
  for (int p = 0; p < 128; ++p) {
    for (int i = 0; i < 128; ++i) keys[i] = (uint32_t)i;
    keys[p] = 0xffffffffu;
    if (check(keys, "one large")) return 1;
    keys[p] = (uint32_t)p;
    for (int i = 0; i < 128; ++i) keys[i] = 0x80000000u + (uint32_t)i;
    keys[p] = 0u;
    if (check(keys, "one small")) return 1;
  }
  // random distinct keys; half of the trials from a small range (near-ties in
  // the high bits, as equal magnitudes give)
  for (int t = 0; t < trials; ++t) {
    std::vector<uint32_t> pool;
    const uint32_t range = (t & 1) ? 512u : 0xffffffffu;
    while ((int)pool.size() < 128) {
      const uint32_t x = (uint32_t)(gen() % range);
      if (std::find(pool.begin(), pool.end(), x) == pool.end()) pool.push_back(x);
    }
    if (check(pool, "random")) return 1;
  }
  std::printf("ok %d\n", trials);
  return 0;
}
