// Counter-based generator behind the synthetic test and benchmark inputs.
#pragma once

#include <stdint.h>

namespace seedq {

// Output number i (0-based) of splitmix64 started at state key (Steele, Lea,
// Flood 2014).
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t key, uint64_t i) {
  uint64_t z = key + (i + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

}  // namespace seedq
