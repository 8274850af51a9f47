// Per-device once-flags for settings that CUDA keeps per device, such as a
// kernel's dynamic shared-memory limit (cudaFuncSetAttribute applies to the
// current device only).  Host code only; no CUDA types, so a plain C++ test can
// exercise it without a GPU.
#pragma once

#include <atomic>
#include <cstdint>

namespace seedq {

// One bit per device ordinal below 64.  run(dev, apply) calls apply() unless it
// has already succeeded on device dev; a failed apply() leaves the bit clear,
// so the next call tries again.  Safe from several host threads: two first
// calls on one device may both apply the setting, which must therefore be
// idempotent.  forget(dev) clears the bit (after the device's context was
// destroyed, e.g. by cudaDeviceReset, its settings are gone).  Devices at or
// above 64 apply the setting on every call.
class DeviceOnce {
 public:
  template <typename F>
  int run(int dev, F &&apply) {
    if (dev >= 0 && dev < 64 && ((bits_.load(std::memory_order_acquire) >> dev) & 1u)) return 0;
    const int r = apply();
    if (r == 0 && dev >= 0 && dev < 64) bits_.fetch_or(1ull << dev, std::memory_order_acq_rel);
    return r;
  }
  void forget(int dev) {
    if (dev >= 0 && dev < 64) bits_.fetch_and(~(1ull << dev), std::memory_order_acq_rel);
  }
  bool done(int dev) const {
    return dev >= 0 && dev < 64 && ((bits_.load(std::memory_order_acquire) >> dev) & 1u);
  }

 private:
  std::atomic<uint64_t> bits_{0};
};

}  // namespace seedq
