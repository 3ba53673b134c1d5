// Thread-safe table of one value per CUDA device, filled on first use.
//
// Device properties and per-device settings (multiprocessor count, a kernel's
// shared-memory opt-in, a symbol's device address) differ between devices and
// must be looked up with that device current, so the library keeps one slot
// per device ordinal instead of one process-wide value.  The header has no
// CUDA dependency, so its logic is tested on the host.
#pragma once

#include <mutex>

namespace fademem {

template <typename T, int kMaxDevices = 64>
class PerDevice {
 public:
  // The value of device `dev`.  On first use `init(dev, &value)` computes it;
  // the value is kept only if init returns true (a failed lookup is retried
  // on the next call).  Returns false for a device ordinal outside the table
  // or a failed init.  Concurrent callers are serialised.
  template <typename Init>
  bool get(int dev, Init&& init, T* out) {
    if (dev < 0 || dev >= kMaxDevices) return false;
    std::lock_guard<std::mutex> lock(mu_);
    if (!have_[dev]) {
      T v{};
      if (!init(dev, &v)) return false;
      val_[dev] = v;
      have_[dev] = true;
    }
    *out = val_[dev];
    return true;
  }

 private:
  std::mutex mu_;
  bool have_[kMaxDevices] = {};
  T val_[kMaxDevices] = {};
};

}  // namespace fademem
