// jf_once.h -- one-time set-up per CUDA device (plain C++, no CUDA types).
//
// Kernel attributes such as the dynamic shared-memory limit belong to the device that was current
// when they were set, so a set-up step guarded by one process-wide flag would be skipped on every
// device after the first. PerDeviceOnce keeps one flag per device ordinal, under a mutex, and
// records a device as done only when its set-up succeeded (a failed set-up runs again next call).
#ifndef JF_ONCE_H
#define JF_ONCE_H

#include <mutex>

namespace jf {

struct PerDeviceOnce {
  static constexpr int kMaxDevices = 64;
  std::mutex mu;
  bool done[kMaxDevices] = {};

  // Runs fn() (returning 0 on success, else an error code) unless it already succeeded for `dev`.
  // Returns 0, fn's error code, or -1 for a device ordinal outside [0, kMaxDevices).
  template <class Fn>
  int run(int dev, Fn&& fn) {
    if (dev < 0 || dev >= kMaxDevices) return -1;
    std::lock_guard<std::mutex> lock(mu);
    if (done[dev]) return 0;
    const int e = static_cast<int>(fn());
    if (e == 0) done[dev] = true;
    return e;
  }
};

}  // namespace jf

#endif  // JF_ONCE_H
