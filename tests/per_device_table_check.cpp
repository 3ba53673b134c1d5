// Host-side check of the library's per-device table (csrc/per_device.h):
// values are kept per device ordinal, computed once per device, a failed
// lookup is retried, ordinals outside the table are refused, and concurrent
// first uses of one device run its lookup once.  Prints "ok" and exits 0.
#include <atomic>
#include <cstdio>
#include <thread>
#include <vector>

#include "per_device.h"

#define CHECK(c)                                             \
  do {                                                       \
    if (!(c)) {                                              \
      std::printf("check failed at line %d: %s\n", __LINE__, #c); \
      return 1;                                              \
    }                                                        \
  } while (0)

int main() {
  fademem::PerDevice<int, 8> table;
  int calls[8] = {};
  auto sm_count = [&calls](int dev, int* v) {
    ++calls[dev];
    *v = 100 + dev;  // a different value per device, like two GPU models
    return true;
  };
  int v = 0;
  CHECK(table.get(0, sm_count, &v) && v == 100);
  CHECK(table.get(1, sm_count, &v) && v == 101);  // the second device gets its own value
  CHECK(table.get(0, sm_count, &v) && v == 100);
  CHECK(table.get(1, sm_count, &v) && v == 101);
  CHECK(calls[0] == 1 && calls[1] == 1);          // looked up once per device
  CHECK(!table.get(8, sm_count, &v) && !table.get(-1, sm_count, &v));

  // A failed lookup stores nothing and is retried.
  int tries = 0;
  auto flaky = [&tries](int, int* v) {
    ++tries;
    *v = 7;
    return tries >= 2;
  };
  v = -1;
  CHECK(!table.get(3, flaky, &v) && v == -1);
  CHECK(table.get(3, flaky, &v) && v == 7 && tries == 2);
  CHECK(table.get(3, flaky, &v) && v == 7 && tries == 2);

  // Concurrent first use of each device: one lookup per device, one value seen by all.
  fademem::PerDevice<int, 8> shared;
  std::atomic<int> lookups[4];
  for (auto& a : lookups) a = 0;
  std::atomic<int> wrong{0};
  std::vector<std::thread> threads;
  for (int t = 0; t < 16; ++t) {
    threads.emplace_back([&, t] {
      for (int r = 0; r < 1000; ++r) {
        const int dev = (t + r) % 4;
        int x = 0;
        const bool ok = shared.get(dev, [&lookups](int d, int* v) {
          lookups[d].fetch_add(1);
          *v = 1000 * (d + 1);
          return true;
        }, &x);
        if (!ok || x != 1000 * (dev + 1)) wrong.fetch_add(1);
      }
    });
  }
  for (auto& th : threads) th.join();
  CHECK(wrong.load() == 0);
  for (auto& a : lookups) CHECK(a.load() == 1);
  std::printf("ok\n");
  return 0;
}
