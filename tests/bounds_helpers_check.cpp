// Host-side check of the range test behind the bounds-checking build
// (csrc/fademem_internal.h, range_holds): an access [p, p + bytes) passes only
// if it lies inside [lo, hi).  Prints "ok" and exits 0.
#include <cstdio>

#include "fademem_internal.h"

#define CHECK(c)                                                   \
  do {                                                             \
    if (!(c)) {                                                    \
      std::printf("check failed at line %d: %s\n", __LINE__, #c); \
      return 1;                                                    \
    }                                                              \
  } while (0)

int main() {
  static char buf[4096];
  const fademem::DevRange r = fademem::dev_range(buf + 256, 1024);  // [buf+256, buf+1280)
  using fademem::range_holds;
  CHECK(range_holds(r, buf + 256, 16));           // first vector
  CHECK(range_holds(r, buf + 1264, 16));          // last vector, ends exactly at hi
  CHECK(range_holds(r, buf + 256, 1024));         // the whole range
  CHECK(range_holds(r, buf + 1280, 0));           // empty access at hi
  CHECK(!range_holds(r, buf + 1265, 16));         // one byte past the end
  CHECK(!range_holds(r, buf + 1280, 16));         // starts at hi
  CHECK(!range_holds(r, buf + 240, 16));          // ends exactly at lo: before the range
  CHECK(!range_holds(r, buf + 255, 16));          // one byte before lo
  CHECK(!range_holds(r, buf + 256, 1025));        // longer than the range
  CHECK(!range_holds(r, buf + 512, ~(size_t)0));  // a length that would wrap the end pointer
  const fademem::DevRange empty = fademem::dev_range(buf, 0);
  CHECK(!range_holds(empty, buf, 16));            // nothing fits an empty buffer
  CHECK(range_holds(empty, buf, 0));
  std::printf("ok\n");
  return 0;
}
