// Test shim: the library's host Task Scheduler header compiled on its own
// (no CUDA), exposed through a minimal C interface, so that copies of the
// header with planted mistakes can be checked against the same traces as
// the library.  Built by tests/test_library_mutations.py.
#include <cstdint>
#include <new>

#include "fo_sched.hpp"

extern "C" {
void* shim_create(int K, int omega, int depth, int policy) {
  return new (std::nothrow) fo::TaskScheduler(K, omega, depth, policy);
}
void shim_destroy(void* s) { delete static_cast<fo::TaskScheduler*>(s); }
int shim_put(void* s, int k, int32_t* slot) {
  *slot = -1;
  return static_cast<fo::TaskScheduler*>(s)->put(k, slot);
}
int shim_peek(void* s, int k, int32_t* slot) {
  *slot = -1;
  return static_cast<const fo::TaskScheduler*>(s)->peek(k, slot);
}
int shim_get(void* s, int* k, int32_t* slot) {
  *k = -1;
  *slot = -1;
  return static_cast<fo::TaskScheduler*>(s)->get(k, slot);
}
int shim_set_active(void* s, int k, int active) { return static_cast<fo::TaskScheduler*>(s)->set_active(k, active); }
void shim_counters(void* s, uint64_t* c) {
  const auto& v = static_cast<fo::TaskScheduler*>(s)->counters();
  for (size_t i = 0; i < v.size(); ++i) c[i] = v[i];
}
void shim_sender(void* s, uint8_t* on) {
  const auto& v = static_cast<fo::TaskScheduler*>(s)->sender_on();
  for (size_t i = 0; i < v.size(); ++i) on[i] = v[i];
}
int shim_queued(void* s) { return static_cast<fo::TaskScheduler*>(s)->queued_total(); }
}
