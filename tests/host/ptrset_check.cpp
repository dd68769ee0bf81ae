// Randomised check of pcs::PtrSet (the session table's set of live handles)
// against std::unordered_set: inserts, erases, membership of values that were
// never inserted, reserve, clear and enumeration, with address patterns that
// make long probe runs and many erased slots.  Prints "ok" or the first
// mismatch.  Usage: ptrset_check <seed> <operations>
#include <cstdio>
#include <cstdlib>
#include <random>
#include <unordered_set>
#include <vector>

#include "pcs_ptrset.h"

struct Obj {};

int main(int argc, char** argv) {
  const unsigned seed = argc > 1 ? static_cast<unsigned>(std::atoi(argv[1])) : 1u;
  const long ops = argc > 2 ? std::atol(argv[2]) : 200000;
  std::mt19937_64 rng(seed);
  // Candidate addresses: a dense run (neighbouring objects), a strided run
  // (equal low bits) and scattered ones; all multiples of 8 and never 0 or 1.
  std::vector<uintptr_t> pool;
  for (uintptr_t i = 0; i < 3000; ++i) pool.push_back(0x7f0000001000ull + 96 * i);
  for (uintptr_t i = 0; i < 3000; ++i) pool.push_back(0x550000000000ull + (i << 20));
  for (int i = 0; i < 3000; ++i) pool.push_back((rng() & 0x0000FFFFFFFFFFF8ull) | 8u);
  pcs::PtrSet<Obj> set;
  std::unordered_set<uintptr_t> ref;
  for (long op = 0; op < ops; ++op) {
    const uintptr_t a = pool[rng() % pool.size()];
    Obj* p = reinterpret_cast<Obj*>(a);
    const unsigned what = static_cast<unsigned>(rng() % 100);
    if (what < 45) {
      set.insert(p);
      ref.insert(a);
    } else if (what < 85) {
      const bool got = set.erase(p), want = ref.erase(a) > 0;
      if (got != want) {
        std::printf("erase mismatch at op %ld\n", op);
        return 1;
      }
    } else if (what < 98) {
      const uintptr_t probe = (what & 1) ? a : (rng() & 0x0000FFFFFFFFFFF8ull) | 8u;
      if (set.count(reinterpret_cast<Obj*>(probe)) != (ref.count(probe) > 0)) {
        std::printf("count mismatch at op %ld\n", op);
        return 1;
      }
    } else if (what < 99) {
      set.reserve(static_cast<size_t>(rng() % 5000));
    } else if (rng() % 50 == 0) {
      set.clear();
      ref.clear();
    }
    if (set.size() != ref.size()) {
      std::printf("size mismatch at op %ld: %zu vs %zu\n", op, set.size(), ref.size());
      return 1;
    }
    if (set.count(nullptr)) {
      std::printf("null reported live at op %ld\n", op);
      return 1;
    }
  }
  size_t seen = 0;
  bool all_known = true;
  set.for_each([&](Obj* p) {
    ++seen;
    all_known = all_known && ref.count(reinterpret_cast<uintptr_t>(p)) > 0;
  });
  for (uintptr_t a : ref)
    if (!set.count(reinterpret_cast<Obj*>(a))) all_known = false;
  if (seen != ref.size() || !all_known) {
    std::printf("enumeration mismatch: %zu listed, %zu live\n", seen, ref.size());
    return 1;
  }
  std::printf("ok\n");
  return 0;
}
