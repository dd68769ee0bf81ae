// Open-addressed set of pointers (host only, no CUDA): the session table's
// set of live snapshot handles.
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>

namespace pcs {

// A set of pointers in one open-addressed table (linear probing, erased
// slots marked): no allocation per insert, and a membership test never
// dereferences the pointer it is asked about, so any value a caller passes
// as a handle can be checked.
template <class T>
class PtrSet {
 public:
  size_t size() const { return n_; }
  bool count(const T* p) const {
    if (slot_.empty() || !p) return false;
    const uintptr_t k = reinterpret_cast<uintptr_t>(p);
    for (size_t i = hash(k) & mask();; i = (i + 1) & mask()) {
      if (slot_[i] == k) return true;
      if (slot_[i] == kEmpty) return false;
    }
  }
  void reserve(size_t n) {
    if ((used_ + n) * 2 > slot_.size()) rehash(n_ + n);
  }
  void insert(T* p) {
    reserve(1);
    const uintptr_t k = reinterpret_cast<uintptr_t>(p);
    size_t gone = SIZE_MAX;
    for (size_t i = hash(k) & mask();; i = (i + 1) & mask()) {
      if (slot_[i] == k) return;
      if (slot_[i] == kGone && gone == SIZE_MAX) gone = i;
      if (slot_[i] == kEmpty) {
        if (gone != SIZE_MAX) {
          i = gone;
        } else {
          ++used_;
        }
        slot_[i] = k;
        ++n_;
        return;
      }
    }
  }
  bool erase(const T* p) {
    if (slot_.empty() || !p) return false;
    const uintptr_t k = reinterpret_cast<uintptr_t>(p);
    for (size_t i = hash(k) & mask();; i = (i + 1) & mask()) {
      if (slot_[i] == k) {
        slot_[i] = kGone;
        --n_;
        return true;
      }
      if (slot_[i] == kEmpty) return false;
    }
  }
  template <class F>
  void for_each(F f) const {
    for (uintptr_t k : slot_)
      if (k != kEmpty && k != kGone) f(reinterpret_cast<T*>(k));
  }
  void clear() {
    slot_.clear();
    n_ = used_ = 0;
  }

 private:
  static constexpr uintptr_t kEmpty = 0, kGone = 1;  // never valid object addresses
  std::vector<uintptr_t> slot_;  // a power of two of slots, at most half in use
  size_t n_ = 0, used_ = 0;      // live entries; live + erased slots
  size_t mask() const { return slot_.size() - 1; }
  static size_t hash(uintptr_t x) {
    uint64_t z = static_cast<uint64_t>(x);
    z ^= z >> 33;
    z *= 0xFF51AFD7ED558CCDull;  // MurmurHash3's 64-bit finaliser constant
    z ^= z >> 33;
    return static_cast<size_t>(z);
  }
  void rehash(size_t want) {
    size_t cap = 16;
    while (cap < want * 2 + 2) cap <<= 1;
    std::vector<uintptr_t> old;
    old.swap(slot_);
    slot_.assign(cap, kEmpty);
    n_ = used_ = 0;
    for (uintptr_t k : old)
      if (k != kEmpty && k != kGone) insert(reinterpret_cast<T*>(k));
  }
};

}  // namespace pcs
