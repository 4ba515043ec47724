// Device primitives of the key -> tier-mask table (layout beside kSlots in
// smetric_impl.cuh): lookup, insert of a tier bit, removal of a tier bit
// that gives the slot back once the key holds no tier.
//
// Concurrency contract: inserts run concurrently with inserts, removals with
// removals and lookups, never inserts with removals (they are separate
// kernels in stream order). Under that contract a key occupies at most one
// slot: slots only fill during an insert kernel, so two inserters of one key
// walking the same bucket order meet at the slot the first of them claimed.
#pragma once

#include "smetric_impl.cuh"

namespace smetric {

constexpr uint64_t kDeleting = 1;  // key word of a slot being given back (keys are >= 2)

__device__ __forceinline__ uint4 load_tags_volatile(const uint8_t* p) {
  const volatile uint32_t* q = reinterpret_cast<const volatile uint32_t*>(p);
  return make_uint4(q[0], q[1], q[2], q[3]);
}

// Adds d (+1 or -1) to the overflow count of bucket b unless it is saturated
// at 255 (a saturated count stays: it only costs later lookups a bucket).
__device__ __forceinline__ void overflow_add(uint8_t* tags, uint64_t b, int d) {
  unsigned int* w = reinterpret_cast<unsigned int*>(tags + b * kBucket) + 3;
  unsigned int old = *reinterpret_cast<volatile unsigned int*>(w);
  for (;;) {
    const unsigned int c = old >> 24;
    if (c == 255u || (d < 0 && c == 0u)) return;
    const unsigned int nw = d > 0 ? old + (1u << 24) : old - (1u << 24);
    const unsigned int prev = atomicCAS(w, old, nw);
    if (prev == old) return;
    old = prev;
  }
}

// Slot of `key` (bucket * kSlots + slot), or -1 when absent. VOLATILE reads
// the tags and keys around the cache for kernels that change the table.
template <bool VOLATILE>
__device__ __forceinline__ int64_t find_slot(const uint8_t* __restrict__ tags, const uint64_t* __restrict__ table,
                                             int ew, uint64_t n_buckets, uint64_t key) {
  const uint32_t tg = key_tag(key);
  uint64_t b = home_bucket(key, n_buckets);
  const uint64_t mb = max_buckets(n_buckets);
  for (uint64_t t = 0; t < mb; ++t) {
    const uint4 tv = VOLATILE ? load_tags_volatile(tags + b * kBucket)
                              : *reinterpret_cast<const uint4*>(tags + b * kBucket);
    uint32_t cand = slot_match(tv, tg);
    while (cand) {
      const int sl = __ffs(cand) - 1;
      cand &= cand - 1;
      const uint64_t slot = b * kSlots + sl;
      const uint64_t k = VOLATILE ? *reinterpret_cast<const volatile uint64_t*>(table + slot * ew)
                                  : table[slot * ew];
      if (k == key) return (int64_t)slot;
    }
    if (overflow_count(tv) == 0) return -1;  // no key stored past this bucket came through it
    if (++b == n_buckets) b = 0;
  }
  return -1;
}

// Sets tier bit m of mask word `word` of `key`, taking a slot if the key is
// new. Pass 1 looks the key up; pass 2 walks from the home bucket again and,
// in each bucket, first takes the key if a concurrent inserter has just
// placed it there, then tries each empty slot with a CAS on its key word.
// The winner publishes the tag after a fence and counts itself in every
// bucket it passed. A CAS that fails on this very key (claimed, tag not yet
// published) uses that slot. Returns false when no slot was found.
__device__ __forceinline__ bool insert_key(uint8_t* tags, uint64_t* table, int ew, uint64_t n_buckets,
                                           uint64_t key, int word, unsigned long long m) {
  const int64_t found = find_slot<true>(tags, table, ew, n_buckets, key);
  if (found >= 0) {
    atomicOr(reinterpret_cast<unsigned long long*>(table + found * ew) + 1 + word, m);
    return true;
  }
  const uint32_t tg = key_tag(key);
  const uint64_t home = home_bucket(key, n_buckets);
  uint64_t b = home;
  const uint64_t mb = max_buckets(n_buckets);
  for (uint64_t t = 0; t < mb; ++t) {
    const uint4 tv = load_tags_volatile(tags + b * kBucket);
    uint32_t cand = slot_match(tv, tg);
    while (cand) {
      const int sl = __ffs(cand) - 1;
      cand &= cand - 1;
      unsigned long long* e = reinterpret_cast<unsigned long long*>(table + (b * kSlots + sl) * ew);
      if (*reinterpret_cast<volatile unsigned long long*>(e) == key) {
        atomicOr(e + 1 + word, m);
        return true;
      }
    }
    uint32_t empty = slot_match(tv, 0);
    while (empty) {
      const int sl = __ffs(empty) - 1;
      empty &= empty - 1;
      unsigned long long* e = reinterpret_cast<unsigned long long*>(table + (b * kSlots + sl) * ew);
      const unsigned long long old = atomicCAS(e, (unsigned long long)kEmpty, (unsigned long long)key);
      if (old == kEmpty) {
        __threadfence();
        atomicOr(reinterpret_cast<unsigned int*>(tags + b * kBucket) + (sl >> 2), tg << (8 * (sl & 3)));
        for (uint64_t p = home, q = 0; q < t; ++q) {
          overflow_add(tags, p, +1);
          if (++p == n_buckets) p = 0;
        }
        atomicOr(e + 1 + word, m);
        return true;
      }
      if (old == key) {
        atomicOr(e + 1 + word, m);
        return true;
      }
    }
    if (++b == n_buckets) b = 0;
  }
  return false;
}

// Clears tier bit m of mask word `word` of `key` (absent pairs are ignored).
// When that leaves the key in no tier, the slot is given back: one thread
// (the winner of a CAS of the key word to kDeleting) clears the tag,
// decrements the overflow count of every bucket between the home bucket and
// the slot's, and zeroes the key word. With W > 1 mask words, a fence
// between clearing the bit and reading the other words makes at least one of
// two threads that clear the last bits of different words see all of them
// zero.
__device__ __forceinline__ void remove_tier(uint8_t* tags, uint64_t* table, int ew, int W, uint64_t n_buckets,
                                            uint64_t key, int word, unsigned long long m) {
  const int64_t slot = find_slot<true>(tags, table, ew, n_buckets, key);
  if (slot < 0) return;
  unsigned long long* e = reinterpret_cast<unsigned long long*>(table + slot * ew);
  const unsigned long long old = atomicAnd(e + 1 + word, ~m);
  if (!(old & m) || (old & ~m)) return;  // the bit was clear, or this word keeps other tiers
  __threadfence();
  for (int w = 0; w < W; ++w)
    if (w != word && *reinterpret_cast<volatile unsigned long long*>(e + 1 + w) != 0ull) return;
  if (atomicCAS(e, (unsigned long long)key, (unsigned long long)kDeleting) != key) return;
  const uint64_t b = (uint64_t)slot / kSlots;
  const int sl = (int)((uint64_t)slot % kSlots);
  atomicAnd(reinterpret_cast<unsigned int*>(tags + b * kBucket) + (sl >> 2), ~(0xFFu << (8 * (sl & 3))));
  for (uint64_t p = home_bucket(key, n_buckets); p != b;) {
    overflow_add(tags, p, -1);
    if (++p == n_buckets) p = 0;
  }
  __threadfence();
  atomicExch(e, (unsigned long long)kEmpty);
}

}  // namespace smetric
