// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "smetric.h"

namespace smetric {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kEmpty = 0;  // key of a never-used slot

// SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014; Stafford's
// Mix13 multipliers). Two xor-shift-multiply rounds and a final xor-shift.
__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// The table is an array of buckets of kSlots = 15 slots. A bucket's 16-byte
// tag group (in a tag array of its own) holds a one-byte tag per slot (0:
// empty; otherwise 0x80 | low 7 key bits) and, in byte 15, the bucket's
// overflow count: how many keys stored past this bucket probed through it
// (saturating at 255, which then stays). Entries (key + tier-mask words) are
// in the entry array, slot sl of bucket b at b * kSlots + sl. A key's home
// bucket is the high 64 bits of key * n_buckets (Lemire's range reduction);
// an insert takes the first empty slot in bucket order from the home bucket
// (linear probing over buckets) and counts itself in the overflow byte of
// every bucket it passed; a lookup stops at the first bucket without the key
// whose overflow count is 0. A key that leaves its last tier gives its slot
// back (tag and key zeroed, the passed buckets' counts decremented), so the
// table holds live keys only and no tombstones. At load factor 0.7 about 98%
// of keys sit in their home bucket: a lookup is one tag read plus one entry
// read.
constexpr int kBucket = 16;  // bytes of a bucket's tag group
constexpr int kSlots = 15;   // slots of a bucket
constexpr uint32_t kSlotBits = (1u << kSlots) - 1;

// mix64 on 32-bit halves, for the serial chain where only latency counts:
// the high word of each product is one three-input sum of the low-by-low
// high half and the two cross products. Same value as mix64.
__device__ __forceinline__ uint64_t mix64_halves(uint64_t z) {
  uint32_t lo = (uint32_t)z, hi = (uint32_t)(z >> 32);
  auto xs = [&](int s) {
    lo ^= __funnelshift_r(lo, hi, s);
    hi ^= hi >> s;
  };
  auto mul = [&](uint64_t c) {
    const uint32_t cl = (uint32_t)c, ch = (uint32_t)(c >> 32);
    const uint32_t x1 = lo * ch, x2 = hi * cl;
    hi = __umulhi(lo, cl) + x1 + x2;
    lo = lo * cl;
  };
  xs(30);
  mul(0xBF58476D1CE4E5B9ull);
  xs(27);
  mul(0x94D049BB133111EBull);
  xs(31);
  return ((uint64_t)hi << 32) | lo;
}

__device__ __forceinline__ uint64_t home_bucket(uint64_t key, uint64_t n_buckets) {
  return __umul64hi(key, n_buckets);
}

__host__ __device__ __forceinline__ uint32_t key_tag(uint64_t key) {
  return 0x80u | (uint32_t)(key & 0x7Fu);
}

// Bit s of the result is set where byte s of the 16 tag bytes equals `tag`.
__device__ __forceinline__ uint32_t tag_match(uint4 t, uint32_t tag) {
  const uint32_t rep = tag * 0x01010101u;
  uint32_t m = 0;
  const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t eq = __vcmpeq4(w[i], rep);  // 0xff in each equal byte
    // gather the top bit of each byte into 4 bits
    const uint32_t b = ((eq >> 7) & 1u) | ((eq >> 14) & 2u) | ((eq >> 21) & 4u) | ((eq >> 28) & 8u);
    m |= b << (4 * i);
  }
  return m;
}

// Bit s of the result is set where slot s's tag equals `tag` (byte 15, the
// overflow count, left out).
__device__ __forceinline__ uint32_t slot_match(uint4 t, uint32_t tag) { return tag_match(t, tag) & kSlotBits; }

// A bucket's overflow count (byte 15 of its tag group).
__device__ __forceinline__ uint32_t overflow_count(uint4 t) { return t.w >> 24; }

// Buckets a lookup or an insert visits at most.
__host__ __device__ __forceinline__ uint64_t max_buckets(uint64_t n_buckets) {
  const uint64_t m = SMETRIC_MAX_PROBE / kBucket;
  return n_buckets < m ? n_buckets : m;
}

// First error wins; later ones are dropped until the host reads and clears.
__device__ __forceinline__ void latch_error(int32_t* status, int32_t code) {
  atomicCAS(reinterpret_cast<int*>(status), 0, code);
}

// Entry stride in 64-bit words for W mask words: key + W words, rounded up to
// a power of two so that no entry straddles a 32-byte sector (W = 1: 16 B,
// W = 2..3: 32 B, W = 4..7: 64 B).
__host__ __device__ constexpr int entry_words(int W) { return W == 1 ? 2 : (W <= 3 ? 4 : 8); }

// Route kernels, in launch order; names returned by smetric_profile_kernel_name.
// kChainProbe is k_lead and k_chain_probe in a route (leader flags, then
// chain, group stage and probe in one kernel) and k_chain in the calls that
// only hash.
enum RouteKernel { kPrep = 0, kDigest = 1, kChainProbe = 2, kWalk = 3, kNumRouteKernels = 4 };

struct ProfileSlot {
  cudaEvent_t ev[kNumRouteKernels + 1];
};

}  // namespace smetric

namespace smetric {

// Device-side LRU of the capped tiers (smetric_index_set_lru; kernels in
// lru.cu). Each capped tier keeps its keys in recency order, least recent
// first, in a region of one of two record buffers; a commit rewrites every
// region from one buffer into the other.
struct LruState {
  int64_t local_cap = 0, global_cap = 0;  // blocks; 0 = uncapped
  int n_tiers = 0;                        // N + 1
  uint64_t* ring[2] = {nullptr, nullptr}; // records (keys), tier t's at its region offset
  int cur = 0;                            // the buffer holding the current records
  int64_t* plan = nullptr;                // kLruPlanFields rows of n_tiers + 1 int64 (lru.cu)
  int64_t* req_off = nullptr;             // 2 * max_batch_requests: a request's first touch in its tiers
  uint64_t* touches = nullptr;            // 2 * max_blocks: the batch's touches, tier after tier
  uint64_t* set = nullptr;                // set_entries (key, last touch + 1) pairs
  int64_t set_entries = 0;
  uint8_t* keep = nullptr;                // max_tiles * kLruTile flags
  int64_t* tile_cnt = nullptr;            // max_tiles + 1, then their exclusive scan
  int64_t* tile_off = nullptr;
  int64_t max_tiles = 0;
};

}  // namespace smetric

struct smetric_index {
  smetric_index_config cfg;
  int device;
  int num_sms;
  int W;   // tier-mask words per key
  int EW;  // entry stride in 64-bit words
  uint64_t n_buckets;  // ceil(capacity_slots / kSlots)
  uint64_t* table;     // n_buckets * kSlots entries of EW words
  uint8_t* tags;       // n_buckets tag groups of kBucket bytes
  int32_t* status;  // device: first latched error
  // route scratch
  int64_t* block_off;  // max_batch_requests + 1: first block of each request
  uint64_t* digest;    // max_batch_tokens / B: per-block digests d_b
  uint64_t* hashes;    // max_batch_tokens / B: per-block chain hashes h_b
  uint64_t* masks;     // W * max_batch_tokens / B: per-block tier masks
  uint64_t* chunk_and; // W * (max_batch_tokens / B / 32 + R + 1): AND of each request-aligned 32-block chunk's masks
  uint64_t* groups;    // 2 * group_slots: (first-block hash, INT32_MAX - leader) pairs
  uint64_t group_slots;  // power of two >= 2 * max_batch_requests
  int32_t* lead;       // max_batch_requests: the request whose masks a request shares
  int32_t* share;      // max_batch_requests: leading blocks taken from the leader
  int32_t* summ;       // max_batch_requests * (num_instances + 1): a leader's run ends c_i, then g
  uint64_t* sk_tmp;     // max_batch_requests: session keys nobody reads (session links); a route's leader flags
  int64_t* chunk_off;  // max_batch_requests + 1: first 32-block chunk of each request
  int32_t* batch_ok;   // device flag written by the prep kernel
  // staging for smetric_route_batch_host
  int32_t* st_tokens;
  int64_t* st_offsets;
  int64_t* st_load;
  int32_t* st_out32;    // 3 * max_batch_requests
  uint64_t* st_sk;      // max_batch_requests
  int digest_occ;  // resident digest CTAs per SM (0 until the first route)
  smetric::LruState* lru;  // capped tiers' recency (NULL: no tier capped)
  // observability
  int64_t launches;
  bool profiling;
  std::vector<smetric::ProfileSlot> prof_pool;  // free event sets
  std::vector<smetric::ProfileSlot> prof_used;  // recorded, not yet read
};

namespace smetric {
// Returns SMETRIC_OK if the index is usable from the current device.
int check_device(const smetric_index* idx);
// Maps a CUDA error to SMETRIC_ERR_CUDA (clearing the sticky-free error state).
int cuda_status(cudaError_t e);
// Inserts a routed batch's block hashes into its chosen instances' local tiers
// (and the global tier); block_off must hold the batch's block offsets.
int launch_commit(smetric_index* idx, const int32_t* d_instance, const uint64_t* d_hashes, int32_t n,
                  int64_t max_blocks, bool global, cudaStream_t s);
// After a commit's inserts: the capped tiers' recency lists take the batch's
// touches and evict what exceeds each cap (no-op without an LRU).
int lru_commit(smetric_index* idx, const int32_t* d_instance, const uint64_t* d_hashes, int32_t n, bool global,
               cudaStream_t s);
// Empties every recency list (after the table is cleared).
int lru_reset(smetric_index* idx, cudaStream_t s);
// Frees the LRU state.
void lru_free(smetric_index* idx);
}  // namespace smetric
