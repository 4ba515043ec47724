// Device-side LRU of capped KV$ tiers.
//
// Each serving instance's local KV$ and the global store are bounded and
// evict their least recently used blocks (Section 2: the instance that ran a
// request caches its blocks; capacity is finite). The recency order is the
// one the replay between batches uses: a block touched by request r of a
// batch at block position b has stamp (batch, r, -b), so within a request
// the deepest blocks are the least recent; after a batch's touches a tier
// over its cap evicts its smallest stamps until it is at the cap.
//
// Each capped tier keeps its keys in a record region, least recent first,
// one record per key. A commit rewrites every region from the current record
// buffer into the other one: the old records whose key the batch touched in
// that tier are dropped, the batch's touches of the tier follow in stamp
// order (a key touched several times once, at its last touch), and the
// first (count - cap) records are evicted instead of written. Per batch:
//   k_lru_plan    one warp: per request its first touch position in its
//                 local tier's and in the global tier's touch list (a stable
//                 prefix over the requests routed to each instance); per tier
//                 the touch count, the touch-list, set and tile offsets.
//   k_lru_touch   thread per block: the touch (deepest block first) into
//                 its tiers' touch lists and the batch's (tier, key) -> last
//                 touch sets.
//   k_lru_flags   CTA per tile of 4,096 records-then-touches of one tier:
//                 whether each survives the rewrite, and the tile's count.
//   k_lru_scan    one CTA: exclusive scan of the tile counts; per tier its
//                 surviving count and the excess over its cap.
//   k_lru_write   CTA per tile: each survivor's rank in its tier; the first
//                 `excess` leave the tier (remove_tier, which gives a slot
//                 back when its key leaves its last tier), the rest go to
//                 the other buffer.
//   k_lru_finish  new lengths; the sets cleared for the next batch.

#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <new>

#include "smetric_impl.cuh"
#include "table.cuh"
#include "call_range.cuh"

using namespace smetric;

namespace {

constexpr int kLruThreads = 256;
constexpr int kLruPer = 16;                          // consecutive elements a thread owns in a tile
constexpr int64_t kLruTile = kLruThreads * kLruPer;  // 4,096
constexpr int64_t kMaxCap = 1LL << 40;

// Rows of the per-tier plan (n_tiers + 1 entries each; the extra entry of
// kTile0 is the total tile count).
enum LruPlan {
  kRingOff = 0,  // the tier's record region in each buffer
  kCap,          // its cap (0: not capped)
  kLen,          // records in the current buffer
  kTouches,      // touches this batch
  kTouchOff,     // first touch in the touch lists
  kSetOff,       // first entry of its set
  kSetMask,      // set entries - 1 (-1: no set)
  kTile0,        // first tile
  kExcess,       // records to evict
  kNewLen,       // records after the rewrite
  kLruPlanFields
};

__device__ __forceinline__ int64_t* row(int64_t* plan, int n_tiers, int f) { return plan + (int64_t)f * (n_tiers + 1); }
__device__ __forceinline__ const int64_t* row(const int64_t* plan, int n_tiers, int f) {
  return plan + (int64_t)f * (n_tiers + 1);
}

// Batch set of one tier: open addressing over (key, last touch + 1) pairs,
// key 0 = empty; sized >= 2 x the tier's touches, so a probe always ends.
__device__ __forceinline__ void set_put(uint64_t* set, int64_t mask, uint64_t key, uint64_t v) {
  uint64_t s = key & (uint64_t)mask;
  for (int64_t t = 0; t <= mask; ++t) {
    unsigned long long* e = reinterpret_cast<unsigned long long*>(set + 2 * s);
    const unsigned long long old = atomicCAS(e, 0ull, (unsigned long long)key);
    if (old == 0ull || old == key) {
      atomicMax(e + 1, (unsigned long long)v);
      return;
    }
    s = (s + 1) & (uint64_t)mask;
  }
}

__device__ __forceinline__ uint64_t set_get(const uint64_t* set, int64_t mask, uint64_t key) {
  if (mask < 0) return 0;
  uint64_t s = key & (uint64_t)mask;
  for (int64_t t = 0; t <= mask; ++t) {
    const ulonglong2 e = *reinterpret_cast<const ulonglong2*>(set + 2 * s);
    if (e.x == key) return e.y;
    if (e.x == 0) return 0;
    s = (s + 1) & (uint64_t)mask;
  }
  return 0;
}

__device__ __forceinline__ int64_t next_pow2(int64_t v) {
  int64_t p = 1;
  while (p < v) p <<= 1;
  return p;
}

// One warp. Requests in rounds of 32: within a round, the lanes routed to
// the same instance (__match_any_sync) sum the blocks of their lower lanes;
// the running totals per instance carry across rounds, so req_off[r] is the
// number of blocks of earlier requests routed to r's instance, and
// req_off[R + r] that of all earlier committed requests (global tier).
__global__ void __launch_bounds__(32)
    k_lru_plan(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ instance,
               const int32_t* __restrict__ batch_ok, int N, bool local_capped, bool global_touch, int64_t* plan,
               int64_t* __restrict__ req_off, int64_t R) {
  extern __shared__ int64_t run[];  // N
  const int lane = threadIdx.x;
  const int nt = N + 1;
  for (int i = lane; i < N; i += 32) run[i] = 0;
  __syncwarp();
  const bool ok = *batch_ok != 0;
  int64_t grun = 0;
  for (int32_t base = 0; ok && base < n; base += 32) {
    const int32_t r = base + lane;
    int32_t i = -1;
    int64_t nb = 0;
    if (r < n) {
      i = instance[r];
      nb = block_off[r + 1] - block_off[r];
      if (i < 0 || i >= N) {
        i = -1;
        nb = 0;
      }
    }
    const unsigned peers = __match_any_sync(0xffffffffu, i);
    int64_t acc = 0, gacc = 0;
#pragma unroll 4
    for (int k = 0; k < 32; ++k) {
      const int64_t v = __shfl_sync(0xffffffffu, nb, k);
      if (k < lane) {
        gacc += v;
        if ((peers >> k) & 1u) acc += v;
      }
    }
    if (r < n && i >= 0) {
      req_off[r] = run[i] + acc;
      req_off[R + r] = grun + gacc;
    }
    __syncwarp();
    if (i >= 0 && lane == 31 - __clz(peers)) run[i] += acc + nb;
    grun += __shfl_sync(0xffffffffu, gacc + nb, 31);
    __syncwarp();
  }
  // per tier: touches, then the offsets of the touch lists, sets and tiles
  int64_t t_off = 0, s_off = 0, tile0 = 0;
  for (int base = 0; base < nt; base += 32) {
    const int t = base + lane;
    int64_t T = 0, S = 0, tiles = 0;
    if (t < nt) {
      const bool capped = row(plan, nt, kCap)[t] > 0;
      T = !capped ? 0 : (t < N ? (local_capped ? run[t] : 0) : (global_touch ? grun : 0));
      S = T > 0 ? next_pow2(2 * T) : 0;
      tiles = (row(plan, nt, kLen)[t] + T + kLruTile - 1) / kLruTile;
    }
    int64_t pt = T, ps = S, pl = tiles;  // inclusive warp scans
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int64_t a = __shfl_up_sync(0xffffffffu, pt, d), b = __shfl_up_sync(0xffffffffu, ps, d),
                    c = __shfl_up_sync(0xffffffffu, pl, d);
      if (lane >= d) {
        pt += a;
        ps += b;
        pl += c;
      }
    }
    if (t < nt) {
      row(plan, nt, kTouches)[t] = T;
      row(plan, nt, kTouchOff)[t] = t_off + pt - T;
      row(plan, nt, kSetOff)[t] = s_off + ps - S;
      row(plan, nt, kSetMask)[t] = S - 1;
      row(plan, nt, kTile0)[t] = tile0 + pl - tiles;
    }
    t_off += __shfl_sync(0xffffffffu, pt, 31);
    s_off += __shfl_sync(0xffffffffu, ps, 31);
    tile0 += __shfl_sync(0xffffffffu, pl, 31);
  }
  if (lane == 0) row(plan, nt, kTile0)[nt] = tile0;  // total tiles
  if (lane == 0) row(plan, nt, kSetOff)[nt] = s_off;  // set entries in use
}

// Thread per block f of the batch (request r, position b of n_r): its touch
// position in a tier's list is the tier's count of earlier requests' blocks
// plus n_r - 1 - b (deepest block first).
__global__ void k_lru_touch(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ instance,
                            const uint64_t* __restrict__ H, const int32_t* __restrict__ batch_ok, int N,
                            bool local_capped, bool global_touch, const int64_t* __restrict__ plan,
                            const int64_t* __restrict__ req_off, int64_t R, uint64_t* __restrict__ touches,
                            uint64_t* __restrict__ set) {
  if (!*batch_ok) return;
  const int nt = N + 1;
  const int64_t total = block_off[n];
  int32_t r = 0;
  for (int64_t f = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; f < total;
       f += (int64_t)gridDim.x * blockDim.x) {
    int32_t lo = r, hi = n;  // largest r with block_off[r] <= f
    while (hi - lo > 1) {
      const int32_t mid = (lo + hi) >> 1;
      if (block_off[mid] <= f) lo = mid; else hi = mid;
    }
    r = lo;
    const int32_t i = instance[r];
    const uint64_t key = H[f];
    if (i < 0 || i >= N || key < 2) continue;  // not committed (k_commit latches the invalid ones)
    const int64_t back = block_off[r + 1] - 1 - f;  // n_r - 1 - b
    if (local_capped) {
      const int64_t q = req_off[r] + back;
      touches[row(plan, nt, kTouchOff)[i] + q] = key;
      set_put(set + 2 * row(plan, nt, kSetOff)[i], row(plan, nt, kSetMask)[i], key, (uint64_t)q + 1);
    }
    if (global_touch) {
      const int64_t q = req_off[R + r] + back;
      touches[row(plan, nt, kTouchOff)[N] + q] = key;
      set_put(set + 2 * row(plan, nt, kSetOff)[N], row(plan, nt, kSetMask)[N], key, (uint64_t)q + 1);
    }
  }
}

// The tier of tile k: the largest t with kTile0[t] <= k (tiers without
// tiles share their successor's first tile and are skipped).
__device__ __forceinline__ int tier_of_tile(const int64_t* tile0, int nt, int64_t k) {
  int lo = 0, hi = nt;  // tile0[lo] <= k < tile0[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (tile0[mid] <= k) lo = mid; else hi = mid;
  }
  return lo;
}

// Element j of tier t's rewrite: a record (j < len) or the touch j - len.
// Returns whether it survives and its key.
__device__ __forceinline__ bool survives(const int64_t* plan, int nt, int t, int64_t j, const uint64_t* ring,
                                         const uint64_t* touches, const uint64_t* set, uint64_t& key) {
  const int64_t len = row(plan, nt, kLen)[t];
  const int64_t mask = row(plan, nt, kSetMask)[t];
  const uint64_t* tset = set + 2 * row(plan, nt, kSetOff)[t];
  if (j < len) {
    key = ring[row(plan, nt, kRingOff)[t] + j];
    return set_get(tset, mask, key) == 0;  // not touched again in this batch
  }
  const int64_t q = j - len;
  if (q >= row(plan, nt, kTouches)[t]) return false;  // the tile's tail
  key = touches[row(plan, nt, kTouchOff)[t] + q];
  return set_get(tset, mask, key) == (uint64_t)q + 1;  // the key's last touch in this batch
}

__global__ void __launch_bounds__(kLruThreads)
    k_lru_flags(const int64_t* __restrict__ plan, int nt, const uint64_t* __restrict__ ring,
                const uint64_t* __restrict__ touches, const uint64_t* __restrict__ set, uint8_t* __restrict__ keep,
                int64_t* __restrict__ tile_cnt) {
  const int64_t* tile0 = row(plan, nt, kTile0);
  const int64_t k = blockIdx.x;
  if (k >= tile0[nt]) return;
  const int t = tier_of_tile(tile0, nt, k);
  const int64_t j0 = (k - tile0[t]) * kLruTile + (int64_t)threadIdx.x * kLruPer;
  uint32_t bits[kLruPer / 4] = {0, 0, 0, 0};
  int cnt = 0;
#pragma unroll
  for (int e = 0; e < kLruPer; ++e) {
    uint64_t key;
    const bool s = survives(plan, nt, t, j0 + e, ring, touches, set, key);
    cnt += s;
    bits[e >> 2] |= (uint32_t)s << (8 * (e & 3));
  }
  *reinterpret_cast<uint4*>(keep + k * kLruTile + (int64_t)threadIdx.x * kLruPer) =
      make_uint4(bits[0], bits[1], bits[2], bits[3]);
  // tile count: warp sums, then the first warp
  __shared__ int ws[kLruThreads / 32];
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) cnt += __shfl_down_sync(0xffffffffu, cnt, d);
  if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    int64_t c = 0;
    for (int w = 0; w < kLruThreads / 32; ++w) c += ws[w];
    tile_cnt[k] = c;
  }
}

// One CTA: exclusive scan of the tile counts into tile_off (total at the
// end), then each tier's survivors, excess over its cap and new length.
__global__ void __launch_bounds__(1024)
    k_lru_scan(int64_t* __restrict__ plan, int nt, const int64_t* __restrict__ tile_cnt,
               int64_t* __restrict__ tile_off) {
  __shared__ int64_t ws[32];
  __shared__ int64_t carry;
  const int64_t total = row(plan, nt, kTile0)[nt];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int64_t base = 0; base < total; base += 1024) {
    const int64_t k = base + threadIdx.x;
    const int64_t v = k < total ? tile_cnt[k] : 0;
    int64_t x = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int64_t a = __shfl_up_sync(0xffffffffu, x, d);
      if (lane >= d) x += a;
    }
    if (lane == 31) ws[w] = x;
    __syncthreads();
    if (w == 0) {
      int64_t y = ws[lane];
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int64_t a = __shfl_up_sync(0xffffffffu, y, d);
        if (lane >= d) y += a;
      }
      ws[lane] = y;  // inclusive over warps
    }
    __syncthreads();
    const int64_t before = carry + (w > 0 ? ws[w - 1] : 0) + x - v;
    if (k < total) tile_off[k] = before;
    __syncthreads();
    if (threadIdx.x == 0) carry += ws[31];
    __syncthreads();
  }
  if (threadIdx.x == 0) tile_off[total] = carry;
  __syncthreads();
  const int64_t* tile0 = row(plan, nt, kTile0);
  for (int t = threadIdx.x; t < nt; t += blockDim.x) {
    const int64_t kept = tile_off[tile0[t + 1]] - tile_off[tile0[t]];
    const int64_t cap = row(plan, nt, kCap)[t];
    const int64_t ex = cap > 0 && kept > cap ? kept - cap : 0;
    row(plan, nt, kExcess)[t] = ex;
    row(plan, nt, kNewLen)[t] = kept - ex;
  }
}

__global__ void __launch_bounds__(kLruThreads)
    k_lru_write(const int64_t* __restrict__ plan, int nt, const uint64_t* __restrict__ ring,
                uint64_t* __restrict__ next, const uint64_t* __restrict__ touches, const uint64_t* __restrict__ set,
                const uint8_t* __restrict__ keep, const int64_t* __restrict__ tile_off, uint8_t* tags,
                uint64_t* table, int ew, int W, uint64_t n_buckets) {
  const int64_t* tile0 = row(plan, nt, kTile0);
  const int64_t k = blockIdx.x;
  if (k >= tile0[nt]) return;
  const int t = tier_of_tile(tile0, nt, k);
  const uint4 fl = *reinterpret_cast<const uint4*>(keep + k * kLruTile + (int64_t)threadIdx.x * kLruPer);
  const uint32_t fw[4] = {fl.x, fl.y, fl.z, fl.w};
  int cnt = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) cnt += __popc(fw[q]);  // one bit per flag byte (0 or 1)
  // exclusive scan of the threads' counts
  __shared__ int ws[kLruThreads / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = cnt;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int a = __shfl_up_sync(0xffffffffu, x, d);
    if (lane >= d) x += a;
  }
  if (lane == 31) ws[w] = x;
  __syncthreads();
  int before = x - cnt;
  for (int v = 0; v < w; ++v) before += ws[v];
  int64_t rank = tile_off[k] - tile_off[tile0[t]] + before;
  const int64_t ex = row(plan, nt, kExcess)[t];
  const int64_t j0 = (k - tile0[t]) * kLruTile + (int64_t)threadIdx.x * kLruPer;
  const int64_t dst = row(plan, nt, kRingOff)[t];
  const int bit = t;  // tier t's mask bit (N = the global tier)
  for (int e = 0; e < kLruPer; ++e) {
    if (!((fw[e >> 2] >> (8 * (e & 3))) & 1u)) continue;
    uint64_t key;
    survives(plan, nt, t, j0 + e, ring, touches, set, key);
    if (rank < ex)
      remove_tier(tags, table, ew, W, n_buckets, key, bit >> 6, 1ull << (bit & 63));
    else
      next[dst + rank - ex] = key;
    ++rank;
  }
}

__global__ void k_lru_finish(int64_t* __restrict__ plan, int nt, uint64_t* __restrict__ set) {
  const int64_t used = row(plan, nt, kSetOff)[nt];
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < used;
       i += (int64_t)gridDim.x * blockDim.x)
    reinterpret_cast<ulonglong2*>(set)[i] = make_ulonglong2(0ull, 0ull);
  if (blockIdx.x == 0)
    for (int t = threadIdx.x; t < nt; t += blockDim.x) row(plan, nt, kLen)[t] = row(plan, nt, kNewLen)[t];
}

}  // namespace

namespace smetric {

void lru_free(smetric_index* idx) {
  LruState* L = idx->lru;
  if (!L) return;
  cudaFree(L->ring[0]);
  cudaFree(L->ring[1]);
  cudaFree(L->plan);
  cudaFree(L->req_off);
  cudaFree(L->touches);
  cudaFree(L->set);
  cudaFree(L->keep);
  cudaFree(L->tile_cnt);
  cudaFree(L->tile_off);
  delete L;
  idx->lru = nullptr;
}

int lru_reset(smetric_index* idx, cudaStream_t s) {
  LruState* L = idx->lru;
  if (!L) return SMETRIC_OK;
  return cuda_status(
      cudaMemsetAsync(L->plan + (int64_t)kLen * (L->n_tiers + 1), 0, (L->n_tiers + 1) * sizeof(int64_t), s));
}

int lru_commit(smetric_index* idx, const int32_t* d_instance, const uint64_t* d_hashes, int32_t n, bool global,
               cudaStream_t s) {
  LruState* L = idx->lru;
  if (!L) return SMETRIC_OK;
  const int N = idx->cfg.num_instances, nt = L->n_tiers;
  const bool local_capped = L->local_cap > 0, global_touch = global && L->global_cap > 0;
  const int64_t R = idx->cfg.max_batch_requests;
  const int64_t max_blocks = idx->cfg.max_batch_tokens / idx->cfg.block_size;
  k_lru_plan<<<1, 32, (size_t)N * sizeof(int64_t), s>>>(idx->block_off, n, d_instance, idx->batch_ok, N,
                                                        local_capped, global_touch, L->plan, L->req_off, R);
  const int64_t want = (max_blocks + 255) / 256;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * 8));
  k_lru_touch<<<grid, 256, 0, s>>>(idx->block_off, n, d_instance, d_hashes, idx->batch_ok, N, local_capped,
                                   global_touch, L->plan, L->req_off, R, L->touches, L->set);
  const uint64_t* ring = L->ring[L->cur];
  uint64_t* next = L->ring[L->cur ^ 1];
  k_lru_flags<<<(unsigned)L->max_tiles, kLruThreads, 0, s>>>(L->plan, nt, ring, L->touches, L->set, L->keep,
                                                              L->tile_cnt);
  k_lru_scan<<<1, 1024, 0, s>>>(L->plan, nt, L->tile_cnt, L->tile_off);
  k_lru_write<<<(unsigned)L->max_tiles, kLruThreads, 0, s>>>(L->plan, nt, ring, next, L->touches, L->set,
                                                              L->keep, L->tile_off, idx->tags, idx->table, idx->EW,
                                                              idx->W, idx->n_buckets);
  const int64_t fwant = (L->set_entries + 255) / 256;
  k_lru_finish<<<(unsigned)std::max<int64_t>(1, std::min<int64_t>(fwant, (int64_t)idx->num_sms * 4)), 256, 0, s>>>(
      L->plan, nt, L->set);
  idx->launches += 6;
  L->cur ^= 1;
  return cuda_status(cudaGetLastError());
}

}  // namespace smetric

extern "C" {

int smetric_index_set_lru(smetric_index* idx, int64_t local_cap, int64_t global_cap) {
  CallRange range("smetric_index_set_lru");
  int rc = check_device(idx);
  if (rc) return rc;
  if (local_cap < 0 || global_cap < 0 || local_cap > kMaxCap || global_cap > kMaxCap) return SMETRIC_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return cuda_status(cudaErrorUnknown);
  lru_free(idx);
  if (local_cap == 0 && global_cap == 0) return SMETRIC_OK;
  const int N = idx->cfg.num_instances, nt = N + 1;
  const int64_t R = idx->cfg.max_batch_requests;
  const int64_t max_blocks = idx->cfg.max_batch_tokens / idx->cfg.block_size;
  LruState* L = new (std::nothrow) LruState();
  if (!L) return SMETRIC_ERR_OOM;
  L->local_cap = local_cap;
  L->global_cap = global_cap;
  L->n_tiers = nt;
  // host copies of the static plan rows
  int64_t* h = new (std::nothrow) int64_t[(size_t)kLruPlanFields * (nt + 1)]();
  if (!h) {
    delete L;
    return SMETRIC_ERR_OOM;
  }
  int64_t ring_total = 0;
  for (int t = 0; t < nt; ++t) {
    const int64_t cap = t < N ? local_cap : global_cap;
    h[(int64_t)kRingOff * (nt + 1) + t] = ring_total;
    h[(int64_t)kCap * (nt + 1) + t] = cap;
    ring_total += cap;
  }
  // tiles: each tier's records (<= cap) and touches, rounded up to whole tiles
  L->max_tiles = (ring_total + 2 * max_blocks) / kLruTile + nt + 1;
  L->set_entries = 8 * max_blocks + 2;
  idx->lru = L;
  const bool ok =
      cudaMalloc(&L->ring[0], std::max<int64_t>(ring_total, 1) * sizeof(uint64_t)) == cudaSuccess &&
      cudaMalloc(&L->ring[1], std::max<int64_t>(ring_total, 1) * sizeof(uint64_t)) == cudaSuccess &&
      cudaMalloc(&L->plan, (size_t)kLruPlanFields * (nt + 1) * sizeof(int64_t)) == cudaSuccess &&
      cudaMalloc(&L->req_off, std::max<int64_t>(2 * R, 1) * sizeof(int64_t)) == cudaSuccess &&
      cudaMalloc(&L->touches, std::max<int64_t>(2 * max_blocks, 1) * sizeof(uint64_t)) == cudaSuccess &&
      cudaMalloc(&L->set, L->set_entries * 2 * sizeof(uint64_t)) == cudaSuccess &&
      cudaMalloc(&L->keep, L->max_tiles * kLruTile) == cudaSuccess &&
      cudaMalloc(&L->tile_cnt, (L->max_tiles + 1) * sizeof(int64_t)) == cudaSuccess &&
      cudaMalloc(&L->tile_off, (L->max_tiles + 1) * sizeof(int64_t)) == cudaSuccess &&
      cudaMemcpy(L->plan, h, (size_t)kLruPlanFields * (nt + 1) * sizeof(int64_t), cudaMemcpyHostToDevice) ==
          cudaSuccess &&
      cudaMemset(L->set, 0, L->set_entries * 2 * sizeof(uint64_t)) == cudaSuccess;
  delete[] h;
  if (!ok) {
    (void)cudaGetLastError();
    lru_free(idx);
    return SMETRIC_ERR_OOM;
  }
  return SMETRIC_OK;
}

int smetric_index_lru_sizes(smetric_index* idx, int64_t* d_sizes, smetric_stream_t stream) {
  CallRange range("smetric_index_lru_sizes");
  int rc = check_device(idx);
  if (rc) return rc;
  if (!d_sizes) return SMETRIC_ERR_INVALID_ARG;
  const int nt = idx->cfg.num_instances + 1;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (!idx->lru) return cuda_status(cudaMemsetAsync(d_sizes, 0, nt * sizeof(int64_t), s));
  return cuda_status(cudaMemcpyAsync(d_sizes, idx->lru->plan + (int64_t)kLen * (nt + 1), nt * sizeof(int64_t),
                                     cudaMemcpyDeviceToDevice, s));
}

}  // extern "C"
