// Two-tier KV$ index on the GPU: one bucketed hash table, key -> tier mask.
//
// The paper's KV$ store has a local tier per serving instance and a global
// tier shared by the cluster (Section 2, Figures 1-2); the router needs, per
// block hash, which tiers hold the block. One table serves all tiers: an
// entry is the 64-bit block hash followed by W = ceil((N+1)/64) mask words,
// bit i < N = local tier of instance i, bit N = global tier. Slots are grouped
// in buckets of kSlots; a one-byte tag per slot (0 = empty, else 0x80 | low
// 7 key bits) and the bucket's overflow count live in a separate 16-byte tag
// group, so that a lookup reads one tag group and then only the entry whose
// tag matches. A key that leaves its last tier gives its slot back (the
// primitives and their concurrency contract are in table.cuh), so a table
// sized for the live keys serves any number of inserted and evicted ones.

#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <new>

#include "smetric_impl.cuh"
#include "table.cuh"
#include "call_range.cuh"

using namespace smetric;

namespace smetric {
// The second route scratch set of SMETRIC_FLAG_PIPELINE (defined beside
// smetric_route_batches, which uses it).
int pipeline_attach(smetric_index* x);
void pipeline_release(smetric_index* x);
}  // namespace smetric

namespace smetric {

int cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return SMETRIC_OK;
  (void)cudaGetLastError();
  return SMETRIC_ERR_CUDA;
}

int check_device(const smetric_index* idx) {
  if (!idx) return SMETRIC_ERR_INVALID_ARG;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return cuda_status(cudaErrorInvalidDevice);
  return dev == idx->device ? SMETRIC_OK : SMETRIC_ERR_INVALID_ARG;
}

}  // namespace smetric

namespace {

enum Op { kInsert = 0, kEvict = 1 };

// One thread per (key, tier) pair, grid-stride.
template <int OP>
__global__ void k_update(uint8_t* __restrict__ tags, uint64_t* __restrict__ table, uint64_t n_buckets,
                         int ew, int W, int N, bool lru_local, bool lru_global, const uint64_t* __restrict__ keys,
                         const int32_t* __restrict__ tiers, int64_t n, int32_t* status) {
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < n;
       j += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t key = keys[j];
    const int32_t tier = tiers[j];
    if (key < 2 || tier < -1 || tier >= N) {
      latch_error(status, SMETRIC_ERR_INVALID_ARG);
      continue;
    }
    const int bit = tier < 0 ? N : tier;
    if ((bit < N && lru_local) || (bit == N && lru_global)) {  // the device LRU owns capped tiers
      latch_error(status, SMETRIC_ERR_INVALID_ARG);
      continue;
    }
    const unsigned long long m = 1ull << (bit & 63);
    if (OP == kInsert) {
      if (!insert_key(tags, table, ew, n_buckets, key, bit >> 6, m))
        latch_error(status, SMETRIC_ERR_TABLE_FULL);
    } else {
      remove_tier(tags, table, ew, W, n_buckets, key, bit >> 6, m);
    }
  }
}

__global__ void k_lookup(const uint8_t* __restrict__ tags, const uint64_t* __restrict__ table,
                         uint64_t n_buckets, int ew, int W, const uint64_t* __restrict__ keys,
                         int64_t n, uint64_t* __restrict__ out) {
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < n;
       j += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t key = keys[j];
    const int64_t slot = key >= 2 ? find_slot<false>(tags, table, ew, n_buckets, key) : -1;
    for (int w = 0; w < W; ++w) out[j * W + w] = slot >= 0 ? table[slot * ew + 1 + w] : 0;
  }
}

// Committing a routed batch: thread per block f of the batch (request r, the
// largest with block_off[r] <= f) adds h_f to the local tier of r's chosen
// instance and, with `global`, to the global tier. A request routed to -1
// (an invalid batch) adds nothing; another out-of-range instance latches
// INVALID_ARG.
__global__ void k_commit(uint8_t* __restrict__ tags, uint64_t* __restrict__ table, uint64_t n_buckets,
                         int ew, int N, const int64_t* __restrict__ block_off, int32_t n,
                         const uint64_t* __restrict__ H, const int32_t* __restrict__ instance, int global,
                         const int32_t* __restrict__ batch_ok, int32_t* status) {
  if (!*batch_ok) return;
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
    if (i == -1) continue;
    const uint64_t key = H[f];
    if (i < -1 || i >= N || key < 2) {
      latch_error(status, SMETRIC_ERR_INVALID_ARG);
      continue;
    }
    if (!insert_key(tags, table, ew, n_buckets, key, i >> 6, 1ull << (i & 63)))
      latch_error(status, SMETRIC_ERR_TABLE_FULL);
    if (global && !insert_key(tags, table, ew, n_buckets, key, N >> 6, 1ull << (N & 63)))
      latch_error(status, SMETRIC_ERR_TABLE_FULL);
  }
}

int grid_for(const smetric_index* idx, int64_t n, int threads) {
  int64_t want = (n + threads - 1) / threads;
  int64_t cap = (int64_t)idx->num_sms * 8;
  return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

int update(smetric_index* idx, const uint64_t* d_keys, const int32_t* d_tiers, int64_t n,
           smetric_stream_t stream, int op) {
  int rc = check_device(idx);
  if (rc) return rc;
  if (n < 0 || (n > 0 && (!d_keys || !d_tiers))) return SMETRIC_ERR_INVALID_ARG;
  if (n == 0) return SMETRIC_OK;
  const int threads = 256;
  int grid = grid_for(idx, n, threads);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const bool ll = idx->lru && idx->lru->local_cap > 0, lg = idx->lru && idx->lru->global_cap > 0;
  if (op == kInsert)
    k_update<kInsert><<<grid, threads, 0, s>>>(idx->tags, idx->table, idx->n_buckets, idx->EW, idx->W,
                                               idx->cfg.num_instances, ll, lg, d_keys, d_tiers, n, idx->status);
  else
    k_update<kEvict><<<grid, threads, 0, s>>>(idx->tags, idx->table, idx->n_buckets, idx->EW, idx->W,
                                              idx->cfg.num_instances, ll, lg, d_keys, d_tiers, n, idx->status);
  idx->launches++;
  return cuda_status(cudaGetLastError());
}

}  // namespace

namespace smetric {

int launch_commit(smetric_index* idx, const int32_t* d_instance, const uint64_t* d_hashes, int32_t n,
                  int64_t max_blocks, bool global, cudaStream_t s) {
  const int threads = 256;
  const int grid = grid_for(idx, max_blocks, threads);
  k_commit<<<grid, threads, 0, s>>>(idx->tags, idx->table, idx->n_buckets, idx->EW, idx->cfg.num_instances,
                                    idx->block_off, n, d_hashes, d_instance, global ? 1 : 0, idx->batch_ok,
                                    idx->status);
  idx->launches++;
  return cuda_status(cudaGetLastError());
}

}  // namespace smetric

namespace {

void free_all(smetric_index* x) {
  pipeline_release(x);
  lru_free(x);
  cudaFree(x->table);
  cudaFree(x->tags);
  cudaFree(x->status);
  cudaFree(x->block_off);
  cudaFree(x->digest);
  cudaFree(x->hashes);
  cudaFree(x->masks);
  cudaFree(x->summ);
  cudaFree(x->chunk_and);
  cudaFree(x->sk_tmp);
  cudaFree(x->groups);
  cudaFree(x->lead);
  cudaFree(x->chunk_off);
  cudaFree(x->batch_ok);
  cudaFree(x->st_tokens);
  cudaFree(x->st_offsets);
  cudaFree(x->st_load);
  cudaFree(x->st_out32);
  cudaFree(x->st_sk);
  for (auto& p : x->prof_pool)
    for (auto& e : p.ev) cudaEventDestroy(e);
  for (auto& p : x->prof_used)
    for (auto& e : p.ev) cudaEventDestroy(e);
}

}  // namespace

extern "C" {

int smetric_index_create(const smetric_index_config* cfg, smetric_index** out) {
  CallRange range("smetric_index_create");
  if (!out) return SMETRIC_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg) return SMETRIC_ERR_INVALID_ARG;
  const smetric_index_config c = *cfg;
  if (c.num_instances < 1 || c.num_instances > SMETRIC_MAX_INSTANCES) return SMETRIC_ERR_INVALID_ARG;
  if (c.block_size < 2 || c.block_size > 256 || (c.block_size & 1)) return SMETRIC_ERR_INVALID_ARG;
  if (c.session_blocks < 1 || c.capacity_slots < 1) return SMETRIC_ERR_INVALID_ARG;
  if (c.max_batch_requests < 0 || c.max_batch_requests > INT32_MAX - 1) return SMETRIC_ERR_INVALID_ARG;
  if (c.max_batch_tokens < 0) return SMETRIC_ERR_INVALID_ARG;
  if (c.flags & ~(SMETRIC_FLAG_HOST_STAGING | SMETRIC_FLAG_PIPELINE)) return SMETRIC_ERR_INVALID_ARG;
  const int W = (c.num_instances + 1 + 63) / 64;
  // slots (rounded up to whole buckets) * entry bytes must not overflow
  if (c.capacity_slots > (UINT64_MAX / 16) / (uint64_t)entry_words(W)) return SMETRIC_ERR_INVALID_ARG;

  smetric_index* x = new (std::nothrow) smetric_index();
  if (!x) return SMETRIC_ERR_OOM;
  x->cfg = c;
  x->W = W;
  x->EW = entry_words(W);
  x->n_buckets = (c.capacity_slots + kSlots - 1) / kSlots;
  if (cudaGetDevice(&x->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&x->num_sms, cudaDevAttrMultiProcessorCount, x->device) != cudaSuccess) {
    delete x;
    return cuda_status(cudaErrorInvalidDevice);
  }
  const size_t slots = (size_t)x->n_buckets * kSlots;
  const size_t table_bytes = slots * x->EW * sizeof(uint64_t);
  const size_t tag_bytes = (size_t)x->n_buckets * kBucket;
  const size_t max_blocks = (size_t)(c.max_batch_tokens / c.block_size);
  const size_t R = (size_t)c.max_batch_requests;
  x->group_slots = 64;
  while (x->group_slots < 2 * (uint64_t)R) x->group_slots <<= 1;
  bool ok = cudaMalloc(&x->table, table_bytes) == cudaSuccess &&
            cudaMalloc(&x->tags, tag_bytes) == cudaSuccess &&
            cudaMalloc(&x->status, sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&x->block_off, (R + 1) * sizeof(int64_t)) == cudaSuccess &&
            // two spare words: k_chain_probe copies a chunk's digests in whole 16-byte pieces
            cudaMalloc(&x->digest, (max_blocks + 2) * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&x->hashes, (max_blocks > 0 ? max_blocks : 1) * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&x->masks, (max_blocks > 0 ? max_blocks : 1) * W * sizeof(uint64_t)) == cudaSuccess &&
            // one per request-aligned 32-block chunk: at most max_blocks / 32 + R
            cudaMalloc(&x->chunk_and, (max_blocks / 32 + R + 1) * W * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&x->groups, 2 * x->group_slots * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&x->lead, 2 * (R + 1) * sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&x->chunk_off, (R + 1) * sizeof(int64_t)) == cudaSuccess &&
            cudaMalloc(&x->sk_tmp, (R + 1) * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&x->summ, (R > 0 ? R : 1) * ((size_t)c.num_instances + 1) * sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&x->batch_ok, sizeof(int32_t)) == cudaSuccess;
  if (ok) x->share = x->lead + (R + 1);
  if (ok && (c.flags & SMETRIC_FLAG_HOST_STAGING)) {
    const size_t T = (size_t)(c.max_batch_tokens > 0 ? c.max_batch_tokens : 1);
    ok = cudaMalloc(&x->st_tokens, T * sizeof(int32_t)) == cudaSuccess &&
         cudaMalloc(&x->st_offsets, (R + 1) * sizeof(int64_t)) == cudaSuccess &&
         cudaMalloc(&x->st_load, (size_t)c.num_instances * sizeof(int64_t)) == cudaSuccess &&
         cudaMalloc(&x->st_out32, (3 * R + 1) * sizeof(int32_t)) == cudaSuccess &&
         cudaMalloc(&x->st_sk, (R + 1) * sizeof(uint64_t)) == cudaSuccess;
  }
  if (ok && (c.flags & SMETRIC_FLAG_PIPELINE)) ok = pipeline_attach(x) == SMETRIC_OK;
  if (ok) ok = cudaMemset(x->table, 0, table_bytes) == cudaSuccess &&
               cudaMemset(x->tags, 0, tag_bytes) == cudaSuccess &&
               cudaMemset(x->status, 0, sizeof(int32_t)) == cudaSuccess &&
               cudaMemset(x->groups, 0, 2 * x->group_slots * sizeof(uint64_t)) == cudaSuccess &&
               cudaDeviceSynchronize() == cudaSuccess;
  if (!ok) {
    (void)cudaGetLastError();
    free_all(x);
    delete x;
    return SMETRIC_ERR_OOM;
  }
  *out = x;
  return SMETRIC_OK;
}

int smetric_index_destroy(smetric_index* idx) {
  CallRange range("smetric_index_destroy");
  if (!idx) return SMETRIC_OK;
  int dev = -1;
  cudaGetDevice(&dev);
  if (dev != idx->device) cudaSetDevice(idx->device);
  cudaDeviceSynchronize();
  free_all(idx);
  int rc = cuda_status(cudaGetLastError());
  if (dev >= 0 && dev != idx->device) cudaSetDevice(dev);
  delete idx;
  return rc;
}

int smetric_index_clear(smetric_index* idx, smetric_stream_t stream) {
  CallRange range("smetric_index_clear");
  int rc = check_device(idx);
  if (rc) return rc;
  const size_t slots = (size_t)idx->n_buckets * kSlots;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(idx->table, 0, slots * idx->EW * sizeof(uint64_t), s) != cudaSuccess ||
      cudaMemsetAsync(idx->tags, 0, (size_t)idx->n_buckets * kBucket, s) != cudaSuccess)
    return cuda_status(cudaErrorUnknown);
  return lru_reset(idx, s);
}

int smetric_index_insert(smetric_index* idx, const uint64_t* d_keys, const int32_t* d_tiers,
                         int64_t n, smetric_stream_t stream) {
  CallRange range("smetric_index_insert");
  return update(idx, d_keys, d_tiers, n, stream, kInsert);
}

int smetric_index_evict(smetric_index* idx, const uint64_t* d_keys, const int32_t* d_tiers,
                        int64_t n, smetric_stream_t stream) {
  CallRange range("smetric_index_evict");
  return update(idx, d_keys, d_tiers, n, stream, kEvict);
}

int smetric_index_lookup(smetric_index* idx, const uint64_t* d_keys, int64_t n, uint64_t* d_masks,
                         smetric_stream_t stream) {
  CallRange range("smetric_index_lookup");
  int rc = check_device(idx);
  if (rc) return rc;
  if (n < 0 || (n > 0 && (!d_keys || !d_masks))) return SMETRIC_ERR_INVALID_ARG;
  if (n == 0) return SMETRIC_OK;
  const int threads = 256;
  k_lookup<<<grid_for(idx, n, threads), threads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      idx->tags, idx->table, idx->n_buckets, idx->EW, idx->W, d_keys, n, d_masks);
  idx->launches++;
  return cuda_status(cudaGetLastError());
}

int32_t smetric_index_mask_words(const smetric_index* idx) { return idx ? idx->W : 0; }

int smetric_status(smetric_index* idx, smetric_stream_t stream) {
  CallRange range("smetric_status");
  int rc = check_device(idx);
  if (rc) return rc;
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return cuda_status(cudaErrorUnknown);
  int32_t h = 0;
  if (cudaMemcpy(&h, idx->status, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess)
    return cuda_status(cudaErrorUnknown);
  if (h != 0 && cudaMemset(idx->status, 0, sizeof(int32_t)) != cudaSuccess)
    return cuda_status(cudaErrorUnknown);
  return h;
}

const char* smetric_strerror(int code) {
  switch (code) {
    case SMETRIC_OK: return "ok";
    case SMETRIC_ERR_INVALID_ARG: return "invalid argument";
    case SMETRIC_ERR_OOM: return "device allocation failed";
    case SMETRIC_ERR_TABLE_FULL: return "index table full";
    case SMETRIC_ERR_CUDA: return "CUDA runtime error";
    case SMETRIC_ERR_OVERFLOW: return "value outside the exact integer range";
    case SMETRIC_ERR_TOO_LARGE: return "batch larger than the fixed no-allocation scratch";
    default: return "unknown error";
  }
}

int64_t smetric_launch_count(const smetric_index* idx) { return idx ? idx->launches : 0; }

}  // extern "C"
