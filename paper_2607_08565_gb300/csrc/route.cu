// Batched routing: block chain hash, session key, two-tier longest-prefix
// match, integer cost and argmin (Figure 6 and Figure 10 of the paper, with
// every request of the batch routed against one snapshot of index and load).
//
// Three kernels per batch, in stream order:
//   k_prep    one CTA: validates offsets and loads, exclusive-scans the
//             per-request full-block counts into block_off.
//   k_digest  HBM-bound: one warp per 32 consecutive blocks of the flattened
//             batch. The warp stages the tokens of its 32 blocks into shared
//             memory with coalesced 8-byte cp.async copies (evict-first in
//             L2), laid out with one pad word per row so that lane j reading
//             word k of block j hits a distinct bank; then lane j folds its
//             block's B/2 words into the digest d_b. Two stages per warp let
//             the next chunk's copy overlap this chunk's arithmetic.
//   k_walk    one thread per request: the serial chain h_b over the digests,
//             home-slot probes issued eight blocks at a time, the running
//             AND of local-tier masks and the global-tier run, then the cost
//             of every instance and the lowest-id argmin.

#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "smetric_impl.cuh"

using namespace smetric;

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kChunk = 32;        // blocks per digest task (one per lane)
constexpr int kDigestWarps = 8;   // most warps per digest CTA (fewer for large B)
constexpr size_t kDigestSmem = 200 * 1024;  // shared-memory budget of one digest CTA
constexpr int kStages = 2;        // shared-memory stages per warp
constexpr int kSpanBlocks = 36;   // staged span: 32 blocks + room for request tails
constexpr int kWalkThreads = 64;  // requests per walk CTA
constexpr int kGroup = 8;         // probes issued together per request

// ---------------------------------------------------------------------------
// prep
// ---------------------------------------------------------------------------

__device__ __forceinline__ int64_t warp_incl_scan(int64_t v, int lane) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    int64_t t = __shfl_up_sync(kFull, v, d);
    if (lane >= d) v += t;
  }
  return v;
}

__global__ void __launch_bounds__(1024) k_prep(const int64_t* __restrict__ off, int32_t n,
                                              int64_t n_tokens, int B, const int64_t* __restrict__ load,
                                              int n_load, int64_t* __restrict__ block_off,
                                              int32_t* batch_ok, int32_t* status) {
  __shared__ int64_t warp_tot[32];
  __shared__ int bad_all;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) bad_all = 0;
  int bad = 0;  // bit 0: invalid offsets, bit 1: out-of-range length or load
  for (int i = tid; i < n_load; i += blockDim.x) {
    const int64_t v = load[i];
    if (v < 0 || v > SMETRIC_MAX_LOAD) bad |= 2;
  }
  const int per = (n + (int)blockDim.x - 1) / (int)blockDim.x;
  const int r0 = min(n, tid * per), r1 = min(n, r0 + per);
  int64_t sum = 0;
  for (int r = r0; r < r1; ++r) {
    const int64_t a = off[r], b = off[r + 1];
    if (a < 0 || b < a || b > n_tokens) { bad |= 1; continue; }
    if (b - a > (int64_t)INT32_MAX) { bad |= 2; continue; }
    sum += (b - a) / B;
  }
  int64_t incl = warp_incl_scan(sum, lane);
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (bad) atomicOr(&bad_all, bad);
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    int64_t t = lane < nw ? warp_tot[lane] : 0;
    int64_t ti = warp_incl_scan(t, lane);
    if (lane < nw) warp_tot[lane] = ti - t;  // exclusive
  }
  __syncthreads();
  int64_t run = warp_tot[warp] + incl - sum;
  for (int r = r0; r < r1; ++r) {
    block_off[r] = run;
    const int64_t a = off[r], b = off[r + 1];
    if (a >= 0 && b >= a && b - a <= (int64_t)INT32_MAX) run += (b - a) / B;
  }
  if (tid == (int)blockDim.x - 1) block_off[n] = warp_tot[warp] + incl;
  __syncthreads();
  if (tid == 0) {
    const int ba = bad_all;
    *batch_ok = ba == 0;
    if (ba & 1) latch_error(status, SMETRIC_ERR_INVALID_ARG);
    else if (ba & 2) latch_error(status, SMETRIC_ERR_OVERFLOW);
  }
}

// ---------------------------------------------------------------------------
// digest
// ---------------------------------------------------------------------------

// Largest r in [0, n) with block_off[r] <= f, given block_off[0] <= f < block_off[n].
__device__ __forceinline__ int32_t find_request(const int64_t* __restrict__ block_off, int32_t n,
                                                int64_t f) {
  int32_t lo = 0, hi = n;
  while (hi - lo > 1) {
    const int32_t mid = (lo + hi) >> 1;
    if (__ldg(block_off + mid) <= f) lo = mid; else hi = mid;
  }
  return lo;
}

struct Chunk {
  int64_t tok0;  // first token of this lane's block
  int64_t u_lo;  // first staged 64-bit word (warp-uniform)
  int32_t nq;    // staged words (warp-uniform)
  bool valid;    // this lane has a block
  bool fast;     // the chunk is staged through shared memory (warp-uniform)
};

__device__ __forceinline__ void locate(Chunk& ch, int64_t c, int64_t total,
                                       const int64_t* __restrict__ off,
                                       const int64_t* __restrict__ block_off, int32_t n, int B,
                                       int lane, int q_max) {
  const int64_t f = c * kChunk + lane;
  ch.valid = f < total;
  int64_t t0 = 0;
  if (ch.valid) {
    const int32_t r = find_request(block_off, n, f);
    t0 = __ldg(off + r) + (f - __ldg(block_off + r)) * B;
  }
  ch.tok0 = t0;
  const unsigned vm = __ballot_sync(kFull, ch.valid);
  const int last = 31 - __clz(vm);
  const int64_t lo = __shfl_sync(kFull, t0, 0);
  const int64_t hi = __shfl_sync(kFull, t0, last) + B;  // end of the last block
  ch.u_lo = lo >> 1;
  const int64_t u_hi = (hi + 1) >> 1;  // one extra word when blocks start on odd tokens
  const int64_t nq = u_hi - ch.u_lo;
  ch.fast = nq <= q_max;
  ch.nq = ch.fast ? (int32_t)nq : 0;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void stage_copy(const Chunk& ch, const int32_t* __restrict__ tokens,
                                           int64_t n_tokens, uint64_t* stage, int rowshift,
                                           int lane, uint64_t policy) {
  const uint32_t base = smem_u32(stage);
  for (int q = lane; q < ch.nq; q += 32) {
    const int64_t t = 2 * (ch.u_lo + q);  // first token of this word
    const uint32_t dst = base + 8u * (uint32_t)(q + (q >> rowshift));
    const int32_t* src = tokens + t;
    if (t + 1 < n_tokens) {
      asm volatile("cp.async.ca.shared.global.L2::cache_hint [%0], [%1], 8, %2;\n" ::"r"(dst),
                   "l"(src), "l"(policy));
    } else if (t < n_tokens) {
      asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(dst), "l"(src));
    }
  }
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

// Digest of one block from the staged words. HB = B/2 when known at compile
// time (0: runtime hb).
template <int HB>
__device__ __forceinline__ uint64_t digest_staged(const uint64_t* stage, int q0, bool odd, int hb,
                                                  int rowshift, uint64_t d) {
  const int n = HB > 0 ? HB : hb;
  if (!odd) {
#pragma unroll 8
    for (int k = 0; k < n; ++k) {
      const int q = q0 + k;
      d = mix64(d ^ stage[q + (q >> rowshift)]);
    }
  } else {
    uint64_t x = stage[q0 + (q0 >> rowshift)];
#pragma unroll 8
    for (int k = 0; k < n; ++k) {
      const int q = q0 + k + 1;
      const uint64_t y = stage[q + (q >> rowshift)];
      d = mix64(d ^ ((x >> 32) | (y << 32)));
      x = y;
    }
  }
  return d;
}

__device__ __forceinline__ uint64_t digest_global(const int32_t* __restrict__ tokens, int64_t t0,
                                                  int hb, uint64_t d) {
  for (int k = 0; k < hb; ++k) {
    const uint64_t lo = (uint32_t)__ldg(tokens + t0 + 2 * k);
    const uint64_t hi = (uint32_t)__ldg(tokens + t0 + 2 * k + 1);
    d = mix64(d ^ (lo | (hi << 32)));
  }
  return d;
}

template <int HB>
__global__ void __launch_bounds__(kDigestWarps * 32)
    k_digest(const int32_t* __restrict__ tokens, int64_t n_tokens, const int64_t* __restrict__ off,
             const int64_t* __restrict__ block_off, int32_t n, int B, uint64_t d_init,
             int rowshift, int q_max, int stage_words, const int32_t* __restrict__ batch_ok,
             uint64_t* __restrict__ digest) {
  extern __shared__ uint64_t dsm[];
  if (!*batch_ok) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, warps = blockDim.x >> 5;
  const int64_t total = block_off[n];
  const int64_t n_chunks = (total + kChunk - 1) / kChunk;
  const int64_t tw = (int64_t)gridDim.x * warps;
  int64_t c = (int64_t)blockIdx.x * warps + warp;
  if (c >= n_chunks) return;
  uint64_t* const stages = dsm + (size_t)warp * kStages * stage_words;  // this warp's stages
  uint64_t policy;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(policy));
  const int hb = B >> 1;

  Chunk cur, nxt;
  locate(cur, c, total, off, block_off, n, B, lane, q_max);
  stage_copy(cur, tokens, n_tokens, stages, rowshift, lane, policy);
  cp_async_commit();
  for (int it = 0; c < n_chunks; ++it, c += tw) {
    const int64_t cn = c + tw;
    if (cn < n_chunks) {
      locate(nxt, cn, total, off, block_off, n, B, lane, q_max);
      stage_copy(nxt, tokens, n_tokens, stages + ((it + 1) & 1) * stage_words, rowshift, lane, policy);
    }
    cp_async_commit();
    cp_async_wait<1>();
    __syncwarp();
    if (cur.valid) {
      uint64_t d;
      if (cur.fast) {
        const int64_t rel = cur.tok0 - 2 * cur.u_lo;
        d = digest_staged<HB>(stages + (it & 1) * stage_words, (int)(rel >> 1), (rel & 1) != 0, hb,
                                 rowshift, d_init);
      } else {
        d = digest_global(tokens, cur.tok0, hb, d_init);
      }
      digest[c * kChunk + lane] = d;
    }
    __syncwarp();
    cur = nxt;
  }
  cp_async_wait<0>();
}

// ---------------------------------------------------------------------------
// walk
// ---------------------------------------------------------------------------

// Tier masks of key h whose home slot s holds (k0, m0) in its first 16 bytes.
template <int W>
__device__ __forceinline__ void resolve(const uint64_t* __restrict__ table, uint64_t cap, uint64_t h,
                                        uint64_t s, uint64_t k0, uint64_t m0, uint64_t (&M)[W]) {
  constexpr int EW = entry_words(W);
  const uint64_t max_probe = cap < SMETRIC_MAX_PROBE ? cap : SMETRIC_MAX_PROBE;
  uint64_t k = k0, t = 0;
  const uint64_t* e = table + s * EW;
  while (true) {
    if (k == h) {
      M[0] = t == 0 ? m0 : __ldg(e + 1);
#pragma unroll
      for (int w = 1; w < W; ++w) M[w] = __ldg(e + 1 + w);
      return;
    }
    if (k == kEmpty || ++t >= max_probe) break;
    if (++s == cap) s = 0;
    e = table + s * EW;
    k = __ldg(e);
  }
#pragma unroll
  for (int w = 0; w < W; ++w) M[w] = 0;
}

template <int W, bool PROBE>
__global__ void __launch_bounds__(kWalkThreads)
    k_walk(const uint64_t* __restrict__ table, uint64_t cap, int N, int B, int S, uint64_t h_init,
           const int64_t* __restrict__ off, const int64_t* __restrict__ block_off, int32_t n,
           const int64_t* __restrict__ load, int64_t w_load, int64_t w_miss, int64_t w_glob,
           const uint64_t* __restrict__ digest, const int32_t* __restrict__ batch_ok,
           int32_t* __restrict__ inst_out, int32_t* __restrict__ lhit_out,
           int32_t* __restrict__ ghit_out, uint64_t* __restrict__ sk_out,
           uint64_t* __restrict__ hash_out) {
  constexpr int EW = entry_words(W);
  extern __shared__ int64_t wsm[];
  int64_t* load_s = wsm;                                    // [N]
  int32_t* death = reinterpret_cast<int32_t*>(wsm + N);     // [N][kWalkThreads]
  const int tid = threadIdx.x;
  if (PROBE)
    for (int i = tid; i < N; i += blockDim.x) load_s[i] = load[i];
  __syncthreads();
  const int32_t r = blockIdx.x * kWalkThreads + tid;
  if (r >= n) return;
  if (!*batch_ok) {
    if (PROBE) { inst_out[r] = -1; lhit_out[r] = 0; ghit_out[r] = 0; }
    sk_out[r] = 0;
    return;
  }
  const int64_t L = off[r + 1] - off[r];
  const int64_t nb = L / B;
  const int64_t bo = block_off[r];
  const int64_t kS = (nb < S ? nb : S) - 1;

  uint64_t alive[W];  // local tiers still holding every block so far
#pragma unroll
  for (int w = 0; w < W; ++w) {
    const int lo = w * 64;
    alive[w] = N >= lo + 64 ? ~0ull : (N > lo ? (1ull << (N - lo)) - 1 : 0ull);
  }
  int64_t g = 0;
  bool galive = PROBE;
  bool walking = PROBE && nb > 0;
  uint64_t h = h_init, sk = 0;
  const int gword = N >> 6;                  // mask word holding the global-tier bit
  const uint64_t gbit = 1ull << (N & 63);

  for (int64_t b0 = 0; b0 < nb; b0 += kGroup) {
    const int cnt = (int)min((int64_t)kGroup, nb - b0);
    uint64_t hs[kGroup];
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      if (j < cnt) {
        h = mix64((h + kGamma) ^ __ldg(digest + bo + b0 + j));
        if (h < 2) h |= 2;
        hs[j] = h;
        if (hash_out) hash_out[bo + b0 + j] = h;
        if (b0 + j == kS) sk = h;
      }
    }
    if (PROBE && walking) {
      uint64_t slot[kGroup], k0[kGroup], m0[kGroup];
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        if (j < cnt) {
          slot[j] = home_slot(hs[j], cap);
          const ulonglong2 v = __ldg(reinterpret_cast<const ulonglong2*>(table + slot[j] * EW));
          k0[j] = v.x;
          m0[j] = v.y;
        }
      }
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        if (j < cnt && walking) {
          uint64_t M[W];
          resolve<W>(table, cap, hs[j], slot[j], k0[j], m0[j], M);
          const int32_t b = (int32_t)(b0 + j);
          bool any = false;
#pragma unroll
          for (int w = 0; w < W; ++w) {
            uint64_t dead = alive[w] & ~M[w];
            while (dead) {
              const int i = w * 64 + __ffsll((long long)dead) - 1;
              death[i * kWalkThreads + tid] = b;
              dead &= dead - 1;
            }
            alive[w] &= M[w];
            any |= alive[w] != 0;
          }
          if (galive) {
            uint64_t mg = 0;
#pragma unroll
            for (int w = 0; w < W; ++w) if (w == gword) mg = M[w];
            if (mg & gbit) g = b + 1;
            else galive = false;
          }
          walking = any || galive;
        }
      }
    }
    if (!walking && !hash_out && b0 + cnt > kS) break;
  }
  sk_out[r] = nb > 0 ? sk : 0;
  if (!PROBE) return;

  int32_t best = 0;
  int64_t best_cost = INT64_MAX, best_c = 0;
#pragma unroll
  for (int w = 0; w < W; ++w) {
    const uint64_t aw = alive[w];
    const int iend = N < 64 * (w + 1) ? N : 64 * (w + 1);
    for (int i = 64 * w; i < iend; ++i) {
      const int64_t ci = ((aw >> (i - 64 * w)) & 1) ? nb : (int64_t)death[i * kWalkThreads + tid];
      const int64_t gi = ci > g ? ci : g;
      const int64_t cost = w_load * load_s[i] + w_miss * (L - B * gi) + w_glob * B * (gi - ci);
      if (cost < best_cost) { best_cost = cost; best = i; best_c = ci; }
    }
  }
  const int64_t gb = best_c > g ? best_c : g;
  inst_out[r] = best;
  lhit_out[r] = (int32_t)(B * best_c);
  ghit_out[r] = (int32_t)(B * (gb - best_c));
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

int log2_floor(int x) { int s = 0; while ((1 << (s + 1)) <= x) ++s; return s; }

struct DigestPlan {
  int rowshift, q_max, stage_words, warps;
  size_t smem;
};

DigestPlan digest_plan(int B) {
  DigestPlan p;
  const int hb = B / 2;
  const bool pow2 = (hb & (hb - 1)) == 0;
  p.rowshift = (pow2 && hb >= 4) ? log2_floor(hb) : 4;
  p.q_max = kSpanBlocks * hb + 2;
  p.stage_words = p.q_max + (p.q_max >> p.rowshift) + 2;
  const size_t per_warp = (size_t)kStages * p.stage_words * sizeof(uint64_t);
  p.warps = (int)std::max<size_t>(1, std::min<size_t>(kDigestWarps, kDigestSmem / per_warp));
  p.smem = (size_t)p.warps * per_warp;
  return p;
}

template <int HB>
int launch_digest(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                  const int64_t* d_offsets, int32_t n, cudaStream_t s) {
  const int B = idx->cfg.block_size;
  const DigestPlan p = digest_plan(B);
  auto kern = k_digest<HB>;
  if (idx->digest_occ == 0) {  // once per index: B, and so the plan, is fixed
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem) != cudaSuccess)
      return cuda_status(cudaErrorInvalidValue);
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, p.warps * 32, p.smem) != cudaSuccess)
      return cuda_status(cudaErrorInvalidValue);
    idx->digest_occ = occ < 1 ? 1 : occ;
  }
  const int occ = idx->digest_occ;
  const int64_t max_chunks = (n_tokens / B + kChunk - 1) / kChunk;
  const int64_t want = (max_chunks + p.warps - 1) / p.warps;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * occ));
  const uint64_t d_init = mix64(idx->cfg.hash_seed ^ (uint64_t)B);
  kern<<<(unsigned)grid, p.warps * 32, p.smem, s>>>(d_tokens, n_tokens, d_offsets, idx->block_off, n, B,
                                                          d_init, p.rowshift, p.q_max, p.stage_words,
                                                          idx->batch_ok, idx->digest);
  idx->launches++;
  return cuda_status(cudaGetLastError());
}

template <int W, bool PROBE>
int launch_walk(smetric_index* idx, const int64_t* d_offsets, int32_t n, const int64_t* d_load,
                smetric_weights w, int32_t* inst, int32_t* lhit, int32_t* ghit, uint64_t* sk,
                uint64_t* hashes, cudaStream_t s) {
  const int N = idx->cfg.num_instances;
  const size_t smem = PROBE ? (size_t)N * sizeof(int64_t) + (size_t)N * kWalkThreads * sizeof(int32_t) : 0;
  auto kern = k_walk<W, PROBE>;
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return cuda_status(cudaErrorInvalidValue);
  const unsigned grid = (unsigned)((n + kWalkThreads - 1) / kWalkThreads);
  const uint64_t h_init = mix64(idx->cfg.hash_seed + kGamma);
  kern<<<grid, kWalkThreads, smem, s>>>(idx->table, idx->cfg.capacity_slots, N, idx->cfg.block_size,
                                        idx->cfg.session_blocks, h_init, d_offsets, idx->block_off, n,
                                        d_load, w.w_load, w.w_miss, w.w_glob, idx->digest, idx->batch_ok,
                                        inst, lhit, ghit, sk, hashes);
  idx->launches++;
  return cuda_status(cudaGetLastError());
}

template <bool PROBE>
int dispatch_walk(smetric_index* idx, const int64_t* d_offsets, int32_t n, const int64_t* d_load,
                  smetric_weights w, int32_t* inst, int32_t* lhit, int32_t* ghit, uint64_t* sk,
                  uint64_t* hashes, cudaStream_t s) {
  if (!PROBE) return launch_walk<1, false>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s);
  switch (idx->W) {
    case 1: return launch_walk<1, PROBE>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s);
    case 2: return launch_walk<2, PROBE>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s);
    case 3: return launch_walk<3, PROBE>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s);
    case 4: return launch_walk<4, PROBE>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s);
    case 5: return launch_walk<5, PROBE>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s);
    default: return SMETRIC_ERR_INVALID_ARG;
  }
}

int dispatch_digest(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                    const int64_t* d_offsets, int32_t n, cudaStream_t s) {
  switch (idx->cfg.block_size) {
    case 16: return launch_digest<8>(idx, d_tokens, n_tokens, d_offsets, n, s);
    case 32: return launch_digest<16>(idx, d_tokens, n_tokens, d_offsets, n, s);
    case 64: return launch_digest<32>(idx, d_tokens, n_tokens, d_offsets, n, s);
    default: return launch_digest<0>(idx, d_tokens, n_tokens, d_offsets, n, s);
  }
}

ProfileSlot* profile_begin(smetric_index* idx, cudaStream_t s) {
  if (!idx->profiling) return nullptr;
  ProfileSlot slot;
  if (!idx->prof_pool.empty()) {
    slot = idx->prof_pool.back();
    idx->prof_pool.pop_back();
  } else {
    for (auto& e : slot.ev)
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  }
  idx->prof_used.push_back(slot);
  cudaEventRecord(idx->prof_used.back().ev[0], s);
  return &idx->prof_used.back();
}

void profile_mark(smetric_index* idx, int k, cudaStream_t s) {
  if (idx->profiling && !idx->prof_used.empty()) cudaEventRecord(idx->prof_used.back().ev[k + 1], s);
}

bool weights_ok(const smetric_weights& w) {
  auto in = [](int64_t v) { return v >= 0 && v <= SMETRIC_MAX_WEIGHT; };
  return in(w.w_load) && in(w.w_miss) && in(w.w_glob);
}

template <bool PROBE>
int route_common(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens, const int64_t* d_offsets,
                 int32_t n, const int64_t* d_load, smetric_weights w, int32_t* inst, int32_t* lhit,
                 int32_t* ghit, uint64_t* sk, uint64_t* hashes, int64_t hashes_cap, cudaStream_t s) {
  int rc = check_device(idx);
  if (rc) return rc;
  const smetric_index_config& c = idx->cfg;
  if (n < 0 || n > c.max_batch_requests || n_tokens < 0 || n_tokens > c.max_batch_tokens)
    return SMETRIC_ERR_INVALID_ARG;
  if (n == 0) return SMETRIC_OK;
  if (!d_offsets || !sk || (n_tokens > 0 && !d_tokens)) return SMETRIC_ERR_INVALID_ARG;
  if (d_tokens && (reinterpret_cast<uintptr_t>(d_tokens) & 15)) return SMETRIC_ERR_INVALID_ARG;
  if (PROBE && (!d_load || !inst || !lhit || !ghit || !weights_ok(w))) return SMETRIC_ERR_INVALID_ARG;
  if (hashes && hashes_cap < n_tokens / c.block_size) return SMETRIC_ERR_INVALID_ARG;
  if (!PROBE && !hashes) return SMETRIC_ERR_INVALID_ARG;

  profile_begin(idx, s);
  k_prep<<<1, 1024, 0, s>>>(d_offsets, n, n_tokens, c.block_size, d_load, PROBE ? c.num_instances : 0,
                            idx->block_off, idx->batch_ok, idx->status);
  idx->launches++;
  if ((rc = cuda_status(cudaGetLastError()))) return rc;
  profile_mark(idx, kPrep, s);
  if (n_tokens / c.block_size > 0) {
    if ((rc = dispatch_digest(idx, d_tokens, n_tokens, d_offsets, n, s))) return rc;
  }
  profile_mark(idx, kDigest, s);
  if ((rc = dispatch_walk<PROBE>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, sk, hashes, s))) return rc;
  profile_mark(idx, kWalk, s);
  return SMETRIC_OK;
}

}  // namespace

extern "C" {

int smetric_route_batch(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                        const int64_t* d_offsets, int32_t n_requests, const int64_t* d_load,
                        smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                        int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                        int64_t hashes_cap, smetric_stream_t stream) {
  return route_common<true>(idx, d_tokens, n_tokens, d_offsets, n_requests, d_load, w, d_instance,
                            d_local_hit, d_global_hit, d_session_key, d_block_hashes, hashes_cap,
                            reinterpret_cast<cudaStream_t>(stream));
}

int smetric_block_hashes(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                         const int64_t* d_offsets, int32_t n_requests, uint64_t* d_session_key,
                         uint64_t* d_block_hashes, int64_t hashes_cap, smetric_stream_t stream) {
  smetric_weights w{0, 0, 0};
  return route_common<false>(idx, d_tokens, n_tokens, d_offsets, n_requests, nullptr, w, nullptr,
                             nullptr, nullptr, d_session_key, d_block_hashes, hashes_cap,
                             reinterpret_cast<cudaStream_t>(stream));
}

int smetric_route_batch_host(smetric_index* idx, const int32_t* h_tokens, int64_t n_tokens,
                             const int64_t* h_offsets, int32_t n_requests, const int64_t* h_load,
                             smetric_weights w, int32_t* h_instance, int32_t* h_local_hit,
                             int32_t* h_global_hit, uint64_t* h_session_key, smetric_stream_t stream) {
  int rc = check_device(idx);
  if (rc) return rc;
  if (!(idx->cfg.flags & SMETRIC_FLAG_HOST_STAGING)) return SMETRIC_ERR_INVALID_ARG;
  const smetric_index_config& c = idx->cfg;
  if (n_requests < 0 || n_requests > c.max_batch_requests || n_tokens < 0 || n_tokens > c.max_batch_tokens)
    return SMETRIC_ERR_INVALID_ARG;
  if (n_requests == 0) return SMETRIC_OK;
  if (!h_offsets || !h_load || !h_instance || !h_local_hit || !h_global_hit || !h_session_key ||
      (n_tokens > 0 && !h_tokens))
    return SMETRIC_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const size_t R = (size_t)n_requests;
  bool ok = true;
  if (n_tokens > 0)
    ok = ok && cudaMemcpyAsync(idx->st_tokens, h_tokens, (size_t)n_tokens * sizeof(int32_t),
                               cudaMemcpyHostToDevice, s) == cudaSuccess;
  ok = ok && cudaMemcpyAsync(idx->st_offsets, h_offsets, (R + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, s) == cudaSuccess;
  ok = ok && cudaMemcpyAsync(idx->st_load, h_load, (size_t)c.num_instances * sizeof(int64_t),
                             cudaMemcpyHostToDevice, s) == cudaSuccess;
  if (!ok) return cuda_status(cudaErrorUnknown);
  int32_t* o = idx->st_out32;
  rc = smetric_route_batch(idx, idx->st_tokens, n_tokens, idx->st_offsets, n_requests, idx->st_load, w,
                           o, o + R, o + 2 * R, idx->st_sk, nullptr, 0, stream);
  if (rc) return rc;
  ok = cudaMemcpyAsync(h_instance, o, R * sizeof(int32_t), cudaMemcpyDeviceToHost, s) == cudaSuccess &&
       cudaMemcpyAsync(h_local_hit, o + R, R * sizeof(int32_t), cudaMemcpyDeviceToHost, s) == cudaSuccess &&
       cudaMemcpyAsync(h_global_hit, o + 2 * R, R * sizeof(int32_t), cudaMemcpyDeviceToHost, s) == cudaSuccess &&
       cudaMemcpyAsync(h_session_key, idx->st_sk, R * sizeof(uint64_t), cudaMemcpyDeviceToHost, s) == cudaSuccess;
  if (!ok) return cuda_status(cudaErrorUnknown);
  return smetric_status(idx, stream);
}

int smetric_profile_enable(smetric_index* idx, int32_t on) {
  if (!idx) return SMETRIC_ERR_INVALID_ARG;
  idx->profiling = on != 0;
  return SMETRIC_OK;
}

int smetric_profile_read(smetric_index* idx, int32_t max_kernels, double* ms, int64_t* launches) {
  if (!idx || max_kernels < 0 || (max_kernels > 0 && (!ms || !launches))) return SMETRIC_ERR_INVALID_ARG;
  const int k = std::min<int>(max_kernels, kNumRouteKernels);
  for (int i = 0; i < k; ++i) { ms[i] = 0; launches[i] = 0; }
  int rc = SMETRIC_OK;
  for (auto& slot : idx->prof_used) {
    if (cudaEventSynchronize(slot.ev[kNumRouteKernels]) != cudaSuccess) { rc = cuda_status(cudaErrorUnknown); continue; }
    for (int i = 0; i < k; ++i) {
      float t = 0;
      if (cudaEventElapsedTime(&t, slot.ev[i], slot.ev[i + 1]) == cudaSuccess) {
        ms[i] += t;
        launches[i] += 1;
      } else {
        (void)cudaGetLastError();
      }
    }
    idx->prof_pool.push_back(slot);
  }
  idx->prof_used.clear();
  return rc ? rc : kNumRouteKernels;
}

const char* smetric_profile_kernel_name(int32_t k) {
  switch (k) {
    case kPrep: return "k_prep";
    case kDigest: return "k_digest";
    case kWalk: return "k_walk";
    default: return "";
  }
}

}  // extern "C"
