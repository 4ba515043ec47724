// Batched routing: block chain hash, session key, two-tier longest-prefix
// match, integer cost and argmin (Figure 6 and Figure 10 of the paper, with
// every request of the batch routed against one snapshot of index and load).
//
// Kernels per batch, in stream order:
//   k_prep        one CTA: validates offsets and loads; scans the per-request
//                 full-block counts into block_off and the 32-block chunk
//                 counts into chunk_off.
//   k_digest_tma  HBM-bound block digests d_b: chunk q of request r is its
//                 blocks 32q..32q+31, one 2D TMA tile of 32 overlapping rows
//                 (each block's bytes rounded out to 16-byte boundaries); a
//                 CTA takes a contiguous range of chunks, its warps
//                 interleaved over it; lane j folds block j's B/2 words.
//                 The lane holding a request's first block also inserts the
//                 request's group key (its first-block hash) into the group
//                 table. (k_digest and k_digest_any cover block sizes the
//                 tensor maps do not.)
//   k_lead        one thread per request: whether it leads its group (the
//                 group's lowest request index).
//   k_chain_probe one CTA per SM. Chain warps (one lane per request the CTA
//                 owns) run the serial chain h_b over the digests and write
//                 the session key; beside them, probe warps find each
//                 member's shared prefix with its leader and probe every
//                 block not shared: the tier masks of h_b from the index (16
//                 tags of the home bucket, then the matching entry), and the
//                 AND of each 32-block chunk's masks.
//   k_walk        one warp per request walks the runs of the local tiers and
//                 the global tier (a member over its leader's probes up to
//                 its shared prefix), 32 chunks per step from the chunk ANDs
//                 and block by block where a run ends; then lanes =
//                 instances for the cost and a shuffle argmin with ties to
//                 the lowest id (or one of the policy scores).

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <utility>
#include <atomic>
#include <cstring>

#include "smetric_impl.cuh"

using namespace smetric;

namespace {

constexpr unsigned kFull = 0xffffffffu;

// Programmatic dependent launch: a route kernel launched with programmatic
// stream serialisation is set up while its predecessor still runs and waits
// here until that predecessor has finished and its writes are visible (a
// no-op for an ordinary launch). No kernel triggers its successor early:
// successors waiting on the SMs during a kernel's run measured slower.
__device__ __forceinline__ void pdl_enter() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
constexpr int kChunk = 32;        // blocks per digest task (one per lane)
constexpr int kDigestWarps = 8;   // most warps per digest CTA
constexpr int kTmaWarps = 24;     // warps per TMA digest CTA (two CTAs per SM)
constexpr int kTmaStages = 1;     // copy stages per TMA digest warp
constexpr int kChainThreads = 32;   // one warp per CTA: chains spread over every SM
constexpr int kChainAhead = 16;   // digests prefetched per request
constexpr int kMatchWarps = 8;    // warps per walk CTA
constexpr int kGroupAhead = 8;    // 32-block rounds of hashes a group warp compares at once

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

constexpr int kPrepRounds = 8;  // rounds of 32 consecutive requests per warp per pass

__global__ void __launch_bounds__(1024) k_prep(const int64_t* __restrict__ off, int32_t n,
                                              int64_t n_tokens, int B, const int64_t* __restrict__ load,
                                              int n_load, int64_t* __restrict__ block_off,
                                              int64_t* __restrict__ chunk_off, int32_t* batch_ok,
                                              int32_t* status, int64_t max_load, int64_t max_len,
                                              const int64_t* __restrict__ est_hit,
                                              const int64_t* __restrict__ aux0 = nullptr, int64_t aux0_max = 0,
                                              const int64_t* __restrict__ aux1 = nullptr, int64_t aux1_max = 0) {
  constexpr int NS = 2;  // scans: full blocks, and 32-block chunks (when chunk_off is wanted)
  constexpr int R = kPrepRounds;
  __shared__ int64_t warp_tot[NS][32];
  __shared__ int64_t pass_tot[NS];
  __shared__ int bad_all;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  if (tid == 0) bad_all = 0;
  __syncthreads();
  int bad = 0;  // bit 0: invalid offsets, bit 1: out-of-range length or load
  for (int i = tid; i < n_load; i += blockDim.x) {
    const int64_t v = load[i];
    if (v < 0 || v > max_load) bad |= 2;
    if (aux0 && (aux0[i] < 0 || aux0[i] > aux0_max)) bad |= 2;  // further per-instance inputs
    if (aux1 && (aux1[i] < 0 || aux1[i] > aux1_max)) bad |= 2;
  }
  if (est_hit)  // the policy's expected hits, each in [0, 2^31)
    for (int64_t r = tid; r < n; r += blockDim.x) {
      const int64_t v = est_hit[r];
      if (v < 0 || v > (int64_t)INT32_MAX) bad |= 2;
    }
  // A pass gives each warp R rounds of 32 consecutive requests (lane = request),
  // so that offsets are loaded and both outputs stored coalesced. Every offset
  // of the pass is loaded before any is used; the counts stay in registers
  // between the warp sums and the scans that write the outputs.
  int64_t carry[NS] = {0, 0};
  for (int64_t base = 0; base < n; base += (int64_t)blockDim.x * R) {
    const int64_t seg = base + (int64_t)warp * 32 * R + lane;
    int64_t a[R], b[R];
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int64_t r = seg + 32 * i;
      a[i] = r < n ? off[r] : 0;
      b[i] = r < n ? off[r + 1] : 0;
    }
    uint32_t nbv[R];
#pragma unroll
    for (int i = 0; i < R; ++i) {
      uint32_t v = 0;
      if (seg + 32 * i < n) {
        if (a[i] < 0 || b[i] < a[i] || b[i] > n_tokens) bad |= 1;
        else if (b[i] - a[i] > max_len) bad |= 2;
        else v = (uint32_t)(b[i] - a[i]) / (uint32_t)B;
      }
      nbv[i] = v;
    }
    auto cnt = [&](int k, int i) -> int64_t { return k == 0 ? nbv[i] : (nbv[i] + 31) >> 5; };
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      int64_t t = 0;
#pragma unroll
      for (int i = 0; i < R; ++i) t += cnt(k, i);
#pragma unroll
      for (int d = 16; d > 0; d >>= 1) t += __shfl_xor_sync(kFull, t, d);
      if (lane == 0) warp_tot[k][warp] = t;
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
      for (int k = 0; k < NS; ++k) {
        const int64_t t = lane < nw ? warp_tot[k][lane] : 0;
        const int64_t ti = warp_incl_scan(t, lane);
        if (lane < nw) warp_tot[k][lane] = ti - t;  // exclusive
        if (lane == 31) pass_tot[k] = ti;
      }
    }
    __syncthreads();
    // both scans side by side, so that their shuffle chains overlap; rounds
    // past the last request are skipped (the test is warp-uniform)
    int64_t run[NS];
#pragma unroll
    for (int k = 0; k < NS; ++k) run[k] = carry[k] + warp_tot[k][warp];  // this warp's exclusive start
#pragma unroll
    for (int i = 0; i < R; ++i) {
      if (seg - lane + 32 * i >= n) break;
      const int64_t r = seg + 32 * i;
      const int64_t c0 = cnt(0, i), c1 = cnt(1, i);
      const int64_t i0 = warp_incl_scan(c0, lane), i1 = warp_incl_scan(c1, lane);
      if (r < n) {
        block_off[r] = run[0] + i0 - c0;
        if (chunk_off) chunk_off[r] = run[1] + i1 - c1;
      }
      run[0] += __shfl_sync(kFull, i0, 31);
      run[1] += __shfl_sync(kFull, i1, 31);
    }
#pragma unroll
    for (int k = 0; k < NS; ++k) carry[k] += pass_tot[k];
    __syncthreads();  // warp_tot and pass_tot are rewritten by the next pass
  }
  if (bad) atomicOr(&bad_all, bad);
  __syncthreads();
  if (tid == 0) {
    block_off[n] = carry[0];
    if (chunk_off) chunk_off[n] = carry[1];
    const int ba = bad_all;
    *batch_ok = ba == 0;
    if (ba & 1) latch_error(status, SMETRIC_ERR_INVALID_ARG);
    else if (ba & 2) latch_error(status, SMETRIC_ERR_OVERFLOW);
  }
}

// ---------------------------------------------------------------------------
// digest
// ---------------------------------------------------------------------------

// The group stage works from the digests, so that it needs no finished chain:
// a request's first-block hash h_0 = chain step from h_init over d_0 is the
// group key, and the shared-prefix length is the number of leading blocks
// whose digests equal the leader's. Equal digests from equal previous hashes
// give equal hashes, so the leader's masks serve those blocks exactly.
__device__ __forceinline__ uint64_t first_hash(uint64_t h_init, uint64_t d0) {
  uint64_t h = mix64((h_init + kGamma) ^ d0);
  return h < 2 ? (h | 2) : h;
}

// Requests whose first block hashes are equal form a group; its leader is
// the lowest request id. Table of (key, INT32_MAX - leader) word pairs,
// key 0 = empty (block hashes are >= 2), linear probing, at most half full.
__device__ __forceinline__ void group_insert(uint64_t* __restrict__ groups, uint64_t gmask, uint64_t key,
                                             int32_t r) {
  uint64_t s = key & gmask;
  for (uint64_t t = 0; t <= gmask; ++t) {
    unsigned long long* const slot = reinterpret_cast<unsigned long long*>(groups + 2 * s);
    const unsigned long long k = atomicCAS(slot, 0ull, (unsigned long long)key);
    if (k == 0ull || k == key) {
      atomicMax(slot + 1, (unsigned long long)(INT32_MAX - r));
      return;
    }
    s = (s + 1) & gmask;
  }
}

// Largest r in [lo, n) with block_off[r] <= f, given block_off[lo] <= f < block_off[n].
__device__ __forceinline__ int32_t find_request(const int64_t* __restrict__ block_off, int32_t lo,
                                                int32_t n, int64_t f) {
  int32_t hi = n;
  while (hi - lo > 1) {
    const int32_t mid = (lo + hi) >> 1;
    if (__ldg(block_off + mid) <= f) lo = mid; else hi = mid;
  }
  return lo;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Digest of one block from its shared-memory row. `row` points at the 8-byte
// word holding the block's first token (its low half when the block starts on
// an even token, its high half when on an odd one).
template <int HB>
__device__ __forceinline__ uint64_t digest_row(const uint64_t* row, bool odd, int hb, uint64_t d) {
  const int n = HB > 0 ? HB : hb;
  if (!odd) {
#pragma unroll 16
    for (int k = 0; k < n; ++k) d = mix64(d ^ row[k]);
  } else {
    uint64_t x = row[0];
#pragma unroll 16
    for (int k = 0; k < n; ++k) {
      const uint64_t y = row[k + 1];
      d = mix64(d ^ ((x >> 32) | (y << 32)));
      x = y;
    }
  }
  return d;
}

// 16 bytes of the token buffer at byte offset `a`, of which only the first
// `avail` bytes (a multiple of 4) are read when fewer than 16 remain.
__device__ __forceinline__ uint4 load_piece(const char* base, int64_t a, int64_t avail) {
  if (avail >= 16) return __ldg(reinterpret_cast<const uint4*>(base + a));
  uint32_t w[4] = {0, 0, 0, 0};
#pragma unroll
  for (int q = 0; q < 4; ++q)
    if (4 * q < avail) w[q] = __ldg(reinterpret_cast<const uint32_t*>(base + a) + q);
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Row layout shared by both digest kernels: row j holds the bytes of block j
// rounded out to 16-byte boundaries, [a_j, a_j + 16*NP) with
// a_j = (4*first token) & ~15, so lane j reading word k of its own block hits
// bank group (row stride * j + 8k) mod 128 and rows of 16*NP bytes keep the
// 32 lanes spread over the banks.

// B = 2*HB with B % 4 == 0 (HB even). A chunk whose 32 blocks belong to one
// request is one contiguous byte span; the warp loads it with coalesced
// 16-byte loads (piece p = lane + 32 i) into registers one chunk ahead, and
// scatters each piece into the row(s) that contain it: piece p lies in row
// p / PB and, when it starts a block, also ends row p / PB - 1.
template <int HB>
__global__ void __launch_bounds__(kDigestWarps * 32)
    k_digest(const int32_t* __restrict__ tokens, int64_t n_tokens, const int64_t* __restrict__ off,
             const int64_t* __restrict__ block_off, int32_t n, uint64_t d_init,
             const int32_t* __restrict__ batch_ok, uint64_t* __restrict__ digest,
             uint64_t* __restrict__ groups, uint64_t gmask, uint64_t h_init) {
  pdl_enter();
  constexpr int B = 2 * HB;
  constexpr int PB = HB > 0 ? HB / 2 : 1;  // 16-byte pieces per block (k_digest<0> is never launched)
  constexpr int NP = PB + 1;  // pieces per row (the block plus its misalignment)
  extern __shared__ uint4 dsm[];
  if (!*batch_ok) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, warps = blockDim.x >> 5;
  const int64_t total = block_off[n];
  const int64_t n_chunks = (total + kChunk - 1) / kChunk;
  const int64_t tw = (int64_t)gridDim.x * warps;
  const int64_t per = (n_chunks + tw - 1) / tw;
  const int64_t c_lo = ((int64_t)blockIdx.x * warps + warp) * per;
  const int64_t c_hi = min(n_chunks, c_lo + per);
  if (c_lo >= c_hi) return;
  uint4* const st = dsm + (size_t)warp * kChunk * NP;
  const int64_t token_bytes = 4 * n_tokens;
  const char* const tb = reinterpret_cast<const char*>(tokens);

  int32_t r = find_request(block_off, 0, n, min(c_lo * kChunk + lane, total - 1));

  struct Chunk {
    int64_t tok0;  // this lane's first token
    int64_t a0;    // byte offset of piece 0 (fast path)
    int nv;        // valid lanes (a prefix of the warp)
    int32_t req;   // this lane's request
    bool valid, fast, head;  // head: the lane's block is its request's block 0
  };
  uint4 buf[NP];
  // locate chunk c and load its bytes into registers
  auto load = [&](int64_t c, Chunk& ch) {
    const int64_t f = c * kChunk + lane;
    ch.valid = f < total;
    ch.head = false;
    ch.req = r;
    if (ch.valid) {
      if (__ldg(block_off + r + 1) <= f) r = find_request(block_off, r + 1, n, f);
      ch.tok0 = __ldg(off + r) + (f - __ldg(block_off + r)) * B;
      ch.head = f == __ldg(block_off + r);
      ch.req = r;
    } else {
      ch.tok0 = 0;
    }
    ch.nv = __popc(__ballot_sync(kFull, ch.valid));
    const int32_t r0 = __shfl_sync(kFull, r, 0);
    ch.a0 = (4 * __shfl_sync(kFull, ch.tok0, 0)) & ~(int64_t)15;
    const int npieces = ch.nv * PB + 1;
    ch.fast = __all_sync(kFull, !ch.valid || r == r0) && ch.a0 + 16 * (int64_t)npieces <= token_bytes;
    if (ch.fast) {
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        const int p = lane + 32 * i;
        if (p < npieces) buf[i] = __ldg(reinterpret_cast<const uint4*>(tb + ch.a0) + p);
      }
    } else if (ch.valid) {
      const int64_t a = (4 * ch.tok0) & ~(int64_t)15;
#pragma unroll
      for (int i = 0; i < NP; ++i) buf[i] = load_piece(tb, a + 16 * i, token_bytes - (a + 16 * i));
    }
  };
  auto store = [&](const Chunk& ch) {
    if (ch.fast) {
      const int npieces = ch.nv * PB + 1;
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        const int p = lane + 32 * i;
        if (p < npieces) {
          const int j = p / PB, q = p - j * PB;
          if (j < ch.nv) st[j * NP + q] = buf[i];
          if (q == 0 && j >= 1) st[(j - 1) * NP + PB] = buf[i];
        }
      }
    } else if (ch.valid) {
#pragma unroll
      for (int i = 0; i < NP; ++i) st[lane * NP + i] = buf[i];
    }
  };

  Chunk cur, nxt;
  load(c_lo, cur);
  for (int64_t c = c_lo; c < c_hi; ++c) {
    store(cur);
    __syncwarp();
    if (c + 1 < c_hi) load(c + 1, nxt);  // in flight during this chunk's arithmetic
    if (cur.valid) {
      const int delta = (int)((cur.tok0 * 4) & 15);  // 0, 4, 8 or 12
      const uint64_t* row = reinterpret_cast<const uint64_t*>(st + lane * NP) + (delta >> 3);
      const uint64_t d = digest_row<HB>(row, (delta & 4) != 0, HB, d_init);
      digest[c * kChunk + lane] = d;
      if (groups && cur.head) group_insert(groups, gmask, first_hash(h_init, d), cur.req);
    }
    __syncwarp();
    cur = nxt;
  }
}

// ---- TMA tensor path -------------------------------------------------------
//
// For B % 4 == 0, block j of a request starts 4B*j bytes after block 0, so the
// rows a_j = (4*first token of block j) & ~15 of one request form a strided
// 2D region: rows of 4B+16 bytes at stride 4B. A 2D tensor map per 16-byte
// phase k (base = tokens + 16k) with row stride 4B and row length 4B+16 lets
// one TMA tile load of 32 rows bring a whole chunk into the padded layout.
// Rows past the end of the map are zero-filled by the TMA unit; a chunk that
// needs such a row, or whose blocks span two requests, is copied by its lanes
// instead.

constexpr int kMaxPhases = 16;  // 4B / 16 for B <= 64
constexpr uint32_t kSpinLimit = 1u << 22;  // bounded mbarrier waits

struct TokenMaps {
  CUtensorMap map[kMaxPhases];
  uint32_t rows[kMaxPhases];  // rows addressable through map k
};

__device__ __forceinline__ void mbar_init(uint32_t mbar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(mbar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t mbar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(mbar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t mbar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(done) : "r"(mbar), "r"(parity) : "memory");
  return done != 0;
}
// Bounded wait for the phase with the given parity; false on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t mbar, uint32_t parity) {
  for (uint32_t i = 0; i < kSpinLimit; ++i)
    if (mbar_try_wait(mbar, parity)) return true;
  return false;
}
__device__ __forceinline__ void tma_rows(uint32_t dst, const CUtensorMap* map, int32_t y, uint32_t mbar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;\n" ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(0),
      "r"(y), "r"(mbar), "l"(policy)
      : "memory");
}

template <int HB, int STAGES>
__global__ void __launch_bounds__(kTmaWarps * 32)
    k_digest_tma(const __grid_constant__ TokenMaps maps, const int32_t* __restrict__ tokens,
                 int64_t n_tokens, const int64_t* __restrict__ off, const int64_t* __restrict__ block_off,
                 const int64_t* __restrict__ chunk_off, int32_t n, uint64_t d_init, const int32_t* __restrict__ batch_ok,
                 uint64_t* __restrict__ digest, int32_t* status, uint64_t* __restrict__ groups, uint64_t gmask,
                 uint64_t h_init) {
  pdl_enter();
  constexpr int B = 2 * HB;
  constexpr int NP = HB / 2 + 1;           // 16-byte pieces per row
  constexpr uint32_t ROW = 16u * NP;       // = 4B + 16
  constexpr uint32_t STAGE = kChunk * ROW;
  extern __shared__ __align__(128) unsigned char dsm_raw[];
  if (!*batch_ok) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, warps = blockDim.x >> 5;
  // chunk c is chunk q of request r: its blocks 32q .. 32q+31, so a chunk
  // never spans two requests
  const int64_t n_chunks = chunk_off[n];
  // A CTA takes a contiguous range of chunks and its warps interleave over it
  // (warp w: chunks w, w + warps, ...), so that the copies a CTA has in flight
  // cover one stretch of consecutive tokens.
  const int64_t per = (n_chunks + gridDim.x - 1) / gridDim.x;  // chunks per CTA
  const int64_t k_lo = (int64_t)blockIdx.x * per;
  const int64_t c_hi = min(n_chunks, k_lo + per);
  const int64_t c_lo = k_lo + warp;  // then every warps-th chunk of the CTA's range
  if (c_lo >= c_hi) return;
  unsigned char* const stages = dsm_raw + (size_t)warp * STAGES * STAGE;
  const uint32_t mbar0 = smem_u32(dsm_raw + (size_t)warps * STAGES * STAGE) + 8u * STAGES * (uint32_t)warp;
  if (lane == 0) {
#pragma unroll
    for (int s = 0; s < STAGES; ++s) mbar_init(mbar0 + 8u * s, 1);
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  __syncwarp();
  uint64_t policy;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(policy));
  const int64_t token_bytes = 4 * n_tokens;
  const char* const tb = reinterpret_cast<const char*>(tokens);
  int32_t r = find_request(chunk_off, 0, n, c_lo);  // warp-uniform

  // Start the copy of chunk c into stage s; returns this lane's first token
  // and sets its digest index and its request (`head` when the lane has the
  // request's block 0, whose digest also gives the request's group key).
  auto issue = [&](int64_t c, int s, bool& valid, int64_t& gidx, int32_t& req, bool& head) -> int64_t {
    for (int i = 0; i < 4 && __ldg(chunk_off + r + 1) <= c; ++i) ++r;  // usually a step or two
    if (__ldg(chunk_off + r + 1) <= c) r = find_request(chunk_off, r + 1, n, c);
    const int64_t bo = __ldg(block_off + r), nbr = __ldg(block_off + r + 1) - bo;
    const int64_t b = (c - __ldg(chunk_off + r)) * kChunk + lane;  // block of request r
    valid = b < nbr;
    const int64_t tok0 = __ldg(off + r) + b * B;
    gidx = bo + b;
    req = r;
    head = b == 0;
    const int nv = (int)min((int64_t)kChunk, nbr - (b - lane));
    const int64_t a0 = (4 * __shfl_sync(kFull, tok0, 0)) & ~(int64_t)15;
    const int k = (int)((a0 % (4 * B)) >> 4);
    const int64_t y0 = a0 / (4 * B);
    unsigned char* const st = stages + (size_t)s * STAGE;
    const uint32_t mbar = mbar0 + 8u * (uint32_t)s;
    if (y0 + nv <= (int64_t)maps.rows[k]) {
      if (lane == 0) {
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
        mbar_arrive_expect_tx(mbar, STAGE);
        tma_rows(smem_u32(st), &maps.map[k], (int32_t)y0, mbar, policy);
      }
    } else {
      // lanes copy their own rows; the stage's barrier completes on lane 0's
      // arrival with no bytes expected
      if (valid) {
        const int64_t a = (4 * tok0) & ~(int64_t)15;
        uint4* row = reinterpret_cast<uint4*>(st + lane * ROW);
#pragma unroll
        for (int i = 0; i < NP; ++i) row[i] = load_piece(tb, a + 16 * i, token_bytes - (a + 16 * i));
      }
      __syncwarp();
      if (lane == 0) mbar_arrive_expect_tx(mbar, 0);
    }
    return tok0;
  };

  uint32_t phase = 0;
  bool failed = false;
  bool v[STAGES], hd[STAGES];
  int64_t t[STAGES], gi[STAGES];
  int32_t rq[STAGES];
#pragma unroll
  for (int s = 0; s < STAGES; ++s)
    if (c_lo + s * warps < c_hi) t[s] = issue(c_lo + s * warps, s, v[s], gi[s], rq[s], hd[s]);
  int s = 0;
  for (int64_t c = c_lo; c < c_hi; c += warps) {
    if (!mbar_wait(mbar0 + 8u * (uint32_t)s, (phase >> s) & 1)) { failed = true; break; }
    phase ^= 1u << s;
    bool vc = false, hc = false;
    int64_t tc = 0, gc = 0;
    int32_t rc = 0;
#pragma unroll
    for (int q = 0; q < STAGES; ++q) if (q == s) { vc = v[q]; tc = t[q]; gc = gi[q]; rc = rq[q]; hc = hd[q]; }
    if (vc) {
      const int delta = (int)((tc * 4) & 15);  // 0, 4, 8 or 12
      const uint64_t* row = reinterpret_cast<const uint64_t*>(stages + (size_t)s * STAGE + lane * ROW) + (delta >> 3);
      const uint64_t d = digest_row<HB>(row, (delta & 4) != 0, HB, d_init);
      digest[gc] = d;
      if (groups && hc) group_insert(groups, gmask, first_hash(h_init, d), rc);
    }
    __syncwarp();
    if (c + STAGES * warps < c_hi) {
      bool vn, hn;
      int64_t gn = 0;
      int32_t rn = 0;
      const int64_t tn = issue(c + STAGES * warps, s, vn, gn, rn, hn);
#pragma unroll
      for (int q = 0; q < STAGES; ++q) if (q == s) { v[q] = vn; t[q] = tn; gi[q] = gn; rq[q] = rn; hd[q] = hn; }
    }
    s = s + 1 == STAGES ? 0 : s + 1;
  }
  if (failed) {
    // a copy never completed: report it and give copies in flight a bounded
    // chance to land before the shared memory is released
    if (lane == 0) latch_error(status, SMETRIC_ERR_CUDA);
#pragma unroll
    for (int q = 0; q < STAGES; ++q) mbar_wait(mbar0 + 8u * q, (phase >> q) & 1);
  }
}

// Any even B: each lane copies its own row straight from global memory.
__global__ void __launch_bounds__(kDigestWarps * 32)
    k_digest_any(const int32_t* __restrict__ tokens, int64_t n_tokens, const int64_t* __restrict__ off,
                 const int64_t* __restrict__ block_off, int32_t n, int B, int nch, uint64_t d_init,
                 const int32_t* __restrict__ batch_ok, uint64_t* __restrict__ digest,
                 uint64_t* __restrict__ groups, uint64_t gmask, uint64_t h_init) {
  pdl_enter();
  extern __shared__ uint4 dsm[];
  if (!*batch_ok) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, warps = blockDim.x >> 5;
  const int64_t total = block_off[n];
  const int64_t n_chunks = (total + kChunk - 1) / kChunk;
  const int64_t tw = (int64_t)gridDim.x * warps;
  const int64_t per = (n_chunks + tw - 1) / tw;
  const int64_t c_lo = ((int64_t)blockIdx.x * warps + warp) * per;
  const int64_t c_hi = min(n_chunks, c_lo + per);
  if (c_lo >= c_hi) return;
  uint4* const row = dsm + ((size_t)warp * kChunk + lane) * nch;
  const int64_t token_bytes = 4 * n_tokens;
  const char* const tb = reinterpret_cast<const char*>(tokens);
  int32_t r = find_request(block_off, 0, n, min(c_lo * kChunk + lane, total - 1));
  for (int64_t c = c_lo; c < c_hi; ++c) {
    const int64_t f = c * kChunk + lane;
    if (f >= total) continue;
    if (__ldg(block_off + r + 1) <= f) r = find_request(block_off, r + 1, n, f);
    const int64_t tok0 = __ldg(off + r) + (f - __ldg(block_off + r)) * B;
    const int64_t a = (4 * tok0) & ~(int64_t)15;
    for (int i = 0; i < nch; ++i) row[i] = load_piece(tb, a + 16 * i, token_bytes - (a + 16 * i));
    const int delta = (int)((tok0 * 4) & 15);
    const uint64_t d = digest_row<0>(reinterpret_cast<const uint64_t*>(row) + (delta >> 3), (delta & 4) != 0,
                                     B >> 1, d_init);
    digest[f] = d;
    if (groups && f == __ldg(block_off + r)) group_insert(groups, gmask, first_hash(h_init, d), r);
  }
}

// ---------------------------------------------------------------------------
// chain
// ---------------------------------------------------------------------------

// 32-byte global load (read-only path) and store of four 64-bit words; the
// address must be 32-byte aligned.
__device__ __forceinline__ void ld_nc_v4(const uint64_t* p, uint64_t (&v)[4]) {
  asm volatile("ld.global.nc.v4.u64 {%0,%1,%2,%3}, [%4];\n"
               : "=l"(v[0]), "=l"(v[1]), "=l"(v[2]), "=l"(v[3])
               : "l"(p));
}
__device__ __forceinline__ void st_v4(uint64_t* p, uint64_t a, uint64_t b, uint64_t c, uint64_t d) {
  asm volatile("st.global.v4.u64 [%0], {%1,%2,%3,%4};\n" ::"l"(p), "l"(a), "l"(b), "l"(c), "l"(d) : "memory");
}

// End of a request's chain: the session key is read back rather than tested
// at every serial step.
__device__ __forceinline__ void nb_done(int32_t r, int64_t nb, const uint64_t* hout, int64_t kS,
                                        uint64_t* __restrict__ sk_out) {
  sk_out[r] = nb > 0 ? hout[kS] : 0;
}

__global__ void __launch_bounds__(kChainThreads)
    k_chain(const int64_t* __restrict__ off, const int64_t* __restrict__ block_off, int32_t n, int B,
            int S, uint64_t h_init, const int32_t* __restrict__ batch_ok,
            const uint64_t* __restrict__ digest, uint64_t* __restrict__ hashes,
            uint64_t* __restrict__ sk_out) {
  pdl_enter();
  const int32_t r = blockIdx.x * kChainThreads + threadIdx.x;
  if (r >= n) return;
  if (!*batch_ok) { sk_out[r] = 0; return; }
  const int64_t bo = block_off[r];
  const int64_t nb = block_off[r + 1] - bo;
  const uint64_t* const d = digest + bo;
  uint64_t* const hout = hashes + bo;
  const int64_t kS = (nb < S ? nb : S) - 1;
  uint64_t h = h_init;
  auto step = [](uint64_t hp, uint64_t db) {
    uint64_t x = mix64_halves((hp + kGamma) ^ db);
    if (x < 2) x |= 2;
    return x;
  };
  // Digests are read and hashes written four blocks per 32-byte access (a
  // lane's accesses are its own request's and do not coalesce across the
  // warp, and fewer instructions shorten every serial step): single blocks
  // up to a 32-byte boundary and after the last whole quad. A caller hash
  // buffer in another 32-byte phase than the digests takes one block per
  // access throughout.
  if (((reinterpret_cast<uintptr_t>(d) ^ reinterpret_cast<uintptr_t>(hout)) & 31) != 0) {
    for (int64_t k = 0; k < nb; ++k) {
      h = step(h, __ldg(d + k));
      hout[k] = h;
    }
    nb_done(r, nb, hout, kS, sk_out);
    return;
  }
  int64_t b = 0;
  while (b < nb && (reinterpret_cast<uintptr_t>(d + b) & 31)) {
    h = step(h, __ldg(d + b));
    hout[b] = h;
    ++b;
  }
  const uint64_t* const dq = d + b;
  uint64_t* const hq = hout + b;
  const int64_t nq = (nb - b) >> 2;  // whole quads
  constexpr int Q = kChainAhead / 4;
  uint64_t c[Q][4], x[Q][4];
#pragma unroll
  for (int j = 0; j < Q; ++j)
    if (j < nq) ld_nc_v4(dq + 4 * j, c[j]);
  for (int64_t q0 = 0; q0 < nq; q0 += Q) {
#pragma unroll
    for (int j = 0; j < Q; ++j)
      if (q0 + Q + j < nq) ld_nc_v4(dq + 4 * (q0 + Q + j), x[j]);
#pragma unroll
    for (int j = 0; j < Q; ++j) {
      if (q0 + j < nq) {
        const uint64_t a0 = step(h, c[j][0]), a1 = step(a0, c[j][1]), a2 = step(a1, c[j][2]);
        h = step(a2, c[j][3]);
        st_v4(hq + 4 * (q0 + j), a0, a1, a2, h);
      }
    }
#pragma unroll
    for (int j = 0; j < Q; ++j)
#pragma unroll
      for (int k = 0; k < 4; ++k) c[j][k] = x[j][k];
  }
  for (int64_t k = b + 4 * nq; k < nb; ++k) {
    h = step(h, __ldg(d + k));
    hout[k] = h;
  }
  nb_done(r, nb, hout, kS, sk_out);
}

// ---------------------------------------------------------------------------
// group
// ---------------------------------------------------------------------------

// ---------------------------------------------------------------------------
// match
// ---------------------------------------------------------------------------

// Tier masks of key h (zeros when absent) from the read-only table: the home
// bucket's 15 tags, then the entry of each tag match, then later buckets while
// the bucket just read has keys stored past it (its overflow count).
template <int W>
__device__ __forceinline__ void probe_one(const uint8_t* __restrict__ tags, const uint64_t* __restrict__ table,
                                          uint64_t n_buckets, uint64_t h, uint64_t (&M)[W]) {
  constexpr int EW = entry_words(W);
  constexpr int NV = (W + 2) / 2;  // 16-byte loads covering key + W mask words
#pragma unroll
  for (int w = 0; w < W; ++w) M[w] = 0;
  const uint32_t tg = key_tag(h);
  uint64_t b = home_bucket(h, n_buckets);
  const uint64_t mb = max_buckets(n_buckets);
  for (uint64_t t = 0; t < mb; ++t) {
    const uint4 tv = __ldg(reinterpret_cast<const uint4*>(tags + b * kBucket));
    uint32_t cand = slot_match(tv, tg);
    while (cand) {
      const int sl = __ffs(cand) - 1;
      cand &= cand - 1;
      const ulonglong2* e = reinterpret_cast<const ulonglong2*>(table + (b * kSlots + sl) * EW);
      ulonglong2 v[NV];
#pragma unroll
      for (int q = 0; q < NV; ++q) v[q] = __ldg(e + q);
      if (v[0].x == h) {
#pragma unroll
        for (int w = 0; w < W; ++w) M[w] = (w & 1) ? v[(w + 1) >> 1].x : v[(w + 1) >> 1].y;
        return;
      }
    }
    if (overflow_count(tv) == 0) return;
    if (++b == n_buckets) b = 0;
  }
}

// ---------------------------------------------------------------------------
// chain, shared prefix and probe in one kernel
// ---------------------------------------------------------------------------
//
// The chain is bound by the latency of its dependent mix64 steps and the
// probe by random memory accesses, so one kernel runs both at once. One CTA
// of 32 warps per SM; the SM deals a CTA's warps to its four schedulers in
// turn (warp w to scheduler w mod 4). The chain warps (lane = request) are
// warps 0 .. chain_warps - 1, one per scheduler, beside probe warps that
// mostly wait on memory, so their dependent steps seldom wait for issue. The
// other warps first find each request's group leader and shared prefix, then
// probe the index for each 32-block chunk as soon as its chain has published
// it.
//
// CTA c owns requests c, c + gridDim, c + 2 gridDim, ..., taken in groups of
// up to 32 * chain_warps (one chain lane each). Chunk q of request r is its
// blocks 32q .. 32q + 31; the chunk ANDs the walk reads are kept per such
// request-aligned chunk, at index chunk_off[r] + q.
constexpr int kCpWarps = 32;
constexpr int kCpMaxChainWarps = 4;  // warps 0 .. 3, one per scheduler
constexpr int kCpMaxGroup = 32 * kCpMaxChainWarps;
constexpr int kCpRingDigests = 34;   // a chunk's 32 digests and one neighbour on each side
constexpr int kCpRingBytes = 560;    // two such slots per chain lane, in 16-byte pieces
constexpr int kCpProbes = 2;         // chunks a probe warp takes at once (probes in flight per lane)
constexpr int kCpDealMax = 512;      // requests a CTA can own when leaders are dealt out

__device__ __forceinline__ int32_t ld_acquire_cta(const int32_t* p) {
  int32_t v;
  asm volatile("ld.acquire.cta.shared::cta.s32 %0, [%1];\n" : "=r"(v) : "r"(smem_u32(p)) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_cta(int32_t* p, int32_t v) {
  asm volatile("st.release.cta.shared::cta.s32 [%0], %1;\n" ::"r"(smem_u32(p)), "r"(v) : "memory");
}
// A chain hash another warp of this CTA has published (ordered by ld_acquire_cta).
__device__ __forceinline__ uint64_t ld_relaxed_cta(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.cta.global.u64 %0, [%1];\n" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

// One chain step: h_b from h_{b-1} and d_b, with the sentinel remap.
__device__ __forceinline__ uint64_t chain_step(uint64_t hp, uint64_t db) {
  uint64_t x = mix64_halves((hp + kGamma) ^ db);
  if (x < 2) x |= 2;
  return x;
}

// Bounded wait until a shared counter exceeds v; false on timeout.
__device__ __forceinline__ bool wait_above(const int32_t* p, int32_t v) {
  for (uint32_t i = 0; i < kSpinLimit; ++i) {
    if (ld_acquire_cta(p) > v) return true;
    __nanosleep(256);  // a long sleep keeps waiting warps off the chain warps' schedulers
  }
  return false;
}

// Tier masks of U keys at once: the home-bucket tags of all, then the first
// tag match's entry of all, so that U pairs of dependent reads are in flight
// together. A key whose first candidate is not it (another key with the same
// tag, or a key stored past its home bucket) takes the full probe_one.
template <int W, int U>
__device__ __forceinline__ void probe_many(const uint8_t* __restrict__ tags, const uint64_t* __restrict__ table,
                                           uint64_t n_buckets, const bool (&act)[U], const uint64_t (&h)[U],
                                           uint64_t (&M)[U][W]) {
  constexpr int EW = entry_words(W);
  constexpr int NV = (W + 2) / 2;
  uint64_t bk[U];
  uint4 tv[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    bk[u] = act[u] ? home_bucket(h[u], n_buckets) : 0;
    if (act[u]) tv[u] = __ldg(reinterpret_cast<const uint4*>(tags + bk[u] * kBucket));
  }
  ulonglong2 v[U][NV];
  uint32_t cand[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    cand[u] = act[u] ? slot_match(tv[u], key_tag(h[u])) : 0;
    if (cand[u]) {
      const ulonglong2* e = reinterpret_cast<const ulonglong2*>(table + (bk[u] * kSlots + __ffs(cand[u]) - 1) * EW);
#pragma unroll
      for (int q = 0; q < NV; ++q) v[u][q] = __ldg(e + q);
    }
  }
#pragma unroll
  for (int u = 0; u < U; ++u) {
#pragma unroll
    for (int w = 0; w < W; ++w) M[u][w] = 0;
    if (!act[u]) continue;
    if (cand[u] && v[u][0].x == h[u]) {
#pragma unroll
      for (int w = 0; w < W; ++w) M[u][w] = (w & 1) ? v[u][(w + 1) >> 1].x : v[u][(w + 1) >> 1].y;
    } else if ((cand[u] & (cand[u] - 1)) || overflow_count(tv[u])) {
      probe_one<W>(tags, table, n_buckets, h[u], M[u]);  // more candidates, or later buckets
    }
    // else: no candidate left and no key stored past the home bucket: absent
  }
}

// One thread per request: 1 if the request leads its group (the group
// table's lowest request with its first-block hash), else 0.
__global__ void __launch_bounds__(256)
    k_lead(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ batch_ok,
           const uint64_t* __restrict__ D, uint64_t h_init, const uint64_t* __restrict__ groups, uint64_t gmask,
           uint8_t* __restrict__ lead_flag) {
  pdl_enter();
  const int32_t r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= n || !*batch_ok) return;
  const int64_t bo = block_off[r];
  uint8_t f = 0;
  if (block_off[r + 1] > bo) {
    const uint64_t key = first_hash(h_init, __ldg(D + bo));
    uint64_t sl = key & gmask;
    for (uint64_t t = 0; t <= gmask; ++t, sl = (sl + 1) & gmask) {
      const ulonglong2 pr = *reinterpret_cast<const ulonglong2*>(groups + 2 * sl);
      if (pr.x == key) {
        f = INT32_MAX - (int32_t)pr.y == r;
        break;
      }
      if (pr.x == 0) break;
    }
  }
  lead_flag[r] = f;
}

template <int W>
__global__ void __launch_bounds__(kCpWarps * 32, 1)
    k_chain_probe(const int64_t* __restrict__ block_off, const int64_t* __restrict__ chunk_off, int32_t n, int S,
                  uint64_t h_init, const int32_t* __restrict__ batch_ok, const uint64_t* __restrict__ D,
                  uint64_t* __restrict__ hashes, uint64_t* __restrict__ sk_out, const uint64_t* __restrict__ groups,
                  uint64_t gmask, int32_t* __restrict__ lead, int32_t* __restrict__ share,
                  const uint8_t* __restrict__ tags,
                  const uint64_t* __restrict__ table, uint64_t n_buckets, uint64_t* __restrict__ masks,
                  uint64_t* __restrict__ chunk_and, const uint8_t* __restrict__ lead_flag, int chain_warps,
                  int32_t* status) {
  pdl_enter();
  extern __shared__ __align__(128) unsigned char csm[];  // chain lanes' digest rings
  __shared__ int32_t s_ready[kCpMaxGroup];  // chunks chained, per request of the group
  __shared__ int32_t s_share[kCpMaxGroup];  // shared prefix per request (-1 until known)
  __shared__ int32_t s_dead[kCpMaxGroup];   // first chunk whose AND is empty (INT32_MAX until one is)
  __shared__ int32_t s_fin[kCpMaxGroup];    // chunks finished in order from the first unshared one
  __shared__ int64_t s_bo[kCpMaxGroup];     // per request of the group: first block in the batch,
  __shared__ int64_t s_cb[kCpMaxGroup];     // first request-aligned chunk,
  __shared__ int32_t s_nb[kCpMaxGroup];     // and full blocks
  __shared__ int32_t s_next0;               // work counter: share tasks
  __shared__ unsigned long long s_next1;    // work counter: probe items
  __shared__ int32_t s_maxch;               // most chunks of a request in the group
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // The CTAs' requests. A group leader (the lowest request with its first
  // block, which probes its whole prefix) costs a member (which probes only
  // past its shared prefix) many times over, so leaders are dealt round robin
  // over the CTAs in request order, then the members after them: every CTA
  // gets its share of each. k_lead has marked the leaders. Past 32 requests
  // a thread, or kCpDealMax a CTA, requests are taken as blockIdx.x +
  // k * gridDim.x instead.
  __shared__ int32_t s_mine[kCpDealMax];
  __shared__ int32_t s_nmine;
  __shared__ int32_t s_wsum[kCpWarps];
  const int32_t stride = (int32_t)gridDim.x;
  const int32_t per_t = (n + (int32_t)blockDim.x - 1) / (int32_t)blockDim.x;
  const bool dealt = *batch_ok && per_t <= 32 && (n + stride - 1) / stride <= kCpDealMax;
  if (dealt) {
    if (threadIdx.x == 0) s_nmine = 0;
    const int32_t a = min(n, (int32_t)threadIdx.x * per_t), e = min(n, a + per_t);
    uint32_t lead_bits = 0;  // bit i: request a + i leads its group (from k_lead)
    for (int32_t r = a; r < e; ++r) lead_bits |= (uint32_t)__ldg(lead_flag + r) << (r - a);
    // exclusive scan of the leader counts over the threads, in request order
    const int32_t cnt = __popc(lead_bits);
    int32_t incl = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int32_t y = __shfl_up_sync(kFull, incl, d);
      if (lane >= d) incl += y;
    }
    if (lane == 31) s_wsum[warp] = incl;
    __syncthreads();
    int32_t before = 0, total = 0;
    for (int w2 = 0; w2 < kCpWarps; ++w2) {
      const int32_t v = s_wsum[w2];
      if (w2 < warp) before += v;
      total += v;
    }
    int32_t lrank = before + incl - cnt;  // leaders before request a
    for (int32_t r = a; r < e; ++r) {
      const bool isl = (lead_bits >> (r - a)) & 1u;
      // leaders by leader rank; members by member rank, continuing the deal
      const int32_t cta = isl ? lrank % stride : (total + (r - lrank)) % stride;
      if (isl) ++lrank;
      if (cta == (int32_t)blockIdx.x) s_mine[atomicAdd(&s_nmine, 1)] = r;
    }
    __syncthreads();
  }
  const int32_t m = dealt ? s_nmine : n > (int32_t)blockIdx.x ? (n - (int32_t)blockIdx.x + stride - 1) / stride : 0;
  auto req_of = [&](int32_t k) { return dealt ? s_mine[k] : (int32_t)blockIdx.x + k * stride; };
  if (!*batch_ok) {
    for (int32_t k = (int32_t)threadIdx.x; k < m; k += blockDim.x) sk_out[req_of(k)] = 0;
    return;
  }
  // chain warps: warp k on scheduler k (one each); every other warp probes
  const int cw = warp;
  const bool chain = warp < chain_warps;
  const bool prober = warp >= chain_warps;
  const int G = 32 * chain_warps;

  for (int32_t g0 = 0; g0 < m; g0 += G) {
    const int mg = min(G, m - g0);
    if ((int)threadIdx.x < mg) {
      s_ready[threadIdx.x] = 0;
      s_share[threadIdx.x] = -1;
      s_dead[threadIdx.x] = INT32_MAX;
      s_fin[threadIdx.x] = 0;
      const int32_t r = req_of(g0 + (int32_t)threadIdx.x);
      const int64_t bo = block_off[r];
      s_bo[threadIdx.x] = bo;
      s_nb[threadIdx.x] = (int32_t)(block_off[r + 1] - bo);
      s_cb[threadIdx.x] = chunk_off[r];
    }
    if (threadIdx.x == 0) {
      s_next0 = 0;
      s_next1 = 0;
      s_maxch = 0;
    }
    __syncthreads();
    if ((int)threadIdx.x < mg)
      atomicMax(&s_maxch, (int32_t)(chunk_off[req_of(g0 + threadIdx.x) + 1] - chunk_off[req_of(g0 + threadIdx.x)]));
    __syncthreads();
    const int32_t maxch = s_maxch;
    if (chain) {
      // lane = request j of the group: the chain over its digests, one chunk
      // at a time from a two-slot ring in shared memory (slot q & 1 holds
      // chunk q; chunk q + 1 is copied in while chunk q is chained)
      const int j = 32 * cw + lane;
      const bool act = j < mg;
      const int32_t r = act ? req_of(g0 + j) : 0;
      int64_t bo = 0, nb = 0;
      if (act) {
        bo = __ldg(block_off + r);
        nb = __ldg(block_off + r + 1) - bo;
      }
      const int32_t nch = (int32_t)((nb + kChunk - 1) / kChunk);
      int32_t wmax = nch;
#pragma unroll
      for (int dd = 16; dd > 0; dd >>= 1) wmax = max(wmax, __shfl_xor_sync(kFull, wmax, dd));
      unsigned char* const ring = csm + (size_t)j * kCpRingBytes;
      const uint32_t ring_s = smem_u32(ring);
      // copies chunk q's digests [first, first + nv) in 16-byte pieces from the
      // even index at or below first into slot q & 1
      auto fetch = [&](int32_t q) {
        const int64_t first = bo + (int64_t)kChunk * q;
        const int64_t a = first & ~(int64_t)1;
        const int nv = (int)min((int64_t)kChunk, nb - (int64_t)kChunk * q);
        const int pieces = (int)((first + nv - a + 1) >> 1);
        const uint32_t dst = ring_s + (uint32_t)((q & 1) * kCpRingDigests * 8);
        for (int i = 0; i < pieces; ++i) cp_async16(dst + 16u * i, D + a + 2 * i);
      };
      if (act && nch > 0) fetch(0);
      cp_async_commit();
      uint64_t h = h_init;
      for (int32_t q = 0; q < wmax; ++q) {
        cp_async_wait_all();
        if (q + 1 < nch) fetch(q + 1);
        cp_async_commit();
        if (q < nch) {
          const int64_t b0 = (int64_t)kChunk * q;
          const int nv = (int)min((int64_t)kChunk, nb - b0);
          const uint64_t* dsm =
              reinterpret_cast<const uint64_t*>(ring + (q & 1) * kCpRingDigests * 8) + ((bo + b0) & 1);
          uint64_t* const ho = hashes + bo + b0;
          for (int i = 0; i < nv; ++i) {
            h = chain_step(h, dsm[i]);
            ho[i] = h;
          }
          __threadfence_block();
          st_release_cta(&s_ready[j], q + 1);  // the chunk's hashes are out
        }
      }
      cp_async_wait_all();
      if (act) sk_out[r] = nb > 0 ? hashes[bo + (nb < S ? nb : (int64_t)S) - 1] : 0;
    } else if (prober) {
      // Phase 1, a warp per request (taken from a counter): the group leader
      // (lowest request id with the same first-block hash, from the table the
      // digest kernel filled) and the number of leading blocks whose digests
      // equal the leader's.
      for (;;) {
        int32_t j = 0;
        if (lane == 0) j = atomicAdd(&s_next0, 1);
        j = __shfl_sync(kFull, j, 0);
        if (j >= mg) break;
        const int32_t r = req_of(g0 + j);
        const int64_t bo = __ldg(block_off + r), nb = __ldg(block_off + r + 1) - bo;
        int32_t l = r;
        int64_t sh = 0;
        if (nb > 0) {
          const uint64_t key = first_hash(h_init, __ldg(D + bo));
          const uint64_t s0 = key & gmask;
          for (uint64_t t = 0; t <= gmask; t += 32) {
            const uint64_t sl = (s0 + t + lane) & gmask;
            const uint64_t k = groups[2 * sl];
            const unsigned hit = __ballot_sync(kFull, k == key), emp = __ballot_sync(kFull, k == 0);
            const unsigned stop = hit | emp;
            if (stop) {
              const int first = __ffs(stop) - 1;
              if (hit & (1u << first)) l = INT32_MAX - (int32_t)groups[2 * ((s0 + t + first) & gmask) + 1];
              break;
            }
          }
          if (l != r && l >= 0 && l < n) {
            const int64_t lo = __ldg(block_off + l), nl = __ldg(block_off + l + 1) - lo;
            const int64_t m = nb < nl ? nb : nl;
            sh = m;
            for (int64_t b = 0; b < m; b += 32 * kGroupAhead) {
              bool ne[kGroupAhead];
#pragma unroll
              for (int u = 0; u < kGroupAhead; ++u) {
                const int64_t bb = b + 32 * u + lane;
                ne[u] = bb < m && __ldg(D + bo + bb) != __ldg(D + lo + bb);
              }
              int64_t first = -1;
#pragma unroll
              for (int u = 0; u < kGroupAhead; ++u) {
                const unsigned x = __ballot_sync(kFull, ne[u]);
                if (x && first < 0) first = 32 * u + __ffs(x) - 1;
              }
              if (first >= 0) {
                sh = b + first;
                break;
              }
            }
          } else {
            l = r;
          }
        }
        if (lane == 0) {
          lead[r] = l;
          share[r] = (int32_t)sh;
          st_release_cta(&s_share[j], (int32_t)sh);
        }
      }
      // Phase 2: items (q, j) in chunk-major order, kCpProbes at a time: the
      // tier masks of chunk q's blocks of request j at or past its shared
      // prefix, once its chain has published the chunk; and the chunk's AND
      // (a block not probed counts as all ones). Skipped with no wait: a chunk
      // wholly inside the shared prefix (the walk reads the leader's). Skipped
      // after waiting: any chunk after one whose AND is empty (that chunk
      // lacks a block of every tier, so every run has ended there: the walk
      // stops before reaching later chunks). When the probers' items in
      // flight would span more than two rounds of the group (few requests per
      // CTA), a request's chunk q starts only once its chunk q - 2 has
      // finished (chunks then finish in order), so at most two of its chunks
      // are probed ahead of knowing whether its runs are over.
      const bool paced = (kCpWarps - chain_warps) * kCpProbes > 2 * mg;
      const int64_t items = (int64_t)maxch * mg;
      for (;;) {
        int64_t t0 = 0;
        if (lane == 0) t0 = (int64_t)atomicAdd(&s_next1, (unsigned long long)kCpProbes);
        t0 = __shfl_sync(kFull, t0, 0);
        if (t0 >= items) break;
        // item t is chunk t / mg of request t % mg; one division per grab
        int32_t q0 = (int32_t)(t0 < INT32_MAX ? (uint32_t)t0 / (uint32_t)mg : t0 / mg);
        int32_t j0 = (int32_t)(t0 - (int64_t)q0 * mg);
        bool act[kCpProbes];
        uint64_t hv[kCpProbes];
        int64_t f[kCpProbes], cidx[kCpProbes];
        int32_t qs[kCpProbes], js[kCpProbes], rel[kCpProbes];  // rel: chunk index counted from the first unshared one
#pragma unroll
        for (int u = 0; u < kCpProbes; ++u) {
          act[u] = false;
          hv[u] = 0;
          f[u] = 0;
          cidx[u] = -1;
          rel[u] = -1;
          const int64_t t = t0 + u;
          const int32_t q = q0, j = j0;
          if (++j0 == mg) {
            j0 = 0;
            ++q0;
          }
          if (t >= items) continue;
          qs[u] = q;
          js[u] = j;
          const int64_t bo = s_bo[j], nb = s_nb[j];
          if ((int64_t)kChunk * q >= nb) continue;  // the request has no chunk q
          if (!wait_above(&s_share[j], -1)) {
            if (lane == 0) latch_error(status, SMETRIC_ERR_CUDA);
            continue;
          }
          const int64_t sh = s_share[j];
          if ((int64_t)kChunk * (q + 1) <= sh) continue;
          rel[u] = paced ? q - (int32_t)(sh / kChunk) : -1;
          if (paced && !wait_above(&s_fin[j], rel[u] - 2)) {  // chunk q - 2 has finished
            if (lane == 0) latch_error(status, SMETRIC_ERR_CUDA);
            rel[u] = -1;
            continue;
          }
          if (ld_acquire_cta(&s_dead[j]) < q) continue;  // finished as skipped below
          if (!wait_above(&s_ready[j], q)) {
            if (lane == 0) latch_error(status, SMETRIC_ERR_CUDA);
            continue;
          }
          const int64_t b = (int64_t)kChunk * q + lane;
          act[u] = b < nb && b >= sh;
          f[u] = bo + b;
          cidx[u] = s_cb[j] + q;
          if (act[u]) hv[u] = ld_relaxed_cta(hashes + bo + b);
        }
        uint64_t M[kCpProbes][W];
        probe_many<W, kCpProbes>(tags, table, n_buckets, act, hv, M);
#pragma unroll
        for (int u = 0; u < kCpProbes; ++u) {
          if (cidx[u] < 0) continue;  // warp-uniform
          if (act[u]) {
#pragma unroll
            for (int w = 0; w < W; ++w) masks[f[u] * W + w] = M[u][w];
          }
          bool empty = true;
#pragma unroll
          for (int w = 0; w < W; ++w) {
            const uint64_t x = act[u] ? M[u][w] : ~0ull;
            const uint64_t a = (uint64_t)__reduce_and_sync(kFull, (unsigned)x) |
                               ((uint64_t)__reduce_and_sync(kFull, (unsigned)(x >> 32)) << 32);
            if (lane == w) chunk_and[cidx[u] * W + w] = a;
            empty &= a == 0;
          }
          if (empty && lane == 0) atomicMin(&s_dead[js[u]], qs[u]);
        }
        // chunks finish in order: after the request's previous chunk
#pragma unroll
        for (int u = 0; u < kCpProbes; ++u) {
          if (rel[u] < 0) continue;  // warp-uniform
          if (lane == 0) {
            if (!wait_above(&s_fin[js[u]], rel[u] - 1)) latch_error(status, SMETRIC_ERR_CUDA);
            st_release_cta(&s_fin[js[u]], rel[u] + 1);
          }
          __syncwarp();
        }
      }
    }
    __syncthreads();  // the group's shared state is rewritten by the next group
  }
}

// The session-centric policy (Figure 10) as the walk's decision; off for
// the argmin cost of smetric_route_batch.
enum Decide { kArgmin = 0, kSession = 1, kColoc = 2, kBailian = 3, kLMetric = 4 };

struct WalkPolicy {
  int on;    // a Decide value; 0 = the argmin cost
  int64_t c_lin, c_att, d0, d1, hit_num, hit_den;
  int32_t rr_base;
  const int32_t* turn;
  const int64_t* est_hit;
  int32_t* stick;
  const int64_t* tpot;  // colocation: prefill cost each instance's live decodes absorb
  const int64_t* nreq;  // colocation: requests each instance runs; baselines: batch sizes
  int64_t lam_num, lam_den;  // Bailian's weight
};

// One warp per request, lanes = 32 consecutive blocks. The masks are
// AND-scanned across lanes; lane j's "death set" is the local tiers held
// through block j-1 but not through block j. Lanes with a non-empty death set
// append an event (block, set) to the warp's list in shared memory; a request
// has at most one event per instance and usually two or three in all. The
// global-tier run is the first lane whose block the global tier lacks. Then
// lanes = instances: c_i = the block of the first event containing i (or n_r
// if i held every block), the cost, and a shuffle argmin with ties to the
// lowest id.
//
// One pass over every request. A member's blocks before `share` are its
// leader's, whose masks and chunk ANDs the probe wrote (the member's own were
// not probed there): its walk reads them from the leader up to block
// `share` (a 32-block chunk that straddles `share` block by block), then its
// own. Every request's run ends (c_i for every instance, then g) go to
// `summ` for the sequential variant.
template <int W, int DECIDE>
__global__ void __launch_bounds__(kMatchWarps * 32, 5)
    k_walk(int N, int B, const int64_t* __restrict__ off, const int64_t* __restrict__ block_off, int32_t n,
           const int64_t* __restrict__ load, int64_t w_load, int64_t w_miss, int64_t w_glob,
           const uint64_t* __restrict__ masks, const uint64_t* __restrict__ chunk_and,
           const int64_t* __restrict__ chunk_off, const int32_t* __restrict__ batch_ok,
           const int32_t* __restrict__ lead, const int32_t* __restrict__ share, int32_t* __restrict__ summ,
           int32_t* __restrict__ inst_out, int32_t* __restrict__ lhit_out,
           int32_t* __restrict__ ghit_out, uint4* __restrict__ groups, int64_t group_vecs,
           const WalkPolicy pol) {
  pdl_enter();
  extern __shared__ int64_t msm[];
  int64_t* load_s = msm;                                                     // [N]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // per warp: N events of (block, W mask words)
  uint64_t* ev_mask = reinterpret_cast<uint64_t*>(msm + N) + (size_t)warp * N * W;
  int64_t* ev_pos = msm + N + (size_t)kMatchWarps * N * W + (size_t)warp * N;
  for (int i = threadIdx.x; i < N; i += blockDim.x) load_s[i] = load[i];
  __syncthreads();
  const bool ok = *batch_ok != 0;
  const int gword = N >> 6;
  const uint64_t gbit = 1ull << (N & 63);
  const int64_t tw = (int64_t)gridDim.x * kMatchWarps;
  const unsigned lt = (1u << lane) - 1;

  if (!ok)
    for (int64_t r = (int64_t)blockIdx.x * kMatchWarps + warp; r < n; r += tw)
      if (lane == 0) {
        inst_out[r] = -1; lhit_out[r] = 0; ghit_out[r] = 0;
        if (DECIDE == kSession || DECIDE == kColoc) pol.stick[r] = 0;
      }
  for (int64_t r = (int64_t)blockIdx.x * kMatchWarps + warp; ok && r < n; r += tw) {
    const int64_t L = off[r + 1] - off[r];
    const int64_t nb = L / B;
    const int64_t bo = block_off[r];
    const int64_t sh = share[r];  // 0 for a leader
    const int32_t l = sh > 0 ? lead[r] : (int32_t)r;
    // chunk ANDs are per request-aligned chunk: blocks 32q .. 32q + 31 of
    // request r at index chunk_off[r] + q; block p < sh of the request is
    // block p of its leader
    const int64_t cbase = __ldg(chunk_off + r);
    const int64_t lbo = sh > 0 ? __ldg(block_off + l) : bo;
    const int64_t lcb = sh > 0 ? __ldg(chunk_off + l) : cbase;
    auto mask_at = [&](int64_t p, int w) -> uint64_t {  // block p of the request
      return __ldg(masks + ((p < sh ? lbo : bo) + p) * W + w);
    };
    auto and_at = [&](int64_t q, int w) -> uint64_t {  // its chunk q; 0 where the chunk straddles sh
      if (32 * (q + 1) <= sh) return __ldg(chunk_and + (lcb + q) * W + w);
      if (32 * q < sh) return 0ull;  // walked block by block
      return __ldg(chunk_and + (cbase + q) * W + w);
    };
    int64_t f = bo;
    const int64_t F1 = bo + nb;
    const bool head_single = F1 - f < 32;
    uint64_t pre[W];
#pragma unroll
    for (int w = 0; w < W; ++w) {
      if (head_single) {
        const int64_t len = F1 - f;
        pre[w] = lane < len ? mask_at(lane, w) : ~0ull;
      } else {
        pre[w] = lane < (nb >> 5) ? and_at(lane, w) : 0;
      }
    }
    constexpr int CT = 2 * W;  // groups of 32 covering the N + 1 <= 64 W tiers
    uint64_t A[W];  // local tiers holding every block so far (warp-uniform)
    bool galive = true;
    int64_t g = 0;
#pragma unroll
    for (int w = 0; w < W; ++w) {
      const int lo = w * 64;
      A[w] = N >= lo + 64 ? ~0ull : (N > lo ? (1ull << (N - lo)) - 1 : 0ull);
    }
    int ne = 0;
    // `len` consecutive blocks from request block `base`, lane j < len holding
    // block base + j (lanes past len hold all ones): the runs that end there
    // become events; returns true once no run is alive
    auto span = [&](int64_t base, int len, const uint64_t (&x)[W]) -> bool {
      if (galive) {
        uint64_t mg = 0;
#pragma unroll
        for (int w = 0; w < W; ++w) if (w == gword) mg = x[w];
        const unsigned miss = __ballot_sync(kFull, !(mg & gbit));
        if (miss) { g = base + __ffs(miss) - 1; galive = false; }
        else g = base + len;
      }
      bool dies = false, any = false;
      uint64_t X[W];
#pragma unroll
      for (int w = 0; w < W; ++w) {
        uint64_t v = x[w];
#pragma unroll
        for (int dd = 1; dd < 32; dd <<= 1) {
          const uint64_t y = __shfl_up_sync(kFull, v, dd);
          if (lane >= dd) v &= y;
        }
        v &= A[w];                                     // held through block base + lane
        const uint64_t prev = __shfl_up_sync(kFull, v, 1);
        X[w] = (lane ? prev : A[w]) & ~v;              // runs that end at block base + lane
        dies |= X[w] != 0;
        A[w] = __shfl_sync(kFull, v, 31);
        any |= A[w] != 0;
      }
      const unsigned ev = __ballot_sync(kFull, dies);
      if (dies) {
        const int at = ne + __popc(ev & lt);
        ev_pos[at] = base + lane;
#pragma unroll
        for (int w = 0; w < W; ++w) ev_mask[at * W + w] = X[w];
      }
      ne += __popc(ev);
      return !any && !galive;
    };
    bool dead = !galive;
#pragma unroll
    for (int w = 0; w < W; ++w) dead &= A[w] == 0;
    // From block sh: single blocks up to a 32-aligned request position, then
    // 32 chunks per step from their AND summaries (lane = chunk); the first
    // chunk that ends an alive run is walked block by block, and the request's
    // last partial chunk too. The first step uses the loads issued above.
    bool first = true;
    while (!dead && f < F1) {
      uint64_t x[W];
      if (((f - bo) & 31) || F1 - f < 32) {
        const int len = (int)min((int64_t)(32 - ((f - bo) & 31)), F1 - f);
#pragma unroll
        for (int w = 0; w < W; ++w)
          x[w] = first ? pre[w] : lane < len ? mask_at(f - bo + lane, w) : ~0ull;
        first = false;
        dead = span(f - bo, len, x);
        f += len;
        continue;
      }
      const int64_t nfull = (F1 - f) >> 5;
#pragma unroll
      for (int w = 0; w < W; ++w) x[w] = first ? pre[w] : lane < nfull ? and_at(((f - bo) >> 5) + lane, w) : 0;
      first = false;
      bool stop = lane >= nfull;
#pragma unroll
      for (int w = 0; w < W; ++w) {
        stop |= (x[w] & A[w]) != A[w];
        if (w == gword && galive) stop |= !(x[w] & gbit);
      }
      const unsigned sm = __ballot_sync(kFull, stop);
      const int j = sm ? __ffs(sm) - 1 : 32;
      f += 32 * (int64_t)j;  // chunks that keep every alive run
      if (galive) g = f - bo;
      if (j < nfull && j < 32) {
#pragma unroll
        for (int w = 0; w < W; ++w) x[w] = mask_at(f - bo + lane, w);
        dead = span(f - bo, 32, x);
        f += 32;
      }
    }
    if (galive) g = nb;  // the global run reaches the last block
    __syncwarp();
    // per instance (lanes = instances): c_i, then the decision
    int64_t best_cost = INT64_MAX;
    int32_t best = N;
    int64_t best_c = 0;
    // policies: prev = argmax c (lowest id); the balance key per instance:
    // 2*estimate_load (Figure 10), or the 128-bit product 2*estimate_load *
    // requests (colocation: over the candidates passing the TPOT check, and
    // over all instances for when none passes); ties rotate from s0
    int64_t pc = -1, pe = INT64_MAX, pec = 0;
    int32_t pi = N, prot = N;
    bool meets_any = false, cand_any = false;
    uint64_t ahi = ~0ull, alo = ~0ull, chi = ~0ull, clo = ~0ull;
    int32_t arot = N, crot = N;
    int64_t ac = 0, cc = 0;
    auto less128 = [](uint64_t h1, uint64_t l1, int32_t r1, uint64_t h2, uint64_t l2, int32_t r2) {
      return h1 < h2 || (h1 == h2 && (l1 < l2 || (l1 == l2 && r1 < r2)));
    };
    int64_t lmax = 0;  // Bailian: the largest batch size
    if (DECIDE == kBailian) {
      for (int i = lane; i < N; i += 32) lmax = max(lmax, __ldg(pol.nreq + i));
#pragma unroll
      for (int dd = 16; dd > 0; dd >>= 1) lmax = max(lmax, __shfl_xor_sync(kFull, lmax, dd));
    }
    const int32_t s0 = DECIDE == kSession || DECIDE == kColoc ? (int32_t)(((int64_t)pol.rr_base + r) % N) : 0;
    const int64_t budget2 = DECIDE == kSession || DECIDE == kColoc ? 2 * (pol.d0 + pol.d1 * L) : 0;
    int32_t* const out_c = summ + r * (N + 1);
#pragma unroll
    for (int t = 0; t < CT; ++t) {
      const int i = 32 * t + lane;
      if (i >= N) break;
      const int wi = i >> 6;
      const uint64_t bi = 1ull << (i & 63);
      uint64_t aw = 0;
#pragma unroll
      for (int w = 0; w < W; ++w) if (w == wi) aw = A[w];
      int64_t ci = nb;
      if (!(aw & bi)) {
        for (int e = 0; e < ne; ++e)
          if (ev_mask[e * W + wi] & bi) { ci = ev_pos[e]; break; }
      }
      out_c[i] = (int32_t)ci;  // every request's run ends (for the sequential variant)
      if (DECIDE == kArgmin) {
        const int64_t gi = ci > g ? ci : g;
        const int64_t cost = w_load * load_s[i] + w_miss * (L - B * gi) + w_glob * B * (gi - ci);
        if (cost < best_cost) { best_cost = cost; best = i; best_c = ci; }
      } else if (DECIDE == kLMetric) {
        // (q_i + L - B c_i) * l_i, below 2^61
        const int64_t f = (load_s[i] + L - B * ci) * __ldg(pol.nreq + i);
        if (less128(0, (uint64_t)f, i, ahi, alo, arot)) { ahi = 0; alo = (uint64_t)f; arot = i; ac = ci; }
      } else if (DECIDE == kBailian) {
        // f_i * LAM_DEN * max l * L = (LAM_DEN - LAM_NUM) l_i L + LAM_NUM (L - B c_i) max l, in 128 bits
        const uint64_t Lm = lmax > 0 ? (uint64_t)lmax : 1, Lr = L > 0 ? (uint64_t)L : 1;
        const uint64_t a1 = lmax > 0 ? (uint64_t)((pol.lam_den - pol.lam_num) * __ldg(pol.nreq + i)) : 0;
        const uint64_t a2 = (uint64_t)pol.lam_num * (L > 0 ? (uint64_t)(L - B * ci) : 1);
        const uint64_t l1 = a1 * Lr, h1 = __umul64hi(a1, Lr), l2 = a2 * Lm, h2 = __umul64hi(a2, Lm);
        const uint64_t lo = l1 + l2, hi = h1 + h2 + (lo < l1 ? 1 : 0);
        if (less128(hi, lo, i, ahi, alo, arot)) { ahi = hi; alo = lo; arot = i; ac = ci; }
      } else {
        // Eq. 1 doubled: 2*c_lin*n + c_att*n*(2L - n), n = new tokens, plus 2*q_i
        const int64_t nn = L - B * ci;
        const int64_t cost2 = 2 * pol.c_lin * nn + pol.c_att * nn * (2 * L - nn);
        const int64_t est2 = 2 * load_s[i] + cost2;
        meets_any |= est2 <= budget2;
        if (ci > pc) { pc = ci; pi = i; }  // lanes see their instances in increasing order
        const int32_t rot = (int32_t)((i - s0 + N) % N);
        if (DECIDE == kSession) {
          if (est2 < pe || (est2 == pe && rot < prot)) { pe = est2; prot = rot; pec = ci; }
        } else {
          const bool cand = cost2 <= 2 * __ldg(pol.tpot + i);
          const uint64_t R = (uint64_t)__ldg(pol.nreq + i);
          const uint64_t lo = (uint64_t)est2 * R, hi = __umul64hi((uint64_t)est2, R);
          cand_any |= cand;
          if (less128(hi, lo, rot, ahi, alo, arot)) { ahi = hi; alo = lo; arot = rot; ac = ci; }
          if (cand && less128(hi, lo, rot, chi, clo, crot)) { chi = hi; clo = lo; crot = rot; cc = ci; }
        }
      }
    }
    if (lane == 0) out_c[N] = (int32_t)g;
    if (DECIDE == kBailian || DECIDE == kLMetric) {
#pragma unroll
      for (int dd = 16; dd > 0; dd >>= 1) {
        const uint64_t oh = __shfl_xor_sync(kFull, ahi, dd), ol = __shfl_xor_sync(kFull, alo, dd);
        const int32_t oi = __shfl_xor_sync(kFull, arot, dd);
        const int64_t oc2 = __shfl_xor_sync(kFull, ac, dd);
        if (less128(oh, ol, oi, ahi, alo, arot)) { ahi = oh; alo = ol; arot = oi; ac = oc2; }
      }
      if (lane == 0) {
        const int64_t gb = ac > g ? ac : g;
        inst_out[r] = arot;
        lhit_out[r] = (int32_t)(B * ac);
        ghit_out[r] = (int32_t)(B * (gb - ac));
      }
    } else if (DECIDE == kArgmin) {
#pragma unroll
      for (int dd = 16; dd > 0; dd >>= 1) {
        const int64_t oc = __shfl_xor_sync(kFull, best_cost, dd);
        const int32_t oi = __shfl_xor_sync(kFull, best, dd);
        const int64_t ocb = __shfl_xor_sync(kFull, best_c, dd);
        if (oc < best_cost || (oc == best_cost && oi < best)) { best_cost = oc; best = oi; best_c = ocb; }
      }
      if (lane == 0) {
        const int64_t gb = best_c > g ? best_c : g;
        inst_out[r] = best;
        lhit_out[r] = (int32_t)(B * best_c);
        ghit_out[r] = (int32_t)(B * (gb - best_c));
      }
    } else {
#pragma unroll
      for (int dd = 16; dd > 0; dd >>= 1) {
        const int64_t oc = __shfl_xor_sync(kFull, pc, dd);
        const int32_t oi = __shfl_xor_sync(kFull, pi, dd);
        if (oc > pc || (oc == pc && oi < pi)) { pc = oc; pi = oi; }
        if (DECIDE == kSession) {
          const int64_t oe = __shfl_xor_sync(kFull, pe, dd);
          const int32_t orot = __shfl_xor_sync(kFull, prot, dd);
          const int64_t oec = __shfl_xor_sync(kFull, pec, dd);
          if (oe < pe || (oe == pe && orot < prot)) { pe = oe; prot = orot; pec = oec; }
        } else {
          uint64_t oh = __shfl_xor_sync(kFull, ahi, dd), ol = __shfl_xor_sync(kFull, alo, dd);
          int32_t orot = __shfl_xor_sync(kFull, arot, dd);
          int64_t oc2 = __shfl_xor_sync(kFull, ac, dd);
          if (less128(oh, ol, orot, ahi, alo, arot)) { ahi = oh; alo = ol; arot = orot; ac = oc2; }
          oh = __shfl_xor_sync(kFull, chi, dd);
          ol = __shfl_xor_sync(kFull, clo, dd);
          orot = __shfl_xor_sync(kFull, crot, dd);
          oc2 = __shfl_xor_sync(kFull, cc, dd);
          if (less128(oh, ol, orot, chi, clo, crot)) { chi = oh; clo = ol; crot = orot; cc = oc2; }
        }
      }
      const bool any = __any_sync(kFull, meets_any);
      const bool cands = __any_sync(kFull, cand_any);
      if (lane == 0) {
        const int64_t np = L - B * pc;
        const int64_t cost2p = 2 * pol.c_lin * np + pol.c_att * np * (2 * L - np);
        const int64_t est2p = 2 * load_s[pi] + cost2p;
        const bool cached = B * pc * pol.hit_den > pol.hit_num * pol.est_hit[r];
        bool stick;
        int32_t to;
        int64_t ct;
        if (DECIDE == kSession) {
          stick = pol.turn[r] != 0 && cached && (est2p <= budget2 || !any);
          to = stick ? pi : (int32_t)((s0 + prot) % N);
          ct = stick ? pc : pec;
        } else {
          const bool prev_cand = !cands || cost2p <= 2 * __ldg(pol.tpot + pi);
          stick = pol.turn[r] != 0 && cached && est2p <= budget2 && prev_cand;
          to = stick ? pi : (int32_t)((s0 + (cands ? crot : arot)) % N);
          ct = stick ? pc : (cands ? cc : ac);
        }
        const int64_t gt = ct > g ? ct : g;
        inst_out[r] = to;
        lhit_out[r] = (int32_t)(B * ct);
        ghit_out[r] = (int32_t)(B * (gt - ct));
        pol.stick[r] = stick ? 1 : 0;
      }
    }
    __syncwarp();
  }
  // the group stage has read the group table: empty it for the next route
  // (it is zero from index creation before the first)
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < group_vecs;
       i += (int64_t)gridDim.x * blockDim.x)
    groups[i] = make_uint4(0, 0, 0, 0);
}

// ---------------------------------------------------------------------------
// sequential-update variant
// ---------------------------------------------------------------------------

// One warp, requests in batch order: the a4-a5 argmin over the run ends the
// walk recorded (summ: c_i for every instance, then g) with the current
// loads, then the chosen load grows by L_r - B*c_{i*}. The next request's
// row is loaded while this one is decided.
__global__ void __launch_bounds__(32)
    k_seq(int N, int B, const int64_t* __restrict__ off, int32_t n, const int64_t* __restrict__ load,
          int64_t w_load, int64_t w_miss, int64_t w_glob, const int32_t* __restrict__ summ,
          const int32_t* __restrict__ batch_ok, int32_t* __restrict__ inst_out, int32_t* __restrict__ lhit_out,
          int32_t* __restrict__ ghit_out, int64_t* __restrict__ load_after, int32_t* status) {
  __shared__ int64_t q[SMETRIC_MAX_INSTANCES];
  const int lane = threadIdx.x;
  if (!*batch_ok) return;  // the route already wrote the invalid batch's outputs
  int64_t top = 0;
  for (int i = lane; i < N; i += 32) { q[i] = load[i]; top = max(top, q[i]); }
#pragma unroll
  for (int dd = 16; dd > 0; dd >>= 1) top = max(top, __shfl_xor_sync(kFull, top, dd));
  if (top + (off[n] - off[0]) > (1LL << 42)) {
    for (int32_t r = lane; r < n; r += 32) { inst_out[r] = -1; lhit_out[r] = 0; ghit_out[r] = 0; }
    if (lane == 0) latch_error(status, SMETRIC_ERR_OVERFLOW);
    return;
  }
  __syncwarp();
  constexpr int MT = (SMETRIC_MAX_INSTANCES + 1 + 31) / 32;  // row entries per lane
  int32_t cur[MT], nxt[MT];
  auto load_row = [&](int32_t r, int32_t (&dst)[MT]) {
#pragma unroll
    for (int t = 0; t < MT; ++t) {
      const int i = 32 * t + lane;
      dst[t] = r < n && i <= N ? summ[(int64_t)r * (N + 1) + i] : 0;
    }
  };
  load_row(0, cur);
  for (int32_t r = 0; r < n; ++r) {
    load_row(r + 1, nxt);
    const int64_t L = off[r + 1] - off[r];
    const int32_t g = __shfl_sync(kFull, cur[N >> 5], N & 31);
    int64_t best_cost = INT64_MAX, best_c = 0;
    int32_t best = N;
#pragma unroll
    for (int t = 0; t < MT; ++t) {
      const int i = 32 * t + lane;
      if (i < N) {
        const int64_t ci = cur[t], gi = ci > g ? ci : g;
        const int64_t cost = w_load * q[i] + w_miss * (L - B * gi) + w_glob * B * (gi - ci);
        if (cost < best_cost) { best_cost = cost; best = i; best_c = ci; }
      }
    }
#pragma unroll
    for (int dd = 16; dd > 0; dd >>= 1) {
      const int64_t oc = __shfl_xor_sync(kFull, best_cost, dd);
      const int32_t oi = __shfl_xor_sync(kFull, best, dd);
      const int64_t ocb = __shfl_xor_sync(kFull, best_c, dd);
      if (oc < best_cost || (oc == best_cost && oi < best)) { best_cost = oc; best = oi; best_c = ocb; }
    }
    if (lane == 0) {
      const int64_t gb = best_c > g ? best_c : g;
      inst_out[r] = best;
      lhit_out[r] = (int32_t)(B * best_c);
      ghit_out[r] = (int32_t)(B * (gb - best_c));
      q[best] += L - B * best_c;
    }
    __syncwarp();
#pragma unroll
    for (int t = 0; t < MT; ++t) cur[t] = nxt[t];
  }
  if (load_after)
    for (int i = lane; i < N; i += 32) load_after[i] = q[i];
}

// ---------------------------------------------------------------------------
// reuse breakdown
// ---------------------------------------------------------------------------

uint64_t reuse_slots_for(int64_t n_blocks) {
  uint64_t g = 64;
  while (g < 2 * (uint64_t)n_blocks) g <<= 1;
  return g;
}

// The first table tried holds an eighth of the window's blocks at load 1/2
// (67 MB for 16M blocks, so it stays in L2); windows whose distinct blocks
// exceed that fall back on the device to the full table, sized for every
// block distinct.
uint64_t reuse_small_slots_for(int64_t n_blocks) { return reuse_slots_for((n_blocks + 7) / 8); }
constexpr int kReuseSmallProbe = 64;  // longer probes in the first table also fall back

// Workspace header after the table: [0] the fallback flag, [1] distinct keys
// in the first table.
struct ReuseHeader {
  int32_t big;
  uint32_t distinct;
  uint32_t next[3];  // work counters of the two inserts and the walk
  uint32_t pad[3];
};

// Warps take requests from a counter in arrival order, so that a warp done
// with a short request takes the next one instead of idling behind a long one.
__device__ __forceinline__ int64_t next_request(uint32_t* ctr, int lane) {
  uint32_t r = 0;
  if (lane == 0) r = atomicAdd(ctr, 1u);
  return __shfl_sync(kFull, r, 0);
}

// Rounds of 32 blocks that a warp loads ahead before it uses them.
constexpr int kReuseAhead = 4;

// Warp per request, 32 blocks per round: each block's hash into the table
// with the earliest request holding it and that request's session, packed as
// (INT32_MAX - request) << 32 | session so that atomicMax keeps the earliest.
// A slot that already names an earlier (or the same) request is left alone,
// which spares most atomics: warps take requests in arrival order, so the
// first holder of a shared block is usually in before its later ones. The
// pre-checks are plain loads, so a block every request shares (a system
// prompt) is read from L1; a stale copy only shows an empty key or a smaller
// value, and both fall through to the atomics. The order of a request's
// blocks does not matter, so each request starts at a round of its own and
// wraps around, which spreads the requests in flight over the table.
// BIG = false fills the first table and raises the fallback flag when it
// runs full (more distinct keys than limit, or a probe longer than
// kReuseSmallProbe); BIG = true runs only after that, on the cleared full
// table.
template <bool BIG>
__global__ void __launch_bounds__(256)
    k_reuse_insert(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ batch_ok,
                   const uint64_t* __restrict__ H, const int32_t* __restrict__ sessions,
                   uint64_t* __restrict__ table, uint64_t mask, ReuseHeader* hdr, uint32_t limit) {
  if (!*batch_ok) return;
  if (BIG && !__ldcg(&hdr->big)) return;
  const int lane = threadIdx.x & 31;
  for (int64_t r = next_request(&hdr->next[BIG], lane); r < n; r = next_request(&hdr->next[BIG], lane)) {
    if (!BIG && __shfl_sync(kFull, lane == 0 ? __ldcg(&hdr->big) : 0, 0)) return;
    const int64_t bo = block_off[r], nb = block_off[r + 1] - bo;
    const unsigned long long val = ((unsigned long long)(INT32_MAX - r) << 32) | (uint32_t)sessions[r];
    const int64_t rounds = (nb + 31) >> 5;
    const int64_t start = rounds ? r % rounds : 0;
    uint32_t fresh_n = 0;
    for (int64_t i = 0; i < rounds; i += kReuseAhead) {
      int64_t b[kReuseAhead];
      uint64_t key[kReuseAhead];
      ulonglong2 sl[kReuseAhead];
#pragma unroll
      for (int u = 0; u < kReuseAhead; ++u) {
        int64_t rd = start + i + u;
        rd = rd >= rounds ? rd - rounds : rd;
        b[u] = i + u < rounds ? rd * 32 + lane : nb;
        key[u] = b[u] < nb ? H[bo + b[u]] : 0;
      }
#pragma unroll
      for (int u = 0; u < kReuseAhead; ++u)
        if (b[u] < nb) sl[u] = *reinterpret_cast<const ulonglong2*>(table + 2 * (key[u] & mask));
      bool full = false;
#pragma unroll
      for (int u = 0; u < kReuseAhead; ++u) {
        // already held by this or an earlier request: nothing to do
        if (b[u] >= nb || (sl[u].x == key[u] && sl[u].y >= val)) continue;
        uint64_t s = key[u] & mask;
        const uint64_t probes = BIG ? mask + 1 : kReuseSmallProbe;
        bool placed = false;
        for (uint64_t t = 0; t < probes; ++t) {
          unsigned long long* const slot = reinterpret_cast<unsigned long long*>(table + 2 * s);
          unsigned long long k = slot[0];
          if (k == 0ull) {
            k = atomicCAS(slot, 0ull, (unsigned long long)key[u]);
            fresh_n += k == 0ull;
          }
          if (k == 0ull || k == key[u]) {
            if (slot[1] < val) atomicMax(slot + 1, val);
            placed = true;
            break;
          }
          s = (s + 1) & mask;
        }
        full |= !placed;
      }
      if (!BIG && __any_sync(kFull, full)) {
        if (lane == 0) atomicExch(&hdr->big, 1);
        return;
      }
    }
    if (!BIG) {
      for (int o = 16; o; o >>= 1) fresh_n += __shfl_xor_sync(kFull, fresh_n, o);
      if (lane == 0 && fresh_n && atomicAdd(&hdr->distinct, fresh_n) + fresh_n > limit) atomicExch(&hdr->big, 1);
    }
  }
}

// Clears the full table once the first one has run full.
__global__ void __launch_bounds__(256) k_reuse_clear(const ReuseHeader* hdr, uint4* table, int64_t n16) {
  if (!*reinterpret_cast<const volatile int32_t*>(&hdr->big)) return;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16; i += (int64_t)gridDim.x * blockDim.x)
    table[i] = make_uint4(0, 0, 0, 0);
}

// Warp per request, 32 blocks per round: block b is reused when its earliest
// holder precedes the request; the run stops at the first block that is not.
// Reused blocks split into system prompt (b < sys_r), intra-session (the
// holder is of r's session) and inter-session.
__global__ void __launch_bounds__(256)
    k_reuse_walk(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ batch_ok,
                 const uint64_t* __restrict__ H, const uint64_t* __restrict__ table, uint64_t mask_small,
                 uint64_t mask_big, ReuseHeader* hdr, const int32_t* __restrict__ sessions,
                 const int32_t* __restrict__ sys_blocks,
                 int32_t* __restrict__ hit, int32_t* __restrict__ sys, int32_t* __restrict__ intra,
                 int32_t* __restrict__ inter, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const bool ok = *batch_ok != 0;
  const uint64_t mask = hdr->big ? mask_big : mask_small;
  for (int64_t r = next_request(&hdr->next[2], lane); r < n; r = next_request(&hdr->next[2], lane)) {
    int32_t nh = 0, ns = 0, ni = 0, ne = 0;
    if (ok) {
      const int64_t bo = block_off[r], nb = block_off[r + 1] - bo;
      int64_t sb = sys_blocks[r];
      if (sb < 0) {
        if (lane == 0) latch_error(status, SMETRIC_ERR_INVALID_ARG);
        sb = 0;
      }
      const int32_t sr = sessions[r];
      bool stop = false;
      for (int64_t base = 0; base < nb && !stop; base += 32 * kReuseAhead) {
        uint64_t key[kReuseAhead];
        ulonglong2 sl[kReuseAhead];
#pragma unroll
        for (int u = 0; u < kReuseAhead; ++u) {
          const int64_t b = base + 32 * u + lane;
          key[u] = b < nb ? H[bo + b] : 0;
        }
#pragma unroll
        for (int u = 0; u < kReuseAhead; ++u)
          if (base + 32 * u + lane < nb) sl[u] = *reinterpret_cast<const ulonglong2*>(table + 2 * (key[u] & mask));
#pragma unroll
        for (int u = 0; u < kReuseAhead; ++u) {
          const int64_t b = base + 32 * u + lane;
          int32_t producer = INT32_MAX, psess = 0;
          if (b < nb) {
            uint64_t s = key[u] & mask;
            ulonglong2 e = sl[u];
            for (uint64_t t = 0; t <= mask; ++t) {
              if (e.x == key[u]) {
                producer = INT32_MAX - (int32_t)(e.y >> 32);
                psess = (int32_t)(uint32_t)e.y;
                break;
              }
              if (e.x == 0) break;
              s = (s + 1) & mask;
              e = *reinterpret_cast<const ulonglong2*>(table + 2 * s);
            }
          }
          const bool reused = b < nb && producer < r;
          const unsigned miss = __ballot_sync(kFull, !reused);
          const unsigned run = miss ? (1u << (__ffs(miss) - 1)) - 1 : kFull;  // lanes before the first miss
          const bool in = (run >> lane) & 1;
          const bool is_sys = in && b < sb;
          const bool is_intra = in && !is_sys && psess == sr;
          nh += __popc(run);
          ns += __popc(__ballot_sync(kFull, is_sys));
          ni += __popc(__ballot_sync(kFull, is_intra));
          ne += __popc(__ballot_sync(kFull, in && !is_sys && !is_intra));
          if (miss) {
            stop = true;
            break;
          }
        }
      }
    }
    if (lane == 0) {
      hit[r] = ok ? nh : -1;
      sys[r] = ok ? ns : -1;
      intra[r] = ok ? ni : -1;
      inter[r] = ok ? ne : -1;
    }
  }
}

// ---------------------------------------------------------------------------
// session links
// ---------------------------------------------------------------------------

// Fingerprint of (user, turn, number of blocks, last block hash) for the
// session-link table; 0 marks an empty slot.
__device__ __forceinline__ uint64_t link_key(int64_t user, int64_t turn, int64_t nb, uint64_t last) {
  uint64_t x = mix64((uint64_t)user ^ kGamma);
  x = mix64(x ^ (uint64_t)turn);
  x = mix64(x ^ (uint64_t)nb);
  x = mix64(x ^ last);
  return x ? x : 1;
}

// Thread per request p: (key, p) into the table (a multi-map: every request
// takes its own slot), and parent[p] = -1.
__global__ void __launch_bounds__(256)
    k_link_insert(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ batch_ok,
                  const uint64_t* __restrict__ H, const int64_t* __restrict__ users,
                  const int32_t* __restrict__ turns, uint64_t* __restrict__ table, uint64_t gmask,
                  int32_t* __restrict__ parent) {
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= n || !*batch_ok) return;
  parent[p] = -1;
  const int64_t bo = block_off[p], nb = block_off[p + 1] - bo;
  const uint64_t key = link_key(users[p], turns[p], nb, nb ? H[bo + nb - 1] : 0);
  uint64_t s = key & gmask;
  for (uint64_t t = 0; t <= gmask; ++t) {
    unsigned long long* const slot = reinterpret_cast<unsigned long long*>(table + 2 * s);
    if (atomicCAS(slot, 0ull, (unsigned long long)key) == 0ull) {
      slot[1] = (unsigned long long)p;
      return;
    }
    s = (s + 1) & gmask;
  }
}

// Thread per (request r, prefix length k <= n_r): the latest earlier request
// of r's user, of turn turn_r - 1, with exactly k blocks, the last equal to
// r's block k - 1, raises parent[r] to it. Candidates from the table are
// checked field by field.
__global__ void __launch_bounds__(256)
    k_link_find(const int64_t* __restrict__ block_off, int32_t n, const int32_t* __restrict__ batch_ok,
                const uint64_t* __restrict__ H, const int64_t* __restrict__ users,
                const int32_t* __restrict__ turns, const uint64_t* __restrict__ table, uint64_t gmask,
                int32_t* __restrict__ parent) {
  if (!*batch_ok) return;
  const int64_t total = block_off[n] + n;  // sum over r of n_r + 1
  int32_t r = 0;
  for (int64_t f = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; f < total;
       f += (int64_t)gridDim.x * blockDim.x) {
    int32_t lo = r, hi = n;  // largest r with block_off[r] + r <= f
    while (hi - lo > 1) {
      const int32_t mid = (lo + hi) >> 1;
      if (__ldg(block_off + mid) + mid <= f) lo = mid; else hi = mid;
    }
    r = lo;
    const int64_t bo = __ldg(block_off + r), k = f - (bo + r);
    const int64_t user = users[r], turn = (int64_t)turns[r] - 1;
    const uint64_t last = k ? __ldg(H + bo + k - 1) : 0;
    const uint64_t key = link_key(user, turn, k, last);
    int32_t best = -1;
    uint64_t s = key & gmask;
    for (uint64_t t = 0; t <= gmask; ++t) {
      const uint64_t kk = __ldg(table + 2 * s);
      if (kk == 0) break;
      if (kk == key) {
        const int32_t p = (int32_t)__ldg(table + 2 * s + 1);
        const int64_t pbo = __ldg(block_off + p);
        if (p < r && p > best && users[p] == user && (int64_t)turns[p] == turn &&
            __ldg(block_off + p + 1) - pbo == k && (k == 0 || __ldg(H + pbo + k - 1) == last))
          best = p;
      }
      s = (s + 1) & gmask;
    }
    if (best >= 0) atomicMax(parent + r, best);
  }
}

// One CTA: session[r] = the head of r's chain of parents (pointer jumping;
// parents are earlier requests, so every chain ends), then the link table
// emptied for the next route.
__global__ void __launch_bounds__(1024)
    k_link_heads(int32_t n, const int32_t* __restrict__ batch_ok, int32_t* __restrict__ parent,
                 int32_t* __restrict__ session, uint4* __restrict__ table, int64_t table_vecs) {
  if (*batch_ok) {
    for (int32_t r = threadIdx.x; r < n; r += blockDim.x) session[r] = parent[r] < 0 ? r : parent[r];
    __syncthreads();
    for (int64_t span = 1; span < n; span <<= 1) {
      for (int32_t r = threadIdx.x; r < n; r += blockDim.x) {
        const int32_t a = session[r];
        session[r] = session[a];  // an ancestor either way: the heads are reached all the same
      }
      __syncthreads();
    }
  } else {  // invalid offsets: no links
    for (int32_t r = threadIdx.x; r < n; r += blockDim.x) { parent[r] = -1; session[r] = -1; }
  }
  for (int64_t i = threadIdx.x; i < table_vecs; i += blockDim.x) table[i] = make_uint4(0, 0, 0, 0);
}

// ---------------------------------------------------------------------------
// commit
// ---------------------------------------------------------------------------

// Checks of a batch to commit and the queue drain: one CTA checks every
// request's instance (in [-1, N)) and local hit (in [0, L_r]); a bad value
// clears the batch flag, so that nothing is committed and the loads stay as
// they were. Otherwise, with `load`, it sums per instance the tokens each
// request routed there must prefill or fetch (L_r - local hit) and sets
// load_i <- (load_i + that sum) >> 1. Integer sums, so the order of the
// atomics does not matter.
__global__ void __launch_bounds__(1024)
    k_drain(const int64_t* __restrict__ off, int32_t n, int N, const int32_t* __restrict__ instance,
            const int32_t* __restrict__ local_hit, int32_t* __restrict__ batch_ok,
            int64_t* __restrict__ load, int32_t* status) {
  __shared__ unsigned long long acc[SMETRIC_MAX_INSTANCES];
  __shared__ int bad;
  if (threadIdx.x == 0) bad = 0;
  for (int i = threadIdx.x; i < N; i += blockDim.x) acc[i] = 0;
  __syncthreads();
  if (!*batch_ok) return;  // invalid offsets
  for (int64_t r = threadIdx.x; r < n; r += blockDim.x) {
    const int32_t i = instance[r];
    const int64_t L = off[r + 1] - off[r], h = local_hit ? local_hit[r] : 0;
    if (i < -1 || i >= N || h < 0 || h > L) { bad = 1; continue; }
    if (i >= 0 && load) atomicAdd(&acc[i], (unsigned long long)(L - h));
  }
  __syncthreads();
  if (bad) {
    if (threadIdx.x == 0) {
      *batch_ok = 0;
      latch_error(status, SMETRIC_ERR_INVALID_ARG);
    }
    return;
  }
  if (load)
    for (int i = threadIdx.x; i < N; i += blockDim.x) load[i] = (load[i] + (int64_t)acc[i]) >> 1;
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

void profile_mark(smetric_index* idx, int k, cudaStream_t s);

// How a batch shares the GPU with the batch after it (smetric_route_batches
// on two scratch sets): an event recorded once its chain and probe are
// enqueued, which the next batch's first kernel waits for.
struct Overlap {
  cudaEvent_t after_chain;
};

// Launches a route kernel; with pdl the launch may begin while the previous
// kernel on the stream is still running (the kernel waits in pdl_enter).
template <typename... KArgs, typename... Args>
int launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl,
             Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = pdl ? attr : nullptr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cuda_status(cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...));
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, looked up once (thread-safe static init).
EncodeTiledFn tensor_map_encoder() {
  static const EncodeTiledFn fn = [] {
    EncodeTiledFn f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&f), 12000,
                                         cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      f = nullptr;
    return f;
  }();
  return fn;
}

// One map per 16-byte phase k of a row start: base tokens + 16k, rows of
// 4B+16 bytes at stride 4B, as many rows as fit inside the token buffer.
bool make_token_maps(TokenMaps& m, const int32_t* tokens, int64_t n_tokens, int B) {
  EncodeTiledFn enc = tensor_map_encoder();
  if (!enc) return false;
  memset(&m, 0, sizeof(m));
  const int64_t bytes = 4 * n_tokens, row = 4 * B + 16, stride = 4 * B;
  for (int k = 0; k < B / 4; ++k) {
    const int64_t base = 16 * k;
    if (bytes < base + row) continue;  // rows[k] = 0: chunks fall back to lane copies
    int64_t rows = (bytes - base - row) / stride + 1;
    if (rows > INT32_MAX) rows = INT32_MAX;
    const cuuint64_t dims[2] = {(cuuint64_t)(B + 4), (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)stride};
    const cuuint32_t box[2] = {(cuuint32_t)(B + 4), (cuuint32_t)kChunk};
    const cuuint32_t es[2] = {1, 1};
    if (enc(&m.map[k], CU_TENSOR_MAP_DATA_TYPE_UINT32, 2,
            const_cast<char*>(reinterpret_cast<const char*>(tokens)) + base, dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return false;
    m.rows[k] = (uint32_t)rows;
  }
  return true;
}

// Group-table slots a batch of n requests uses: a power of two >= 2n.
uint64_t group_slots_for(int32_t n) {
  uint64_t g = 64;
  while (g < 2 * (uint64_t)n) g <<= 1;
  return g;
}

// The digest kernel for the index's block size; with `group` it also puts
// each request's first-block hash into the group table.
template <int HB>
int launch_digest(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                  const int64_t* d_offsets, int32_t n, cudaStream_t s, bool group) {
  const int B = idx->cfg.block_size;
  const uint64_t d_init = mix64(idx->cfg.hash_seed ^ (uint64_t)B);
  const uint64_t h_init = mix64(idx->cfg.hash_seed + kGamma);
  uint64_t* const groups = group ? idx->groups : nullptr;
  const uint64_t gmask = group_slots_for(n) - 1;
  // request-aligned chunks (TMA kernel) number at most blocks / 32 + n
  const int64_t max_chunks = (n_tokens / B + kChunk - 1) / kChunk + (HB > 0 ? n : 0);
  // rows of 16*nch bytes: a block's 4B bytes start at most 12 bytes past a
  // 16-byte boundary
  const int nch = HB > 0 ? HB / 2 + 1 : (4 * B + 12 + 15) / 16;
  if (HB > 0 && B / 4 <= kMaxPhases) {
    static thread_local TokenMaps maps;
    if (make_token_maps(maps, d_tokens, n_tokens, B)) {
      auto kern = k_digest_tma<(HB > 0 ? HB : 2), kTmaStages>;
      const size_t per_warp = (size_t)kTmaStages * kChunk * nch * 16 + 8 * kTmaStages;
      const int warps = kTmaWarps;
      const size_t smem = (size_t)warps * per_warp;
      if (idx->digest_occ == 0) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
          return cuda_status(cudaErrorInvalidValue);
        int occ = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, warps * 32, smem) != cudaSuccess)
          return cuda_status(cudaErrorInvalidValue);
        idx->digest_occ = occ < 1 ? 1 : occ;
      }
      const int64_t want = (max_chunks + warps - 1) / warps;
      const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * idx->digest_occ));
      idx->launches++;
      return launch_k(kern, dim3((unsigned)grid), dim3(warps * 32), smem, s, !idx->profiling, maps, d_tokens,
                      n_tokens, d_offsets, (const int64_t*)idx->block_off, (const int64_t*)idx->chunk_off, n, d_init,
                      (const int32_t*)idx->batch_ok, idx->digest, idx->status, groups, gmask, h_init);
    }
  }
  const size_t per_warp = (size_t)kChunk * nch * 16;
  const int warps = (int)std::max<size_t>(1, std::min<size_t>(kDigestWarps, (200 * 1024) / per_warp));
  const size_t smem = (size_t)warps * per_warp;
  auto kern = HB > 0 ? k_digest<HB> : nullptr;
  const void* fn = HB > 0 ? (const void*)kern : (const void*)k_digest_any;
  if (idx->digest_occ == 0) {  // once per index: B, and so the plan, is fixed
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return cuda_status(cudaErrorInvalidValue);
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fn, warps * 32, smem) != cudaSuccess)
      return cuda_status(cudaErrorInvalidValue);
    idx->digest_occ = occ < 1 ? 1 : occ;
  }
  const int64_t want = (max_chunks + warps - 1) / warps;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * idx->digest_occ));
  idx->launches++;
  if (HB > 0)
    return launch_k(kern, dim3((unsigned)grid), dim3(warps * 32), smem, s, !idx->profiling, d_tokens, n_tokens,
                    d_offsets, (const int64_t*)idx->block_off, n, d_init, (const int32_t*)idx->batch_ok,
                    idx->digest, groups, gmask, h_init);
  return launch_k(k_digest_any, dim3((unsigned)grid), dim3(warps * 32), smem, s, !idx->profiling, d_tokens,
                  n_tokens, d_offsets, (const int64_t*)idx->block_off, n, B, nch, d_init,
                  (const int32_t*)idx->batch_ok, idx->digest, groups, gmask, h_init);
}

int dispatch_digest(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                    const int64_t* d_offsets, int32_t n, cudaStream_t s, bool group) {
  switch (idx->cfg.block_size) {
    case 16: return launch_digest<8>(idx, d_tokens, n_tokens, d_offsets, n, s, group);
    case 32: return launch_digest<16>(idx, d_tokens, n_tokens, d_offsets, n, s, group);
    case 64: return launch_digest<32>(idx, d_tokens, n_tokens, d_offsets, n, s, group);
    default: return launch_digest<0>(idx, d_tokens, n_tokens, d_offsets, n, s, group);
  }
}

int launch_chain(smetric_index* idx, const int64_t* d_offsets, int32_t n, uint64_t* hashes,
                 uint64_t* sk, bool pdl, cudaStream_t s) {
  const unsigned grid = (unsigned)((n + kChainThreads - 1) / kChainThreads);
  const uint64_t h_init = mix64(idx->cfg.hash_seed + kGamma);
  idx->launches++;
  return launch_k(k_chain, dim3(grid), dim3(kChainThreads), 0, s, pdl, d_offsets, idx->block_off, n,
                  idx->cfg.block_size, idx->cfg.session_blocks, h_init, idx->batch_ok, idx->digest,
                  hashes ? hashes : idx->hashes, sk);
}

template <int W>
int launch_match(smetric_index* idx, const int64_t* d_offsets, int32_t n, const int64_t* d_load,
                 smetric_weights w, int32_t* inst, int32_t* lhit, int32_t* ghit, uint64_t* hashes,
                 uint64_t* sk, int64_t max_blocks, const WalkPolicy& pol, cudaStream_t s,
                 const Overlap* ov) {
  const cudaEvent_t after_chain = ov ? ov->after_chain : nullptr;
  const int N = idx->cfg.num_instances;
  int rc;
  {
    // chain, group leaders and shared prefixes, and probe: one CTA per SM,
    // a chain lane for each request a CTA owns (1 to 4 warps; more requests
    // are taken in groups)
    const int grid = idx->num_sms;
    const int64_t per_cta = ((int64_t)n + grid - 1) / grid;
    const int chain_warps = (int)std::max<int64_t>(1, std::min<int64_t>(kCpMaxChainWarps, (per_cta + 31) / 32));
    const size_t smem = (size_t)chain_warps * 32 * kCpRingBytes;
    // leader flags, one byte a request, in the scratch words k_link_sessions uses for its keys
    uint8_t* const flags = reinterpret_cast<uint8_t*>(idx->sk_tmp);
    idx->launches++;
    if ((rc = launch_k(k_lead, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, !idx->profiling,
                       (const int64_t*)idx->block_off, n, (const int32_t*)idx->batch_ok, (const uint64_t*)idx->digest,
                       mix64(idx->cfg.hash_seed + kGamma), (const uint64_t*)idx->groups, group_slots_for(n) - 1,
                       flags)))
      return rc;
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(k_chain_probe<W>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return cuda_status(cudaErrorInvalidValue);
    idx->launches++;
    if ((rc = launch_k(k_chain_probe<W>, dim3((unsigned)grid), dim3(kCpWarps * 32), smem, s, !idx->profiling,
                       (const int64_t*)idx->block_off, (const int64_t*)idx->chunk_off, n, idx->cfg.session_blocks,
                       mix64(idx->cfg.hash_seed + kGamma), (const int32_t*)idx->batch_ok,
                       (const uint64_t*)idx->digest, hashes ? hashes : idx->hashes, sk, (const uint64_t*)idx->groups,
                       group_slots_for(n) - 1, idx->lead, idx->share, (const uint8_t*)idx->tags,
                       (const uint64_t*)idx->table, idx->n_buckets, idx->masks, idx->chunk_and,
                       (const uint8_t*)flags, chain_warps, idx->status)))
      return rc;
    if (after_chain && cudaEventRecord(after_chain, s) != cudaSuccess) return cuda_status(cudaErrorUnknown);
  }
  profile_mark(idx, kChainProbe, s);
  const size_t smem = (size_t)N * sizeof(int64_t) + (size_t)kMatchWarps * N * (W + 1) * sizeof(uint64_t);
  const int64_t want = ((int64_t)n + kMatchWarps - 1) / kMatchWarps;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * 8));
  // every request in one pass (members read their leaders' probes)
  using WalkKernel = decltype(&k_walk<W, kArgmin>);  // every instantiation has this signature
  const WalkKernel kerns[5] = {k_walk<W, kArgmin>, k_walk<W, kSession>, k_walk<W, kColoc>, k_walk<W, kBailian>,
                               k_walk<W, kLMetric>};
  const WalkKernel kern = kerns[pol.on];
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return cuda_status(cudaErrorInvalidValue);
  idx->launches++;
  if ((rc = launch_k(kern, dim3((unsigned)grid), dim3(kMatchWarps * 32), smem, s, !idx->profiling, N,
                     idx->cfg.block_size, d_offsets, idx->block_off, n, d_load, w.w_load, w.w_miss, w.w_glob,
                     idx->masks, idx->chunk_and, (const int64_t*)idx->chunk_off, idx->batch_ok, idx->lead,
                     idx->share, idx->summ, inst, lhit, ghit, reinterpret_cast<uint4*>(idx->groups),
                     (int64_t)group_slots_for(n), pol)))
    return rc;
  return SMETRIC_OK;
}

int dispatch_match(smetric_index* idx, const int64_t* d_offsets, int32_t n, const int64_t* d_load,
                   smetric_weights w, int32_t* inst, int32_t* lhit, int32_t* ghit, uint64_t* hashes,
                   uint64_t* sk, int64_t max_blocks, const WalkPolicy& pol, cudaStream_t s,
                   const Overlap* ov) {
  switch (idx->W) {
    case 1: return launch_match<1>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, hashes, sk, max_blocks, pol, s, ov);
    case 2: return launch_match<2>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, hashes, sk, max_blocks, pol, s, ov);
    case 3: return launch_match<3>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, hashes, sk, max_blocks, pol, s, ov);
    case 4: return launch_match<4>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, hashes, sk, max_blocks, pol, s, ov);
    case 5: return launch_match<5>(idx, d_offsets, n, d_load, w, inst, lhit, ghit, hashes, sk, max_blocks, pol, s, ov);
    default: return SMETRIC_ERR_INVALID_ARG;
  }
}

void profile_begin(smetric_index* idx, cudaStream_t s) {
  if (!idx->profiling) return;
  ProfileSlot slot;
  if (!idx->prof_pool.empty()) {
    slot = idx->prof_pool.back();
    idx->prof_pool.pop_back();
  } else {
    for (auto& e : slot.ev)
      if (cudaEventCreate(&e) != cudaSuccess) return;
  }
  idx->prof_used.push_back(slot);
  cudaEventRecord(idx->prof_used.back().ev[0], s);
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
                 int32_t* ghit, uint64_t* sk, uint64_t* hashes, int64_t hashes_cap, cudaStream_t s,
                 const WalkPolicy* pol = nullptr, const Overlap* ov = nullptr) {
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
  // the policies' Eq. 1 arithmetic has its own limits on queues and lengths
  const bool eq1 = pol && (pol->on == kSession || pol->on == kColoc);
  k_prep<<<1, 1024, 0, s>>>(d_offsets, n, n_tokens, c.block_size, d_load, PROBE ? c.num_instances : 0,
                            idx->block_off, idx->chunk_off, idx->batch_ok, idx->status,
                            eq1 ? SMETRIC_POLICY_MAX_QUEUED : SMETRIC_MAX_LOAD,
                            eq1 ? SMETRIC_POLICY_MAX_LEN : (int64_t)INT32_MAX, pol ? pol->est_hit : nullptr,
                            pol ? pol->tpot : nullptr, SMETRIC_POLICY_MAX_TPOT,
                            pol ? pol->nreq : nullptr, SMETRIC_POLICY_MAX_REQUESTS);
  idx->launches++;
  if ((rc = cuda_status(cudaGetLastError()))) return rc;
  profile_mark(idx, kPrep, s);
  // a route's digests also fill the group table (each request's first-block hash)
  if (n_tokens / c.block_size > 0) {
    if ((rc = dispatch_digest(idx, d_tokens, n_tokens, d_offsets, n, s, PROBE)))
      return rc;
  }
  profile_mark(idx, kDigest, s);
  if (PROBE) {
    const WalkPolicy off_pol = {};
    if ((rc = dispatch_match(idx, d_offsets, n, d_load, w, inst, lhit, ghit, hashes, sk,
                             n_tokens / c.block_size, pol ? *pol : off_pol, s, ov)))
      return rc;
  } else {
    if ((rc = launch_chain(idx, d_offsets, n, hashes, sk, !idx->profiling, s))) return rc;
    profile_mark(idx, kChainProbe, s);
  }
  profile_mark(idx, kWalk, s);
  return SMETRIC_OK;
}

int route_policy(smetric_index* idx, int mode, const int32_t* d_tokens, int64_t n_tokens,
                 const int64_t* d_offsets, int32_t n_requests, const int64_t* d_queued,
                 const int64_t* d_tpot, const int64_t* d_nreq, const int32_t* d_turn,
                 const int64_t* d_est_hit, smetric_policy p, int32_t* d_instance, int32_t* d_local_hit,
                 int32_t* d_global_hit, int32_t* d_stick, uint64_t* d_session_key, uint64_t* d_block_hashes,
                 int64_t hashes_cap, smetric_stream_t stream) {
  if (!idx) return SMETRIC_ERR_INVALID_ARG;
  const int64_t N = idx->cfg.num_instances;
  if (p.c_lin < 0 || p.c_lin > (1LL << 20) || p.c_att < 0 || p.c_att > (1LL << 12) || p.ttft_d0 < 0 ||
      p.ttft_d0 > (1LL << 60) || p.ttft_d1 < 0 || p.ttft_d1 > (1LL << 35) || p.hit_den < 1 ||
      p.hit_den > (1LL << 20) || p.hit_num < 0 || p.hit_num > p.hit_den || p.rr_base < 0 || p.rr_base >= N ||
      p.reserved != 0)
    return SMETRIC_ERR_INVALID_ARG;
  if (n_requests > 0 && (!d_turn || !d_est_hit || !d_stick)) return SMETRIC_ERR_INVALID_ARG;
  WalkPolicy pol;
  pol.on = mode;
  pol.c_lin = p.c_lin;
  pol.c_att = p.c_att;
  pol.d0 = p.ttft_d0;
  pol.d1 = p.ttft_d1;
  pol.hit_num = p.hit_num;
  pol.hit_den = p.hit_den;
  pol.rr_base = p.rr_base;
  pol.turn = d_turn;
  pol.est_hit = d_est_hit;
  pol.stick = d_stick;
  pol.tpot = d_tpot;
  pol.nreq = d_nreq;
  // the argmin weights are unused by the policy; any valid ones pass the checks
  return route_common<true>(idx, d_tokens, n_tokens, d_offsets, n_requests, d_queued, smetric_weights{0, 0, 0},
                            d_instance, d_local_hit, d_global_hit, d_session_key, d_block_hashes, hashes_cap,
                            reinterpret_cast<cudaStream_t>(stream), &pol);
}

}  // namespace

#include <mutex>
#include <new>
#include <unordered_map>

#include "call_range.cuh"

// ---------------------------------------------------------------------------
// batches overlapped on two scratch sets
// ---------------------------------------------------------------------------

namespace smetric {

// The second route scratch set of an index created with SMETRIC_FLAG_PIPELINE:
// the same buffers, with the same sizes, as the index's own set.
struct RouteScratchSet {
  int64_t* block_off = nullptr;
  int64_t* chunk_off = nullptr;
  uint64_t* digest = nullptr;
  uint64_t* hashes = nullptr;
  uint64_t* masks = nullptr;
  uint64_t* chunk_and = nullptr;
  uint64_t* groups = nullptr;
  int32_t* lead = nullptr;  // lead, then share at lead + max_batch_requests + 1
  int32_t* summ = nullptr;
  uint64_t* sk_tmp = nullptr;
  int32_t* batch_ok = nullptr;
};

struct Pipeline {
  RouteScratchSet alt;
  cudaStream_t stream = nullptr;                   // runs the batches that use `alt`
  cudaEvent_t chain_done[2] = {nullptr, nullptr};  // per set: its latest batch's chain has finished
  cudaEvent_t start = nullptr, finish = nullptr;   // the caller's stream to `stream`, and back
};

// Both live until the process ends and are never destroyed, so that an index
// destroyed late in process exit still finds them.
static std::mutex& pipeline_mutex() {
  static std::mutex* m = new std::mutex;
  return *m;
}

// Indexes created with SMETRIC_FLAG_PIPELINE and their second sets (kept
// beside the index so that the index's layout stays as it is).
static std::unordered_map<const smetric_index*, Pipeline*>& pipelines() {
  static auto* table = new std::unordered_map<const smetric_index*, Pipeline*>;
  return *table;
}

static Pipeline* pipeline_of(const smetric_index* idx) {
  std::lock_guard<std::mutex> lock(pipeline_mutex());
  auto it = pipelines().find(idx);
  return it == pipelines().end() ? nullptr : it->second;
}

static void free_pipeline(Pipeline* p) {
  RouteScratchSet& a = p->alt;
  cudaFree(a.block_off);
  cudaFree(a.chunk_off);
  cudaFree(a.digest);
  cudaFree(a.hashes);
  cudaFree(a.masks);
  cudaFree(a.chunk_and);
  cudaFree(a.groups);
  cudaFree(a.lead);
  cudaFree(a.summ);
  cudaFree(a.sk_tmp);
  cudaFree(a.batch_ok);
  if (p->stream) cudaStreamDestroy(p->stream);
  for (cudaEvent_t e : {p->chain_done[0], p->chain_done[1], p->start, p->finish})
    if (e) cudaEventDestroy(e);
  delete p;
}

// Exchanges the index's route scratch with set `a` (host pointers only: a
// launch takes the pointers current when it is enqueued).
static void swap_scratch(smetric_index* x, RouteScratchSet& a) {
  std::swap(x->block_off, a.block_off);
  std::swap(x->chunk_off, a.chunk_off);
  std::swap(x->digest, a.digest);
  std::swap(x->hashes, a.hashes);
  std::swap(x->masks, a.masks);
  std::swap(x->chunk_and, a.chunk_and);
  std::swap(x->groups, a.groups);
  std::swap(x->lead, a.lead);
  x->share = x->lead + (x->cfg.max_batch_requests + 1);
  std::swap(x->summ, a.summ);
  std::swap(x->sk_tmp, a.sk_tmp);
  std::swap(x->batch_ok, a.batch_ok);
}

// Allocates the second set of index x (called by smetric_index_create once
// the index's own set exists). The sizes are those of the index's own set.
int pipeline_attach(smetric_index* x) {
  const smetric_index_config& c = x->cfg;
  const size_t R = (size_t)c.max_batch_requests;
  const size_t max_blocks = (size_t)(c.max_batch_tokens / c.block_size);
  const size_t nb = max_blocks > 0 ? max_blocks : 1;
  const size_t W = (size_t)x->W;
  Pipeline* p = new (std::nothrow) Pipeline();
  if (!p) return SMETRIC_ERR_OOM;
  RouteScratchSet& a = p->alt;
  bool ok = cudaMalloc(&a.block_off, (R + 1) * sizeof(int64_t)) == cudaSuccess &&
            cudaMalloc(&a.digest, (nb + 2) * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&a.hashes, nb * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&a.masks, nb * W * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&a.chunk_and, (max_blocks / 32 + R + 1) * W * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&a.groups, 2 * x->group_slots * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&a.lead, 2 * (R + 1) * sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&a.chunk_off, (R + 1) * sizeof(int64_t)) == cudaSuccess &&
            cudaMalloc(&a.sk_tmp, (R + 1) * sizeof(uint64_t)) == cudaSuccess &&
            cudaMalloc(&a.summ, (R > 0 ? R : 1) * ((size_t)c.num_instances + 1) * sizeof(int32_t)) == cudaSuccess &&
            cudaMalloc(&a.batch_ok, sizeof(int32_t)) == cudaSuccess &&
            cudaMemset(a.groups, 0, 2 * x->group_slots * sizeof(uint64_t)) == cudaSuccess &&
            cudaStreamCreateWithFlags(&p->stream, cudaStreamNonBlocking) == cudaSuccess;
  for (cudaEvent_t* e : {&p->chain_done[0], &p->chain_done[1], &p->start, &p->finish})
    ok = ok && cudaEventCreateWithFlags(e, cudaEventDisableTiming) == cudaSuccess;
  if (!ok) {
    (void)cudaGetLastError();
    free_pipeline(p);
    return SMETRIC_ERR_OOM;
  }
  std::lock_guard<std::mutex> lock(pipeline_mutex());
  pipelines()[x] = p;
  return SMETRIC_OK;
}

// Frees the second set of index x, if it has one (the device is idle).
void pipeline_release(smetric_index* x) {
  Pipeline* p = nullptr;
  {
    std::lock_guard<std::mutex> lock(pipeline_mutex());
    auto it = pipelines().find(x);
    if (it == pipelines().end()) return;
    p = it->second;
    pipelines().erase(it);
  }
  free_pipeline(p);
}

}  // namespace smetric

namespace {

// smetric_route_batches: the host checks of route_common for every batch
// first, then the batches, alternating between the two sets when the index
// has a second one. Batch j's first kernel waits for batch j - 1's chain and
// probe kernel, so that batch j's prep and digests (bound by the integer
// pipe) run beside batch j - 1's walk (bound by latency), and batch j - 1's
// chain does not share the GPU with batch j's digests.
int route_batches(smetric_index* idx, int32_t nb, const int32_t* const* tok, const int64_t* ntok,
                  const int64_t* const* off, const int32_t* nreq, const int64_t* const* load, smetric_weights w,
                  int32_t* const* inst, int32_t* const* lhit, int32_t* const* ghit, uint64_t* const* sk,
                  cudaStream_t s) {
  int rc = check_device(idx);
  if (rc) return rc;
  if (nb < 0 || (nb > 0 && (!tok || !ntok || !off || !nreq || !load || !inst || !lhit || !ghit || !sk)))
    return SMETRIC_ERR_INVALID_ARG;
  const smetric_index_config& c = idx->cfg;
  for (int32_t j = 0; j < nb; ++j) {
    const int32_t n = nreq[j];
    const int64_t nt = ntok[j];
    if (n < 0 || n > c.max_batch_requests || nt < 0 || nt > c.max_batch_tokens) return SMETRIC_ERR_INVALID_ARG;
    if (n == 0) continue;
    if (!off[j] || !sk[j] || (nt > 0 && !tok[j])) return SMETRIC_ERR_INVALID_ARG;
    if (tok[j] && (reinterpret_cast<uintptr_t>(tok[j]) & 15)) return SMETRIC_ERR_INVALID_ARG;
    if (!load[j] || !inst[j] || !lhit[j] || !ghit[j] || !weights_ok(w)) return SMETRIC_ERR_INVALID_ARG;
  }
  Pipeline* p = pipeline_of(idx);
  if (!p || idx->profiling || nb < 2) {
    for (int32_t j = 0; j < nb; ++j)
      if ((rc = route_common<true>(idx, tok[j], ntok[j], off[j], nreq[j], load[j], w, inst[j], lhit[j], ghit[j],
                                   sk[j], nullptr, 0, s)))
        return rc;
    return SMETRIC_OK;
  }
  // the second stream starts from everything enqueued on the caller's stream
  if (cudaEventRecord(p->start, s) != cudaSuccess || cudaStreamWaitEvent(p->stream, p->start, 0) != cudaSuccess)
    return cuda_status(cudaErrorUnknown);
  for (int32_t j = 0; j < nb && rc == SMETRIC_OK; ++j) {
    const int set = j & 1;
    cudaStream_t sj = set ? p->stream : s;
    if (j > 0 && cudaStreamWaitEvent(sj, p->chain_done[set ^ 1], 0) != cudaSuccess) {
      rc = cuda_status(cudaErrorUnknown);
      break;
    }
    if (set) swap_scratch(idx, p->alt);
    const Overlap ov = {p->chain_done[set]};
    rc = route_common<true>(idx, tok[j], ntok[j], off[j], nreq[j], load[j], w, inst[j], lhit[j], ghit[j], sk[j],
                            nullptr, 0, sj, nullptr, &ov);
    if (set) swap_scratch(idx, p->alt);
  }
  // the caller's stream continues after the second stream's batches
  if (cudaEventRecord(p->finish, p->stream) != cudaSuccess || cudaStreamWaitEvent(s, p->finish, 0) != cudaSuccess)
    return rc ? rc : cuda_status(cudaErrorUnknown);
  return rc;
}

// smetric_index_commit_batch's steps; with prep the batch's block offsets
// and validity are computed here, else a route call just left them.
int commit_common(smetric_index* idx, const int64_t* d_offsets, int32_t n_requests, const int32_t* d_instance,
                  const int32_t* d_local_hit, const uint64_t* d_block_hashes, int32_t flags, int64_t* d_load,
                  cudaStream_t s, bool prep) {
  int rc = check_device(idx);
  if (rc) return rc;
  const smetric_index_config& c = idx->cfg;
  if (n_requests < 0 || n_requests > c.max_batch_requests || (flags & ~SMETRIC_COMMIT_GLOBAL))
    return SMETRIC_ERR_INVALID_ARG;
  if (n_requests == 0) return SMETRIC_OK;
  if (!d_offsets || !d_instance || !d_block_hashes || (d_load && !d_local_hit)) return SMETRIC_ERR_INVALID_ARG;
  if (prep) {
    // block offsets of the batch (and the offsets' checks) into the index's scratch
    k_prep<<<1, 1024, 0, s>>>(d_offsets, n_requests, c.max_batch_tokens, c.block_size, nullptr, 0, idx->block_off,
                              nullptr, idx->batch_ok, idx->status, SMETRIC_MAX_LOAD, (int64_t)INT32_MAX, nullptr);
    idx->launches++;
    if ((rc = cuda_status(cudaGetLastError()))) return rc;
  }
  // the checks (and the drain) first: a bad output commits nothing
  k_drain<<<1, 1024, 0, s>>>(d_offsets, n_requests, c.num_instances, d_instance, d_local_hit, idx->batch_ok,
                             d_load, idx->status);
  idx->launches++;
  if ((rc = cuda_status(cudaGetLastError()))) return rc;
  if ((rc = launch_commit(idx, d_instance, d_block_hashes, n_requests, c.max_batch_tokens / c.block_size,
                          (flags & SMETRIC_COMMIT_GLOBAL) != 0, s)))
    return rc;
  return lru_commit(idx, d_instance, d_block_hashes, n_requests, (flags & SMETRIC_COMMIT_GLOBAL) != 0, s);
}

}  // namespace

extern "C" {

int smetric_route_batch(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                        const int64_t* d_offsets, int32_t n_requests, const int64_t* d_load,
                        smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                        int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                        int64_t hashes_cap, smetric_stream_t stream) {
  CallRange range("smetric_route_batch");
  return route_common<true>(idx, d_tokens, n_tokens, d_offsets, n_requests, d_load, w, d_instance,
                            d_local_hit, d_global_hit, d_session_key, d_block_hashes, hashes_cap,
                            reinterpret_cast<cudaStream_t>(stream));
}

int smetric_route_batches(smetric_index* idx, int32_t n_batches, const int32_t* const* d_tokens,
                          const int64_t* n_tokens, const int64_t* const* d_offsets, const int32_t* n_requests,
                          const int64_t* const* d_load, smetric_weights w, int32_t* const* d_instance,
                          int32_t* const* d_local_hit, int32_t* const* d_global_hit,
                          uint64_t* const* d_session_key, smetric_stream_t stream) {
  CallRange range("smetric_route_batches");
  return route_batches(idx, n_batches, d_tokens, n_tokens, d_offsets, n_requests, d_load, w, d_instance,
                       d_local_hit, d_global_hit, d_session_key, reinterpret_cast<cudaStream_t>(stream));
}

int smetric_route_batch_sequential(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                                   const int64_t* d_offsets, int32_t n_requests, const int64_t* d_load,
                                   smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                                   int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                   int64_t hashes_cap, int64_t* d_load_after, smetric_stream_t stream) {
  CallRange range("smetric_route_batch_sequential");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int rc = route_common<true>(idx, d_tokens, n_tokens, d_offsets, n_requests, d_load, w, d_instance, d_local_hit,
                              d_global_hit, d_session_key, d_block_hashes, hashes_cap, s);
  if (rc || n_requests == 0) return rc;
  k_seq<<<1, 32, 0, s>>>(idx->cfg.num_instances, idx->cfg.block_size, d_offsets, n_requests, d_load, w.w_load,
                         w.w_miss, w.w_glob, idx->summ, idx->batch_ok, d_instance, d_local_hit, d_global_hit,
                         d_load_after, idx->status);
  idx->launches++;
  return cuda_status(cudaGetLastError());
}

int smetric_route_batch_baseline(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                                 const int64_t* d_offsets, int32_t n_requests, int32_t scorer,
                                 const int64_t* d_queued, const int64_t* d_batch, int64_t lam_num,
                                 int64_t lam_den, int32_t* d_instance, int32_t* d_local_hit,
                                 int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                 int64_t hashes_cap, smetric_stream_t stream) {
  CallRange range("smetric_route_batch_baseline");
  if (!idx || !d_batch || (scorer != SMETRIC_SCORER_BAILIAN && scorer != SMETRIC_SCORER_LMETRIC) ||
      lam_den < 1 || lam_den > (1LL << 20) || lam_num < 0 || lam_num > lam_den)
    return SMETRIC_ERR_INVALID_ARG;
  WalkPolicy pol = {};
  pol.on = scorer == SMETRIC_SCORER_BAILIAN ? kBailian : kLMetric;
  pol.nreq = d_batch;
  pol.lam_num = lam_num;
  pol.lam_den = lam_den;
  return route_common<true>(idx, d_tokens, n_tokens, d_offsets, n_requests, d_queued, smetric_weights{0, 0, 0},
                            d_instance, d_local_hit, d_global_hit, d_session_key, d_block_hashes, hashes_cap,
                            reinterpret_cast<cudaStream_t>(stream), &pol);
}

int smetric_route_batch_policy_coloc(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                                     const int64_t* d_offsets, int32_t n_requests, const int64_t* d_queued,
                                     const int64_t* d_tpot_budget, const int64_t* d_num_requests,
                                     const int32_t* d_turn, const int64_t* d_est_hit, smetric_policy p,
                                     int32_t* d_instance, int32_t* d_local_hit, int32_t* d_global_hit,
                                     int32_t* d_stick, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                     int64_t hashes_cap, smetric_stream_t stream) {
  CallRange range("smetric_route_batch_policy_coloc");
  if (!idx || !d_tpot_budget || !d_num_requests) return SMETRIC_ERR_INVALID_ARG;
  return route_policy(idx, kColoc, d_tokens, n_tokens, d_offsets, n_requests, d_queued, d_tpot_budget,
                      d_num_requests, d_turn, d_est_hit, p, d_instance, d_local_hit, d_global_hit, d_stick,
                      d_session_key, d_block_hashes, hashes_cap, stream);
}

int smetric_route_batch_policy(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                               const int64_t* d_offsets, int32_t n_requests, const int64_t* d_queued,
                               const int32_t* d_turn, const int64_t* d_est_hit, smetric_policy p,
                               int32_t* d_instance, int32_t* d_local_hit, int32_t* d_global_hit,
                               int32_t* d_stick, uint64_t* d_session_key, uint64_t* d_block_hashes,
                               int64_t hashes_cap, smetric_stream_t stream) {
  CallRange range("smetric_route_batch_policy");
  return route_policy(idx, kSession, d_tokens, n_tokens, d_offsets, n_requests, d_queued, nullptr, nullptr,
                      d_turn, d_est_hit, p, d_instance, d_local_hit, d_global_hit, d_stick, d_session_key,
                      d_block_hashes, hashes_cap, stream);
}


int smetric_index_commit_batch(smetric_index* idx, const int64_t* d_offsets, int32_t n_requests,
                               const int32_t* d_instance, const int32_t* d_local_hit,
                               const uint64_t* d_block_hashes, int32_t flags, int64_t* d_load,
                               smetric_stream_t stream) {
  CallRange range("smetric_index_commit_batch");
  return commit_common(idx, d_offsets, n_requests, d_instance, d_local_hit, d_block_hashes, flags, d_load,
                       reinterpret_cast<cudaStream_t>(stream), true);
}

int smetric_route_commit_batch(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                               const int64_t* d_offsets, int32_t n_requests, int64_t* d_load,
                               smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                               int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                               int64_t hashes_cap, int32_t flags, smetric_stream_t stream) {
  CallRange range("smetric_route_commit_batch");
  if ((flags & ~SMETRIC_COMMIT_GLOBAL) || !d_block_hashes) return SMETRIC_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int rc = route_common<true>(idx, d_tokens, n_tokens, d_offsets, n_requests, d_load, w, d_instance,
                                    d_local_hit, d_global_hit, d_session_key, d_block_hashes, hashes_cap, s);
  if (rc) return rc;
  // the route's prep left this batch's block offsets and validity in the scratch
  return commit_common(idx, d_offsets, n_requests, d_instance, d_local_hit, d_block_hashes, flags, d_load, s,
                       false);
}

int64_t smetric_reuse_workspace_bytes(int64_t n_blocks) {
  return n_blocks < 0 ? 0 : (int64_t)(2 * sizeof(uint64_t) * reuse_slots_for(n_blocks) + sizeof(ReuseHeader));
}

int smetric_reuse_breakdown(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                            const int64_t* d_offsets, int32_t n_requests, const int32_t* d_sessions,
                            const int32_t* d_sys_blocks, void* d_workspace, int64_t workspace_bytes,
                            int32_t* d_hit, int32_t* d_sys, int32_t* d_intra, int32_t* d_inter,
                            smetric_stream_t stream) {
  CallRange range("smetric_reuse_breakdown");
  int rc = check_device(idx);
  if (rc) return rc;
  if (n_requests < 0 || n_requests > idx->cfg.max_batch_requests || n_tokens < 0) return SMETRIC_ERR_INVALID_ARG;
  if (n_requests == 0) return SMETRIC_OK;
  const int64_t n_blocks = n_tokens / idx->cfg.block_size;
  if (!d_sessions || !d_sys_blocks || !d_hit || !d_sys || !d_intra || !d_inter || !d_workspace ||
      workspace_bytes < smetric_reuse_workspace_bytes(n_blocks) || (reinterpret_cast<uintptr_t>(d_workspace) & 15))
    return SMETRIC_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((rc = route_common<false>(idx, d_tokens, n_tokens, d_offsets, n_requests, nullptr, smetric_weights{0, 0, 0},
                                nullptr, nullptr, nullptr, idx->sk_tmp, idx->hashes, n_blocks, s)))
    return rc;
  const uint64_t slots = reuse_slots_for(n_blocks), small = reuse_small_slots_for(n_blocks);
  uint64_t* table = static_cast<uint64_t*>(d_workspace);
  ReuseHeader* hdr = reinterpret_cast<ReuseHeader*>(table + 2 * slots);
  if (cudaMemsetAsync(table, 0, 2 * sizeof(uint64_t) * small, s) != cudaSuccess ||
      cudaMemsetAsync(hdr, 0, sizeof(ReuseHeader), s) != cudaSuccess)
    return cuda_status(cudaErrorUnknown);
  const unsigned wgrid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(((int64_t)n_requests + 7) / 8,
                                                                          (int64_t)idx->num_sms * 8));
  k_reuse_insert<false><<<wgrid, 256, 0, s>>>(idx->block_off, n_requests, idx->batch_ok, idx->hashes, d_sessions,
                                              table, small - 1, hdr, (uint32_t)(small / 2));
  k_reuse_clear<<<idx->num_sms * 8, 256, 0, s>>>(hdr, reinterpret_cast<uint4*>(table), (int64_t)slots);
  k_reuse_insert<true><<<wgrid, 256, 0, s>>>(idx->block_off, n_requests, idx->batch_ok, idx->hashes, d_sessions,
                                             table, slots - 1, hdr, 0);
  k_reuse_walk<<<wgrid, 256, 0, s>>>(idx->block_off, n_requests, idx->batch_ok, idx->hashes, table, small - 1,
                                     slots - 1, hdr, d_sessions, d_sys_blocks, d_hit, d_sys, d_intra, d_inter,
                                     idx->status);
  idx->launches += 4;
  return cuda_status(cudaGetLastError());
}

int smetric_link_sessions(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                          const int64_t* d_offsets, int32_t n_requests, const int64_t* d_users,
                          const int32_t* d_turns, int32_t* d_parent, int32_t* d_session,
                          smetric_stream_t stream) {
  CallRange range("smetric_link_sessions");
  int rc = check_device(idx);
  if (rc) return rc;
  if (n_requests < 0 || n_requests > idx->cfg.max_batch_requests) return SMETRIC_ERR_INVALID_ARG;
  if (n_requests == 0) return SMETRIC_OK;
  if (!d_users || !d_turns || !d_parent || !d_session) return SMETRIC_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // block hashes of the batch into the index's scratch
  if ((rc = route_common<false>(idx, d_tokens, n_tokens, d_offsets, n_requests, nullptr, smetric_weights{0, 0, 0},
                                nullptr, nullptr, nullptr, idx->sk_tmp, idx->hashes,
                                n_tokens / idx->cfg.block_size, s)))
    return rc;
  const uint64_t gmask = group_slots_for(n_requests) - 1;
  const unsigned g = (unsigned)((n_requests + 255) / 256);
  k_link_insert<<<g, 256, 0, s>>>(idx->block_off, n_requests, idx->batch_ok, idx->hashes, d_users, d_turns,
                                  idx->groups, gmask, d_parent);
  const int64_t want = (n_tokens / idx->cfg.block_size + n_requests + 255) / 256;
  const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)idx->num_sms * 8));
  k_link_find<<<grid, 256, 0, s>>>(idx->block_off, n_requests, idx->batch_ok, idx->hashes, d_users, d_turns,
                                   idx->groups, gmask, d_parent);
  k_link_heads<<<1, 1024, 0, s>>>(n_requests, idx->batch_ok, d_parent, d_session,
                                  reinterpret_cast<uint4*>(idx->groups), (int64_t)(gmask + 1));
  idx->launches += 3;
  return cuda_status(cudaGetLastError());
}

int smetric_block_hashes(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                         const int64_t* d_offsets, int32_t n_requests, uint64_t* d_session_key,
                         uint64_t* d_block_hashes, int64_t hashes_cap, smetric_stream_t stream) {
  CallRange range("smetric_block_hashes");
  smetric_weights w{0, 0, 0};
  return route_common<false>(idx, d_tokens, n_tokens, d_offsets, n_requests, nullptr, w, nullptr,
                             nullptr, nullptr, d_session_key, d_block_hashes, hashes_cap,
                             reinterpret_cast<cudaStream_t>(stream));
}

int smetric_route_batch_host(smetric_index* idx, const int32_t* h_tokens, int64_t n_tokens,
                             const int64_t* h_offsets, int32_t n_requests, const int64_t* h_load,
                             smetric_weights w, int32_t* h_instance, int32_t* h_local_hit,
                             int32_t* h_global_hit, uint64_t* h_session_key, smetric_stream_t stream) {
  CallRange range("smetric_route_batch_host");
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
    case kChainProbe: return "k_chain_probe";
    case kWalk: return "k_walk";
    default: return "";
  }
}

}  // extern "C"

// ---------------------------------------------------------------------------
// block hashes with fixed scratch and no allocation
// ---------------------------------------------------------------------------

namespace {

// Word layout of the fixed scratch: the batch-valid flag, the per-request
// first-block offsets, the per-block digests. Each part starts on a 256-byte
// boundary. Nothing in it needs an initial value: every call writes the flag
// and the offsets before any kernel reads them, and the digests of exactly
// the blocks the chain reads.
constexpr int64_t kNaFlagWords = 32;
constexpr int64_t kNaOffWords = (SMETRIC_NOALLOC_MAX_REQUESTS + 1 + 31) / 32 * 32;
constexpr int64_t kNaWords = kNaFlagWords + kNaOffWords + SMETRIC_NOALLOC_MAX_BLOCKS;
static_assert(kNaWords * 8 == 295424, "the header states the scratch size");

static __device__ __align__(256) uint64_t na_scratch[kNaWords];

constexpr int kNaMaxDevices = 64;
std::atomic<uint64_t*> na_addr[kNaMaxDevices];

// Device address of na_scratch on the current device, looked up once per
// device (the first call on a device should not be under stream capture).
// The cached address is not refreshed after a device reset (a reset
// recreates the context and reloads the module).
int na_scratch_for(int dev, uint64_t** out) {
  if (dev < 0 || dev >= kNaMaxDevices) return SMETRIC_ERR_INVALID_ARG;
  uint64_t* p = na_addr[dev].load(std::memory_order_acquire);
  if (!p) {
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&p), na_scratch) != cudaSuccess)
      return cuda_status(cudaErrorInvalidSymbol);
    na_addr[dev].store(p, std::memory_order_release);
  }
  *out = p;
  return SMETRIC_OK;
}

template <int HB>
int na_digest(const int32_t* d_tokens, int64_t n_tokens, const int64_t* d_offsets, const int64_t* block_off,
              int32_t n, int B, int num_sms, uint64_t d_init, const int32_t* ok, uint64_t* digest,
              cudaStream_t s) {
  const int64_t max_chunks = (n_tokens / B + kChunk - 1) / kChunk;
  const int nch = HB > 0 ? HB / 2 + 1 : (4 * B + 12 + 15) / 16;
  const size_t per_warp = (size_t)kChunk * nch * 16;
  const int warps = (int)std::max<size_t>(1, std::min<size_t>(kDigestWarps, (200 * 1024) / per_warp));
  const size_t smem = (size_t)warps * per_warp;
  const void* fn = HB > 0 ? (const void*)k_digest<(HB > 0 ? HB : 2)> : (const void*)k_digest_any;
  int occ = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fn, warps * 32, smem) != cudaSuccess)
    return cuda_status(cudaErrorInvalidValue);
  const int64_t want = (max_chunks + warps - 1) / warps;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)num_sms * std::max(occ, 1)));
  if (HB > 0)
    k_digest<(HB > 0 ? HB : 2)><<<(unsigned)grid, warps * 32, smem, s>>>(d_tokens, n_tokens, d_offsets,
                                                                        block_off, n, d_init, ok, digest,
                                                                        nullptr, 0, 0);
  else
    k_digest_any<<<(unsigned)grid, warps * 32, smem, s>>>(d_tokens, n_tokens, d_offsets, block_off, n, B, nch,
                                                          d_init, ok, digest, nullptr, 0, 0);
  return cuda_status(cudaGetLastError());
}

}  // namespace

extern "C" int smetric_block_hashes_noalloc(const int32_t* d_tokens, int64_t n_tokens,
                                            const int64_t* d_offsets, int32_t n_requests, int32_t block_size,
                                            int32_t session_blocks, uint64_t hash_seed,
                                            uint64_t* d_session_key, uint64_t* d_block_hashes,
                                            int64_t hashes_cap, int32_t* d_status, smetric_stream_t stream) {
  const int B = block_size;
  if (B < 2 || B > 256 || (B & 1) || session_blocks < 1 || n_requests < 0 || n_tokens < 0)
    return SMETRIC_ERR_INVALID_ARG;
  if (n_requests > SMETRIC_NOALLOC_MAX_REQUESTS || n_tokens / B > SMETRIC_NOALLOC_MAX_BLOCKS)
    return SMETRIC_ERR_TOO_LARGE;
  if (n_requests == 0) return SMETRIC_OK;
  if (!d_offsets || !d_session_key || !d_block_hashes || !d_status || (n_tokens > 0 && !d_tokens))
    return SMETRIC_ERR_INVALID_ARG;
  if (d_tokens && (reinterpret_cast<uintptr_t>(d_tokens) & 15)) return SMETRIC_ERR_INVALID_ARG;
  if (hashes_cap < n_tokens / B) return SMETRIC_ERR_INVALID_ARG;
  int dev = 0, num_sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return cuda_status(cudaErrorInvalidDevice);
  uint64_t* scratch = nullptr;
  int rc = na_scratch_for(dev, &scratch);
  if (rc) return rc;
  int32_t* ok = reinterpret_cast<int32_t*>(scratch);
  int64_t* block_off = reinterpret_cast<int64_t*>(scratch + kNaFlagWords);
  uint64_t* digest = scratch + kNaFlagWords + kNaOffWords;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  k_prep<<<1, 1024, 0, s>>>(d_offsets, n_requests, n_tokens, B, nullptr, 0, block_off, nullptr, ok, d_status,
                            SMETRIC_MAX_LOAD, (int64_t)INT32_MAX, nullptr);
  if ((rc = cuda_status(cudaGetLastError()))) return rc;
  if (n_tokens / B > 0) {
    const uint64_t d_init = mix64(hash_seed ^ (uint64_t)B);
    switch (B) {
      case 16: rc = na_digest<8>(d_tokens, n_tokens, d_offsets, block_off, n_requests, B, num_sms, d_init, ok, digest, s); break;
      case 32: rc = na_digest<16>(d_tokens, n_tokens, d_offsets, block_off, n_requests, B, num_sms, d_init, ok, digest, s); break;
      case 64: rc = na_digest<32>(d_tokens, n_tokens, d_offsets, block_off, n_requests, B, num_sms, d_init, ok, digest, s); break;
      default: rc = na_digest<0>(d_tokens, n_tokens, d_offsets, block_off, n_requests, B, num_sms, d_init, ok, digest, s);
    }
    if (rc) return rc;
  }
  const unsigned grid = (unsigned)((n_requests + kChainThreads - 1) / kChainThreads);
  k_chain<<<grid, kChainThreads, 0, s>>>(d_offsets, block_off, n_requests, B, session_blocks,
                                         mix64(hash_seed + kGamma), ok, digest, d_block_hashes, d_session_key);
  return cuda_status(cudaGetLastError());
}
