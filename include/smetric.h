/*
 * smetric.h - C ABI of the batched routing path of balanced session-centric
 * scheduling (SMetric, arXiv 2607.08565), for one NVIDIA GB300 (sm_103a).
 *
 * For a batch of agent requests the library
 *   (a) chain-hashes each prompt's int32 tokens in blocks of B tokens,
 *   (b) derives a stateless session key from the leading S blocks,
 *   (c) longest-prefix-matches the block-hash chain against a two-tier KV$
 *       index (one local tier per serving instance plus one global tier),
 *   (d) scores every instance with an integer cost and takes the argmin.
 * The paper's router scores instances per request (Section 4.1, Figure 6:
 * each request goes to the instance minimising a function of c_i, the
 * prompt's prefix hit in instance i's local KV$, and l_i, its load) and keeps only
 * per-instance state (Section 4.2, Challenge 1); the two-tier store is the
 * local GPU tier plus the cluster-wide global tier (Section 2, Figure 2).
 *
 * Definitions (exact; every output is bit-reproducible):
 *   mix64(z)  SplitMix64 output function: z ^= z>>30; z *= 0xBF58476D1CE4E5B9;
 *             z ^= z>>27; z *= 0x94D049BB133111EB; z ^= z>>31 (mod 2^64).
 *   GAMMA     0x9E3779B97F4A7C15.
 *   w_{b,k}   (uint32)t[bB+2k] | (uint32)t[bB+2k+1] << 32, k < B/2.
 *   d_b       x = mix64(seed ^ B); for k: x = mix64(x ^ w_{b,k}); d_b = x.
 *   h_b       h_{-1} = mix64(seed + GAMMA); h_b = mix64((h_{b-1}+GAMMA) ^ d_b),
 *             then h_b |= 2 if h_b < 2. Only the n_r = floor(L_r/B) full
 *             blocks are hashed.
 *   sk_r      h_{min(n_r,S)-1}, or 0 if n_r = 0.
 *   c_i       largest k <= n_r with h_0..h_{k-1} all in instance i's local tier.
 *   g         largest k <= n_r with h_0..h_{k-1} all in the global tier.
 *   cost_i    w_load*load_i + w_miss*(L_r - B*max(c_i,g))
 *             + w_glob*B*(max(c_i,g) - c_i), in int64.
 *   i*        smallest i with minimal cost_i.
 * Every request of one batch sees the same index and load (snapshot).
 *
 * Conventions
 *   - "d_" pointers are device memory of the device that was current at
 *     smetric_index_create; "h_" pointers are host memory (pinned memory
 *     gives the fastest copies). The caller owns every buffer it passes.
 *   - Calls are stream-ordered: inserts, evictions and routes enqueued on one
 *     stream see each other's effects in enqueue order. Calls on one index
 *     share that index's scratch, so they must not run concurrently on
 *     different streams.
 *   - Host-detectable errors return immediately with nothing enqueued.
 *     Device-detectable errors (bad offsets, out-of-range tiers or loads, a
 *     full table) are latched in the index and reported by smetric_status.
 *   - Nothing here allocates device memory except smetric_index_create.
 */
#ifndef SMETRIC_H
#define SMETRIC_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* smetric_stream_t;

typedef struct smetric_index smetric_index; /* opaque, library-owned */

enum {
  SMETRIC_OK = 0,
  SMETRIC_ERR_INVALID_ARG = -1, /* bad argument, offsets, tier or key */
  SMETRIC_ERR_OOM = -2,         /* device allocation failed at create */
  SMETRIC_ERR_TABLE_FULL = -3,  /* an insert found no free slot */
  SMETRIC_ERR_CUDA = -4,        /* a CUDA runtime call failed */
  SMETRIC_ERR_OVERFLOW = -5,    /* a load or prompt length outside the exact int64 range */
  SMETRIC_ERR_TOO_LARGE = -6    /* batch larger than smetric_block_hashes_noalloc's fixed scratch */
};

/* Instance limit and the limits that keep every cost exact in int64:
 * |cost| < 3 * 2^20 * 2^40 < 2^63. */
#define SMETRIC_MAX_INSTANCES 256
#define SMETRIC_MAX_WEIGHT (1LL << 20)
#define SMETRIC_MAX_LOAD (1LL << 40)
/* An insert that visits SMETRIC_MAX_PROBE / 16 buckets (of 15 slots) without
 * finding its key or a free slot reports SMETRIC_ERR_TABLE_FULL; lookups
 * visit as many buckets at most. */
#define SMETRIC_MAX_PROBE 65536

/* smetric_index_config.flags */
#define SMETRIC_FLAG_HOST_STAGING 1 /* allocate device staging buffers for smetric_route_batch_host */
#define SMETRIC_FLAG_PIPELINE 2     /* allocate a second route scratch set for smetric_route_batches */

typedef struct {
  int32_t num_instances;      /* N, 1..SMETRIC_MAX_INSTANCES (local tiers 0..N-1) */
  int32_t block_size;         /* B, even, 2..256 tokens */
  int32_t session_blocks;     /* S >= 1: blocks that form the session key */
  int32_t flags;              /* SMETRIC_FLAG_* */
  uint64_t capacity_slots;    /* index slots, >= 1; size for a load factor <= 0.7 of the live keys */
  uint64_t hash_seed;         /* seed of the chain hash */
  int64_t max_batch_requests; /* largest n_requests a route call accepts */
  int64_t max_batch_tokens;   /* largest n_tokens a route call accepts */
} smetric_index_config;

/* Integer cost weights, each in [0, SMETRIC_MAX_WEIGHT]. */
typedef struct {
  int64_t w_load; /* per queued token of the instance (Figure 10(c): q_i) */
  int64_t w_miss; /* per token the instance must prefill */
  int64_t w_glob; /* per token fetched from the global tier (Section 1: slower, limited bandwidth) */
} smetric_weights;

/* Create an empty index and its route scratch on the current device.
 * The table holds capacity_slots (rounded up to a multiple of 15) entries of
 * 16, 32 or 64 bytes (key plus ceil((N+1)/64) tier-mask words, padded to a
 * power of two) and a 16-byte tag group per 15 slots (a tag byte per slot
 * and the bucket's overflow count). A key occupies a slot while some tier
 * holds it: evictions give slots back. The route scratch holds, in 64-bit
 * words, (2 + W) * (max_batch_tokens/B) for per-block digests, hashes and
 * tier masks, 2 * (max_batch_requests + 1) for per-request offsets, group
 * leaders and shared-block counts, and 2 * G for the group table, G the
 * smallest power of two >= max(64, 2 * max_batch_requests);
 * W = ceil((N+1)/64). SMETRIC_FLAG_PIPELINE allocates a second route scratch
 * of the same size (and two streams) for smetric_route_batches.
 * Returns SMETRIC_ERR_INVALID_ARG for an out-of-range field and
 * SMETRIC_ERR_OOM when a device allocation fails; *out is NULL then. */
int smetric_index_create(const smetric_index_config* cfg, smetric_index** out);

/* Free the index and its device memory. Waits for the device first.
 * NULL is accepted. */
int smetric_index_destroy(smetric_index* idx);

/* Empty every tier (Section 2, Figure 2: the KV$ store's contents). */
int smetric_index_clear(smetric_index* idx, smetric_stream_t stream);

/* Tier membership updates (Section 2: the local tier of each instance and the
 * global tier each cache KV$ blocks; the serving side reports which blocks
 * each tier holds). For each j < n: add key d_keys[j] to tier d_tiers[j]
 * (0..N-1 = local tier of that instance, -1 = global tier). Keys are block
 * hashes (>= 2). Set semantics: idempotent and order-independent within a
 * call. Errors latched: a key < 2 or tier out of range (INVALID_ARG, that
 * pair skipped), no free slot (TABLE_FULL). A tier the device LRU caps
 * (smetric_index_set_lru) is INVALID_ARG here: its keys enter through
 * smetric_index_commit_batch only. */
int smetric_index_insert(smetric_index* idx, const uint64_t* d_keys, const int32_t* d_tiers,
                         int64_t n, smetric_stream_t stream);

/* Remove key d_keys[j] from tier d_tiers[j]; absent pairs are ignored. A key
 * that leaves its last tier gives its slot back for later inserts. A tier the
 * device LRU caps is INVALID_ARG here (latched, pair skipped): it evicts on
 * its own. */
int smetric_index_evict(smetric_index* idx, const uint64_t* d_keys, const int32_t* d_tiers,
                        int64_t n, smetric_stream_t stream);

/* Tier masks of n keys: d_masks[j*W + w] is word w of key j's tier set
 * (bit i < N: local tier of instance i; bit N: global tier; zeros for an
 * absent key), W = smetric_index_mask_words(idx). */
int smetric_index_lookup(smetric_index* idx, const uint64_t* d_keys, int64_t n,
                         uint64_t* d_masks, smetric_stream_t stream);

/* W = ceil((N+1)/64), the number of 64-bit tier-mask words per key; 0 for NULL. */
int32_t smetric_index_mask_words(const smetric_index* idx);

/* The routing step (Figure 6 and Figure 10: per request, the local hit c of
 * every instance, then argmin over instances of the cost).
 *   d_tokens   int32 [n_tokens], 16-byte aligned; request r is
 *              d_tokens[d_offsets[r] .. d_offsets[r+1]).
 *   d_offsets  int64 [n_requests+1], non-decreasing, d_offsets[0] >= 0,
 *              d_offsets[n_requests] <= n_tokens, every length < 2^31.
 *   d_load     int64 [N], each in [0, SMETRIC_MAX_LOAD].
 *   outputs    int32 d_instance[r] = i*, d_local_hit[r] = B*c_{i*},
 *              d_global_hit[r] = B*(max(c_{i*},g) - c_{i*}),
 *              uint64 d_session_key[r] = sk_r.
 *   d_block_hashes  NULL, or uint64 [hashes_cap] receiving every request's
 *              full-block hashes h_0..h_{n_r-1}, request after request;
 *              hashes_cap must be >= n_tokens / B.
 * 0 <= n_requests <= max_batch_requests and 0 <= n_tokens <= max_batch_tokens.
 * With invalid offsets or loads the call latches INVALID_ARG or OVERFLOW and
 * writes instance -1, zero hits and key 0 for every request. */
int smetric_route_batch(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                        const int64_t* d_offsets, int32_t n_requests, const int64_t* d_load,
                        smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                        int32_t* d_global_hit, uint64_t* d_session_key,
                        uint64_t* d_block_hashes, int64_t hashes_cap, smetric_stream_t stream);

/* Limits of the session-centric policy's inputs (its integer arithmetic
 * stays below 2^63 within them). */
#define SMETRIC_POLICY_MAX_LEN (1LL << 24)     /* prompt tokens per request */
#define SMETRIC_POLICY_MAX_QUEUED (1LL << 59)  /* an instance's queued cost */
#define SMETRIC_POLICY_MAX_TPOT (1LL << 60)    /* colocation: a TPOT budget */
#define SMETRIC_POLICY_MAX_REQUESTS (1LL << 20) /* colocation: an instance's request count */

/* Parameters of the session-centric policy (Figure 10), integers:
 *   c_lin, c_att  Eq. 1's coefficients: the prefill cost of n new tokens in
 *                 an L-token prompt is c_lin*n + c_att*n*(L - n/2) cost units;
 *                 c_lin in [0, 2^20], c_att in [0, 2^12].
 *   ttft_d0, ttft_d1  the TTFT deadline in cost units,
 *                 D(L) = ttft_d0 + ttft_d1*L (SLACK * PREFILL_RATE * the
 *                 SLO b + a*L); ttft_d0 in [0, 2^60], ttft_d1 in [0, 2^35].
 *   hit_num, hit_den  HIT_RATIO = hit_num / hit_den,
 *                 0 <= hit_num <= hit_den, 1 <= hit_den <= 2^20.
 *   rr_base       where request 0's round robin over equal loads starts,
 *                 [0, N). */
typedef struct smetric_policy {
  int64_t c_lin;
  int64_t c_att;
  int64_t ttft_d0;
  int64_t ttft_d1;
  int64_t hit_num;
  int64_t hit_den;
  int32_t rr_base;
  int32_t reserved; /* 0 */
} smetric_policy;

/* The routing step with the session-centric policy of Figure 10 as its
 * decision (the second epilogue over the same local hits c_i and global run
 * g as smetric_route_batch; Section 4.2's basic policy with SLO-aware
 * migration). Per request r, with n_i = L - B*c_i its new tokens on
 * instance i and est_i = d_queued[i] + c_lin*n_i + c_att*n_i*(L - n_i/2)
 * (Figure 10(c), Eq. 1):
 *   prev   = argmax_i c_i, lowest id among equals;
 *   cached = B*c_prev > HIT_RATIO * d_est_hit[r]          (session_cached)
 *   meets(i) = est_i <= D(L)                              (Figure 10(b))
 *   stick  = d_turn[r] != 0 and cached and (meets(prev) or no i meets);
 *   i*     = prev if stick, else the first minimal est_i scanning
 *            i = s, s+1, ..., N-1, 0, ..., s-1 with s = (rr_base + r) mod N.
 * All comparisons are exact (computed on 2*est_i in int64).
 *   d_queued   int64 [N], each in [0, SMETRIC_POLICY_MAX_QUEUED]: the cost
 *              already queued on each instance, in Eq. 1's units.
 *   d_turn     int32 [n_requests]: 0 marks a session's first request.
 *   d_est_hit  int64 [n_requests], each in [0, 2^31): the hit in tokens
 *              that the request's history leads one to expect.
 *   outputs    as smetric_route_batch for i*, plus int32 d_stick[r] = 1 when
 *              the request stuck to prev, else 0.
 * Other arguments and the other rules as smetric_route_batch; every prompt
 * must be at most SMETRIC_POLICY_MAX_LEN tokens. Parameters out of range
 * return SMETRIC_ERR_INVALID_ARG with nothing enqueued; queued costs,
 * expected hits or prompt lengths out of range latch SMETRIC_ERR_OVERFLOW
 * and the batch's outputs are instance -1, zero hits, stick 0 and key 0. */
int smetric_route_batch_policy(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                               const int64_t* d_offsets, int32_t n_requests, const int64_t* d_queued,
                               const int32_t* d_turn, const int64_t* d_est_hit, smetric_policy p,
                               int32_t* d_instance, int32_t* d_local_hit, int32_t* d_global_hit,
                               int32_t* d_stick, uint64_t* d_session_key, uint64_t* d_block_hashes,
                               int64_t hashes_cap, smetric_stream_t stream);

/* The session-centric policy under PD colocation (Appendix B): as
 * smetric_route_batch_policy, with two changes.
 *   TPOT check: with cost_i = c_lin*n_i + c_att*n_i*(L - n_i/2) (the request's
 *   own prefill on instance i), instance i is a candidate when
 *   cost_i <= d_tpot_budget[i], the prefill the live decodes on i absorb
 *   within their TPOT SLO (PREFILL_RATE times their smallest slack, in cost
 *   units; SMETRIC_POLICY_MAX_TPOT for an instance with none); when no
 *   instance passes, every instance is a candidate.
 *   stick = d_turn[r] != 0 and cached and meets(prev) and prev is a
 *   candidate (no last resort);
 *   i* = prev if stick, else the first minimal est_i * d_num_requests[i]
 *   over the candidates in the rotation order (LMetric's product, compared
 *   exactly in 128 bits).
 *   d_tpot_budget   int64 [N], each in [0, SMETRIC_POLICY_MAX_TPOT].
 *   d_num_requests  int64 [N], each in [0, SMETRIC_POLICY_MAX_REQUESTS].
 * Out-of-range values of either latch SMETRIC_ERR_OVERFLOW like the queued
 * costs. */
int smetric_route_batch_policy_coloc(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                                     const int64_t* d_offsets, int32_t n_requests, const int64_t* d_queued,
                                     const int64_t* d_tpot_budget, const int64_t* d_num_requests,
                                     const int32_t* d_turn, const int64_t* d_est_hit, smetric_policy p,
                                     int32_t* d_instance, int32_t* d_local_hit, int32_t* d_global_hit,
                                     int32_t* d_stick, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                     int64_t hashes_cap, smetric_stream_t stream);

/* KV$ reuse breakdown of a trace window (Section 3.1, Findings 1-3):
 * against an unbounded store of every earlier request's blocks (requests in
 * arrival order), request r reuses its longest block prefix the store holds.
 * Each reused block b counts as system prompt when b < d_sys_blocks[r], else
 * as intra-session when the earliest request holding it has r's session
 * (d_sessions, e.g. from smetric_link_sessions), else as inter-session.
 * Outputs (int32 [n_requests], blocks): d_hit = d_sys + d_intra + d_inter.
 * The caller provides a 16-byte aligned device workspace of at least
 * smetric_reuse_workspace_bytes(n_tokens / block_size) bytes (nothing is
 * allocated). Uses the index's hashing and route scratch. Invalid offsets
 * latch INVALID_ARG and write -1 everywhere; a negative system span latches
 * INVALID_ARG and counts as 0. */
int64_t smetric_reuse_workspace_bytes(int64_t n_blocks);
int smetric_reuse_breakdown(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                            const int64_t* d_offsets, int32_t n_requests, const int32_t* d_sessions,
                            const int32_t* d_sys_blocks, void* d_workspace, int64_t workspace_bytes,
                            int32_t* d_hit, int32_t* d_sys, int32_t* d_intra, int32_t* d_inter,
                            smetric_stream_t stream);

/* Windowed load imbalance (Section 3.2, Figure 3(c)): an instance's load in
 * a time window is its average number of running requests there; the
 * window's imbalance is the maximum load over the mean across the index's N
 * instances. Request r runs on instance d_instance[r] over the integer time
 * interval [d_start[r], d_end[r]) (ticks of the caller's choosing). Window
 * w < n_windows is [w*window, (w+1)*window); running time after the last
 * window is not counted. With S_i(w) the ticks instance i's requests run
 * inside window w, the outputs (device, [n_windows]) are d_max[w] =
 * max_i S_i(w) (int64), d_argmax[w] = the lowest instance attaining it
 * (int32) and d_sum[w] = sum_i S_i(w) (int64); the imbalance is
 * N * d_max[w] / d_sum[w] (no running request: all three are 0). The caller
 * provides an 8-byte aligned device workspace of at least
 * smetric_imbalance_workspace_bytes(n_windows, N) bytes. Limits: 1 <= window
 * <= SMETRIC_IMBALANCE_MAX_WINDOW, n_windows * window <= 2^62, n_requests <=
 * SMETRIC_IMBALANCE_MAX_REQUESTS, n_windows * N <= SMETRIC_IMBALANCE_MAX_CELLS
 * (else INVALID_ARG before any launch). A request with an instance outside
 * [0, N), a negative start or end < start latches INVALID_ARG and is left
 * out; the others are counted. Does not touch the index's tables or route
 * scratch. */
#define SMETRIC_IMBALANCE_MAX_WINDOW (1LL << 36)
#define SMETRIC_IMBALANCE_MAX_REQUESTS (1 << 26)
#define SMETRIC_IMBALANCE_MAX_CELLS (1LL << 31)
int64_t smetric_imbalance_workspace_bytes(int32_t n_windows, int32_t num_instances);
int smetric_window_imbalance(smetric_index* idx, const int32_t* d_instance, const int64_t* d_start,
                             const int64_t* d_end, int32_t n_requests, int64_t window, int32_t n_windows,
                             void* d_workspace, int64_t workspace_bytes, int64_t* d_max, int32_t* d_argmax,
                             int64_t* d_sum, smetric_stream_t stream);

/* Session reconstruction from block hashes (Appendix A): in a batch of
 * requests in arrival order, request r follows the latest earlier request p
 * of the same user (d_users) with d_turns[p] = d_turns[r] - 1 whose
 * block-hash sequence is a prefix of r's (equal and empty sequences
 * included); d_parent[r] = p, or -1. d_session[r] = the first request of
 * r's chain of parents. Hashes are the index's (its block size and seed);
 * same token and offset rules as smetric_route_batch. Uses the index's
 * route scratch (no route may run on the index concurrently). Invalid
 * offsets latch INVALID_ARG and write -1 to both outputs. Prefixes are
 * compared by the hash of p's last block, which decides as a full comparison
 * does up to a 64-bit collision of the chain hash. */
int smetric_link_sessions(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                          const int64_t* d_offsets, int32_t n_requests, const int64_t* d_users,
                          const int32_t* d_turns, int32_t* d_parent, int32_t* d_session,
                          smetric_stream_t stream);

/* smetric_route_batch with the loads updated request by request (Figure 10
 * routes one request at a time, so each request sees the queues the batch's
 * earlier requests joined): requests in batch order, each takes the argmin
 * cost with the current loads, then load_{i*} += L_r - B*c_{i*}. The hits
 * are those of the index snapshot, as in smetric_route_batch. The decisions
 * run on one warp, request after request. d_load_after (int64 [N], may be
 * NULL) receives the loads after the batch; d_load is read, not written.
 * The largest load plus the batch's tokens must be at most 2^42, else the
 * call latches OVERFLOW and writes instance -1 and zero hits. */
int smetric_route_batch_sequential(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                                   const int64_t* d_offsets, int32_t n_requests, const int64_t* d_load,
                                   smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                                   int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                   int64_t hashes_cap, int64_t* d_load_after, smetric_stream_t stream);

/* Baseline scorers of Section 5.1 as the routing decision (argmin over the
 * same local hits c_i, ties to the lowest id). */
#define SMETRIC_SCORER_BAILIAN 1 /* (1-lambda)*l_i/max_j l_j + lambda*(1 - B*c_i/L) */
#define SMETRIC_SCORER_LMETRIC 2 /* (q_i + L - B*c_i) * l_i */

/*   d_queued  int64 [N], each in [0, SMETRIC_MAX_LOAD]: queued prefill tokens
 *             q_i (LMetric; unused by Bailian's score but still checked).
 *   d_batch   int64 [N], each in [0, SMETRIC_POLICY_MAX_REQUESTS]: batch
 *             sizes l_i. Bailian normalises them by their maximum (the load
 *             term is 0 when every l_j is 0) and takes the hit ratio as 0 for
 *             an empty prompt; lambda = lam_num / lam_den,
 *             0 <= lam_num <= lam_den, 1 <= lam_den <= 2^20. Scores are
 *             compared exactly (128-bit integers).
 * Outputs as smetric_route_batch. Out-of-range parameters return
 * INVALID_ARG; out-of-range queues or batch sizes latch OVERFLOW. */
int smetric_route_batch_baseline(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                                 const int64_t* d_offsets, int32_t n_requests, int32_t scorer,
                                 const int64_t* d_queued, const int64_t* d_batch, int64_t lam_num,
                                 int64_t lam_den, int32_t* d_instance, int32_t* d_local_hit,
                                 int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                 int64_t hashes_cap, smetric_stream_t stream);

/* Flags of smetric_index_commit_batch. */
#define SMETRIC_COMMIT_GLOBAL 1 /* also add every block to the global tier */

/* Device-side index maintenance after a routed batch, with no host round
 * trip (the replay step between batches: Section 2, the serving side caches
 * a request's KV$ blocks on the instance that ran it). For every request r
 * with d_instance[r] >= 0, its full-block hashes join the local tier of
 * d_instance[r] (and the global tier with SMETRIC_COMMIT_GLOBAL). Then, when
 * d_load is not NULL, each instance's queue drains:
 *   d_load[i] <- (d_load[i] + sum over r routed to i of (L_r - d_local_hit[r])) >> 1.
 *   d_offsets      the routed batch's offsets (int64 [n_requests+1]).
 *   d_instance, d_local_hit  the route's outputs (int32 [n_requests]).
 *   d_block_hashes the route's block hashes (request after request, as
 *                  smetric_route_batch writes them).
 *   d_load         int64 [N], read and written; NULL skips the drain.
 * Stream-ordered after the route; set semantics as smetric_index_insert
 * (inserting a key a tier holds is a no-op). Tiers capped by
 * smetric_index_set_lru then evict their least recently used blocks down to
 * the cap; other capped tiers are the caller's to evict
 * (smetric_index_evict). Errors
 * latched: invalid offsets, an instance outside [-1, N) or a local hit
 * outside [0, L_r] (INVALID_ARG: nothing is committed and the loads are left
 * as they were), no free slot (TABLE_FULL). d_local_hit may be NULL when
 * d_load is. */
int smetric_index_commit_batch(smetric_index* idx, const int64_t* d_offsets, int32_t n_requests,
                               const int32_t* d_instance, const int32_t* d_local_hit,
                               const uint64_t* d_block_hashes, int32_t flags, int64_t* d_load,
                               smetric_stream_t stream);

/* One replay step on the device: smetric_route_batch, then
 * smetric_index_commit_batch of its outputs, on one stream with no host
 * round trip in between. d_load (int64 [N]) is read by the route and then
 * drained in place by the commit. d_block_hashes is required (the commit
 * reads it); flags as smetric_index_commit_batch. Arguments and errors as
 * the two calls; an invalid batch routes every request to -1 and commits
 * nothing. */
int smetric_route_commit_batch(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                               const int64_t* d_offsets, int32_t n_requests, int64_t* d_load,
                               smetric_weights w, int32_t* d_instance, int32_t* d_local_hit,
                               int32_t* d_global_hit, uint64_t* d_session_key, uint64_t* d_block_hashes,
                               int64_t hashes_cap, int32_t flags, smetric_stream_t stream);

/* Device-side LRU for capped tiers (Section 2: an instance's local KV$ and
 * the global store are bounded and keep their most recently used blocks).
 * local_cap > 0 caps every local tier at that many blocks, global_cap > 0
 * the global tier; 0 leaves a tier uncapped, and (0, 0) turns the LRU off.
 * After each smetric_index_commit_batch, a capped tier holds its cap most
 * recent blocks: a block touched by request r of a commit at block position
 * b has recency (commit, r, -b) (later commits, later requests and, within a
 * request, leading blocks are more recent), and the least recent leave
 * first. Call it while the capped tiers are empty (after create or
 * smetric_index_clear): keys already in them are not tracked. Synchronises
 * the device; any earlier recency state is dropped. Device memory: 16 B per
 * capped block (two record buffers), plus 16 B x 2 x max_blocks of touch
 * lists, 16 B x 8 x max_blocks of per-batch sets and a byte per record and
 * touch (max_blocks = max_batch_tokens / B).
 * Errors: a negative cap or one above 2^40 (INVALID_ARG), an allocation
 * failure (OOM: the LRU is off then). */
int smetric_index_set_lru(smetric_index* idx, int64_t local_cap, int64_t global_cap);

/* d_sizes[t] (int64 [N+1], device) = blocks the LRU tracks in tier t (local
 * tiers 0..N-1, the global tier at N); 0 for uncapped tiers. Stream-ordered. */
int smetric_index_lru_sizes(smetric_index* idx, int64_t* d_sizes, smetric_stream_t stream);

/* Step (a)-(b) alone: block hashes and session keys of a batch, without
 * index lookups (Appendix A: a request's block-hash sequence starts with its
 * parent's). Same argument rules as smetric_route_batch; d_block_hashes is
 * required here. */
int smetric_block_hashes(smetric_index* idx, const int32_t* d_tokens, int64_t n_tokens,
                         const int64_t* d_offsets, int32_t n_requests, uint64_t* d_session_key,
                         uint64_t* d_block_hashes, int64_t hashes_cap, smetric_stream_t stream);

/* Limits of smetric_block_hashes_noalloc's fixed scratch. */
#define SMETRIC_NOALLOC_MAX_REQUESTS 4096
#define SMETRIC_NOALLOC_MAX_BLOCKS 32768

/* smetric_block_hashes without an index and without allocating anything.
 * The paper has no counterpart: this is a library convenience.
 *
 * Who needs it: a caller that must not allocate device memory at call time
 * and has no index -- for example a request front-end that computes session
 * keys and block hashes on a GPU whose memory a serving engine has already
 * reserved in its own pools, or a latency-critical loop in which the device
 * synchronisation that cudaMalloc/cudaFree imply would stall other streams.
 * smetric_block_hashes needs an index, and smetric_index_create allocates the
 * table and per-batch scratch; this call allocates nothing: no cudaMalloc,
 * no cudaFree, no allocating library call.
 *
 * Scratch: one statically sized device array compiled into the library
 * (request offsets and per-block digests, 295,424 bytes, one copy per device,
 * existing from module load). The first call on each device, with that
 * device current, looks up the array's device address once
 * (cudaGetSymbolAddress) and caches it; make that first call before any
 * stream capture on the device. The cached address belongs to the device's
 * context as it was at that first call: after cudaDeviceReset (or anything
 * else that destroys and recreates the primary context) it is stale, so do
 * not call this function again in that process after such a reset.
 *
 * Limits: n_requests <= SMETRIC_NOALLOC_MAX_REQUESTS and
 * n_tokens / block_size <= SMETRIC_NOALLOC_MAX_BLOCKS; a larger batch returns
 * SMETRIC_ERR_TOO_LARGE with nothing enqueued.
 *
 * Arguments are those of smetric_block_hashes, with the index configuration
 * given directly (block_size B even in 2..256, session_blocks S >= 1, the
 * hash seed) and one more:
 *   d_status   int32 in device memory, owned by the caller; it MUST be 0 when
 *              the call's kernels start. Invalid offsets latch
 *              SMETRIC_ERR_INVALID_ARG and lengths of 2^31 or more latch
 *              SMETRIC_ERR_OVERFLOW into it (first error wins); session keys
 *              are then 0 and no hash is written.
 * Host-detectable errors return immediately with nothing enqueued.
 *
 * Concurrency: every call on one device uses the same scratch. Calls whose
 * kernels overlap (different streams or host threads without ordering
 * between them) race on it and produce wrong results; order them on one
 * stream or with events. */
int smetric_block_hashes_noalloc(const int32_t* d_tokens, int64_t n_tokens, const int64_t* d_offsets,
                                 int32_t n_requests, int32_t block_size, int32_t session_blocks,
                                 uint64_t hash_seed, uint64_t* d_session_key, uint64_t* d_block_hashes,
                                 int64_t hashes_cap, int32_t* d_status, smetric_stream_t stream);

/* smetric_route_batch from host buffers: copies tokens, offsets and load to
 * the index's staging buffers (the index must have been created with
 * SMETRIC_FLAG_HOST_STAGING), routes, copies the four outputs back and waits
 * for the stream. Returns the call's status including any error the device
 * latched, which it clears. */
int smetric_route_batch_host(smetric_index* idx, const int32_t* h_tokens, int64_t n_tokens,
                             const int64_t* h_offsets, int32_t n_requests, const int64_t* h_load,
                             smetric_weights w, int32_t* h_instance, int32_t* h_local_hit,
                             int32_t* h_global_hit, uint64_t* h_session_key,
                             smetric_stream_t stream);

/* Several batches routed in one call: batch j < n_batches is routed exactly
 * as smetric_route_batch would route it with no block-hash output (tokens
 * d_tokens[j] of n_tokens[j], offsets d_offsets[j], n_requests[j] requests,
 * loads d_load[j], outputs d_instance[j], d_local_hit[j], d_global_hit[j],
 * d_session_key[j]). Each d_ argument is a host array of n_batches device
 * pointers; n_tokens and n_requests are host arrays of counts; the weights
 * are shared. Every batch sees the index as of the call (routes do not
 * change it) and its own loads, so the outputs equal those of n_batches
 * smetric_route_batch calls in a row, and when the call returns every output
 * is complete in `stream` order.
 *
 * With an index created with SMETRIC_FLAG_PIPELINE (and profiling off), the
 * batches alternate between the index's two scratch sets and two streams,
 * so that batch j+1's token read (the block digests, bound by HBM
 * bandwidth) runs while batch j's tier lookups and walk (bound by random
 * accesses and latency) finish: batch j+1 starts once batch j's hash chain
 * is done. Without the flag the batches run one after another on `stream`.
 * The outputs of different batches must not overlap (two batches may run at
 * once); inputs may be shared. Nothing is allocated (the second set comes
 * with the index). Host-detectable errors in any batch return before
 * anything is enqueued; device-detected errors latch as for
 * smetric_route_batch (a bad batch gets the invalid-batch outputs, the
 * others are routed). */
int smetric_route_batches(smetric_index* idx, int32_t n_batches, const int32_t* const* d_tokens,
                          const int64_t* n_tokens, const int64_t* const* d_offsets, const int32_t* n_requests,
                          const int64_t* const* d_load, smetric_weights w, int32_t* const* d_instance,
                          int32_t* const* d_local_hit, int32_t* const* d_global_hit,
                          uint64_t* const* d_session_key, smetric_stream_t stream);

/* Wait for `stream`, then return and clear the first error the device latched
 * for this index since the last call (SMETRIC_OK if none). */
int smetric_status(smetric_index* idx, smetric_stream_t stream);

/* Static description of an error code. */
const char* smetric_strerror(int code);

/* Observability. With profiling on, each route records CUDA events around
 * each of its kernels on the launch stream. smetric_profile_read waits for
 * them and returns, per kernel k < min(max_kernels, count), the summed device
 * milliseconds ms[k] and launches[k] since the previous read, then resets;
 * it returns the number of kernels a route launches (or a negative error).
 * smetric_profile_kernel_name(k) names kernel k. */
int smetric_profile_enable(smetric_index* idx, int32_t on);
int smetric_profile_read(smetric_index* idx, int32_t max_kernels, double* ms, int64_t* launches);
const char* smetric_profile_kernel_name(int32_t k);

/* Kernels this index has launched since it was created. */
int64_t smetric_launch_count(const smetric_index* idx);

#ifdef __cplusplus
}
#endif

#endif /* SMETRIC_H */
