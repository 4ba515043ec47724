/*
 * CPU oracle for the batched routing decision of balanced session-centric
 * scheduling (SMetric, arXiv 2607.08565).
 *
 * TEST INFRASTRUCTURE ONLY. Only the test suite, the package smoke check and
 * the benchmark's CPU-baseline leg may load this library. It shares no code,
 * header, table or constant generator with the CUDA path; it is written from
 * the definitions below so that a reader can check it against them by eye.
 * It is deliberately plain: scalar loops, a chained hash map, a block-by-block
 * prefix walk per tier and an exhaustive argmin.
 *
 * What it computes (per request r of a batch):
 *
 *  Block chain hash (Section 3.1: reuse is measured at KV$ block granularity;
 *  Appendix A: a follow-up request's block-hash sequence starts with its
 *  parent's, so the hash of block b must identify the whole prefix up to b).
 *  The paper fixes no hash function; the definition here is SplitMix64-style:
 *    mix64(z): the SplitMix64 output function (Steele, Lea & Flood, OOPSLA
 *              2014, with Stafford's "Mix13" multipliers).
 *    word k of block b: the little-endian u64 made of tokens bB+2k (low half)
 *              and bB+2k+1 (high half), each as u32.
 *    digest:   d_b = fold over k = 0..B/2-1 of x <- mix64(x ^ w_k), starting
 *              from x = mix64(seed ^ B).
 *    chain:    h_{-1} = mix64(seed + GAMMA);
 *              h_b = mix64((h_{b-1} + GAMMA) ^ d_b), then h_b |= 2 when
 *              h_b < 2 (0 and 1 are reserved), and the remapped value chains.
 *    Only full blocks are hashed: n_r = floor(L_r / B); a partial tail block
 *    is never a hit (Section 3.1 counts reuse in whole hit blocks).
 *
 *  Session key (Section 4.2, basic solution: a session is recognised from
 *  the request itself, with no per-session state): sk_r = h_{min(n_r,S)-1},
 *  or 0 when n_r = 0.
 *
 *  Two-tier longest prefix match (Figure 6 and Figure 10: the router asks the
 *  KV$ for the prompt's prefix hit on each instance; Section 2 and Section
 *  4.2: a local miss can be fetched from the global tier):
 *    c_i = largest k <= n_r with h_0..h_{k-1} all in instance i's local tier,
 *    g   = largest k <= n_r with h_0..h_{k-1} all in the global tier,
 *    g_i = max(c_i, g).
 *
 *  Integer cost and argmin (Figure 6: the request goes to the instance that
 *  minimises a function of its hit and its load; Figure 10(c): the load is
 *  the queued prefill plus the request's own new tokens):
 *    miss_i  = L_r - B*g_i            (tokens instance i must prefill)
 *    fetch_i = B*(g_i - c_i)          (tokens fetched from the global tier)
 *    cost_i  = w_load*load_i + w_miss*miss_i + w_glob*fetch_i   (int64)
 *    i*      = smallest i attaining the minimum cost.
 *  Outputs: instance = i*, local_hit = B*c_{i*}, global_hit = fetch_{i*},
 *  session_key = sk_r.
 *
 * Every request of a batch sees the same index and load (snapshot semantics).
 *
 * Session-centric policy (Figure 10, second epilogue over the same c_i and
 * g; oracle_route_batch_policy). Figure 10(c), Eq. 1: the prefill cost of n
 * new tokens in an L-token prompt is C_LIN*n + C_ATT*n*(L - n/2); here in
 * fixed point and doubled so that it stays an integer:
 *    n_i     = L_r - B*c_i
 *    est2_i  = 2*q_i + 2*C_LIN*n_i + C_ATT*n_i*(2*L_r - n_i)
 *              (= 2 * estimate_load(req, i), q_i = instance i's queued cost)
 * Figure 10(a):
 *    prev    = argmax_i c_i (lowest id among equals)
 *    cached  = B*c_prev*HIT_DEN > HIT_NUM*est_hit_r   (session_cached; the
 *              ratio HIT_RATIO = HIT_NUM/HIT_DEN, est_hit_r = the hit the
 *              request's history leads one to expect)
 * Figure 10(b): meets(i) = est2_i <= 2*(D0 + D1*L_r), the TTFT deadline in
 * cost units (SLACK * PREFILL_RATE * (b + a*L)), none_meets = no i meets.
 *    stick   = turn_r != 0 and cached and (meets(prev) or none_meets)
 *    i*      = prev if stick, else the first minimal est2_i in the order
 *              s, s+1, ..., N-1, 0, ..., s-1 with s = (rr_base + r) mod N
 *              (rr_argmin: equal loads are taken in turn).
 * Outputs: instance = i*, stick, local_hit = B*c_{i*}, global_hit =
 * B*(max(c_{i*}, g) - c_{i*}), session_key as above.
 *
 * The same policy under PD colocation (Appendix B; oracle_route_batch_coloc):
 *    cost2_i = 2*C_LIN*n_i + C_ATT*n_i*(2*L_r - n_i)   (2 * prefill_cost)
 *    tpot(i) = cost2_i <= 2*T_i, T_i the prefill cost instance i's live
 *              decodes can absorb within their TPOT SLO (PREFILL_RATE times
 *              the smallest slack); cand = {i : tpot(i)}, or every instance
 *              when no instance passes.
 *    stick   = turn_r != 0 and cached and meets(prev) and prev in cand
 *              (no last resort here)
 *    i*      = prev if stick, else the first minimal est2_i * R_i over cand
 *              in the rotation order above, R_i = the requests instance i
 *              runs (LMetric's multiplicative score), compared exactly in
 *              128 bits.
 *
 * Sequential-update variant (oracle_route_batch_sequential; Figure 10 routes
 * one request at a time, so each request sees the queues its predecessors
 * in the batch joined): requests in order, each takes the argmin cost above
 * with the current loads, then load_{i*} += L_r - B*c_{i*} (the tokens the
 * chosen instance must prefill or fetch). Limits: max_i load_i plus the
 * batch's tokens at most 2^42.
 *
 * Baseline scorers of Section 5.1 (oracle_route_batch_baseline), argmin with
 * ties to the lowest id over the same c_i:
 *    Bailian: f_i = (1 - LAMBDA) * l_i / max_j l_j + LAMBDA * (1 - B*c_i / L_r)
 *             (l_i instance i's batch size; the load term is 0 when every
 *             l_j is 0 and the hit ratio is 0 for an empty prompt);
 *             LAMBDA = LAM_NUM / LAM_DEN; compared exactly on f_i times
 *             LAM_DEN * max_j l_j * L_r in 128 bits.
 *    LMetric: f_i = (q_i + L_r - B*c_i) * l_i (q_i the queued prefill tokens).
 *
 * Reuse breakdown (Section 3.1, Findings 1-3; oracle_reuse_breakdown): against
 * an idealised KV$ store of unbounded capacity holding every block of every
 * earlier request, request r's hit is its longest block prefix whose blocks
 * the store holds (hash h_b occurs in some earlier request). Each hit block
 * is attributed to the earliest request p holding it: to the system prompt
 * when b < sys_r (the request's leading system-prompt blocks), else
 * intra-session when session_p = session_r, else inter-session.
 *
 * Windowed load imbalance (Section 3.2, Figure 3(c); oracle_window_imbalance):
 * request r runs on instance inst_r over the integer time interval
 * [start_r, end_r). Window w is [w*T, (w+1)*T). Instance i's load in window w
 * is its average number of running requests there, S_i(w) / T with
 *    S_i(w) = sum over r with inst_r = i of |[start_r, end_r) ∩ window w|
 * (running-request time in ticks), and the window's imbalance is the maximum
 * load over the mean across all N instances, N * max_i S_i(w) / sum_i S_i(w).
 * Outputs per window: max_i S_i(w), its lowest maximising instance, and
 * sum_i S_i(w) (exact integers; the ratio is formed by the caller).
 *
 * Session reconstruction (Appendix A; oracle_link_sessions): request r
 * follows request p when p is earlier (p < r, requests in arrival order), of
 * the same user, of turn turn_r - 1, and p's block-hash sequence is a prefix
 * of r's (h_p[b] = h_r[b] for every b < n_p; the empty sequence is a prefix
 * of every sequence). parent_r is the latest such p, or -1; session_r is the
 * first request of r's chain of parents.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_GAMMA 0x9E3779B97F4A7C15ULL

enum {
  ORACLE_OK = 0,
  ORACLE_ERR_INVALID_ARG = -1,
  ORACLE_ERR_OOM = -2,
};

/* ------------------------------------------------------------------------ */
/* Hashing                                                                  */
/* ------------------------------------------------------------------------ */

uint64_t oracle_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static uint64_t oracle_word(const int32_t* t, int64_t i) {
  uint64_t lo = (uint64_t)(uint32_t)t[i];
  uint64_t hi = (uint64_t)(uint32_t)t[i + 1];
  return lo | (hi << 32);
}

/* Full-block chain hashes of one request. Writes floor(L/B) values to out and
 * returns that count, or a negative error for an invalid block size. */
int64_t oracle_block_hashes(const int32_t* tokens, int64_t L, int32_t B, uint64_t seed,
                            uint64_t* out) {
  if (B < 2 || (B % 2) != 0 || L < 0) return ORACLE_ERR_INVALID_ARG;
  int64_t n = L / B;
  uint64_t h = oracle_mix64(seed + ORACLE_GAMMA);
  for (int64_t b = 0; b < n; ++b) {
    uint64_t d = oracle_mix64(seed ^ (uint64_t)B);
    for (int32_t k = 0; k < B / 2; ++k) d = oracle_mix64(d ^ oracle_word(tokens, b * B + 2 * k));
    h = oracle_mix64((h + ORACLE_GAMMA) ^ d);
    if (h < 2) h |= 2;
    out[b] = h;
  }
  return n;
}

/* ------------------------------------------------------------------------ */
/* Index: key -> set of tiers (bit i < N: local tier of instance i; bit N:   */
/* global tier). A chained hash map; nodes are never removed, a key whose    */
/* tier set becomes empty is simply a member of no tier.                      */
/* ------------------------------------------------------------------------ */

typedef struct oracle_node {
  uint64_t key;
  struct oracle_node* next;
  uint8_t tiers[]; /* (N + 1) bits */
} oracle_node;

typedef struct oracle_index {
  int32_t N;
  size_t tier_bytes;
  uint64_t nbuckets;
  uint64_t count;
  oracle_node** buckets;
} oracle_index;

oracle_index* oracle_index_create(int32_t N) {
  if (N < 1) return NULL;
  oracle_index* x = (oracle_index*)calloc(1, sizeof(oracle_index));
  if (!x) return NULL;
  x->N = N;
  x->tier_bytes = (size_t)(N + 1 + 7) / 8;
  x->nbuckets = 1024;
  x->buckets = (oracle_node**)calloc(x->nbuckets, sizeof(oracle_node*));
  if (!x->buckets) { free(x); return NULL; }
  return x;
}

void oracle_index_destroy(oracle_index* x) {
  if (!x) return;
  for (uint64_t i = 0; i < x->nbuckets; ++i) {
    oracle_node* p = x->buckets[i];
    while (p) { oracle_node* q = p->next; free(p); p = q; }
  }
  free(x->buckets);
  free(x);
}

static oracle_node* oracle_find(const oracle_index* x, uint64_t key) {
  for (oracle_node* p = x->buckets[key % x->nbuckets]; p; p = p->next)
    if (p->key == key) return p;
  return NULL;
}

static int oracle_grow(oracle_index* x) {
  uint64_t nb = x->nbuckets * 2;
  oracle_node** nbk = (oracle_node**)calloc(nb, sizeof(oracle_node*));
  if (!nbk) return ORACLE_ERR_OOM;
  for (uint64_t i = 0; i < x->nbuckets; ++i) {
    oracle_node* p = x->buckets[i];
    while (p) {
      oracle_node* q = p->next;
      p->next = nbk[p->key % nb];
      nbk[p->key % nb] = p;
      p = q;
    }
  }
  free(x->buckets);
  x->buckets = nbk;
  x->nbuckets = nb;
  return ORACLE_OK;
}

static int oracle_tier_bit(const oracle_index* x, int32_t tier) {
  if (tier == -1) return x->N;
  if (tier >= 0 && tier < x->N) return tier;
  return -1;
}

/* Insert each (keys[j], tiers[j]) pair; tier -1 is the global tier. */
int oracle_index_insert(oracle_index* x, const uint64_t* keys, const int32_t* tiers, int64_t n) {
  if (!x || n < 0) return ORACLE_ERR_INVALID_ARG;
  for (int64_t j = 0; j < n; ++j) {
    int bit = oracle_tier_bit(x, tiers[j]);
    if (bit < 0 || keys[j] < 2) return ORACLE_ERR_INVALID_ARG;
    oracle_node* p = oracle_find(x, keys[j]);
    if (!p) {
      if (x->count >= x->nbuckets && oracle_grow(x) != ORACLE_OK) return ORACLE_ERR_OOM;
      p = (oracle_node*)calloc(1, sizeof(oracle_node) + x->tier_bytes);
      if (!p) return ORACLE_ERR_OOM;
      p->key = keys[j];
      p->next = x->buckets[keys[j] % x->nbuckets];
      x->buckets[keys[j] % x->nbuckets] = p;
      x->count++;
    }
    p->tiers[bit / 8] |= (uint8_t)(1u << (bit % 8));
  }
  return ORACLE_OK;
}

/* Remove each (keys[j], tiers[j]) membership; absent pairs are ignored. */
int oracle_index_evict(oracle_index* x, const uint64_t* keys, const int32_t* tiers, int64_t n) {
  if (!x || n < 0) return ORACLE_ERR_INVALID_ARG;
  for (int64_t j = 0; j < n; ++j) {
    int bit = oracle_tier_bit(x, tiers[j]);
    if (bit < 0) return ORACLE_ERR_INVALID_ARG;
    oracle_node* p = oracle_find(x, keys[j]);
    if (p) p->tiers[bit / 8] &= (uint8_t)~(1u << (bit % 8));
  }
  return ORACLE_OK;
}

/* 1 if key is in the given tier (-1 = global), else 0. */
int oracle_index_contains(const oracle_index* x, uint64_t key, int32_t tier) {
  int bit = oracle_tier_bit(x, tier);
  if (bit < 0) return 0;
  const oracle_node* p = oracle_find(x, key);
  return p && ((p->tiers[bit / 8] >> (bit % 8)) & 1u);
}

/* ------------------------------------------------------------------------ */
/* Routing                                                                  */
/* ------------------------------------------------------------------------ */

/* Prefix hits of one hashed request: c[i] for each instance i and g for the
 * global tier. Each tier's run starts at block 0 and stops at the first block
 * that the tier does not hold; block k's tier set is looked up once and
 * checked against every tier whose run is still going. */
void oracle_prefix_hits(const oracle_index* x, const uint64_t* h, int64_t n, int64_t* c,
                        int64_t* g) {
  const int32_t N = x->N;
  int32_t running = N + 1; /* tiers whose run has not stopped yet */
  for (int32_t i = 0; i < N; ++i) c[i] = -1;
  *g = -1;
  for (int64_t k = 0; k < n && running > 0; ++k) {
    const oracle_node* p = oracle_find(x, h[k]);
    for (int32_t i = 0; i < N; ++i) {
      if (c[i] >= 0) continue;
      int held = p && ((p->tiers[i / 8] >> (i % 8)) & 1u);
      if (!held) { c[i] = k; running--; }
    }
    if (*g < 0) {
      int held = p && ((p->tiers[N / 8] >> (N % 8)) & 1u);
      if (!held) { *g = k; running--; }
    }
  }
  for (int32_t i = 0; i < N; ++i) if (c[i] < 0) c[i] = n; /* held every block */
  if (*g < 0) *g = n;
}

/* Route one batch. offsets has n_requests + 1 entries; tokens holds
 * offsets[n_requests] entries. block_hashes (may be NULL) receives every
 * request's full-block hashes, request after request. n_threads > 1 routes
 * requests in parallel (they are independent under snapshot semantics). */
int oracle_route_batch(const oracle_index* x, int32_t B, int32_t S, uint64_t seed,
                       const int32_t* tokens, const int64_t* offsets, int32_t n_requests,
                       const int64_t* load, int64_t w_load, int64_t w_miss, int64_t w_glob,
                       int32_t* instance, int32_t* local_hit, int32_t* global_hit,
                       uint64_t* session_key, uint64_t* block_hashes, int32_t n_threads) {
  if (!x || B < 2 || (B % 2) != 0 || S < 1 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  for (int32_t r = 0; r < n_requests; ++r)
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0) return ORACLE_ERR_INVALID_ARG;
  const int32_t N = x->N;
  int failed = 0;
  /* first block index of each request in block_hashes */
  int64_t* before = (int64_t*)malloc((size_t)(n_requests + 1) * sizeof(int64_t));
  if (!before) return ORACLE_ERR_OOM;
  before[0] = 0;
  for (int32_t r = 0; r < n_requests; ++r) before[r + 1] = before[r] + (offsets[r + 1] - offsets[r]) / B;
  (void)n_threads;
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads > 0 ? n_threads : 1)
  for (int32_t r = 0; r < n_requests; ++r) {
    int64_t L = offsets[r + 1] - offsets[r];
    int64_t n = L / B;
    uint64_t* h = (uint64_t*)malloc((size_t)(n > 0 ? n : 1) * sizeof(uint64_t));
    int64_t* c = (int64_t*)malloc((size_t)N * sizeof(int64_t));
    if (!h || !c) {
      free(h); free(c);
#pragma omp atomic write
      failed = 1;
      continue;
    }
    oracle_block_hashes(tokens + offsets[r], L, B, seed, h);
    if (block_hashes) memcpy(block_hashes + before[r], h, (size_t)n * sizeof(uint64_t));
    int64_t g;
    oracle_prefix_hits(x, h, n, c, &g);
    int32_t best = -1;
    int64_t best_cost = 0;
    for (int32_t i = 0; i < N; ++i) {
      int64_t gi = c[i] > g ? c[i] : g;
      int64_t miss = L - (int64_t)B * gi;
      int64_t fetch = (int64_t)B * (gi - c[i]);
      int64_t cost = w_load * load[i] + w_miss * miss + w_glob * fetch;
      if (best < 0 || cost < best_cost) { best = i; best_cost = cost; }
    }
    int64_t gb = c[best] > g ? c[best] : g;
    instance[r] = best;
    local_hit[r] = (int32_t)((int64_t)B * c[best]);
    global_hit[r] = (int32_t)((int64_t)B * (gb - c[best]));
    if (n == 0) session_key[r] = 0;
    else session_key[r] = h[(n < S ? n : S) - 1];
    free(h);
    free(c);
  }
  free(before);
  return failed ? ORACLE_ERR_OOM : ORACLE_OK;
}

/* Session-centric policy (Figure 10) over the same hashes and prefix hits.
 * Limits that keep every quantity below 2^63: L_r <= 2^24, C_LIN <= 2^20,
 * C_ATT <= 2^12, 0 <= q_i <= 2^59, D0 <= 2^60, D1 <= 2^35,
 * 0 <= est_hit_r < 2^31, 0 <= HIT_NUM <= HIT_DEN, 1 <= HIT_DEN <= 2^20,
 * 0 <= rr_base < N; anything else returns ORACLE_ERR_INVALID_ARG. */
int oracle_route_batch_policy(const oracle_index* x, int32_t B, int32_t S, uint64_t seed,
                              const int32_t* tokens, const int64_t* offsets, int32_t n_requests,
                              const int64_t* queued, const int32_t* turn, const int64_t* est_hit,
                              int64_t c_lin, int64_t c_att, int64_t d0, int64_t d1, int64_t hit_num,
                              int64_t hit_den, int32_t rr_base, int32_t* instance, int32_t* local_hit,
                              int32_t* global_hit, int32_t* stick, uint64_t* session_key) {
  if (!x || B < 2 || (B % 2) != 0 || S < 1 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  const int32_t N = x->N;
  if (c_lin < 0 || c_lin > (1LL << 20) || c_att < 0 || c_att > (1LL << 12) || d0 < 0 ||
      d0 > (1LL << 60) || d1 < 0 || d1 > (1LL << 35) || hit_den < 1 || hit_den > (1LL << 20) ||
      hit_num < 0 || hit_num > hit_den || rr_base < 0 || rr_base >= N)
    return ORACLE_ERR_INVALID_ARG;
  for (int32_t i = 0; i < N; ++i)
    if (queued[i] < 0 || queued[i] > (1LL << 59)) return ORACLE_ERR_INVALID_ARG;
  for (int32_t r = 0; r < n_requests; ++r) {
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0 || offsets[r + 1] - offsets[r] > (1LL << 24))
      return ORACLE_ERR_INVALID_ARG;
    if (est_hit[r] < 0 || est_hit[r] >= (1LL << 31)) return ORACLE_ERR_INVALID_ARG;
  }
  int64_t* c = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  int64_t* est2 = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  uint64_t* h = NULL;
  int64_t cap = 0;
  int rc = ORACLE_OK;
  if (!c || !est2) rc = ORACLE_ERR_OOM;
  for (int32_t r = 0; r < n_requests && rc == ORACLE_OK; ++r) {
    const int64_t L = offsets[r + 1] - offsets[r];
    const int64_t n = L / B;
    if (n + 1 > cap) {
      free(h);
      cap = n + 1;
      h = (uint64_t*)malloc((size_t)cap * sizeof(uint64_t));
      if (!h) { rc = ORACLE_ERR_OOM; break; }
    }
    oracle_block_hashes(tokens + offsets[r], L, B, seed, h);
    int64_t g;
    oracle_prefix_hits(x, h, n, c, &g);
    /* (c) load model: doubled Eq. 1 plus the queued cost */
    for (int32_t i = 0; i < N; ++i) {
      const int64_t nn = L - (int64_t)B * c[i];
      est2[i] = 2 * queued[i] + 2 * c_lin * nn + c_att * nn * (2 * L - nn);
    }
    /* (a) the instance that likely served the previous turn */
    int32_t prev = 0;
    for (int32_t i = 1; i < N; ++i)
      if (c[i] > c[prev]) prev = i;
    const int cached = (int64_t)B * c[prev] * hit_den > hit_num * est_hit[r];
    /* (b) SLO checks */
    const int64_t budget2 = 2 * (d0 + d1 * L);
    int any_meets = 0;
    for (int32_t i = 0; i < N; ++i)
      if (est2[i] <= budget2) any_meets = 1;
    const int meets_prev = est2[prev] <= budget2;
    const int st = turn[r] != 0 && cached && (meets_prev || !any_meets);
    int32_t to = prev;
    if (!st) {
      /* rr_argmin: the first minimal load in the order starting at s */
      const int32_t s0 = (int32_t)(((int64_t)rr_base + r) % N);
      to = s0;
      for (int32_t k = 1; k < N; ++k) {
        const int32_t i = (s0 + k) % N;
        if (est2[i] < est2[to]) to = i;
      }
    }
    const int64_t gt = c[to] > g ? c[to] : g;
    instance[r] = to;
    stick[r] = st;
    local_hit[r] = (int32_t)((int64_t)B * c[to]);
    global_hit[r] = (int32_t)((int64_t)B * (gt - c[to]));
    session_key[r] = n == 0 ? 0 : h[(n < S ? n : S) - 1];
  }
  free(h);
  free(c);
  free(est2);
  return rc;
}

/* Session-centric policy under PD colocation (Appendix B). Limits as the
 * policy above plus 0 <= T_i <= 2^60 and 0 <= R_i <= 2^20. */
int oracle_route_batch_coloc(const oracle_index* x, int32_t B, int32_t S, uint64_t seed,
                             const int32_t* tokens, const int64_t* offsets, int32_t n_requests,
                             const int64_t* queued, const int64_t* tpot_budget, const int64_t* num_requests,
                             const int32_t* turn, const int64_t* est_hit, int64_t c_lin, int64_t c_att,
                             int64_t d0, int64_t d1, int64_t hit_num, int64_t hit_den, int32_t rr_base,
                             int32_t* instance, int32_t* local_hit, int32_t* global_hit, int32_t* stick,
                             uint64_t* session_key) {
  if (!x || B < 2 || (B % 2) != 0 || S < 1 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  const int32_t N = x->N;
  if (c_lin < 0 || c_lin > (1LL << 20) || c_att < 0 || c_att > (1LL << 12) || d0 < 0 ||
      d0 > (1LL << 60) || d1 < 0 || d1 > (1LL << 35) || hit_den < 1 || hit_den > (1LL << 20) ||
      hit_num < 0 || hit_num > hit_den || rr_base < 0 || rr_base >= N)
    return ORACLE_ERR_INVALID_ARG;
  for (int32_t i = 0; i < N; ++i)
    if (queued[i] < 0 || queued[i] > (1LL << 59) || tpot_budget[i] < 0 || tpot_budget[i] > (1LL << 60) ||
        num_requests[i] < 0 || num_requests[i] > (1LL << 20))
      return ORACLE_ERR_INVALID_ARG;
  for (int32_t r = 0; r < n_requests; ++r) {
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0 || offsets[r + 1] - offsets[r] > (1LL << 24))
      return ORACLE_ERR_INVALID_ARG;
    if (est_hit[r] < 0 || est_hit[r] >= (1LL << 31)) return ORACLE_ERR_INVALID_ARG;
  }
  int64_t* c = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  int64_t* cost2 = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  int64_t* est2 = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  int* cand = (int*)malloc((size_t)N * sizeof(int));
  uint64_t* h = NULL;
  int64_t cap = 0;
  int rc = ORACLE_OK;
  if (!c || !cost2 || !est2 || !cand) rc = ORACLE_ERR_OOM;
  for (int32_t r = 0; r < n_requests && rc == ORACLE_OK; ++r) {
    const int64_t L = offsets[r + 1] - offsets[r];
    const int64_t n = L / B;
    if (n + 1 > cap) {
      free(h);
      cap = n + 1;
      h = (uint64_t*)malloc((size_t)cap * sizeof(uint64_t));
      if (!h) { rc = ORACLE_ERR_OOM; break; }
    }
    oracle_block_hashes(tokens + offsets[r], L, B, seed, h);
    int64_t g;
    oracle_prefix_hits(x, h, n, c, &g);
    for (int32_t i = 0; i < N; ++i) {
      const int64_t nn = L - (int64_t)B * c[i];
      cost2[i] = 2 * c_lin * nn + c_att * nn * (2 * L - nn);
      est2[i] = 2 * queued[i] + cost2[i];
    }
    int32_t prev = 0;
    for (int32_t i = 1; i < N; ++i)
      if (c[i] > c[prev]) prev = i;
    /* the TPOT filter: every live decode of i tolerates the new prefill */
    int n_cand = 0;
    for (int32_t i = 0; i < N; ++i) {
      cand[i] = cost2[i] <= 2 * tpot_budget[i];
      n_cand += cand[i];
    }
    if (n_cand == 0)
      for (int32_t i = 0; i < N; ++i) cand[i] = 1;
    const int cached = (int64_t)B * c[prev] * hit_den > hit_num * est_hit[r];
    const int meets_prev = est2[prev] <= 2 * (d0 + d1 * L);
    const int st = turn[r] != 0 && cached && meets_prev && cand[prev];
    int32_t to = prev;
    if (!st) {
      /* rr_argmin over the candidates of estimate_load * num_requests */
      const int32_t s0 = (int32_t)(((int64_t)rr_base + r) % N);
      to = -1;
      unsigned __int128 best = 0;
      for (int32_t k = 0; k < N; ++k) {
        const int32_t i = (s0 + k) % N;
        if (!cand[i]) continue;
        const unsigned __int128 score = (unsigned __int128)(uint64_t)est2[i] * (uint64_t)num_requests[i];
        if (to < 0 || score < best) { to = i; best = score; }
      }
    }
    const int64_t gt = c[to] > g ? c[to] : g;
    instance[r] = to;
    stick[r] = st;
    local_hit[r] = (int32_t)((int64_t)B * c[to]);
    global_hit[r] = (int32_t)((int64_t)B * (gt - c[to]));
    session_key[r] = n == 0 ? 0 : h[(n < S ? n : S) - 1];
  }
  free(h);
  free(c);
  free(cost2);
  free(est2);
  free(cand);
  return rc;
}

/* Session reconstruction (Appendix A), by definition: every earlier request
 * is compared in full, latest first. users and turns have n_requests
 * entries; parent and session receive n_requests entries. */
int oracle_link_sessions(int32_t B, uint64_t seed, const int32_t* tokens, const int64_t* offsets,
                         int32_t n_requests, const int64_t* users, const int32_t* turns, int32_t* parent,
                         int32_t* session) {
  if (B < 2 || (B % 2) != 0 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  for (int32_t r = 0; r < n_requests; ++r)
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0) return ORACLE_ERR_INVALID_ARG;
  int64_t* first = (int64_t*)malloc((size_t)(n_requests + 1) * sizeof(int64_t));
  if (!first) return ORACLE_ERR_OOM;
  first[0] = 0;
  for (int32_t r = 0; r < n_requests; ++r) first[r + 1] = first[r] + (offsets[r + 1] - offsets[r]) / B;
  uint64_t* h = (uint64_t*)malloc((size_t)(first[n_requests] + 1) * sizeof(uint64_t));
  if (!h) { free(first); return ORACLE_ERR_OOM; }
  for (int32_t r = 0; r < n_requests; ++r)
    oracle_block_hashes(tokens + offsets[r], offsets[r + 1] - offsets[r], B, seed, h + first[r]);
  for (int32_t r = 0; r < n_requests; ++r) {
    const int64_t nr = first[r + 1] - first[r];
    parent[r] = -1;
    for (int32_t p = r - 1; p >= 0; --p) {
      if (users[p] != users[r] || (int64_t)turns[p] != (int64_t)turns[r] - 1) continue;
      const int64_t np = first[p + 1] - first[p];
      if (np > nr) continue;
      int prefix = 1;
      for (int64_t b = 0; b < np && prefix; ++b) prefix = h[first[p] + b] == h[first[r] + b];
      if (prefix) { parent[r] = p; break; }
    }
    session[r] = parent[r] < 0 ? r : session[parent[r]];  /* parents come first */
  }
  free(h);
  free(first);
  return ORACLE_OK;
}

/* Baseline scorers (Section 5.1): scorer 1 = Bailian's weighted sum of the
 * normalised batch size and miss ratio, 2 = LMetric's product. Limits:
 * 0 <= l_i <= 2^20, 0 <= q_i <= 2^40, 0 <= LAM_NUM <= LAM_DEN <= 2^20,
 * LAM_DEN >= 1, L_r < 2^31. */
int oracle_route_batch_baseline(const oracle_index* x, int32_t B, int32_t S, uint64_t seed,
                                const int32_t* tokens, const int64_t* offsets, int32_t n_requests,
                                int32_t scorer, const int64_t* queued, const int64_t* batch, int64_t lam_num,
                                int64_t lam_den, int32_t* instance, int32_t* local_hit, int32_t* global_hit,
                                uint64_t* session_key) {
  if (!x || B < 2 || (B % 2) != 0 || S < 1 || n_requests < 0 || (scorer != 1 && scorer != 2))
    return ORACLE_ERR_INVALID_ARG;
  const int32_t N = x->N;
  if (lam_den < 1 || lam_den > (1LL << 20) || lam_num < 0 || lam_num > lam_den) return ORACLE_ERR_INVALID_ARG;
  int64_t lmax = 0;
  for (int32_t i = 0; i < N; ++i) {
    if (batch[i] < 0 || batch[i] > (1LL << 20) || queued[i] < 0 || queued[i] > (1LL << 40))
      return ORACLE_ERR_INVALID_ARG;
    if (batch[i] > lmax) lmax = batch[i];
  }
  for (int32_t r = 0; r < n_requests; ++r)
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0 || offsets[r + 1] - offsets[r] >= (1LL << 31))
      return ORACLE_ERR_INVALID_ARG;
  int64_t* c = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  uint64_t* h = NULL;
  int64_t cap = 0;
  int rc = c ? ORACLE_OK : ORACLE_ERR_OOM;
  for (int32_t r = 0; r < n_requests && rc == ORACLE_OK; ++r) {
    const int64_t L = offsets[r + 1] - offsets[r];
    const int64_t n = L / B;
    if (n + 1 > cap) {
      free(h);
      cap = n + 1;
      h = (uint64_t*)malloc((size_t)cap * sizeof(uint64_t));
      if (!h) { rc = ORACLE_ERR_OOM; break; }
    }
    oracle_block_hashes(tokens + offsets[r], L, B, seed, h);
    int64_t g;
    oracle_prefix_hits(x, h, n, c, &g);
    int32_t best = -1;
    unsigned __int128 best_f = 0;
    for (int32_t i = 0; i < N; ++i) {
      unsigned __int128 f;
      if (scorer == 2) {
        f = (unsigned __int128)(uint64_t)(queued[i] + L - (int64_t)B * c[i]) * (uint64_t)batch[i];
      } else {
        /* f_i * LAM_DEN * lmax * L, with the load term dropped when lmax = 0
         * and the miss ratio taken as 1 when L = 0 */
        const uint64_t miss = (uint64_t)(L - (int64_t)B * c[i]);
        const uint64_t Lm = (uint64_t)(lmax > 0 ? lmax : 1), Lr = (uint64_t)(L > 0 ? L : 1);
        const unsigned __int128 load_term =
            lmax > 0 ? (unsigned __int128)(uint64_t)((lam_den - lam_num) * batch[i]) * Lr : 0;
        const unsigned __int128 miss_term =
            (unsigned __int128)(uint64_t)lam_num * (L > 0 ? miss : 1) * Lm;
        f = load_term + miss_term;
      }
      if (best < 0 || f < best_f) { best = i; best_f = f; }
    }
    const int64_t gb = c[best] > g ? c[best] : g;
    instance[r] = best;
    local_hit[r] = (int32_t)((int64_t)B * c[best]);
    global_hit[r] = (int32_t)((int64_t)B * (gb - c[best]));
    session_key[r] = n == 0 ? 0 : h[(n < S ? n : S) - 1];
  }
  free(h);
  free(c);
  return rc;
}

/* The argmin cost with the loads updated request by request (one request at
 * a time, as Figure 10 routes). load_after (may be NULL) receives the loads
 * after the batch. */
int oracle_route_batch_sequential(const oracle_index* x, int32_t B, int32_t S, uint64_t seed,
                                  const int32_t* tokens, const int64_t* offsets, int32_t n_requests,
                                  const int64_t* load, int64_t w_load, int64_t w_miss, int64_t w_glob,
                                  int32_t* instance, int32_t* local_hit, int32_t* global_hit,
                                  uint64_t* session_key, int64_t* load_after) {
  if (!x || B < 2 || (B % 2) != 0 || S < 1 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  const int32_t N = x->N;
  int64_t top = 0;
  for (int32_t i = 0; i < N; ++i) {
    if (load[i] < 0) return ORACLE_ERR_INVALID_ARG;
    if (load[i] > top) top = load[i];
  }
  for (int32_t r = 0; r < n_requests; ++r)
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0) return ORACLE_ERR_INVALID_ARG;
  if (n_requests > 0 && top + (offsets[n_requests] - offsets[0]) > (1LL << 42)) return ORACLE_ERR_INVALID_ARG;
  int64_t* q = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  int64_t* c = (int64_t*)malloc((size_t)N * sizeof(int64_t));
  uint64_t* h = NULL;
  int64_t cap = 0;
  int rc = q && c ? ORACLE_OK : ORACLE_ERR_OOM;
  if (rc == ORACLE_OK) memcpy(q, load, (size_t)N * sizeof(int64_t));
  for (int32_t r = 0; r < n_requests && rc == ORACLE_OK; ++r) {
    const int64_t L = offsets[r + 1] - offsets[r];
    const int64_t n = L / B;
    if (n + 1 > cap) {
      free(h);
      cap = n + 1;
      h = (uint64_t*)malloc((size_t)cap * sizeof(uint64_t));
      if (!h) { rc = ORACLE_ERR_OOM; break; }
    }
    oracle_block_hashes(tokens + offsets[r], L, B, seed, h);
    int64_t g;
    oracle_prefix_hits(x, h, n, c, &g);
    int32_t best = -1;
    int64_t best_cost = 0;
    for (int32_t i = 0; i < N; ++i) {
      const int64_t gi = c[i] > g ? c[i] : g;
      const int64_t cost = w_load * q[i] + w_miss * (L - (int64_t)B * gi) + w_glob * (int64_t)B * (gi - c[i]);
      if (best < 0 || cost < best_cost) { best = i; best_cost = cost; }
    }
    q[best] += L - (int64_t)B * c[best];  /* the chosen queue grows before the next request */
    const int64_t gb = c[best] > g ? c[best] : g;
    instance[r] = best;
    local_hit[r] = (int32_t)((int64_t)B * c[best]);
    global_hit[r] = (int32_t)((int64_t)B * (gb - c[best]));
    session_key[r] = n == 0 ? 0 : h[(n < S ? n : S) - 1];
  }
  if (rc == ORACLE_OK && load_after) memcpy(load_after, q, (size_t)N * sizeof(int64_t));
  free(h);
  free(c);
  free(q);
  return rc;
}

/* Reuse breakdown, by definition: for every hit candidate, every earlier
 * request is searched for the block hash, earliest first. Outputs per
 * request (int32): hit blocks and their split into system-prompt,
 * intra-session and inter-session blocks. */
int oracle_reuse_breakdown(int32_t B, uint64_t seed, const int32_t* tokens, const int64_t* offsets,
                           int32_t n_requests, const int32_t* sessions, const int32_t* sys_blocks, int32_t* hit,
                           int32_t* sys, int32_t* intra, int32_t* inter) {
  if (B < 2 || (B % 2) != 0 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  for (int32_t r = 0; r < n_requests; ++r)
    if (offsets[r + 1] < offsets[r] || offsets[r] < 0 || sys_blocks[r] < 0) return ORACLE_ERR_INVALID_ARG;
  int64_t* first = (int64_t*)malloc((size_t)(n_requests + 1) * sizeof(int64_t));
  if (!first) return ORACLE_ERR_OOM;
  first[0] = 0;
  for (int32_t r = 0; r < n_requests; ++r) first[r + 1] = first[r] + (offsets[r + 1] - offsets[r]) / B;
  uint64_t* h = (uint64_t*)malloc((size_t)(first[n_requests] + 1) * sizeof(uint64_t));
  if (!h) { free(first); return ORACLE_ERR_OOM; }
  for (int32_t r = 0; r < n_requests; ++r)
    oracle_block_hashes(tokens + offsets[r], offsets[r + 1] - offsets[r], B, seed, h + first[r]);
  for (int32_t r = 0; r < n_requests; ++r) {
    hit[r] = sys[r] = intra[r] = inter[r] = 0;
    for (int64_t b = 0; b < first[r + 1] - first[r]; ++b) {
      const uint64_t key = h[first[r] + b];
      int32_t producer = -1;  /* the earliest earlier request holding the block */
      for (int32_t p = 0; p < r && producer < 0; ++p)
        for (int64_t k = first[p]; k < first[p + 1]; ++k)
          if (h[k] == key) { producer = p; break; }
      if (producer < 0) break;  /* the prefix ends at the first block the store lacks */
      hit[r]++;
      if (b < sys_blocks[r]) sys[r]++;
      else if (sessions[producer] == sessions[r]) intra[r]++;
      else inter[r]++;
    }
  }
  free(h);
  free(first);
  return ORACLE_OK;
}

/* ------------------------------------------------------------------------ */
/* Windowed load imbalance                                                   */
/* ------------------------------------------------------------------------ */

int oracle_window_imbalance(int32_t N, int64_t T, int32_t n_windows, const int32_t* inst, const int64_t* start,
                            const int64_t* end, int32_t n_requests, int64_t* out_max, int32_t* out_argmax,
                            int64_t* out_sum) {
  if (N < 1 || T < 1 || n_windows < 0 || n_requests < 0) return ORACLE_ERR_INVALID_ARG;
  for (int32_t r = 0; r < n_requests; ++r)
    if (inst[r] < 0 || inst[r] >= N || start[r] < 0 || end[r] < start[r]) return ORACLE_ERR_INVALID_ARG;
  for (int32_t w = 0; w < n_windows; ++w) {
    const int64_t lo = (int64_t)w * T, hi = lo + T;
    out_max[w] = 0;
    out_argmax[w] = 0;
    out_sum[w] = 0;
    for (int32_t i = 0; i < N; ++i) {
      int64_t s = 0; /* running-request ticks of instance i in window w */
      for (int32_t r = 0; r < n_requests; ++r) {
        if (inst[r] != i) continue;
        const int64_t a = start[r] > lo ? start[r] : lo;
        const int64_t b = end[r] < hi ? end[r] : hi;
        if (b > a) s += b - a;
      }
      out_sum[w] += s;
      if (s > out_max[w]) {
        out_max[w] = s;
        out_argmax[w] = i;
      }
    }
  }
  return ORACLE_OK;
}
