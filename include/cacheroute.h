/*
 * cacheroute.h -- C ABI of the GB300 (sm_103a) library for the data-parallel
 * hot path of planned prefix-affinity routing (CacheRoute, arXiv 2608.19677).
 *
 * The method (paper sec. 3): once per control interval a planner turns the
 * measured per-key request rates lambda_b into a routing table T: b -> a set
 * of destinations (Eq. 1 and Algorithm 1); during the interval, a request
 * whose key is in T goes to the least-loaded member of T(b), and any other
 * request goes to the less loaded of two random destinations (power-of-two
 * choices).  Before a table is enabled it is shadow-replayed and its cache
 * hits and per-destination load are compared with cache-blind balancing
 * (sec. 3.2, sec. 5.3).  The calls below are that path, on one GPU:
 *
 *   cr_hash_prefixes  request prefix span -> 64-bit routing key b
 *   cr_build_plan     keys of one interval -> lambda_b, k_b, admission, LPT, table
 *   cr_route_batch    keys -> one destination per (request, replica)
 *   cr_ring_create    consistent-hashing ring of the bounded-load comparison policy
 *   cr_plan_diff      cache and count churn between two plans (replanning under drift)
 *   cr_partition_create, cr_set_resolve_stream
 *                     routing split over two streams on disjoint SM sets
 *   cr_shadow_replay  routed requests -> per-destination LRU hits and load
 *
 * Conventions shared by every call:
 *   - Pointers named d_* are DEVICE pointers owned by the caller (any CUDA
 *     allocation, e.g. a torch tensor's storage on the context's device).
 *     Host pointers carry no prefix.  No call keeps a caller pointer after it
 *     returns, except that work it enqueued reads and writes them later on
 *     the context's stream: keep them alive until that work has finished.
 *   - The library owns cr_ctx, cr_plan and cr_replay objects and every scratch
 *     buffer behind them; it allocates device memory only inside
 *     cr_create/cr_plan_create/cr_replay_create and when a call needs a
 *     larger scratch buffer than it held before.
 *   - Every call returns a status; nothing throws.  Calls are asynchronous on
 *     the context's CUDA stream unless documented as blocking.  Device-side
 *     checks (for example an arithmetic overflow found in a kernel) are
 *     reported by the next blocking call (cr_sync, *_export, *_info).
 *   - All quantities are unsigned integers: results are exact and
 *     deterministic (bit-identical run to run).
 *   - A call whose scratch buffers are already large enough allocates
 *     nothing and does not synchronise, so a sequence of non-blocking calls
 *     can be captured into a CUDA graph after one pass over the same sizes
 *     (stream capture on a stream other than the legacy default one).
 */
#ifndef CACHEROUTE_H
#define CACHEROUTE_H

#include <stdint.h>

#if defined(__GNUC__)
#define CR_API __attribute__((visibility("default")))
#else
#define CR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------- */
#define CR_OK 0        /* success */
#define CR_EINVAL 1    /* an argument is out of range or inconsistent */
#define CR_ENOMEM 2    /* a device allocation failed */
#define CR_ECUDA 3     /* a CUDA runtime call failed (see cr_last_error) */
#define CR_ETIMEOUT 4  /* a bounded device-side wait gave up */
#define CR_EOVERFLOW 5 /* a count or load exceeded its documented range */

/* ---- dispatch policies (cr_replica.policy) -------------------------------- */
#define CR_POLICY_CACHEROUTE 0 /* T(b) from an LPT plan, else P2C (Fig. 1)       */
#define CR_POLICY_CR_NOLPT 1   /* T(b) from a random-placement plan, else P2C    */
#define CR_POLICY_CR_NOREPL 2  /* T(b) from a single-copy LPT plan, else P2C     */
#define CR_POLICY_P2C 3        /* power-of-two choices over all R ("Flat-LB")   */
#define CR_POLICY_RR 4         /* round robin over the global request index      */
#define CR_POLICY_HASH 5       /* sticky: jump consistent hash of the key        */
#define CR_POLICY_CHWBL 6      /* consistent hashing with bounded loads, eps 1/4 */

/* ---- plan variants (cr_plan_params.variant) ------------------------------- */
#define CR_VARIANT_LPT 0    /* Algorithm 1 as printed                            */
#define CR_VARIANT_RANDOM 1 /* Eq. 1 replica counts, random distinct placement  */
#define CR_VARIANT_NOREPL 2 /* k_b = 1 for every key, LPT placement              */
#define CR_VARIANT_SLOTCAP 3 /* LPT with at most W replicas per destination; a key
                                gets min(k_b, destinations with a free slot)       */

/* ---- limits --------------------------------------------------------------- */
#define CR_MAX_R 8192         /* destinations per plan / route call              */
#define CR_MAX_CAP 1024       /* LRU capacity (prefix entries) per simulator     */
#define CR_MAX_CAPS 8         /* capacities replayed together                    */
#define CR_MAX_REPLICAS 256   /* (policy, seed) replicas per route/replay call   */
#define CR_MAX_VNODES 1024    /* ring points per destination (cr_ring_create)    */
#define CR_CTR_FIELDS 5       /* requests, hits, hit tokens, prompt, prefill     */

typedef struct cr_ctx cr_ctx;
typedef struct cr_plan cr_plan;
typedef struct cr_replay cr_replay;
typedef struct cr_ring cr_ring;
typedef struct cr_partition cr_partition;
typedef struct cr_replay_input cr_replay_input;

/* ==== context ============================================================ */

/* Create a context on CUDA device `device` that enqueues its work on
 * `cuda_stream` (a cudaStream_t; NULL = the legacy default stream).
 * *out receives the context.  Errors: CR_EINVAL (out NULL, bad device),
 * CR_ECUDA, CR_ENOMEM. */
CR_API int cr_create(cr_ctx **out, int device, void *cuda_stream);

/* Destroy a context after waiting for its stream.  NULL is accepted. */
CR_API int cr_destroy(cr_ctx *ctx);

/* Switch the stream later calls enqueue on. */
CR_API int cr_set_stream(cr_ctx *ctx, void *cuda_stream);

/* Routing split over two streams: with a non-NULL stream, cr_route_batch runs
 * the per-request candidates (and the load counts of RR / HASH replicas) on
 * the context's stream and the load-dependent resolution on `cuda_stream`,
 * ordered by an event; the resolution's end (on `cuda_stream`) then covers all
 * of the call's writes to d_dest and d_load, and the next call's candidates
 * wait for it.  Callers order later readers of d_dest / d_load after
 * `cuda_stream`.  NULL restores single-stream routing.  Setting the stream the
 * context already has does nothing; switching waits for the old stream.
 * cr_sync also waits for the last resolution enqueued on `cuda_stream`, so an
 * error it raised is reported by the first blocking call after it.
 * Errors: CR_EINVAL, CR_ECUDA. */
CR_API int cr_set_resolve_stream(cr_ctx *ctx, void *cuda_stream);

/* Two CUDA streams whose kernels run on disjoint sets of SMs (green contexts):
 * *small_stream on small_sms SMs, *big_stream on the rest (the driver may round
 * the split to its SM granularity).  Kernels launched through the runtime API
 * into either stream stay on its SMs; other streams may use every SM.  The
 * streams live until cr_partition_destroy.  Errors: CR_EINVAL (bad device or
 * small_sms not in 1 .. SMs - 1), CR_ECUDA (green contexts unavailable),
 * CR_ENOMEM.  The calling thread's current device is the same after the call
 * as before it. */
CR_API int cr_partition_create(int device, uint32_t small_sms, cr_partition **out, void **big_stream,
                               void **small_stream);
/* Waits for both streams, then destroys them and their green contexts.  NULL is accepted. */
CR_API int cr_partition_destroy(cr_partition *p);

/* Blocking: wait for the context's stream (and, when routing is split by
 * cr_set_resolve_stream, for the last resolution enqueued on the resolve
 * stream), then report any error a kernel recorded since the last blocking
 * call (CR_EOVERFLOW, CR_ETIMEOUT, CR_EINVAL) and clear it. */
CR_API int cr_sync(cr_ctx *ctx);

/* Message for the last failing call on this context (static storage; never
 * NULL).  A NULL ctx gives the message of the last failed cr_create. */
CR_API const char *cr_last_error(const cr_ctx *ctx);

/* Number of kernel launches this context has issued since it was created. */
CR_API uint64_t cr_launch_count(const cr_ctx *ctx);

/* ---- per-launch timing (tracing aid; no counterpart in the paper) --------
 * With profiling enabled, the calls below bracket their main kernels with
 * CUDA timing events on the stream the kernels run on, one pair per launch:
 *   CR_PROF_HASH           k_hash_prefixes (cr_hash_prefixes)
 *   CR_PROF_PLAN           the whole plan build (cr_build_plans)
 *   CR_PROF_ROUTE_CAND     the load-independent pass of cr_route_batch
 *   CR_PROF_ROUTE_RESOLVE  its load-dependent pass (on the resolve stream if split)
 *   CR_PROF_PARTITION      the per-destination partition of cr_shadow_replay
 *   CR_PROF_REPLAY         its LRU simulation kernel
 * Every call also opens an NVTX range named after it (visible to profilers).
 * cr_profile_enable(ctx, n) keeps room for n launches (0 turns timing off) and
 * forgets earlier ones; launches beyond n are not timed.  cr_profile_read is
 * blocking: it waits for the recorded events and returns the number of timed
 * launches with `tag` and their summed duration in milliseconds.  Errors:
 * CR_EINVAL (tag out of range), CR_ENOMEM, CR_ECUDA. */
#define CR_PROF_HASH 0
#define CR_PROF_PLAN 1
#define CR_PROF_ROUTE_CAND 2
#define CR_PROF_ROUTE_RESOLVE 3
#define CR_PROF_PARTITION 4
#define CR_PROF_REPLAY 5
#define CR_PROF_TAGS 6
CR_API int cr_profile_enable(cr_ctx *ctx, uint32_t max_launches);
CR_API int cr_profile_read(cr_ctx *ctx, uint32_t tag, uint64_t *launches, double *total_ms);

/* ==== a1: prefix-span routing key ==================================== */
/*
 * The paper routes on an opaque business key b, which it allows to be salted
 * (sec. 3.1; supplement, data handling), and defines no hash.  This library
 * derives b from the request's reusable prefix span:
 *
 *   b = fmix64(salt ^ P) + sum_{i < ceil(P/2)} fmix64(w_i ^ (salt + (i+1)*G))  (mod 2^64)
 *
 * with fmix64 the SplitMix64 finaliser, G = 0x9e3779b97f4a7c15, and
 * w_i = (uint32)t[2i] | (uint32)t[2i+1] << 32 the i-th pair of prefix tokens
 * (t[P] reads as 0 when P is odd).  Only the P prefix tokens are read.
 *
 *   d_tokens  int32 token arena (any layout: records may overlap or be padded)
 *   d_off     uint64[n] token index of request r's first prefix token
 *   d_plen    uint32[n] prefix length P_r in tokens (0 allowed)
 *   n         number of requests (0 allowed: nothing is enqueued)
 *   salt      64-bit salt
 *   d_key_out uint64[n] receives b_r
 * Requests whose prefix starts on a 16-byte boundary (d_off[r] % 4 == 0) take
 * the vectorised path; any other offset is still exact, only slower.
 * Errors: CR_EINVAL (NULL pointer with n > 0). */
CR_API int cr_hash_prefixes(cr_ctx *ctx, const int32_t *d_tokens, const uint64_t *d_off,
                     const uint32_t *d_plen, uint64_t n, uint64_t salt, uint64_t *d_key_out);

/* ==== a2..a6: the plan (Eq. 1, Algorithm 1) ========================== */

typedef struct {
    uint32_t R;               /* destinations, 1..CR_MAX_R                          */
    uint32_t W;               /* warm slots per destination; C = R*W (sec. 3.1)     */
    uint64_t qcap_num;        /* q_cap = qcap_num / qcap_den requests per interval  */
    uint64_t qcap_den;        /*   (den < 2^32, num >= 1)                            */
    uint32_t variant;         /* CR_VARIANT_*                                        */
    uint32_t reserved;        /* must be 0                                           */
    uint64_t seed;            /* CR_VARIANT_RANDOM: placement stream                 */
    uint64_t epoch;           /* CR_VARIANT_RANDOM: e.g. the interval index          */
    const uint64_t *d_init_load; /* uint64[R] starting loads, or NULL for the
                                    cold-tail share floor(cold requests / R)        */
} cr_plan_params;

/* Create an empty plan owned by the library (device buffers grow on demand). */
CR_API int cr_plan_create(cr_ctx *ctx, cr_plan **out);
/* Destroy a plan (waits for the context's stream).  NULL is accepted. */
CR_API int cr_plan_destroy(cr_ctx *ctx, cr_plan *plan);

/*
 * Build n_plans plans from the same interval's keys d_key[n] (uint64, any
 * order, device).  One per-key histogram (lambda_b = number of requests with
 * key b) is shared by all of them; plan j follows params[j]:
 *   k_b   = min(R, max(1, ceil(lambda_b * den / num)))    (Eq. 1; 1 for NOREPL)
 *   order = keys by (lambda_b descending, b ascending)
 *   admit the longest prefix of that order with sum k_b <= C = R*W
 *          (Algorithm 1 admission step: stop at the first key that does not fit)
 *   L[r]  = d_init_load[r], or floor(sum of unadmitted lambda_b / R)
 *   LPT:    for each admitted b in order, T(b) = the k_b smallest (L[r], r),
 *           in that order; lambda_b is split into k_b integer jobs
 *           floor(lambda_b/k_b) (+1 for the first lambda_b mod k_b members),
 *           added to L (Algorithm 1 placement loop).
 *   RANDOM: T(b) = first k_b steps of a Fisher-Yates shuffle of 0..R-1 driven
 *           by Philox4x64-10(key = (seed, 1), counter = (a, s, 1, epoch)),
 *           a = admission position, s = step (sec. 5.2, Table 4 "+replication").
 * The table T is then installed as a device hash table for cr_route_batch.
 * plans[j] must be distinct objects from cr_plan_create; any previous content
 * is replaced.  Blocking: no.  Errors: CR_EINVAL (n >= 2^32, bad params,
 * NULL pointers), CR_ENOMEM, CR_ECUDA; CR_EOVERFLOW is reported by the next
 * blocking call if a load L[r] reaches 2^47. */
CR_API int cr_build_plans(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
                   uint32_t n_plans, cr_plan *const *plans);

/* cr_build_plans with one plan. */
CR_API int cr_build_plan(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
                  cr_plan *plan);

typedef struct {
    uint64_t n;      /* requests the plan was built from                     */
    uint64_t U;      /* distinct keys                                         */
    uint64_t n_adm;  /* admitted keys                                         */
    uint64_t sum_k;  /* sum of k_b over admitted keys (<= C)                  */
    uint64_t cold;   /* requests of unadmitted keys                           */
    uint64_t max_k;  /* largest k_b among admitted keys (0 if none)           */
    uint32_t R, W;
} cr_plan_info;

/* Blocking: plan sizes.  Errors as cr_sync. */
CR_API int cr_plan_get_info(cr_ctx *ctx, const cr_plan *plan, cr_plan_info *out);

/* Blocking: copy a plan to HOST arrays (any may be NULL to skip it), sized
 * from cr_plan_get_info:
 *   ukey[U], ucnt[U]           histogram, keys ascending
 *   adm_key[n_adm], adm_cnt[n_adm], adm_k[n_adm]   admission order
 *   koff[n_adm+1]              member offsets
 *   members[sum_k] (uint16), jobs[sum_k]           T(b) and its expected loads
 *   load[R]                    final L */
CR_API int cr_plan_export(cr_ctx *ctx, const cr_plan *plan, uint64_t *ukey, uint64_t *ucnt,
                   uint64_t *adm_key, uint64_t *adm_cnt, uint32_t *adm_k, uint32_t *koff,
                   uint16_t *members, uint64_t *jobs, uint64_t *load);

/* Blocking: install a plan computed elsewhere -- for example one exported by
 * cr_plan_export from another process, or a host planner's table (the paper's
 * planner runs on the host, sec. 3.1) -- so that cr_route_batch can route
 * with it.  Host arrays in admission order, as cr_plan_export gives them:
 *   adm_key[n_adm], adm_cnt[n_adm], adm_k[n_adm]   keys, their rates, k_b
 *   members[sum k_b]   T(b) of each key in turn (uint16; the first member of
 *                      a key breaks ties first, as in dispatch)
 *   jobs[sum k_b], load[R]   optional (NULL: zeros); kept for export only
 * The plan's histogram becomes the admitted keys with their rates.  Errors:
 * CR_EINVAL (R or W out of range, n_adm or sum k_b above R*W, k_b of 0 or
 * above R, a member >= R or repeated within a key, a repeated key, NULL
 * arrays), CR_ENOMEM, CR_ECUDA. */
CR_API int cr_plan_import(cr_ctx *ctx, cr_plan *plan, uint32_t R, uint32_t W, uint64_t n_adm, const uint64_t *adm_key,
                          const uint64_t *adm_cnt, const uint32_t *adm_k, const uint16_t *members,
                          const uint64_t *jobs, const uint64_t *load);

/* ==== f2: plan difference (replanning under drift) ===================== */

/* Integer counts describing how plan b differs from plan a (supplement
 * "Replanning Under Drift", replan table; sec. 5 "Rate drift and remapping").
 * The assignment set of a plan is its set of (key, destination) pairs.
 *   cache churn = 1 - pairs_common / (pairs_a + pairs_b - pairs_common)
 *   count churn = hist_kb_changed / hist_keys
 * Count churn is taken over every key of either plan's histogram with k_b
 * from Eq. 1 of that plan's rate and q_cap (single-copy plans: 1); a key
 * missing from one histogram has lambda = 0 there, so k_b = 1.  The adm_*
 * counts restrict the comparison to admitted keys (k = 0 and an empty set for
 * a key a plan did not admit). */
typedef struct {
    uint64_t keys_a, keys_b;       /* admitted keys of each plan */
    uint64_t keys_common;          /* keys admitted by both */
    uint64_t pairs_a, pairs_b;     /* (key, destination) pairs = sum of k_b over admitted keys */
    uint64_t pairs_common;         /* pairs in both tables */
    uint64_t adm_k_changed;        /* keys admitted by either plan whose k in T differs */
    uint64_t adm_set_changed;      /* keys admitted by either plan whose destination set differs */
    uint64_t hist_keys;            /* keys in either plan's histogram */
    uint64_t hist_kb_changed;      /* of those, keys whose Eq. 1 k_b differs */
} cr_plan_diff_counts;

/* Blocking: compare two built plans with the same R (device kernels: one warp
 * per admitted key, member sets compared through per-warp bitmaps of R bits;
 * histograms through per-plan hash tables in context scratch, 32 bytes per
 * request of the larger build); *out receives the counts.  The kernels run on
 * ctx's stream: plans built through another context must be complete first
 * (e.g. cr_sync on that context).  Errors: CR_EINVAL (plan not built, R
 * differs), CR_ENOMEM, CR_ECUDA. */
CR_API int cr_plan_diff(cr_ctx *ctx, const cr_plan *a, const cr_plan *b, cr_plan_diff_counts *out);

/* ==== a7: batched dispatch ========================================== */

/*
 * Ring of the bounded-load comparison policy (CHWBL, sec. 4; epsilon = 0.25;
 * consistent hashing with bounded loads, Mirrokni, Thorup and Zadimoghaddam,
 * SODA 2018).  The paper fixes epsilon only; the ring is this library's
 * reading: destination d owns `vnodes` points, point (d, v) being output
 * number k = d*vnodes + v of SplitMix64 from state `seed`, that is
 * fmix64(seed + (k + 1) * 0x9e3779b97f4a7c15) mod 2^64, and the ring lists
 * the R*vnodes points in ascending (point, d) order.
 * cr_ring_create builds it on the device (enqueued on the context's stream;
 * R in 1..CR_MAX_R, vnodes in 1..CR_MAX_VNODES).  Errors: CR_EINVAL,
 * CR_ENOMEM, CR_ECUDA.  The ring is read-only afterwards and may be shared
 * by any number of replicas and calls. */
CR_API int cr_ring_create(cr_ctx *ctx, uint32_t R, uint32_t vnodes, uint64_t seed, cr_ring **out);
/* Destroy (waits for the context's stream).  NULL is accepted. */
CR_API int cr_ring_destroy(cr_ctx *ctx, cr_ring *ring);
/* Blocking: copy the ring to host arrays point[R*vnodes] (ascending) and
 * owner[R*vnodes]. */
CR_API int cr_ring_export(cr_ctx *ctx, const cr_ring *ring, uint64_t *point, uint16_t *owner);

typedef struct {
    uint32_t policy;      /* CR_POLICY_* */
    uint32_t reserved;    /* must be 0 */
    uint64_t seed;        /* RNG / offset / hash seed of this replica */
    const cr_ring *ring;  /* CR_POLICY_CHWBL: its ring (R destinations); else ignored */
} cr_replica;

/*
 * Route requests d_key[n] (device, arrival order, global request indices
 * first_req_index .. first_req_index+n-1) for n_rep replicas at once.
 *   plans[i]  plan used by replica i (CACHEROUTE, CR_NOLPT, CR_NOREPL), or
 *             NULL for P2C, RR, HASH and CHWBL.  Plans may be shared; plan R
 *             must equal R.
 *   reps[i]   policy and seed (host array)
 *   batch_B   requests are taken in batches of batch_B (>= 1); every request
 *             of a batch sees the load vector as it stood when the batch
 *             began; the batch's requests are added to it afterwards.
 *             batch_B = 1 is exact sequential dispatch.
 *   d_load    uint64[n_rep][R] live load, in/out (pass zeros at the start of
 *             an interval to count requests routed in the interval)
 *   d_dest    uint16[n_rep][n] receives the destination of every request
 * Rules (Fig. 1 and sec. 3.1; comparison policies of sec. 4):
 *   CACHEROUTE-type: b in T -> member of T(b) with the smallest
 *     (load, position in T(b)); otherwise P2C with the replica's policy id.
 *   P2C: u = Philox4x64-10(key = (seed, policy), counter = (g, 0, 0, 0)),
 *     d1 = floor(u0 R / 2^64), d2 = (d1 + 1 + floor(u1 (R-1) / 2^64)) mod R;
 *     pick d1 if load[d1] <= load[d2], else d2.
 *   RR: (g + seed) mod R.     HASH: jump_hash(fmix64(b ^ seed), R).
 *   CHWBL: with m = the sum of the load vector the request sees, every
 *     destination may hold cap = ceil(5 (m + 1) / (4 R)) requests; starting
 *     at the first ring point >= fmix64(b ^ seed) (wrapping to the first
 *     point), walk the ring and take the first owner whose load is < cap.
 *     The least-loaded destination is always below cap, so the walk ends.
 * Batches of at most 32 requests are resolved by one warp per replica that
 * takes 32 // batch_B whole batches per step; longer batches by one CTA per
 * replica.  Both give the sequential result defined above.
 * Errors: CR_EINVAL (R == 0 or > CR_MAX_R, n_rep > CR_MAX_REPLICAS, missing
 * or mismatched plan or ring, batch_B == 0, n >= 2^40).  A load sum that
 * has wrapped past 2^64 can leave no destination below cap: the request then
 * takes the owner of its first ring point and the next blocking call
 * reports CR_EOVERFLOW. */
CR_API int cr_route_batch(cr_ctx *ctx, const cr_plan *const *plans, const cr_replica *reps,
                   uint32_t n_rep, uint32_t R, const uint64_t *d_key, uint64_t n,
                   uint64_t first_req_index, uint32_t batch_B, uint64_t *d_load,
                   uint16_t *d_dest);

/* ==== a8, a9: shadow replay ========================================= */

/* Create replay state for n_rep replicas x R destinations x n_caps LRU
 * capacities (caps[] host array, each 1..CR_MAX_CAP, n_caps <= CR_MAX_CAPS).
 * Every simulator starts empty.  Errors: CR_EINVAL, CR_ENOMEM. */
CR_API int cr_replay_create(cr_ctx *ctx, uint32_t n_rep, uint32_t R, const uint32_t *caps,
                     uint32_t n_caps, cr_replay **out);
/* Byte-aware variant (token-weighted capacity; the paper's byte budgets of
 * sec. 3.1 and 6, and the 70B configuration's 24k-token slot budget read as
 * tokens): every simulator holds whole prefixes, most recent first, while their
 * prefix tokens sum to at most its capacity (token_caps[], 1 .. 2^31) and
 * there are at most CR_MAX_CAP of them; an access moves or inserts its key at
 * the front, then the least recent prefixes are evicted until both limits
 * hold.  A key must have the same prefix length at every access (the longest
 * recent run of prefixes that fits is then what every capacity holds, and one
 * list decides all capacities); a key that comes back with another length
 * makes the next blocking call return CR_EINVAL, and the counters of that call
 * are not meaningful.  cr_shadow_replay, cr_replay_reset, cr_replay_destroy
 * and cr_replay_export_state work on it unchanged.  Errors: CR_EINVAL,
 * CR_ENOMEM. */
CR_API int cr_replay_create_tokens(cr_ctx *ctx, uint32_t n_rep, uint32_t R, const uint32_t *token_caps,
                                   uint32_t n_caps, cr_replay **out);
/* Empty every simulator (enqueued on the stream). */
CR_API int cr_replay_reset(cr_ctx *ctx, cr_replay *rp);
/* Destroy (waits for the stream).  NULL is accepted. */
CR_API int cr_replay_destroy(cr_ctx *ctx, cr_replay *rp);

/*
 * Replay n routed requests through every simulator.  For replica i the
 * requests with d_dest[i*n + j] == r reach destination r's caches in
 * arrival order; each (replica, capacity, destination) is a whole-prefix LRU
 * of `cap` entries keyed by the routing key (this library's model of the
 * engine-native prefix cache that admitted and cold-tail traffic share,
 * sec. 3.2).  A request hits when its key is resident: it then becomes most
 * recent and its P prefix tokens are hit tokens; otherwise it is inserted as
 * most recent and, when the cache is full, the least recent entry leaves.
 * State persists across calls (and plan changes) until cr_replay_reset.
 *   d_key uint64[n], d_plen uint32[n], d_slen uint32[n]: per request
 *   d_dest uint16[n_rep][n]: destinations (each < R, checked on device)
 *   d_ctr  uint64[n_rep][n_caps][R][5], ACCUMULATED (+=): requests, hit
 *          requests, hit tokens, prompt tokens (P+S), prefill tokens
 *          (prompt - hit tokens)
 * Errors: CR_EINVAL (NULL pointers with n > 0, n >= 2^31); a destination
 * >= R is skipped and reported as CR_EINVAL by the next blocking call. */
CR_API int cr_shadow_replay(cr_ctx *ctx, cr_replay *rp, const uint64_t *d_key, const uint32_t *d_plen,
                     const uint32_t *d_slen, const uint16_t *d_dest, uint64_t n,
                     uint64_t *d_ctr);

/*
 * cr_shadow_replay in two calls, so that the partition (a8) of later requests
 * can run on another stream while the simulators (a9), which must take the
 * requests in arrival order, work through earlier ones:
 *   cr_replay_partition  splits n routed requests (same arguments as
 *       cr_shadow_replay) into every (replica, destination) stream in arrival
 *       order, into a library-owned input object `in` (its device buffers grow on
 *       demand; growing waits for the whole device).  Enqueued on ctx's stream.
 *   cr_replay_simulate   runs the simulators of `rp` over `in` and accumulates
 *       the counters exactly as cr_shadow_replay does.  Enqueued on ctx's stream,
 *       which the caller orders after the partition (same stream, or an event)
 *       and before any later partition into the same `in`.
 * `in` must have been partitioned for a replay of the same n_rep, R and
 * capacity kind.  cr_shadow_replay is exactly partition + simulate.  Errors:
 * CR_EINVAL (shape mismatch, NULL pointers, n * n_rep >= 2^32 - 1), CR_ENOMEM,
 * CR_ECUDA. */
CR_API int cr_replay_input_create(cr_ctx *ctx, cr_replay_input **out);
CR_API int cr_replay_input_destroy(cr_ctx *ctx, cr_replay_input *in);
CR_API int cr_replay_partition(cr_ctx *ctx, const cr_replay *rp, const uint64_t *d_key, const uint32_t *d_plen,
                               const uint32_t *d_slen, const uint16_t *d_dest, uint64_t n, cr_replay_input *in);
CR_API int cr_replay_simulate(cr_ctx *ctx, cr_replay *rp, const cr_replay_input *in, uint64_t *d_ctr);

/* Blocking: resident keys of one simulator at the largest capacity, most
 * recent first, into keys_out[CR_MAX_CAP] (host); *fill_out = their count.
 * The state at a smaller capacity c is the first min(c, fill) of them. */
CR_API int cr_replay_export_state(cr_ctx *ctx, const cr_replay *rp, uint32_t rep, uint32_t r,
                           uint64_t *keys_out, uint32_t *fill_out);

/* Blocking: set one simulator's resident keys (host array, most recent
 * first, distinct, at most the largest capacity), e.g. from
 * cr_replay_export_state, so that a replay can resume from saved state; the
 * simulators of smaller capacities hold the first min(c, fill) of them.
 * Prefix-count replays only (a token-weighted replay also keeps each prefix's
 * size).  Errors: CR_EINVAL (bad stream, too many keys, repeated key, token
 * replay), CR_ECUDA. */
CR_API int cr_replay_import_state(cr_ctx *ctx, cr_replay *rp, uint32_t rep, uint32_t r, const uint64_t *keys,
                                  uint32_t fill);

/* ==== allocation-free key histogram ================================== */
/*
 * The paper has no counterpart to this call: it exists for callers that
 * cannot allocate device memory at the moment they call in, for example a
 * process whose device memory is owned by another runtime's pool, or a
 * latency-critical path that cannot afford cudaMalloc (which may synchronise
 * the device).  It needs no context: it computes the same per-key histogram
 * as cr_build_plans (lambda_b = requests with key b) with all of its scratch
 * in a fixed array inside the library (about 3.6 MB, held on every GPU that
 * loads the library until the process exits), and calls no allocating
 * function.
 *   d_key   uint64[n] keys (device), n <= CR_NOALLOC_MAX_KEYS
 *   d_ukey  uint64[n] receives the distinct keys, ascending (first *d_U used)
 *   d_ucnt  uint64[n] receives their counts
 *   d_U     uint64[1] (device) receives the number of distinct keys
 *   cuda_stream  stream the work is enqueued on (NULL = legacy default)
 * The first call on a device looks up the array's device address on that
 * device (it must be current); make that first call before any stream
 * capture.  All calls share the one array: calls whose work overlaps on the
 * GPU (different streams, or different host threads) race and must be
 * ordered by the caller.  Every call clears what it needs, so earlier
 * contents never leak into a result.
 * Errors (message via cr_last_error(NULL)): CR_EINVAL (n too large, NULL
 * pointer), CR_ECUDA. */
#define CR_NOALLOC_MAX_KEYS 65536
CR_API int cr_key_histogram_noalloc(const uint64_t *d_key, uint64_t n, uint64_t *d_ukey, uint64_t *d_ucnt,
                                    uint64_t *d_U, void *cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* CACHEROUTE_H */
