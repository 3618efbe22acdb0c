/*
 * CPU oracle for the planned prefix-affinity routing hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file; only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header, table or constant
 * generator with the CUDA library: every definition below was written from
 * the paper (CacheRoute, arXiv 2608.19677) and from the published
 * definitions of the two mixing functions it uses.
 *
 * Plain, slow, single-threaded C.  Every quantity is an unsigned integer
 * (requests, tokens, keys), so results are exact.
 *
 * Functions and the passages they follow:
 *   orc_fmix64, orc_philox4x64_10 .... SplitMix64 finaliser (Steele, Lea and
 *       Flood, OOPSLA 2014); Philox4x64-10 (Salmon et al., SC 2011).
 *   orc_hash_prefixes ................ the routing key b of a request (sec. 3.1,
 *       Appendix "Data handling": b is an opaque, possibly salted key).  The
 *       paper defines no hash; the definition here is this library's reading.
 *   orc_histogram .................... per-key rate lambda_b over one control
 *       interval (Fig. 1 "aggregate telemetry", Algorithm 1 inputs).
 *   orc_build_plan ................... Eq. 1 (k_b), warm-set admission
 *       (sec. 3.1 "Warm-set admission", Algorithm 1 admission step), cold-tail
 *       initialisation and LPT placement (sec. 3.1 "Placement and dispatch",
 *       Algorithm 1 placement loop); random, single-copy and slot-capped
 *       (per-destination budget, this library's reading) variants.
 *   orc_route ........................ dispatch (Fig. 1; sec. 3.1: least-loaded
 *       member of T(b), otherwise power-of-two choices over the fleet) and the
 *       comparison policies of sec. 4 (Flat-LB, sticky hashing, consistent
 *       hashing with bounded loads at epsilon = 0.25) plus round-robin.
 *   orc_ring_* ....................... the consistent-hashing ring of that
 *       bounded-load policy (the ring layout is this library's reading).
 *   orc_replay_* ..................... shadow replay of each destination's
 *       prefix cache as a whole-prefix LRU (deployment gate of sec. 3.2 and 5.3; the paper
 *       replays on hardware, the LRU model is this library's reading).
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_ENOMEM 2

/* ---------------------------------------------------------------------- */
/* Mixing functions                                                        */
/* ---------------------------------------------------------------------- */

/* SplitMix64 output finaliser ("mix64", variant 13 of Stafford's mixers). */
uint64_t orc_fmix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

/* SplitMix64 increment (the golden-ratio "gamma"). */
#define ORC_GAMMA 0x9e3779b97f4a7c15ULL

static void mul128(uint64_t a, uint64_t b, uint64_t *hi, uint64_t *lo)
{
    unsigned __int128 p = (unsigned __int128)a * (unsigned __int128)b;
    *hi = (uint64_t)(p >> 64);
    *lo = (uint64_t)p;
}

/* Philox4x64 with 10 rounds, as defined by Salmon, Moraes, Dror and Shaw,
 * "Parallel random numbers: as easy as 1, 2, 3" (SC 2011). */
void orc_philox4x64_10(const uint64_t ctr_in[4], const uint64_t key_in[2], uint64_t out[4])
{
    uint64_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
    uint64_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        uint64_t hi0, lo0, hi1, lo1;
        mul128(0xD2E7470EE14C6C93ULL, c0, &hi0, &lo0);
        mul128(0xCA5A826395121157ULL, c2, &hi1, &lo1);
        uint64_t n0 = hi1 ^ c1 ^ k0;
        uint64_t n1 = lo1;
        uint64_t n2 = hi0 ^ c3 ^ k1;
        uint64_t n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
        k0 += 0x9E3779B97F4A7C15ULL;
        k1 += 0xBB67AE8584CAA73BULL;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* floor(u * m / 2^64): maps a uniform 64-bit word onto [0, m). */
static uint64_t scale_u64(uint64_t u, uint64_t m)
{
    uint64_t hi, lo;
    mul128(u, m, &hi, &lo);
    return hi;
}

/* ---------------------------------------------------------------------- */
/* a1: prefix-span key                                                     */
/* ---------------------------------------------------------------------- */

/*
 * key = fmix64(salt ^ P) + sum_{i < ceil(P/2)} fmix64(w_i ^ (salt + (i+1)*gamma))   (mod 2^64)
 * where w_i = (uint32)tok[2i] | (uint32)tok[2i+1] << 32, and tok[P] reads as 0
 * when P is odd.  Only the prefix span tok[off, off+P) is read.
 */
uint64_t orc_hash_one(const int32_t *tok, uint32_t P, uint64_t salt)
{
    uint64_t h = orc_fmix64(salt ^ (uint64_t)P);
    uint32_t nwords = (P + 1) / 2;
    for (uint32_t i = 0; i < nwords; ++i) {
        uint64_t lo = (uint32_t)tok[2 * i];
        uint64_t hi = (2 * i + 1 < P) ? (uint32_t)tok[2 * i + 1] : 0;
        uint64_t w = lo | (hi << 32);
        uint64_t k = salt + (uint64_t)(i + 1) * ORC_GAMMA;
        h += orc_fmix64(w ^ k);
    }
    return h;
}

void orc_hash_prefixes(const int32_t *tokens, const uint64_t *off, const uint32_t *plen,
                       uint64_t n, uint64_t salt, uint64_t *key_out)
{
    for (uint64_t r = 0; r < n; ++r)
        key_out[r] = orc_hash_one(tokens + off[r], plen[r], salt);
}

/* ---------------------------------------------------------------------- */
/* a2: per-key rate histogram                                              */
/* ---------------------------------------------------------------------- */

static int cmp_u64(const void *a, const void *b)
{
    uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
    return (x > y) - (x < y);
}

/* lambda_b = number of requests in the interval that carry key b.
 * Output: distinct keys ascending with their counts; returns U. */
uint64_t orc_histogram(const uint64_t *key, uint64_t n, uint64_t *ukey, uint64_t *cnt)
{
    if (n == 0)
        return 0;
    uint64_t *s = (uint64_t *)malloc(n * sizeof(uint64_t));
    memcpy(s, key, n * sizeof(uint64_t));
    qsort(s, n, sizeof(uint64_t), cmp_u64);
    uint64_t U = 0;
    for (uint64_t i = 0; i < n; ++i) {
        if (i == 0 || s[i] != s[i - 1]) {
            ukey[U] = s[i];
            cnt[U] = 0;
            ++U;
        }
        cnt[U - 1] += 1;
    }
    free(s);
    return U;
}

/* ---------------------------------------------------------------------- */
/* a3..a6: the plan (Eq. 1 and Algorithm 1)                                */
/* ---------------------------------------------------------------------- */

enum { ORC_VARIANT_LPT = 0, ORC_VARIANT_RANDOM = 1, ORC_VARIANT_NOREPL = 2, ORC_VARIANT_SLOTCAP = 3 };
enum { ORC_CR = 0, ORC_CR_NOLPT = 1, ORC_CR_NOREPL = 2, ORC_P2C = 3, ORC_RR = 4, ORC_HASH = 5, ORC_CHWBL = 6 };

typedef struct {
    uint32_t R, W;
    uint64_t qcap_num, qcap_den;   /* q_cap = num / den requests per interval */
    uint32_t variant;              /* ORC_VARIANT_* */
    uint64_t seed, epoch;          /* random placement stream (variant RANDOM) */
    const uint64_t *init_load;     /* nullable: cold-tail share */
} orc_plan_params;

/* Output arrays are caller-owned: adm_* sized >= n (distinct keys bound),
 * members/jobs sized >= R*W, load sized R. */
typedef struct {
    uint64_t U, n_adm, sum_k, cold;
    uint64_t *adm_key;   /* admitted keys in admission order (lambda desc, key asc) */
    uint64_t *adm_cnt;   /* their lambda */
    uint32_t *adm_k;     /* their k_b */
    uint32_t *koff;      /* [n_adm+1] offsets into members/jobs */
    uint16_t *members;   /* T(b), in selection order */
    uint64_t *jobs;      /* expected load each member receives */
    uint64_t *load;      /* [R] final L */
} orc_plan;

typedef struct {
    uint64_t key, cnt;
} kc_t;

static int cmp_rate_desc(const void *a, const void *b)
{
    const kc_t *x = (const kc_t *)a, *y = (const kc_t *)b;
    if (x->cnt != y->cnt)
        return x->cnt > y->cnt ? -1 : 1;
    return (x->key > y->key) - (x->key < y->key);
}

/* Eq. 1 with q_cap = num/den, clamped to R (T(b) holds k_b DISTINCT destinations). */
uint32_t orc_kb(uint64_t lambda, uint64_t num, uint64_t den, uint32_t R)
{
    uint64_t a = lambda * den;           /* lambda < 2^32 and den < 2^32 */
    uint64_t k = a / num + (a % num != 0);
    if (k < 1)
        k = 1;
    if (k > R)
        k = R;
    return (uint32_t)k;
}

int orc_build_plan(const uint64_t *key, uint64_t n, const orc_plan_params *p, orc_plan *out)
{
    if (!p || !out || p->R == 0 || p->R > 65535 || p->W == 0 || p->qcap_num == 0 ||
        p->qcap_den == 0 || p->qcap_den >= (1ULL << 32) || n >= (1ULL << 32) || p->variant > 3)
        return ORC_EINVAL;
    const uint32_t R = p->R;
    const uint64_t C = (uint64_t)R * p->W;

    /* rates */
    uint64_t *ukey = (uint64_t *)malloc((n + 1) * sizeof(uint64_t));
    uint64_t *cnt = (uint64_t *)malloc((n + 1) * sizeof(uint64_t));
    uint64_t U = orc_histogram(key, n, ukey, cnt);

    /* sort keys by decreasing lambda (ties: ascending key) */
    kc_t *kc = (kc_t *)malloc((U + 1) * sizeof(kc_t));
    for (uint64_t i = 0; i < U; ++i) {
        kc[i].key = ukey[i];
        kc[i].cnt = cnt[i];
    }
    qsort(kc, U, sizeof(kc_t), cmp_rate_desc);

    /* admit while sum k_b <= C: the longest prefix of that order */
    uint64_t sum = 0, n_adm = 0;
    for (uint64_t i = 0; i < U; ++i) {
        uint32_t k = (p->variant == ORC_VARIANT_NOREPL) ? 1
                                                        : orc_kb(kc[i].cnt, p->qcap_num, p->qcap_den, R);
        if (sum + k > C)
            break;
        sum += k;
        out->adm_key[n_adm] = kc[i].key;
        out->adm_cnt[n_adm] = kc[i].cnt;
        out->adm_k[n_adm] = k;
        ++n_adm;
    }
    uint64_t cold = 0;
    for (uint64_t i = n_adm; i < U; ++i)
        cold += kc[i].cnt;

    /* L[r] starts at the expected cold-tail share */
    for (uint32_t r = 0; r < R; ++r)
        out->load[r] = p->init_load ? p->init_load[r] : cold / R;

    /* placement, in admission (decreasing-rate) order.  Slot-capped variant
     * (per-destination byte budget, this library's reading): a destination
     * holds at most W replicas; a key goes to the k smallest (L[r], r) among
     * destinations with a free slot, k = min(k_b, such destinations), so it
     * may get fewer replicas than Eq. 1 asks, or none (then T has no entry
     * for it and it is routed like a key that was not admitted). */
    uint8_t *taken = (uint8_t *)calloc(R, 1);
    uint32_t *slots = (uint32_t *)calloc(R, sizeof(uint32_t));
    uint64_t placed = 0;
    uint32_t *chosen = (uint32_t *)malloc(R * sizeof(uint32_t));
    uint32_t *perm = (uint32_t *)malloc(R * sizeof(uint32_t));
    uint32_t pos = 0;
    for (uint64_t a = 0; a < n_adm; ++a) {
        uint32_t k = out->adm_k[a];
        uint64_t lam = out->adm_cnt[a];
        out->koff[a] = pos;
        if (p->variant == ORC_VARIANT_SLOTCAP) {
            uint32_t free_dest = 0;
            for (uint32_t r = 0; r < R; ++r)
                free_dest += slots[r] < p->W;
            if (k > free_dest)
                k = free_dest;
            out->adm_k[a] = k;
            if (k == 0)
                continue;
        }
        if (p->variant == ORC_VARIANT_RANDOM) {
            /* k distinct destinations in uniformly random order: the first k
             * steps of a Fisher-Yates shuffle of 0..R-1, step s swapping slot s
             * with slot s + floor(u * (R - s) / 2^64), u the first word of
             * Philox(key = (seed, CR_NOLPT), counter = (a, s, 1, epoch)). */
            for (uint32_t r = 0; r < R; ++r)
                perm[r] = r;
            for (uint32_t s = 0; s < k; ++s) {
                uint64_t ctr[4] = {a, s, 1, p->epoch}, pk[2] = {p->seed, ORC_CR_NOLPT}, o[4];
                orc_philox4x64_10(ctr, pk, o);
                uint32_t t = s + (uint32_t)scale_u64(o[0], (uint64_t)(R - s));
                uint32_t tmp = perm[s];
                perm[s] = perm[t];
                perm[t] = tmp;
                chosen[s] = perm[s];
            }
        } else {
            /* the k smallest (L[r], r), in that order */
            for (uint32_t s = 0; s < k; ++s) {
                int64_t best = -1;
                for (uint32_t r = 0; r < R; ++r) {
                    if (taken[r] || (p->variant == ORC_VARIANT_SLOTCAP && slots[r] >= p->W))
                        continue;
                    if (best < 0 || out->load[r] < out->load[best])
                        best = r;
                }
                taken[best] = 1;
                chosen[s] = (uint32_t)best;
            }
        }
        /* k jobs of lambda/k in integers: the first (lambda mod k) get one more */
        uint64_t q = lam / k, rem = lam % k;
        for (uint32_t s = 0; s < k; ++s) {
            uint64_t job = q + (s < rem ? 1 : 0);
            out->members[pos + s] = (uint16_t)chosen[s];
            out->jobs[pos + s] = job;
            out->load[chosen[s]] += job;
            taken[chosen[s]] = 0;
            slots[chosen[s]] += 1;
        }
        pos += k;
        placed += k;
    }
    out->koff[n_adm] = pos;
    out->U = U;
    out->n_adm = n_adm;
    out->sum_k = p->variant == ORC_VARIANT_SLOTCAP ? placed : sum;
    out->cold = cold;
    free(slots);
    free(taken);
    free(chosen);
    free(perm);
    free(kc);
    free(ukey);
    free(cnt);
    return ORC_OK;
}

/* ---------------------------------------------------------------------- */
/* a7: dispatch                                                            */
/* ---------------------------------------------------------------------- */

/* Jump consistent hash (Lamping and Veach, 2014), with the bucket-jump step
 * evaluated exactly in integers: j = floor((b+1) * 2^31 / ((k >> 33) + 1)). */
uint32_t orc_jump_hash(uint64_t k, uint32_t R)
{
    int64_t b = -1;
    uint64_t j = 0;
    while (j < R) {
        b = (int64_t)j;
        k = k * 2862933555777941757ULL + 1;
        j = ((uint64_t)(b + 1) << 31) / ((k >> 33) + 1);
    }
    return (uint32_t)b;
}

/* sorted view of a plan's admitted keys, for lookup by binary search */
typedef struct {
    uint64_t key;
    uint64_t entry;
} ent_t;

static int cmp_ent(const void *a, const void *b)
{
    uint64_t x = ((const ent_t *)a)->key, y = ((const ent_t *)b)->key;
    return (x > y) - (x < y);
}

static int64_t lookup(const ent_t *tab, uint64_t n, uint64_t key)
{
    uint64_t lo = 0, hi = n;
    while (lo < hi) {
        uint64_t mid = lo + (hi - lo) / 2;
        if (tab[mid].key < key)
            lo = mid + 1;
        else
            hi = mid;
    }
    if (lo < n && tab[lo].key == key)
        return (int64_t)tab[lo].entry;
    return -1;
}

static uint32_t p2c(uint64_t seed, uint32_t policy, uint64_t g, uint32_t R, const uint64_t *snap)
{
    uint64_t ctr[4] = {g, 0, 0, 0}, pk[2] = {seed, policy}, o[4];
    orc_philox4x64_10(ctr, pk, o);
    uint32_t d1 = (uint32_t)scale_u64(o[0], R);
    uint32_t d2 = (uint32_t)((d1 + 1 + scale_u64(o[1], (uint64_t)R - 1)) % R);
    return snap[d1] <= snap[d2] ? d1 : d2;
}

/*
 * Consistent-hashing ring for bounded-load dispatch (the CHWBL comparison
 * policy of sec. 4, epsilon = 0.25; Mirrokni, Thorup and Zadimoghaddam, SODA
 * 2018).  The paper fixes only epsilon; the ring is this library's reading:
 * destination d owns V points, point (d, v) being output number d*V + v of
 * SplitMix64 started from state `seed` (output k = fmix64(seed + (k+1)*gamma)),
 * and the ring lists all R*V points in ascending (point, destination) order.
 */
typedef struct {
    uint32_t R, V;
    uint64_t M;       /* R * V */
    uint64_t *point;  /* ascending */
    uint16_t *owner;
} orc_ring;

typedef struct {
    uint64_t point;
    uint32_t owner;
} ring_ent;

static int cmp_ring_ent(const void *a, const void *b)
{
    const ring_ent *x = (const ring_ent *)a, *y = (const ring_ent *)b;
    if (x->point != y->point)
        return x->point < y->point ? -1 : 1;
    return (x->owner > y->owner) - (x->owner < y->owner);
}

orc_ring *orc_ring_create(uint32_t R, uint32_t V, uint64_t seed)
{
    if (R == 0 || R > 65535 || V == 0)
        return NULL;
    uint64_t M = (uint64_t)R * V;
    ring_ent *e = (ring_ent *)malloc(M * sizeof(ring_ent));
    orc_ring *g = (orc_ring *)calloc(1, sizeof(orc_ring));
    if (!e || !g) {
        free(e);
        free(g);
        return NULL;
    }
    for (uint32_t d = 0; d < R; ++d)
        for (uint32_t v = 0; v < V; ++v) {
            uint64_t k = (uint64_t)d * V + v;
            e[k].point = orc_fmix64(seed + (k + 1) * ORC_GAMMA);
            e[k].owner = d;
        }
    qsort(e, M, sizeof(ring_ent), cmp_ring_ent);
    g->R = R;
    g->V = V;
    g->M = M;
    g->point = (uint64_t *)malloc(M * sizeof(uint64_t));
    g->owner = (uint16_t *)malloc(M * sizeof(uint16_t));
    for (uint64_t j = 0; j < M; ++j) {
        g->point[j] = e[j].point;
        g->owner[j] = (uint16_t)e[j].owner;
    }
    free(e);
    return g;
}

void orc_ring_free(orc_ring *g)
{
    if (!g)
        return;
    free(g->point);
    free(g->owner);
    free(g);
}

void orc_ring_export(const orc_ring *g, uint64_t *point, uint16_t *owner)
{
    memcpy(point, g->point, g->M * sizeof(uint64_t));
    memcpy(owner, g->owner, g->M * sizeof(uint16_t));
}

/* Bounded-load choice for one request.  Every destination may hold at most
 * cap = ceil((1 + 1/4) (m + 1) / R) requests, m being the requests in the
 * load vector; the request goes to the first destination, walking the ring
 * clockwise from its key's position h (the first point >= h, wrapping to the
 * start), whose load is below cap.  The least-loaded destination holds at most
 * m / R < cap, so the walk always ends.  Returns R on an exhausted walk. */
static uint32_t chwbl(const orc_ring *g, uint64_t h, uint32_t R, const uint64_t *snap, uint64_t m)
{
    uint64_t cap = (5 * (m + 1) + 4 * (uint64_t)R - 1) / (4 * (uint64_t)R);
    uint64_t lo = 0, hi = g->M;
    while (lo < hi) {
        uint64_t mid = lo + (hi - lo) / 2;
        if (g->point[mid] < h)
            lo = mid + 1;
        else
            hi = mid;
    }
    uint64_t j = lo == g->M ? 0 : lo;
    for (uint64_t t = 0; t < g->M; ++t) {
        uint32_t d = g->owner[j];
        if (snap[d] < cap)
            return d;
        j = j + 1 == g->M ? 0 : j + 1;
    }
    return R;
}

/*
 * Route n requests (arrival order, global indices g0..g0+n-1) for n_rep replicas.
 * Requests are taken in batches of B; every request of a batch sees the load
 * vector as it stood when the batch began, and the batch's counts are added
 * after it.  load is [n_rep][R] (in/out), dest is [n_rep][n].
 * plans[i] may be NULL for P2C, RR, HASH and CHWBL; rings[i] (R destinations)
 * is needed by CHWBL only.  The key's ring position is fmix64(key ^ seed).
 */
int orc_route(const orc_plan *const *plans, const orc_ring *const *rings, const uint32_t *policy,
              const uint64_t *seed, uint32_t n_rep, uint32_t R, const uint64_t *key, uint64_t n,
              uint64_t g0, uint32_t B, uint64_t *load, uint16_t *dest)
{
    if (R == 0 || R > 65535 || B == 0)
        return ORC_EINVAL;
    uint64_t *snap = (uint64_t *)malloc(R * sizeof(uint64_t));
    for (uint32_t rp = 0; rp < n_rep; ++rp) {
        uint32_t pol = policy[rp];
        const orc_plan *pl = plans ? plans[rp] : NULL;
        const orc_ring *rg = rings ? rings[rp] : NULL;
        if (pol > ORC_CHWBL || (pol <= ORC_CR_NOREPL && !pl) ||
            (pol == ORC_CHWBL && (!rg || rg->R != R))) {
            free(snap);
            return ORC_EINVAL;
        }
        ent_t *tab = NULL;
        uint64_t nt = 0;
        if (pol <= ORC_CR_NOREPL) {
            nt = pl->n_adm;
            tab = (ent_t *)malloc((nt + 1) * sizeof(ent_t));
            for (uint64_t e = 0; e < nt; ++e) {
                tab[e].key = pl->adm_key[e];
                tab[e].entry = e;
            }
            qsort(tab, nt, sizeof(ent_t), cmp_ent);
        }
        uint64_t *L = load + (uint64_t)rp * R;
        uint16_t *D = dest + (uint64_t)rp * n;
        for (uint64_t b0 = 0; b0 < n; b0 += B) {
            uint64_t b1 = b0 + B < n ? b0 + B : n;
            memcpy(snap, L, R * sizeof(uint64_t));
            uint64_t m = 0;
            for (uint32_t r = 0; r < R; ++r)
                m += snap[r];
            for (uint64_t i = b0; i < b1; ++i) {
                uint64_t g = g0 + i;
                uint32_t d;
                if (pol == ORC_RR) {
                    d = (uint32_t)((g + seed[rp]) % R);
                } else if (pol == ORC_HASH) {
                    d = orc_jump_hash(orc_fmix64(key[i] ^ seed[rp]), R);
                } else if (pol == ORC_P2C) {
                    d = p2c(seed[rp], pol, g, R, snap);
                } else if (pol == ORC_CHWBL) {
                    d = chwbl(rg, orc_fmix64(key[i] ^ seed[rp]), R, snap, m);
                    if (d >= R) {
                        free(tab);
                        free(snap);
                        return ORC_EINVAL;
                    }
                } else {
                    int64_t e = lookup(tab, nt, key[i]);
                    if (e >= 0) {
                        /* least-loaded member of T(b); ties keep the earlier member */
                        uint32_t o0 = pl->koff[e], o1 = pl->koff[e + 1];
                        d = pl->members[o0];
                        for (uint32_t m = o0 + 1; m < o1; ++m)
                            if (snap[pl->members[m]] < snap[d])
                                d = pl->members[m];
                    } else {
                        d = p2c(seed[rp], pol, g, R, snap);
                    }
                }
                D[i] = (uint16_t)d;
                L[d] += 1;
            }
        }
        free(tab);
    }
    free(snap);
    return ORC_OK;
}

/* ---------------------------------------------------------------------- */
/* a8, a9: shadow replay with one whole-prefix LRU per (replica, cap, dest) */
/* ---------------------------------------------------------------------- */

typedef struct {
    uint32_t n_rep, R, n_caps;
    uint32_t *caps;
    uint32_t tokens;  /* 0: capacities in prefixes; 1: in prefix tokens */
    uint32_t *fill;   /* [n_rep][n_caps][R] */
    uint64_t **list;  /* [n_rep][n_caps][R] -> keys, most recent first */
    uint32_t **size;  /* token mode: prefix tokens of each listed key */
    uint64_t *total;  /* token mode: tokens held by each simulator */
} orc_replay;

/* A token-weighted simulator also holds at most this many prefixes. */
#define ORC_TOKEN_LRU_MAX_ENTRIES 1024

static orc_replay *replay_new(uint32_t n_rep, uint32_t R, const uint32_t *caps, uint32_t n_caps,
                              uint32_t tokens);

orc_replay *orc_replay_create(uint32_t n_rep, uint32_t R, const uint32_t *caps, uint32_t n_caps)
{
    return replay_new(n_rep, R, caps, n_caps, 0);
}

/* Token-weighted variant (byte-aware capacity): a simulator holds whole
 * prefixes, most recent first, while their prefix tokens sum to at most its
 * capacity (and at most ORC_TOKEN_LRU_MAX_ENTRIES prefixes); an access moves
 * or inserts its key at the front with the request's prefix length, then the
 * least recent prefixes are evicted until both limits hold. */
orc_replay *orc_replay_create_tokens(uint32_t n_rep, uint32_t R, const uint32_t *caps, uint32_t n_caps)
{
    return replay_new(n_rep, R, caps, n_caps, 1);
}

static orc_replay *replay_new(uint32_t n_rep, uint32_t R, const uint32_t *caps, uint32_t n_caps,
                              uint32_t tokens)
{
    if (n_rep == 0 || R == 0 || n_caps == 0)
        return NULL;
    for (uint32_t c = 0; c < n_caps; ++c)
        if (caps[c] == 0)
            return NULL;
    orc_replay *s = (orc_replay *)calloc(1, sizeof(orc_replay));
    s->n_rep = n_rep;
    s->R = R;
    s->n_caps = n_caps;
    s->caps = (uint32_t *)malloc(n_caps * sizeof(uint32_t));
    memcpy(s->caps, caps, n_caps * sizeof(uint32_t));
    s->tokens = tokens;
    uint64_t nsim = (uint64_t)n_rep * n_caps * R;
    s->fill = (uint32_t *)calloc(nsim, sizeof(uint32_t));
    s->list = (uint64_t **)calloc(nsim, sizeof(uint64_t *));
    if (tokens) {
        s->size = (uint32_t **)calloc(nsim, sizeof(uint32_t *));
        s->total = (uint64_t *)calloc(nsim, sizeof(uint64_t));
    }
    for (uint64_t i = 0; i < nsim; ++i) {
        uint32_t c = tokens ? ORC_TOKEN_LRU_MAX_ENTRIES : caps[(i / R) % n_caps];
        s->list[i] = (uint64_t *)malloc((uint64_t)c * sizeof(uint64_t));
        if (tokens)
            s->size[i] = (uint32_t *)malloc((uint64_t)c * sizeof(uint32_t));
    }
    return s;
}

void orc_replay_free(orc_replay *s)
{
    if (!s)
        return;
    uint64_t nsim = (uint64_t)s->n_rep * s->n_caps * s->R;
    for (uint64_t i = 0; i < nsim; ++i) {
        free(s->list[i]);
        if (s->tokens)
            free(s->size[i]);
    }
    free(s->list);
    free(s->size);
    free(s->total);
    free(s->fill);
    free(s->caps);
    free(s);
}

/* Counters per (replica, cap, dest): requests, hit requests, hit tokens,
 * prompt tokens, prefill tokens. */
enum { CTR_REQ = 0, CTR_HIT = 1, CTR_HIT_TOK = 2, CTR_PROMPT = 3, CTR_PREFILL = 4, CTR_N = 5 };

int orc_shadow_replay(orc_replay *s, const uint64_t *key, const uint32_t *plen,
                      const uint32_t *slen, const uint16_t *dest, uint64_t n, uint64_t *ctr)
{
    if (!s)
        return ORC_EINVAL;
    for (uint32_t rp = 0; rp < s->n_rep; ++rp) {
        for (uint64_t i = 0; i < n; ++i) {
            uint32_t r = dest[(uint64_t)rp * n + i];
            if (r >= s->R)
                return ORC_EINVAL;
            for (uint32_t c = 0; c < s->n_caps; ++c) {
                uint64_t sim = ((uint64_t)rp * s->n_caps + c) * s->R + r;
                uint64_t *lst = s->list[sim];
                uint32_t f = s->fill[sim], cap = s->caps[c];
                uint64_t *C = ctr + sim * CTR_N;
                uint32_t at = f;
                for (uint32_t q = 0; q < f; ++q)
                    if (lst[q] == key[i]) {
                        at = q;
                        break;
                    }
                C[CTR_REQ] += 1;
                C[CTR_PROMPT] += (uint64_t)plen[i] + slen[i];
                if (s->tokens) {
                    uint32_t *sz = s->size[sim];
                    uint64_t T = s->total[sim];
                    if (at < f) {
                        C[CTR_HIT] += 1;
                        C[CTR_HIT_TOK] += plen[i];
                        C[CTR_PREFILL] += slen[i];
                        T -= sz[at];
                    } else {
                        C[CTR_PREFILL] += (uint64_t)plen[i] + slen[i];
                        if (f == ORC_TOKEN_LRU_MAX_ENTRIES) {
                            /* a full list: the least recent prefix makes room (the
                             * entry limit would evict it after the insertion) */
                            T -= sz[f - 1];
                            f -= 1;
                        }
                        at = f;
                        f += 1;
                    }
                    memmove(lst + 1, lst, (uint64_t)at * sizeof(uint64_t));
                    memmove(sz + 1, sz, (uint64_t)at * sizeof(uint32_t));
                    lst[0] = key[i];
                    sz[0] = plen[i];
                    T += plen[i];
                    while (f > 0 && T > cap) { /* least recent first */
                        T -= sz[f - 1];
                        f -= 1;
                    }
                    s->fill[sim] = f;
                    s->total[sim] = T;
                    continue;
                }
                if (at < f) {
                    /* hit: move to the most-recent position */
                    memmove(lst + 1, lst, (uint64_t)at * sizeof(uint64_t));
                    lst[0] = key[i];
                    C[CTR_HIT] += 1;
                    C[CTR_HIT_TOK] += plen[i];
                    C[CTR_PREFILL] += slen[i];
                } else {
                    /* miss: insert as most recent; the least recent falls off when full */
                    uint32_t keep = f < cap ? f : cap - 1;
                    memmove(lst + 1, lst, (uint64_t)keep * sizeof(uint64_t));
                    lst[0] = key[i];
                    s->fill[sim] = keep + 1;
                    C[CTR_PREFILL] += (uint64_t)plen[i] + slen[i];
                }
            }
        }
    }
    return ORC_OK;
}

/* Copy out one simulator's resident keys, most recent first; returns the count. */
uint32_t orc_replay_state(const orc_replay *s, uint32_t rep, uint32_t cap_idx, uint32_t r,
                          uint64_t *keys_out)
{
    uint64_t sim = ((uint64_t)rep * s->n_caps + cap_idx) * s->R + r;
    uint32_t f = s->fill[sim];
    memcpy(keys_out, s->list[sim], (uint64_t)f * sizeof(uint64_t));
    return f;
}
