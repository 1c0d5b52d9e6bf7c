/*
 * Plain, slow, single-threaded CPU oracle for the PSS hashed-embedding hot path
 * of "The trade-offs of model size in large recommendation models"
 * (Desai & Shrivastava, arXiv 2207.10731).
 *
 * TEST INFRASTRUCTURE.  Only the tests, the package smoke check and the
 * benchmark's CPU-baseline leg may load this code.  The CUDA library never
 * links, includes or calls it, and it shares no source with the CUDA library.
 *
 * What it computes (each function cites the passage it follows):
 *   - the ROBE-Z mapping of Sec. 2.5: chunk j of the embedding of id i in
 *     table t is the Z-long block M[h(t,i,j) : h(t,i,j)+Z] of one shared 1-D
 *     array, h a universal hash (Sec. 2.5, "Sparse JL with independence
 *     relaxation": S generated on the fly by universal hashing);
 *   - forward(i) = (S e_i)^T M and backward(i, D) = (S e_i) D of Sec. 2.4,
 *     i.e. a gather of the hashed blocks, sum-pooled per bag, and the
 *     scatter-add of the upstream gradient into an M-sized buffer (the dense
 *     branch of Algorithm 1);
 *   - the optimizer step applied to M: SGD (Sec. 4, training-time figure) and
 *     Adagrad.
 *
 * Readings of points the paper leaves open (all integer work is exact):
 *   - hash family: Carter-Wegman affine hash modulo the Mersenne prime
 *     P = 2^61 - 1, followed by "mod R";
 *   - the table id t is folded into the hashed key so equal ids of different
 *     tables map independently: key = ((i*T + t)*J + j);
 *   - block starts are multiples of an alignment G: loc = G * (x mod R) with
 *     R = floor((M - L)/G) + 1 and L = min(Z, d), so every block lies inside M
 *     (the printed range {0..|M_r|} would read past the end);
 *   - Z > d reads the first d values of the block; the last chunk has length
 *     min(Z, d - jZ);
 *   - hash parameters (A, B0) come from the splitmix64 generator (Steele, Lea
 *     & Flood 2014) seeded with the user seed: A = 1 + (s1 mod (P-1)),
 *     B0 = s2 mod P;
 *   - sums are taken in fp64 and rounded to fp32 once; the optimizer update is
 *     done in fp32, one IEEE operation at a time in a fixed order (compile
 *     with -ffp-contract=off so no multiply-add is fused);
 *   - signed hashing (optional; Sec. 2.5 derives the sketch from Achlioptas'
 *     +-1 random projections, ROBE-Z itself has no sign): every (id, chunk)
 *     also gets a sign s = +-1 from a second hash of the same family with its
 *     own parameters A2 = 1 + (s3 mod (P-1)), B2 = s4 mod P (the third and
 *     fourth splitmix64 outputs): s = -1 when (A2*key + B2) mod P is odd.  The
 *     forward adds s * block, the backward adds s * upstream gradient;
 *   - circular array (optional; the other reading of the printed range
 *     {0..|M_r|}): R = M / G block starts (G must divide M), and element z of
 *     the block at loc is M[(loc + z) mod M], so blocks near the end wrap to
 *     the start of the array.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

#define ORACLE_P ((((uint64_t)1) << 61) - 1)

typedef struct {
    int64_t T, d, M, Z, G;        /* tables, dim, shared-array length, chunk, alignment */
    int64_t J, L, R;              /* chunks per embedding, block length read, #starts */
    uint64_t A, B0;               /* hash parameters */
    const int64_t* cards;         /* host, T cardinalities (not owned) */
    int64_t sgn;                  /* 1: signed hashing */
    uint64_t A2, B2;              /* sign-hash parameters */
    int64_t circ;                 /* 1: circular array */
} oracle_pss;

/* splitmix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014): state += golden gamma, then the variant-13 mix. */
static uint64_t oracle_splitmix64(uint64_t* state)
{
    uint64_t z;
    *state += 0x9e3779b97f4a7c15ULL;
    z = *state;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

/* Raw splitmix64 outputs, exported so the tests can check the generator
 * against its published output sequence. */
void oracle_splitmix64_seq(uint64_t seed, int64_t n, uint64_t* out)
{
    uint64_t s = seed;
    for (int64_t k = 0; k < n; ++k) out[k] = oracle_splitmix64(&s);
}

/* Universal-hash parameters drawn from the seed (Sec. 2.5: S "can be generated
 * on-the-fly using universal hashing", O(1) memory for the mapping). */
void oracle_hash_params(uint64_t seed, uint64_t* A, uint64_t* B0)
{
    uint64_t s = seed;
    uint64_t s1 = oracle_splitmix64(&s);
    uint64_t s2 = oracle_splitmix64(&s);
    *A = 1 + (s1 % (ORACLE_P - 1));
    *B0 = s2 % ORACLE_P;
}

/* Sign-hash parameters: the third and fourth splitmix64 outputs of the seed. */
void oracle_sign_params(uint64_t seed, uint64_t* A2, uint64_t* B2)
{
    uint64_t s = seed, s3, s4;
    oracle_splitmix64(&s);
    oracle_splitmix64(&s);
    s3 = oracle_splitmix64(&s);
    s4 = oracle_splitmix64(&s);
    *A2 = 1 + (s3 % (ORACLE_P - 1));
    *B2 = s4 % ORACLE_P;
}

/* Set up one PSS instance.  Returns 0 on success, a negative code when the
 * sizes are invalid (no block fits, or keys would exceed the hash's field). */
int oracle_init(oracle_pss* p, const int64_t* cards, int64_t T, int64_t d, int64_t M,
                int64_t Z, int64_t G, uint64_t seed)
{
    int64_t max_card = 0;
    if (T <= 0 || d <= 0 || Z <= 0 || G <= 0 || M <= 0 || !cards) return -1;
    p->T = T; p->d = d; p->M = M; p->Z = Z; p->G = G;
    p->J = (d + Z - 1) / Z;
    p->L = Z < d ? Z : d;
    if (M < p->L) return -2;
    p->R = (M - p->L) / G + 1;
    for (int64_t t = 0; t < T; ++t) {
        if (cards[t] <= 0) return -3;
        if (cards[t] > max_card) max_card = cards[t];
    }
    /* every key ((i*T + t)*J + j) must lie below P */
    if ((unsigned __int128)max_card * (unsigned __int128)T * (unsigned __int128)p->J
        > (unsigned __int128)ORACLE_P) return -4;
    p->cards = cards;
    oracle_hash_params(seed, &p->A, &p->B0);
    oracle_sign_params(seed, &p->A2, &p->B2);
    p->sgn = 0;
    p->circ = 0;
    return 0;
}

/* Turn the circular array on (1) or off (0).  On: R = M / G block starts
 * (G must divide M; returns -5 otherwise and leaves the instance unchanged). */
int oracle_set_circular(oracle_pss* p, int64_t on)
{
    if (on) {
        if (p->M % p->G) return -5;
        p->R = p->M / p->G;
        p->circ = 1;
    } else {
        p->R = (p->M - p->L) / p->G + 1;
        p->circ = 0;
    }
    return 0;
}

/* Element of the shared array that holds offset z of the block at loc. */
static int64_t elem(const oracle_pss* p, int64_t loc, int64_t z)
{
    int64_t e = loc + z;
    return (p->circ && e >= p->M) ? e - p->M : e;
}

/* Turn signed hashing on (1) or off (0). */
void oracle_set_signed(oracle_pss* p, int64_t on)
{
    p->sgn = on ? 1 : 0;
}

/* h(t, i, j): start of the block that holds chunk j of id i of table t
 * (ROBE-Z mapping, Sec. 2.5), as an element offset into M. */
int64_t oracle_location(const oracle_pss* p, int64_t id, int64_t t, int64_t j)
{
    uint64_t key = ((uint64_t)id * (uint64_t)p->T + (uint64_t)t) * (uint64_t)p->J + (uint64_t)j;
    unsigned __int128 v = (unsigned __int128)p->A * key + p->B0;
    uint64_t x = (uint64_t)(v % ORACLE_P);
    return p->G * (int64_t)(x % (uint64_t)p->R);
}

/* s(t, i, j): +1, or -1 when signed hashing is on and the sign hash of the
 * key is odd. */
int64_t oracle_sign(const oracle_pss* p, int64_t id, int64_t t, int64_t j)
{
    uint64_t key;
    unsigned __int128 v;
    if (!p->sgn) return 1;
    key = ((uint64_t)id * (uint64_t)p->T + (uint64_t)t) * (uint64_t)p->J + (uint64_t)j;
    v = (unsigned __int128)p->A2 * key + p->B2;
    return ((uint64_t)(v % ORACLE_P) & 1u) ? -1 : 1;
}

/* Check the CSR bag layout: offsets non-decreasing, inside [0, nnz]. */
static int check_offsets(const int64_t* off, int64_t nbags, int64_t nnz)
{
    if (off[0] < 0) return -10;
    for (int64_t s = 0; s < nbags; ++s)
        if (off[s + 1] < off[s]) return -10;
    if (off[nbags] > nnz) return -10;
    return 0;
}

static void note_bad(int64_t* first_bad, int64_t q)
{
    if (first_bad && (*first_bad < 0 || q < *first_bad)) *first_bad = q;
}

/* The mapping matrix of Algorithm 1 ("locations from which the output was
 * accessed"), one entry per (id, chunk): locs[q*J + j] = h(t, indices[q], j),
 * or -1 for an id outside [0, n_t).  Bags are table-major: bag (t, b) is
 * slot t*B + b. */
int oracle_locations(const oracle_pss* p, const int64_t* indices, int64_t nnz,
                     const int64_t* offsets, int64_t B, int64_t* locs, int64_t* first_bad)
{
    int rc = check_offsets(offsets, p->T * B, nnz);
    if (rc) return rc;
    for (int64_t q = 0; q < nnz * p->J; ++q) locs[q] = -1;
    for (int64_t t = 0; t < p->T; ++t)
        for (int64_t b = 0; b < B; ++b) {
            int64_t s = t * B + b;
            for (int64_t q = offsets[s]; q < offsets[s + 1]; ++q) {
                int64_t id = indices[q];
                if (id < 0 || id >= p->cards[t]) { note_bad(first_bad, q); continue; }
                for (int64_t j = 0; j < p->J; ++j)
                    locs[q * p->J + j] = oracle_location(p, id, t, j);
            }
        }
    return 0;
}

/* Signs of every (id, chunk), laid out like the locations: signs[q*J + j] =
 * s(t, indices[q], j), 0 for an id outside its table. */
int oracle_signs(const oracle_pss* p, const int64_t* indices, int64_t nnz,
                 const int64_t* offsets, int64_t B, int8_t* signs)
{
    int rc = check_offsets(offsets, p->T * B, nnz);
    if (rc) return rc;
    for (int64_t q = 0; q < nnz * p->J; ++q) signs[q] = 0;
    for (int64_t t = 0; t < p->T; ++t)
        for (int64_t b = 0; b < B; ++b) {
            int64_t s = t * B + b;
            for (int64_t q = offsets[s]; q < offsets[s + 1]; ++q) {
                int64_t id = indices[q];
                if (id < 0 || id >= p->cards[t]) continue;
                for (int64_t j = 0; j < p->J; ++j)
                    signs[q * p->J + j] = (int8_t)oracle_sign(p, id, t, j);
            }
        }
    return 0;
}

/* Sum-pooled forward from given locations (Sec. 2.4 forward, summed over the
 * ids of a bag): out[b][t][jZ+z] = sum_q s_qj * M[locs[q*J+j] + z],
 * z < min(Z, d-jZ), with s_qj = signs[q*J+j] (+1 when signs is NULL).
 * An empty bag gives zeros; an entry with loc < 0 contributes nothing. */
int oracle_pool(const oracle_pss* p, const float* w, const int64_t* locs, int64_t nnz,
                const int64_t* offsets, int64_t B, float* out, const int8_t* signs)
{
    int64_t d = p->d, T = p->T;
    double* acc;
    int rc = check_offsets(offsets, T * B, nnz);
    if (rc) return rc;
    acc = (double*)malloc(sizeof(double) * (size_t)d);
    if (!acc) return -20;
    for (int64_t t = 0; t < T; ++t)
        for (int64_t b = 0; b < B; ++b) {
            int64_t s = t * B + b;
            for (int64_t k = 0; k < d; ++k) acc[k] = 0.0;
            for (int64_t q = offsets[s]; q < offsets[s + 1]; ++q)
                for (int64_t j = 0; j < p->J; ++j) {
                    int64_t loc = locs[q * p->J + j];
                    int64_t Lj = d - j * p->Z < p->Z ? d - j * p->Z : p->Z;
                    double sg = signs ? (double)signs[q * p->J + j] : 1.0;
                    if (loc < 0) continue;
                    for (int64_t z = 0; z < Lj; ++z) acc[j * p->Z + z] += sg * (double)w[elem(p, loc, z)];
                }
            for (int64_t k = 0; k < d; ++k) out[(b * T + t) * d + k] = (float)acc[k];
        }
    free(acc);
    return 0;
}

/* Forward pass: hash every (id, chunk) (and sign it, when signed hashing is
 * on), then gather and sum-pool. */
int oracle_forward(const oracle_pss* p, const float* w, const int64_t* indices, int64_t nnz,
                   const int64_t* offsets, int64_t B, float* out, int64_t* first_bad)
{
    int64_t* locs = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nnz * p->J + 1));
    int8_t* signs = p->sgn ? (int8_t*)malloc((size_t)(nnz * p->J + 1)) : NULL;
    int rc;
    if (!locs || (p->sgn && !signs)) {
        free(locs);
        free(signs);
        return -20;
    }
    rc = oracle_locations(p, indices, nnz, offsets, B, locs, first_bad);
    if (!rc && signs) rc = oracle_signs(p, indices, nnz, offsets, B, signs);
    if (!rc) rc = oracle_pool(p, w, locs, nnz, offsets, B, out, signs);
    free(locs);
    free(signs);
    return rc;
}

/* Dense branch of Algorithm 1 from given locations: g (length M, fp64,
 * zeroed here) receives, for every bag, id and chunk, the upstream gradient of
 * that bag's output chunk, times the chunk's sign (signs[q*J+j], +1 when
 * signs is NULL), added element by element at the block's location
 * (Sec. 2.4 backward(i, D) = (S e_i) D, summed over the ids of each bag). */
int oracle_scatter(const oracle_pss* p, const int64_t* locs, int64_t nnz, const int64_t* offsets,
                   int64_t B, const float* grad_out, double* g, const int8_t* signs)
{
    int64_t d = p->d, T = p->T;
    int rc = check_offsets(offsets, T * B, nnz);
    if (rc) return rc;
    for (int64_t e = 0; e < p->M; ++e) g[e] = 0.0;
    for (int64_t t = 0; t < T; ++t)
        for (int64_t b = 0; b < B; ++b) {
            int64_t s = t * B + b;
            const float* go = grad_out + (b * T + t) * d;
            for (int64_t q = offsets[s]; q < offsets[s + 1]; ++q)
                for (int64_t j = 0; j < p->J; ++j) {
                    int64_t loc = locs[q * p->J + j];
                    int64_t Lj = d - j * p->Z < p->Z ? d - j * p->Z : p->Z;
                    double sg = signs ? (double)signs[q * p->J + j] : 1.0;
                    if (loc < 0) continue;
                    for (int64_t z = 0; z < Lj; ++z) g[elem(p, loc, z)] += sg * (double)go[j * p->Z + z];
                }
        }
    return 0;
}

/* Gradient w.r.t. the whole shared array (dense branch of Algorithm 1). */
int oracle_grad(const oracle_pss* p, const int64_t* indices, int64_t nnz, const int64_t* offsets,
                int64_t B, const float* grad_out, double* g, int64_t* first_bad)
{
    int64_t* locs = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nnz * p->J + 1));
    int8_t* signs = p->sgn ? (int8_t*)malloc((size_t)(nnz * p->J + 1)) : NULL;
    int rc;
    if (!locs || (p->sgn && !signs)) {
        free(locs);
        free(signs);
        return -20;
    }
    rc = oracle_locations(p, indices, nnz, offsets, B, locs, first_bad);
    if (!rc && signs) rc = oracle_signs(p, indices, nnz, offsets, B, signs);
    if (!rc) rc = oracle_scatter(p, locs, nnz, offsets, B, grad_out, g, signs);
    free(locs);
    free(signs);
    return rc;
}

static int64_t lower_bound_i64(const int64_t* a, int64_t n, int64_t x)
{
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        int64_t mid = lo + (hi - lo) / 2;
        if (a[mid] < x) lo = mid + 1; else hi = mid;
    }
    return lo;
}

/* The same gradient, evaluated only at the sorted, distinct element positions
 * elems[0..n_elems): g_at[k] = g[elems[k]].  Used when M is too large for a
 * dense fp64 buffer on the host. */
int oracle_grad_at(const oracle_pss* p, const int64_t* indices, int64_t nnz, const int64_t* offsets,
                   int64_t B, const float* grad_out, const int64_t* elems, int64_t n_elems,
                   double* g_at, int64_t* first_bad)
{
    int64_t d = p->d, T = p->T;
    int rc = check_offsets(offsets, T * B, nnz);
    if (rc) return rc;
    for (int64_t k = 1; k < n_elems; ++k)
        if (elems[k] <= elems[k - 1]) return -11;
    for (int64_t k = 0; k < n_elems; ++k) g_at[k] = 0.0;
    for (int64_t t = 0; t < T; ++t)
        for (int64_t b = 0; b < B; ++b) {
            int64_t s = t * B + b;
            const float* go = grad_out + (b * T + t) * d;
            for (int64_t q = offsets[s]; q < offsets[s + 1]; ++q) {
                int64_t id = indices[q];
                if (id < 0 || id >= p->cards[t]) { note_bad(first_bad, q); continue; }
                for (int64_t j = 0; j < p->J; ++j) {
                    int64_t loc = oracle_location(p, id, t, j);
                    int64_t Lj = d - j * p->Z < p->Z ? d - j * p->Z : p->Z;
                    double sg = (double)oracle_sign(p, id, t, j);
                    if (p->circ && loc + Lj > p->M) {
                        /* a block that wraps: look every element up */
                        for (int64_t z = 0; z < Lj; ++z) {
                            int64_t e = elem(p, loc, z);
                            int64_t k = lower_bound_i64(elems, n_elems, e);
                            if (k < n_elems && elems[k] == e) g_at[k] += sg * (double)go[j * p->Z + z];
                        }
                        continue;
                    }
                    for (int64_t k = lower_bound_i64(elems, n_elems, loc);
                         k < n_elems && elems[k] < loc + Lj; ++k)
                        g_at[k] += sg * (double)go[j * p->Z + (elems[k] - loc)];
                }
            }
        }
    return 0;
}

/* SGD step (Sec. 4 trains with SGD): w <- w - lr*g, in fp32, g already
 * rounded to fp32.  Elements with g == 0 keep their bits. */
void oracle_sgd(float* w, const float* g, int64_t n, float lr)
{
    for (int64_t e = 0; e < n; ++e) {
        float step = lr * g[e];
        w[e] = w[e] - step;
    }
}

/* Adagrad step: G <- G + g*g; w <- w - lr * g / (sqrt(G) + eps), each
 * operation rounded to fp32 in this order; elements with g == 0 are left as
 * they are (their update is exactly zero). */
void oracle_adagrad(float* w, float* Gacc, const float* g, int64_t n, float lr, float eps)
{
    for (int64_t e = 0; e < n; ++e) {
        float ge = g[e];
        float sq, Gn, s, den, q, step;
        if (ge == 0.0f) continue;
        sq = ge * ge;
        Gn = Gacc[e] + sq;
        s = sqrtf(Gn);
        den = s + eps;
        q = ge / den;
        step = lr * q;
        Gacc[e] = Gn;
        w[e] = w[e] - step;
    }
}
