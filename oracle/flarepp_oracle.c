/*
 * FLARE++ routing-chain oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct float64 CPU statement of what the routing chain
 * computes. Only the test suite, the package's smoke check and the benchmark's CPU
 * baseline may load it. It shares no code, header, table or helper with the CUDA
 * library, and the CUDA library never calls it.
 *
 * Definitions followed (FLARE++ paper):
 *   SDPA(Q, K, V) = softmax(s Q K^T) V, the softmax normalising over the N_k keys,
 *                   one D-vector out per query row                    (Sec. 2, eq. sdpa_definition)
 *   call 1  Q_h = SDPA(Qseed_h, Kt_h, Vt_h)                           (Sec. 3.2, eq. flarepp_dynamic_query)
 *   call 2  Z_h = SDPA(Q_h, K_h, V_h)                                 (Sec. 3.2, eq. flarepp_mixer)
 *   call 3  Y_h = SDPA(K_h, Q_h, Z_h)   -- softmax over the M routes  (Sec. 3.2, eq. flarepp_mixer; Fig. 1)
 *   shard statistics  L_r = log sum_j exp(S_r,j),  O_r = softmax(S_r) V_r         (App. A.2)
 *   merge  L_max = max_r L_r, a_r = exp(L_r - L_max), a = sum_r a_r,
 *          U = sum_r a_r O_r, L = L_max + log a, Z = U / a                         (App. A.3)
 *   an attention row with no keys has L = -inf and output 0, never NaN            (App. A.3)
 *   backward of one SDPA with the saved output O and log-normaliser L          (App. A.5):
 *          P = exp(S - L),  c = <dO, O>_D,  dV = P^T dO,  dS = P o (dO V^T - c),
 *          dK = s dS^T Q,  dQ = s dS K
 *   chain backward: the decoder's query gradient is added to the encoder's before call 1's
 *          backward, and each call uses its own saved L                          (App. A.5)
 *
 * Every softmax is two-pass: the exact row maximum first, then exp(x - max) summed in
 * ascending key order. Dot products run in ascending channel order. OpenMP splits only
 * over independent rows, so results do not depend on the thread count.
 *
 * Layouts (all row-major float64, D innermost):
 *   seeds [H, M, D];  Kt, Vt, K, V, Y [B, H, N, D];  Q, Z [B, H, M, D].
 *
 * ORACLE_PLANT (compile-time, default 0) plants one deliberate mistake so that a test
 * can show the pin suite rejects it; a normal build never defines it.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#ifndef ORACLE_PLANT
#define ORACLE_PLANT 0
#endif

int oracle_plant(void) { return ORACLE_PLANT; }

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/*
 * One SDPA query row (eq. sdpa_definition).
 *   q [D], k [nk, D], v [nk, D] -> out [D]; returns the row's log-normaliser
 *   L = log sum_j exp(s <q, k_j>), or -inf when nk == 0 (then out = 0).
 *   sc is caller scratch of nk doubles.
 */
static double sdpa_row(int64_t nk, int64_t D, const double* q, const double* k,
                       const double* v, double s, double* out, double* sc) {
    for (int64_t d = 0; d < D; ++d) out[d] = 0.0;
    if (nk == 0) return -INFINITY;
    /* scores s <q, k_j> */
    for (int64_t j = 0; j < nk; ++j) {
        double dot = 0.0;
        for (int64_t d = 0; d < D; ++d) dot += q[d] * k[j * D + d];
#if ORACLE_PLANT == 4
        sc[j] = s * s * dot; /* planted: scale applied twice */
#else
        sc[j] = s * dot;
#endif
    }
    /* pass 1: exact maximum */
    double mx = sc[0];
    for (int64_t j = 1; j < nk; ++j)
        if (sc[j] > mx) mx = sc[j];
#if ORACLE_PLANT == 1
    mx = 0.0; /* planted: no max subtraction */
#endif
    /* pass 2: exponentials, their sum, and the weighted sum of values */
    double l = 0.0;
#if ORACLE_PLANT == 6
    const int64_t jend = nk > 1 ? nk - 1 : nk; /* planted: last key dropped */
#else
    const int64_t jend = nk;
#endif
    for (int64_t j = 0; j < jend; ++j) {
        const double e = exp(sc[j] - mx);
        l += e;
        for (int64_t d = 0; d < D; ++d) out[d] += e * v[j * D + d];
    }
    for (int64_t d = 0; d < D; ++d) out[d] /= l;
    return mx + log(l);
}

static double* scratch_alloc(int64_t n) {
    return (double*)malloc((size_t)(n > 0 ? n : 1) * sizeof(double));
}

/*
 * Batched SDPA over G independent groups (eq. sdpa_definition):
 *   q [G, nq, D] (or [nq, D] shared by all groups when q_shared != 0),
 *   k, v [G, nk, D] -> out [G, nq, D], lse [G, nq] (lse may be NULL).
 * Returns 0, or -1 if scratch could not be allocated.
 */
int oracle_sdpa_f64(int64_t G, int64_t nq, int64_t nk, int64_t D, const double* q,
                    int q_shared, const double* k, const double* v, double s,
                    double* out, double* lse) {
    int err = 0;
#pragma omp parallel reduction(| : err)
    {
        double* sc = scratch_alloc(nk);
        if (!sc) {
            err = 1;
        } else {
#pragma omp for schedule(static) collapse(2)
            for (int64_t g = 0; g < G; ++g) {
                for (int64_t i = 0; i < nq; ++i) {
                    const double* qi = q + ((q_shared ? 0 : g * nq) + i) * D;
                    const double* kg = k + g * nk * D;
                    const double* vg = v + g * nk * D;
                    double L = sdpa_row(nk, D, qi, kg, vg, s, out + (g * nq + i) * D, sc);
                    if (lse) lse[g * nq + i] = L;
                }
            }
            free(sc);
        }
    }
    return err ? -1 : 0;
}

/*
 * The full routing chain (eqs. flarepp_dynamic_query, flarepp_mixer), per (b, h):
 *   Q = SDPA(seeds_h, Kt, Vt);  Z = SDPA(Q, K, V);  Y = SDPA(K, Q, Z).
 * Q and Z are written to the caller's [B, H, M, D] buffers; Y to [B, H, N, D].
 */
int oracle_route_f64(int64_t B, int64_t H, int64_t N, int64_t M, int64_t D,
                     const double* seeds, const double* Kt, const double* Vt,
                     const double* K, const double* V, double s, double* Q, double* Z,
                     double* Y) {
    const int64_t G = B * H;
    int err = 0;
    /* call 1: the seeds of head h serve every batch element */
#pragma omp parallel reduction(| : err)
    {
        double* sc = scratch_alloc(N);
        if (!sc) {
            err = 1;
        } else {
#pragma omp for schedule(static) collapse(2)
            for (int64_t g = 0; g < G; ++g)
                for (int64_t m = 0; m < M; ++m) {
                    const int64_t h = g % H;
                    sdpa_row(N, D, seeds + (h * M + m) * D, Kt + g * N * D, Vt + g * N * D, s,
                             Q + (g * M + m) * D, sc);
                }
            free(sc);
        }
    }
    if (err) return -1;
    /* call 2: gather the values through the synthesised queries */
    if (oracle_sdpa_f64(G, M, N, D, Q, 0, K, V, s, Z, NULL)) return -1;
    /* call 3: scatter back; queries are the tokens' keys, keys are the routes */
#if ORACLE_PLANT == 2
    /* planted: the query-synthesis keys used as decode queries */
    return oracle_sdpa_f64(G, N, M, D, Kt, 0, Q, Z, s, Y, NULL);
#elif ORACLE_PLANT == 3
    /* planted: decode against the seeds instead of the synthesised queries */
    {
        int e = 0;
        for (int64_t g = 0; g < G && !e; ++g)
            e = oracle_sdpa_f64(1, N, M, D, K + g * N * D, 0, seeds + (g % H) * M * D,
                                Z + g * M * D, s, Y + g * N * D, NULL);
        return e;
    }
#else
    return oracle_sdpa_f64(G, N, M, D, K, 0, Q, Z, s, Y, NULL);
#endif
}

/*
 * Encoder evaluated shard by shard and merged (App. A.2-A.3): the nk keys are cut into
 * consecutive shards of `chunk` keys (the last one shorter), each shard yields (O_r, L_r),
 * and the stable log-sum-exp merge recovers the globally normalised output and L.
 *   q [G, nq, D], k, v [G, nk, D] -> out [G, nq, D], lse [G, nq] (may be NULL).
 * n_empty extra empty shards (L_r = -inf, O_r = 0) are merged in as well, to exercise the
 * empty-row convention.
 */
int oracle_encode_sharded_f64(int64_t G, int64_t nq, int64_t nk, int64_t D, const double* q,
                              const double* k, const double* v, double s, int64_t chunk,
                              int64_t n_empty, double* out, double* lse) {
    if (chunk <= 0) return -2;
    const int64_t R = (nk + chunk - 1) / chunk;
    const int64_t Rt = R + n_empty;
    int err = 0;
#pragma omp parallel reduction(| : err)
    {
        double* sc = scratch_alloc(chunk);
        double* O = scratch_alloc(Rt * D);
        double* L = scratch_alloc(Rt);
        if (!sc || !O || !L) {
            err = 1;
        } else {
#pragma omp for schedule(static) collapse(2)
            for (int64_t g = 0; g < G; ++g) {
                for (int64_t i = 0; i < nq; ++i) {
                    const double* qi = q + (g * nq + i) * D;
                    /* per-shard statistics */
                    for (int64_t r = 0; r < Rt; ++r) {
                        const int64_t j0 = r * chunk;
                        int64_t nr = 0;
                        if (r < R) nr = (nk - j0 < chunk) ? nk - j0 : chunk;
                        const double* kr = k + (g * nk + (r < R ? j0 : 0)) * D;
                        const double* vr = v + (g * nk + (r < R ? j0 : 0)) * D;
                        L[r] = sdpa_row(nr, D, qi, kr, vr, s, O + r * D, sc);
                    }
                    /* stable merge */
                    double Lmax = -INFINITY;
                    for (int64_t r = 0; r < Rt; ++r)
                        if (L[r] > Lmax) Lmax = L[r];
                    double* o = out + (g * nq + i) * D;
                    for (int64_t d = 0; d < D; ++d) o[d] = 0.0;
                    if (Lmax == -INFINITY) {
                        if (lse) lse[g * nq + i] = -INFINITY;
                        continue;
                    }
                    double a = 0.0;
#if ORACLE_PLANT == 5
                    const int64_t rend = Rt > 1 ? Rt - 1 : Rt; /* planted: last shard lost */
#else
                    const int64_t rend = Rt;
#endif
                    for (int64_t r = 0; r < rend; ++r) {
                        const double ar = exp(L[r] - Lmax);
                        a += ar;
                        for (int64_t d = 0; d < D; ++d) o[d] += ar * O[r * D + d];
                    }
                    for (int64_t d = 0; d < D; ++d) o[d] /= a;
                    if (lse) lse[g * nq + i] = Lmax + log(a);
                }
            }
        }
        free(sc);
        free(O);
        free(L);
    }
    return err ? -1 : 0;
}

/*
 * Backward of one SDPA group (App. A.5, one shard), accumulating into dq, dk, dv:
 *   q [nq, D], k, v [nk, D], the forward output o [nq, D] and log-normaliser lse [nq],
 *   the output gradient dO [nq, D]. With S = s q k^T:
 *     P = exp(S - lse)            (the saved L broadcast along the keys)
 *     c_i = <dO_i, o_i>_D
 *     dS = P o (dO v^T - c)
 *     dq += s dS k,  dk += s dS^T q,  dv += P^T dO
 *   P and dS are held as full [nq, nk] matrices; the query-side sums run over rows in
 *   parallel, the key-side sums over key rows in parallel, each in ascending order.
 */
static int sdpa_bwd_group(int64_t nq, int64_t nk, int64_t D, const double* q, const double* k,
                          const double* v, const double* o, const double* lse, const double* dO,
                          double s, double* dq, double* dk, double* dv) {
    if (nq == 0 || nk == 0) return 0;
    double* P = (double*)malloc((size_t)nq * (size_t)nk * sizeof(double));
    double* dS = (double*)malloc((size_t)nq * (size_t)nk * sizeof(double));
    if (!P || !dS) {
        free(P);
        free(dS);
        return -1;
    }
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < nq; ++i) {
        const double* qi = q + i * D;
        const double* dOi = dO + i * D;
        double c = 0.0;
        for (int64_t d = 0; d < D; ++d) c += dOi[d] * o[i * D + d];
#if ORACLE_PLANT == 7
        c = 0.0; /* planted: the <dO, O> correction dropped */
#endif
        for (int64_t j = 0; j < nk; ++j) {
            double dot = 0.0;
            for (int64_t d = 0; d < D; ++d) dot += qi[d] * k[j * D + d];
            const double p = exp(s * dot - lse[i]);
            double dp = 0.0;
            for (int64_t d = 0; d < D; ++d) dp += dOi[d] * v[j * D + d];
            P[i * nk + j] = p;
            dS[i * nk + j] = p * (dp - c);
        }
        for (int64_t j = 0; j < nk; ++j)
            for (int64_t d = 0; d < D; ++d) dq[i * D + d] += s * dS[i * nk + j] * k[j * D + d];
    }
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < nk; ++j) {
        for (int64_t i = 0; i < nq; ++i) {
            const double ds = dS[i * nk + j], p = P[i * nk + j];
            for (int64_t d = 0; d < D; ++d) {
#if ORACLE_PLANT == 8
                dk[j * D + d] += s * ds * k[j * D + d]; /* planted: key gradient through k */
#else
                dk[j * D + d] += s * ds * q[i * D + d];
#endif
                dv[j * D + d] += p * dO[i * D + d];
            }
        }
    }
    free(P);
    free(dS);
    return 0;
}

/*
 * Batched SDPA backward over G independent groups (App. A.5): the shapes of
 * oracle_sdpa_f64 with the forward's out and lse, and dO [G, nq, D]. Writes (not
 * accumulates) dq [G, nq, D], dk, dv [G, nk, D].
 */
int oracle_sdpa_bwd_f64(int64_t G, int64_t nq, int64_t nk, int64_t D, const double* q,
                        const double* k, const double* v, const double* out, const double* lse,
                        const double* dO, double s, double* dq, double* dk, double* dv) {
    memset(dq, 0, (size_t)(G * nq * D) * sizeof(double));
    memset(dk, 0, (size_t)(G * nk * D) * sizeof(double));
    memset(dv, 0, (size_t)(G * nk * D) * sizeof(double));
    for (int64_t g = 0; g < G; ++g) {
        const int64_t qo = g * nq * D, ko = g * nk * D;
        if (sdpa_bwd_group(nq, nk, D, q + qo, k + ko, v + ko, out + qo, lse + g * nq, dO + qo,
                           s, dq + qo, dk + ko, dv + ko))
            return -1;
    }
    return 0;
}

/*
 * Backward of the routing chain (App. A.5 applied to eqs. flarepp_dynamic_query and
 * flarepp_mixer), per (b, h), given dY [B, H, N, D]:
 *   forward again: Q, L1 = SDPA(seeds_h, Kt, Vt); Z, L2 = SDPA(Q, K, V); Y, L3 = SDPA(K, Q, Z)
 *   call 3 (decode; queries K, keys Q, values Z):  dK  = ..., dQ = ..., dZ = ...
 *   call 2 (encode; queries Q, keys K, values V):  dQ += ..., dK += ..., dV = ...
 *   call 1 (encode; queries seeds, keys Kt, values Vt), with the summed dQ as its output
 *          gradient:  dKt, dVt, and the seeds' gradient summed over the batch.
 * Outputs dseeds [H, M, D] and dKt, dVt, dK, dV [B, H, N, D] are overwritten.
 */
int oracle_route_bwd_f64(int64_t B, int64_t H, int64_t N, int64_t M, int64_t D,
                         const double* seeds, const double* Kt, const double* Vt, const double* K,
                         const double* V, double s, const double* dY, double* dseeds, double* dKt,
                         double* dVt, double* dK, double* dV) {
    const int64_t G = B * H;
    const size_t lat = (size_t)(G * M * D), tok = (size_t)(G * N * D);
    double* Qs = (double*)malloc((lat ? lat : 1) * sizeof(double));
    double* Q = (double*)malloc((lat ? lat : 1) * sizeof(double));
    double* Z = (double*)malloc((lat ? lat : 1) * sizeof(double));
    double* Y = (double*)malloc((tok ? tok : 1) * sizeof(double));
    double* L1 = (double*)malloc((size_t)(G * M + 1) * sizeof(double));
    double* L2 = (double*)malloc((size_t)(G * M + 1) * sizeof(double));
    double* L3 = (double*)malloc((size_t)(G * N + 1) * sizeof(double));
    double* dQ = (double*)malloc((lat ? lat : 1) * sizeof(double));
    double* dQ2 = (double*)malloc((lat ? lat : 1) * sizeof(double));
    double* dZ = (double*)malloc((lat ? lat : 1) * sizeof(double));
    double* dK2 = (double*)malloc((tok ? tok : 1) * sizeof(double));
    double* dQs = (double*)malloc((lat ? lat : 1) * sizeof(double));
    int err = !Qs || !Q || !Z || !Y || !L1 || !L2 || !L3 || !dQ || !dQ2 || !dZ || !dK2 || !dQs;
    if (!err) {
        /* the seeds of head h serve every batch element */
        for (int64_t g = 0; g < G; ++g)
            memcpy(Qs + g * M * D, seeds + (g % H) * M * D, (size_t)(M * D) * sizeof(double));
        err = oracle_sdpa_f64(G, M, N, D, Qs, 0, Kt, Vt, s, Q, L1) ||
              oracle_sdpa_f64(G, M, N, D, Q, 0, K, V, s, Z, L2) ||
              oracle_sdpa_f64(G, N, M, D, K, 0, Q, Z, s, Y, L3);
    }
    /* call 3: Y = SDPA(K, Q, Z) */
    if (!err) err = oracle_sdpa_bwd_f64(G, N, M, D, K, Q, Z, Y, L3, dY, s, dK, dQ, dZ);
    /* call 2: Z = SDPA(Q, K, V) with output gradient dZ */
    if (!err) err = oracle_sdpa_bwd_f64(G, M, N, D, Q, K, V, Z, L2, dZ, s, dQ2, dK2, dV);
    if (!err) {
        for (size_t i = 0; i < tok; ++i) dK[i] += dK2[i];
#if ORACLE_PLANT == 9
        /* planted: call 1 sees only the decoder's query gradient */
#else
        for (size_t i = 0; i < lat; ++i) dQ[i] += dQ2[i];
#endif
        /* call 1: Q = SDPA(seeds, Kt, Vt) with output gradient dQ */
        err = oracle_sdpa_bwd_f64(G, M, N, D, Qs, Kt, Vt, Q, L1, dQ, s, dQs, dKt, dVt);
    }
    if (!err) {
        memset(dseeds, 0, (size_t)(H * M * D) * sizeof(double));
#if ORACLE_PLANT == 10
        const int64_t bend = B > 0 ? 1 : 0; /* planted: seeds' gradient from b = 0 only */
#else
        const int64_t bend = B;
#endif
        for (int64_t b = 0; b < bend; ++b)
            for (int64_t h = 0; h < H; ++h)
                for (int64_t i = 0; i < M * D; ++i)
                    dseeds[h * M * D + i] += dQs[(b * H + h) * M * D + i];
    }
    free(Qs);
    free(Q);
    free(Z);
    free(Y);
    free(L1);
    free(L2);
    free(L3);
    free(dQ);
    free(dQ2);
    free(dZ);
    free(dK2);
    free(dQs);
    return err ? -1 : 0;
}
