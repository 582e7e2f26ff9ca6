/*
 * Tsubame per-step logit path -- CPU ORACLE.
 *
 * TEST INFRASTRUCTURE ONLY. This is a plain, slow, single-threaded reference of what the
 * plan / replay / verify path computes, written from the paper (Tsubame: Tree Replay for
 * Diffusion-Based Speculative Decoding) and the works it cites for the sampling and
 * verification rules. Only the test suite, the smoke check and the benchmark's CPU-baseline
 * leg may load it. It shares no code, header, helper or constant table with the CUDA
 * library; both sides follow the same written contract (counter layout, tie rules).
 *
 * Arithmetic: a logit z (bf16 or fp32) is widened exactly to fp32 and multiplied once by
 * invT = fp32(1/T) in fp32, x = fp32(z) * invT (one IEEE rounding, identical on every
 * machine). Everything after that is fp64 with libm, in the order the algorithm states.
 * Build with -ffp-contract=off so no multiply-add is fused behind our back.
 *
 * Every decision taken from floating point (a heap pop, a Gumbel selection, an acceptance
 * test) also reports whether it was a near tie, so the tests can exempt exactly those
 * decisions where a correct fp32 implementation may legitimately decide differently.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_CHUNK 256 /* fixed chunk of the hierarchical replay sampler (contract) */

/* Purposes of the counter-based random stream (contract). */
enum {
    PURPOSE_REPLAY_CHUNK = 0, /* node = parent, draw = chunk index        */
    PURPOSE_REPLAY_ELEM = 1,  /* node = parent, draw = token id           */
    PURPOSE_ACCEPT = 2,       /* node = child being tested, draw = 0      */
    PURPOSE_FINAL = 3,        /* node = where the final token is drawn, draw = token id */
    PURPOSE_BLOCK_ETA = 4,    /* node = chain position i, draw = 0         */
    PURPOSE_FINAL_CHUNK = 5   /* node = where the final token is drawn, draw = chunk index */
};

/* Near ties. A decision taken from floating point is flagged when a uniform that decides it
 * lies within U_BAND of the value that would flip it (the parity contract's 1e-6 band), or
 * when the compared keys differ by less than KEY_BAND times max(1, |key|): an fp32 Gumbel key
 * x + G(U) is formed with at most four roundings at its own magnitude (two logarithms of
 * relative error <= 2^-24 each, the sum, and the shift to the chunk maximum), so a correct
 * fp32 implementation is within 4 * 2^-24 = 2^-22 of it, relative.
 *
 * Planner pops: a candidate's key is Sx - CL[d] (Sx the path's sum of logits, CL[d] the sum of
 * the first d draft rows' log-normalisers). Another implementation that holds Sx exactly and
 * each row's log-normaliser within lse_err, rounding CL[d] and the logits onto a 2^-30 grid,
 * can swap two candidates at depths da and db only when their keys differ by less than
 *     lse_err * |da - db| + 2^-30 * (da + db + 2)
 * (the rows da and db share contribute to both keys alike); plan_band() is that bound. */
static const double U_BAND = 1e-6;
static const double KEY_BAND = 2.384185791015625e-07; /* 2^-22 */
static const double FIX_GRID = 9.313225746154785e-10; /* 2^-30 */

static double plan_band(int da, int db, double lse_err)
{
    return lse_err * (double)(da > db ? da - db : db - da) + FIX_GRID * (double)(da + db + 2);
}

/* ------------------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3",
 * SC 2011, Sec. 3.2). Ten rounds of the 4x32 S-box; the key is bumped by the Weyl
 * constants between rounds.                                                              */
void orc_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4])
{
    uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        uint64_t prod0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
        uint64_t prod1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
        uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
        uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
        uint32_t n0 = hi1 ^ c1 ^ k0;
        uint32_t n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
    }
    out[0] = c0;
    out[1] = c1;
    out[2] = c2;
    out[3] = c3;
}

/* The uniform of one draw: counter {draw/4, node, batch, purpose}, key {seed lo, seed hi},
 * word draw%4; U = (top 24 bits + 1/2) * 2^-24, which lies in (0,1) and is exact in fp32. */
double orc_uniform(uint64_t seed, int32_t purpose, int32_t batch, int32_t node, int32_t draw)
{
    uint32_t ctr[4] = {(uint32_t)draw >> 2, (uint32_t)node, (uint32_t)batch, (uint32_t)purpose};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t w[4];
    orc_philox4x32_10(ctr, key, w);
    uint32_t bits = w[(uint32_t)draw & 3u] >> 8;
    return ((double)bits + 0.5) * (1.0 / 16777216.0);
}

/* Standard Gumbel by inversion, G(U) = -log(-log U). */
static double gumbel_of(double u) { return -log(-log(u)); }

/* dG/dU: how fast a Gumbel key moves per unit of its uniform (used to turn key margins
 * into uniform-space margins). */
static double gumbel_slope(double u) { return 1.0 / (u * -log(u)); }

/* ------------------------------------------------------------------------------------ */
/* Logit tensors: element (b, r, v) sits at data[b*batch_stride + r*row_stride + v].      */
typedef struct {
    const void *data;
    int32_t dtype; /* 0 = fp32, 1 = bf16 (raw 16-bit patterns) */
    int32_t B, R, V;
    int64_t batch_stride, row_stride;
} orc_logits;

/* x_v = fp32(z_v) * invT for one row, widened to double (exactly). */
static void read_row(const orc_logits *t, int b, int r, float invT, double *x)
{
    const int64_t base = (int64_t)b * t->batch_stride + (int64_t)r * t->row_stride;
    for (int v = 0; v < t->V; ++v) {
        float z;
        if (t->dtype == 1) {
            uint32_t bits = (uint32_t)((const uint16_t *)t->data)[base + v] << 16;
            memcpy(&z, &bits, sizeof z);
        } else {
            z = ((const float *)t->data)[base + v];
        }
        float xf = z * invT;
        x[v] = (double)xf;
    }
}

/* log sum_v exp(x_v), shifted by the maximum (plain definition of the softmax normaliser). */
static double logsumexp(const double *x, int n)
{
    double m = -INFINITY;
    for (int v = 0; v < n; ++v)
        if (x[v] > m) m = x[v];
    double s = 0.0;
    for (int v = 0; v < n; ++v) s += exp(x[v] - m);
    return m + log(s);
}

/* softmax into out[], fp64 */
static void softmax(const double *x, int n, double *out)
{
    double lse = logsumexp(x, n);
    for (int v = 0; v < n; ++v) out[v] = exp(x[v] - lse);
}

/* (x desc, id asc): does (xa, a) come before (xb, b)? */
static int before_xv(double xa, int a, double xb, int b) { return xa > xb || (xa == xb && a < b); }

/* Top-K of a row by (x desc, id asc): K rounds of "best element after the previous one". */
static void topk_row(const double *x, int V, int K, int32_t *ids, double *xs)
{
    double px = INFINITY;
    int pid = -1;
    for (int k = 0; k < K; ++k) {
        int best = -1;
        for (int v = 0; v < V; ++v) {
            int after_prev = (x[v] < px) || (x[v] == px && v > pid);
            if (!after_prev) continue;
            if (best < 0 || before_xv(x[v], v, x[best], best)) best = v;
        }
        ids[k] = best;
        xs[k] = x[best];
        px = x[best];
        pid = best;
    }
}

/* Row statistics of step a1: max, log-normaliser, top-K, chunk log-masses.
 * Exposed for the tests (row_lse/topk pins).                                             */
int orc_row_stats(const orc_logits *rows, float temperature, int32_t K, double *row_max, double *row_lse,
                  int32_t *topk_id, float *topk_x, double *chunk_lse)
{
    if (!rows || !(temperature > 0.0f) || K < 1 || K > rows->V) return -1;
    const float invT = 1.0f / temperature;
    const int V = rows->V, C = (V + ORC_CHUNK - 1) / ORC_CHUNK;
    double *x = (double *)malloc(sizeof(double) * V);
    double *xs = (double *)malloc(sizeof(double) * K);
    if (!x || !xs) { free(x); free(xs); return -3; }
    for (int b = 0; b < rows->B; ++b)
        for (int r = 0; r < rows->R; ++r) {
            const int64_t row = (int64_t)b * rows->R + r;
            read_row(rows, b, r, invT, x);
            double m = -INFINITY;
            for (int v = 0; v < V; ++v)
                if (x[v] > m) m = x[v];
            if (row_max) row_max[row] = m;
            if (row_lse) row_lse[row] = logsumexp(x, V);
            if (topk_id || topk_x) {
                int32_t ids[64];
                topk_row(x, V, K, ids, xs);
                for (int k = 0; k < K; ++k) {
                    if (topk_id) topk_id[row * K + k] = ids[k];
                    if (topk_x) topk_x[row * K + k] = (float)xs[k];
                }
            }
            if (chunk_lse)
                for (int c = 0; c < C; ++c) {
                    int lo = c * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
                    chunk_lse[row * C + c] = logsumexp(x + lo, hi - lo);
                }
        }
    free(x);
    free(xs);
    return 0;
}

/* ------------------------------------------------------------------------------------ */
/* PLAN (first pass, Sec. 3.1; max-heap expansion of DDTree as described in Sec. 2.2 and
 * App. B.3): best-first expansion by cumulative draft path log-probability under a node
 * budget. Node 0 is the root; nodes 1..N are numbered in pop order.
 *
 * Path score of a node at depth d reached through ranks (r_1..r_d):
 *     score = sum_j log q_j(y_j) = (sum_j x_{j, r_j}) - (sum_{j<=d} LSE_j)
 * held as the fp64 sum Sx of the x's (added in path order) and key = Sx - CL[d] with
 * CL[d] = LSE_1 + ... + LSE_d. Candidates pop in the order
 *     (key desc, depth asc, parent asc, rank asc).
 * Same-depth candidates share CL[d], so equal Sx always means equal keys on every machine,
 * and the tie goes to the earlier parent, then the lower rank.                           */
typedef struct {
    double key, sx;
    int depth, parent, rank;
} cand;

static int cand_before(const cand *a, const cand *b)
{
    if (a->key != b->key) return a->key > b->key;
    if (a->depth != b->depth) return a->depth < b->depth;
    if (a->parent != b->parent) return a->parent < b->parent;
    return a->rank < b->rank;
}

/* Maximum node count a (K, L) tree can hold besides the root: K + K^2 + ... + K^L. */
static int64_t max_nodes(int K, int L)
{
    int64_t total = 0, level = 1;
    for (int d = 1; d <= L; ++d) {
        level *= K;
        total += level;
        if (total > (int64_t)1 << 40) return total;
    }
    return total;
}

/* pool = 0: path scores use the full-vocabulary log-normaliser of each draft row; pool = P > 0:
 * the log-normaliser of the row's P most probable tokens (the pooled draft law of Sec. 3.1),
 * whose K most probable tokens are the candidates.                                        */
static int plan_impl(const orc_logits *draft, float temperature, int32_t N, int32_t K, int32_t L, int32_t pool,
                     int32_t *parent, int32_t *depth, int32_t *rank, int32_t *plan_token, double *score,
                     int32_t *child_off, int32_t *child_ids, double lse_err, uint8_t *exempt, double *min_margin)
{
    if (!draft || N < 1 || K < 1 || L < 1 || K > 64 || K > draft->V || draft->R < L) return -1;
    if (pool != 0 && (pool < K || pool > draft->V)) return -1;
    if (!(temperature > 0.0f)) return -1;
    if ((int64_t)N > max_nodes(K, L)) return -2;
    const float invT = 1.0f / temperature;
    const int V = draft->V, NN = N + 1;
    double *x = (double *)malloc(sizeof(double) * V);
    double *lse = (double *)malloc(sizeof(double) * L);
    double *CL = (double *)malloc(sizeof(double) * (L + 1));
    int32_t *tid = (int32_t *)malloc(sizeof(int32_t) * L * K);
    double *tx = (double *)malloc(sizeof(double) * L * K);
    double *sxn = (double *)malloc(sizeof(double) * NN);
    cand *front = (cand *)malloc(sizeof(cand) * (2 * (size_t)NN + 2));
    int32_t *nchild = (int32_t *)malloc(sizeof(int32_t) * NN);
    int32_t *pid = (int32_t *)malloc(sizeof(int32_t) * (pool > 0 ? pool : 1));
    double *px = (double *)malloc(sizeof(double) * (pool > 0 ? pool : 1));
    if (!x || !lse || !CL || !tid || !tx || !sxn || !front || !nchild || !pid || !px) return -3;

    for (int b = 0; b < draft->B; ++b) {
        int32_t *par = parent + (int64_t)b * NN, *dep = depth + (int64_t)b * NN;
        int32_t *rk = rank + (int64_t)b * NN, *tok = plan_token + (int64_t)b * NN;
        double *sc = score + (int64_t)b * NN;
        /* per-depth candidate pools: top-K of draft row d (tokens of depth d+1) */
        for (int d = 0; d < L; ++d) {
            read_row(draft, b, d, invT, x);
            if (pool > 0) { /* the pooled law: normalised over the row's P most probable tokens */
                topk_row(x, V, pool, pid, px);
                lse[d] = logsumexp(px, pool);
            } else {
                lse[d] = logsumexp(x, V);
            }
            topk_row(x, V, K, tid + d * K, tx + d * K);
        }
        CL[0] = 0.0;
        for (int d = 1; d <= L; ++d) CL[d] = CL[d - 1] + lse[d - 1];

        par[0] = -1; dep[0] = 0; rk[0] = -1; tok[0] = -1; sc[0] = 0.0; sxn[0] = 0.0;
        int nf = 0;
        front[nf].sx = tx[0];
        front[nf].depth = 1;
        front[nf].parent = 0;
        front[nf].rank = 0;
        front[nf].key = front[nf].sx - CL[1];
        ++nf;
        uint8_t ex = 0;
        double mm = INFINITY;
        for (int i = 1; i <= N; ++i) {
            if (nf == 0) return -4; /* cannot happen when N <= max_nodes */
            int best = 0;
            for (int f = 1; f < nf; ++f)
                if (cand_before(&front[f], &front[best])) best = f;
            /* Near-tie check (plan_band). Keys of different depths depend on the
             * log-normalisers, which another implementation computes with some error; same-depth
             * keys differ only through their exact sums of logits. Same-depth candidates with
             * equal Sx tie exactly everywhere and are not near ties. */
            for (int f = 0; f < nf; ++f) {
                if (f == best) continue;
                if (front[f].depth == front[best].depth && front[f].sx == front[best].sx) continue;
                double margin = front[best].key - front[f].key;
                if (front[f].depth != front[best].depth && margin < mm) mm = margin;
                if (margin < plan_band(front[f].depth, front[best].depth, lse_err)) ex = 1;
            }
            cand c = front[best];
            front[best] = front[--nf];
            par[i] = c.parent;
            dep[i] = c.depth;
            rk[i] = c.rank;
            tok[i] = tid[(c.depth - 1) * K + c.rank];
            sc[i] = c.key;
            sxn[i] = c.sx;
            if (c.rank + 1 < K) { /* next sibling */
                cand s;
                s.depth = c.depth;
                s.parent = c.parent;
                s.rank = c.rank + 1;
                s.sx = sxn[c.parent] + tx[(c.depth - 1) * K + c.rank + 1];
                s.key = s.sx - CL[s.depth];
                front[nf++] = s;
            }
            if (c.depth < L) { /* first child */
                cand f;
                f.depth = c.depth + 1;
                f.parent = i;
                f.rank = 0;
                f.sx = sxn[i] + tx[c.depth * K + 0];
                f.key = f.sx - CL[f.depth];
                front[nf++] = f;
            }
        }
        if (exempt) exempt[b] = ex;
        if (min_margin) min_margin[b] = mm;
        /* child lists (CSR) in slot (= rank = pop) order */
        int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        for (int u = 0; u < NN; ++u) nchild[u] = 0;
        for (int i = 1; i <= N; ++i) nchild[par[i]]++;
        off[0] = 0;
        for (int u = 0; u < NN; ++u) off[u + 1] = off[u] + nchild[u];
        for (int u = 0; u < NN; ++u) nchild[u] = 0;
        for (int i = 1; i <= N; ++i) ids[off[par[i]] + nchild[par[i]]++] = i;
    }
    free(x); free(lse); free(CL); free(tid); free(tx); free(sxn); free(front); free(nchild); free(pid); free(px);
    return 0;
}

int orc_plan(const orc_logits *draft, float temperature, int32_t N, int32_t K, int32_t L,
             int32_t *parent, int32_t *depth, int32_t *rank, int32_t *plan_token, double *score,
             int32_t *child_off, int32_t *child_ids, double lse_err, uint8_t *exempt, double *min_margin)
{
    return plan_impl(draft, temperature, N, K, L, 0, parent, depth, rank, plan_token, score, child_off, child_ids,
                     lse_err, exempt, min_margin);
}

/* First pass with pooled draft laws (Sec. 3.1, App. B.7): as orc_plan, with each depth's law
 * normalised over its P most probable tokens. */
int orc_plan_pooled(const orc_logits *draft, float temperature, int32_t N, int32_t K, int32_t L, int32_t P,
                    int32_t *parent, int32_t *depth, int32_t *rank, int32_t *plan_token, double *score,
                    int32_t *child_off, int32_t *child_ids, double lse_err, uint8_t *exempt, double *min_margin)
{
    if (P < 1) return -1;
    return plan_impl(draft, temperature, N, K, L, P, parent, depth, rank, plan_token, score, child_off, child_ids,
                     lse_err, exempt, min_margin);
}

/* ------------------------------------------------------------------------------------ */
/* REPLAY (second pass, Sec. 3.2, Eq. replay-distribution; WoR as defined in App. A).
 * For each parent u with m_u children, draw m_u tokens without replacement from
 * q_u = softmax(x_row(u)); the j-th draw fills child slot j.
 *
 * WoR draws are the top-m_u of the Gumbel keys x_v + G_v (Gumbel-top-k: Vieira 2014;
 * Kool, van Hoof & Welling 2019). The keys are built top-down (Maddison, Tarlow & Minka
 * 2014, A* sampling; Kool et al. 2019, App. B): chunk keys K_c ~ Gumbel(A_c) with
 * A_c = log sum_{v in c} exp(x_v); inside each of the top-m_u chunks, fresh element keys
 * g_v ~ Gumbel(x_v) are shifted to the law conditional on their maximum being K_c,
 *     k_v = -log(exp(-K_c) - exp(-Z_c) + exp(-g_v)),   Z_c = max_{v in c} g_v,
 * which leaves the joint law of all keys that of flat Gumbel-top-k.                       */

/* stable form of the conditional shift (Kool et al. 2019, App. B) */
static double shift_key(double T, double Z, double g)
{
    double u = T - g + log1p(-exp(g - Z));
    double sp = (u > 0 ? u : 0.0) + log1p(exp(-fabs(u)));
    return T - sp;
}

typedef struct {
    double k;  /* key */
    int v;     /* token id */
    double sens; /* max |d key / d uniform| over the uniforms the key depends on */
} elem_key;

static int elem_before(const elem_key *a, const elem_key *b) { return a->k > b->k || (a->k == b->k && a->v < b->v); }

/* Sort the first n entries so the first `take` are the best in order (selection sort). */
static void partial_sort(elem_key *e, int n, int take)
{
    for (int i = 0; i < take && i < n; ++i) {
        int best = i;
        for (int j = i + 1; j < n; ++j)
            if (elem_before(&e[j], &e[best])) best = j;
        elem_key t = e[i];
        e[i] = e[best];
        e[best] = t;
    }
}

/* Is the decision "a before b" a near tie in uniform space? */
static int near_tie_keys(double ka, double kb, double sens)
{
    double dk = ka - kb;
    double mag = fabs(ka) > 1.0 ? fabs(ka) : 1.0;
    return dk < U_BAND * sens || dk < KEY_BAND * mag;
}

static int near_tie(const elem_key *a, const elem_key *b)
{
    return near_tie_keys(a->k, b->k, a->sens > b->sens ? a->sens : b->sens);
}

/* The Philox batch index of local tree b (callers may pass a sample of a larger batch). */
static int batch_of(const int32_t *batch_ids, int b) { return batch_ids ? batch_ids[b] : b; }

static int replay_row_index(const int32_t *qrow_of_node, const int32_t *depth, int64_t idx) { return qrow_of_node ? qrow_of_node[idx] : depth[idx]; }

int orc_replay(const orc_logits *q, float temperature, const int32_t *qrow_of_node, int32_t N,
               const int32_t *depth, const int32_t *child_off, const int32_t *child_ids, uint64_t seed,
               const int32_t *batch_ids, int32_t *token, uint8_t *exempt_node)
{
    if (!q || N < 0 || !(temperature > 0.0f)) return -1;
    const float invT = 1.0f / temperature;
    const int V = q->V, C = (V + ORC_CHUNK - 1) / ORC_CHUNK, NN = N + 1;
    double *x = (double *)malloc(sizeof(double) * V);
    elem_key *ck = (elem_key *)malloc(sizeof(elem_key) * C);
    double *A = (double *)malloc(sizeof(double) * C);
    elem_key *ek = (elem_key *)malloc(sizeof(elem_key) * (size_t)V);
    if (!x || !ck || !A || !ek) return -3;
    for (int b = 0; b < q->B; ++b) {
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        token[(int64_t)b * NN + 0] = -1;
        for (int u = 0; u < NN; ++u) {
            if (exempt_node) exempt_node[(int64_t)b * NN + u] = 0;
            const int m = off[u + 1] - off[u];
            if (m == 0) continue;
            const int r = replay_row_index(qrow_of_node, depth, (int64_t)b * NN + u);
            if (r < 0 || r >= q->R) return -5;
            read_row(q, b, r, invT, x);
            /* 1. chunk log-masses and chunk keys */
            for (int c = 0; c < C; ++c) {
                int lo = c * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
                A[c] = logsumexp(x + lo, hi - lo);
                double uc = orc_uniform(seed, PURPOSE_REPLAY_CHUNK, batch_of(batch_ids, b), u, c);
                ck[c].k = A[c] + gumbel_of(uc);
                ck[c].v = c;
                ck[c].sens = gumbel_slope(uc);
            }
            /* 2. the top-m chunks by (K desc, c asc) */
            const int msel = m < C ? m : C;
            partial_sort(ck, C, msel + 1 < C ? msel + 1 : C);
            uint8_t ex = 0;
            if (C > msel && near_tie(&ck[msel - 1], &ck[msel])) ex = 1;
            /* 3. element keys inside the selected chunks, shifted to max K_c */
            int ne = 0;
            for (int s = 0; s < msel; ++s) {
                const int c = ck[s].v;
                const double Tc = ck[s].k;
                const double uc_slope = ck[s].sens;
                int lo = c * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
                int first = ne;
                double Z = -INFINITY;
                int jmax = -1;
                double umax = 0.5;
                for (int v = lo; v < hi; ++v) {
                    double uv = orc_uniform(seed, PURPOSE_REPLAY_ELEM, batch_of(batch_ids, b), u, v);
                    double g = x[v] + gumbel_of(uv);
                    ek[ne].k = g; /* raw key for now */
                    ek[ne].v = v;
                    ek[ne].sens = gumbel_slope(uv);
                    if (g > Z) { Z = g; jmax = ne; umax = uv; }
                    ++ne;
                }
                for (int e = first; e < ne; ++e) {
                    if (e == jmax) {
                        ek[e].k = Tc;
                        ek[e].sens = uc_slope;
                    } else {
                        double g = ek[e].k;
                        double k = shift_key(Tc, Z, g);
                        /* sensitivities through g (own uniform), T (chunk uniform), Z (max's uniform) */
                        double s_own = ek[e].sens * exp(k - g);
                        double s_T = uc_slope * exp(k - Tc);
                        double s_Z = gumbel_slope(umax) * exp(k - Z);
                        double s = s_own > s_T ? s_own : s_T;
                        if (s_Z > s) s = s_Z;
                        ek[e].k = k;
                        ek[e].sens = s;
                    }
                }
            }
            /* 4. the top-m keys over the selected chunks are the ordered WoR draws */
            partial_sort(ek, ne, m + 1 < ne ? m + 1 : ne);
            for (int j = 0; j < m; ++j) {
                if (j + 1 < ne && near_tie(&ek[j], &ek[j + 1])) ex = 1;
                token[(int64_t)b * NN + ids[off[u] + j]] = ek[j].v;
            }
            if (exempt_node) exempt_node[(int64_t)b * NN + u] = ex;
        }
    }
    free(x); free(ck); free(A); free(ek);
    return 0;
}

/* Flat Gumbel-top-m over the whole row (independent cross-check of the law only). */
int orc_replay_flat(const orc_logits *q, float temperature, const int32_t *qrow_of_node, int32_t N,
                    const int32_t *depth, const int32_t *child_off, const int32_t *child_ids, uint64_t seed,
                    const int32_t *batch_ids, int32_t *token)
{
    if (!q || N < 0 || !(temperature > 0.0f)) return -1;
    const float invT = 1.0f / temperature;
    const int V = q->V, NN = N + 1;
    double *x = (double *)malloc(sizeof(double) * V);
    elem_key *ek = (elem_key *)malloc(sizeof(elem_key) * (size_t)V);
    if (!x || !ek) return -3;
    for (int b = 0; b < q->B; ++b) {
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        token[(int64_t)b * NN] = -1;
        for (int u = 0; u < NN; ++u) {
            const int m = off[u + 1] - off[u];
            if (m == 0) continue;
            const int r = replay_row_index(qrow_of_node, depth, (int64_t)b * NN + u);
            if (r < 0 || r >= q->R) return -5;
            read_row(q, b, r, invT, x);
            for (int v = 0; v < V; ++v) {
                ek[v].k = x[v] + gumbel_of(orc_uniform(seed, PURPOSE_REPLAY_ELEM, batch_of(batch_ids, b), u, v));
                ek[v].v = v;
                ek[v].sens = 0;
            }
            partial_sort(ek, V, m);
            for (int j = 0; j < m; ++j) token[(int64_t)b * NN + ids[off[u] + j]] = ek[j].v;
        }
    }
    free(x); free(ek);
    return 0;
}

/* ------------------------------------------------------------------------------------ */
/* VERIFY: recursive rejection sampling for WoR candidates down the tree (Sec. 2.3 Eq.
 * rs-overlap for one candidate; App. A for the WoR variant used by Sequoia / EAGLE / RSD).
 * At a node with target law P, draft law Q and children y_1..y_m (in slot order):
 *   slot i: q' = Q(y_i)/t (t = draft mass not yet drawn), p' = P(y_i);
 *           accept iff U_i * q' < p'  (probability min(1, p'/q'));
 *           on reject: R(v) = max(P(v) - Q(v)/t [v not drawn], 0), P <- R / sum R,
 *                      y_i joins the drawn set, t <- t - Q(y_i).
 * If a child is accepted its token is emitted and the walk continues there; if all are
 * rejected the final token is drawn from the last residual R; at a leaf the bonus token
 * is drawn from the node's target row. Losslessness: Prop. 1. A residual with no mass after
 * a rejection cannot occur in exact arithmetic (a rejection needs p' < q', so some token has
 * p > q); should rounding produce one, the final token is drawn from the node's target row. */

static double draft_ratio(double qv, double t) { return (qv > 0.0 && t > 0.0) ? qv / t : 0.0; }

/* One rejection step: unnormalised residual R and its mass. */
static double rrs_residual(int V, const double *P, const double *Q, double t, const uint8_t *drawn, double *R)
{
    double Z = 0.0;
    for (int v = 0; v < V; ++v) {
        double qv = drawn[v] ? 0.0 : draft_ratio(Q[v], t);
        double r = P[v] - qv;
        R[v] = r > 0.0 ? r : 0.0;
        Z += R[v];
    }
    return Z;
}

/* Final-token draw from the law proportional to w (w >= 0), two-level Gumbel-max:
 *   chunk keys  K_c = log(sum_{v in c} w_v) + G(U[FINAL_CHUNK, node, c]) over chunks of
 *               ORC_CHUNK tokens with positive mass; the best chunk c* by (K desc, c asc);
 *   token       argmax_{v in c*, w_v > 0} log w_v + G(U[FINAL, node, v]) by (key desc, v asc).
 * P(c*) = mass(c)/total and, independently, P(v | c*) = w_v / mass(c*), so the token has law
 * w / total exactly (the m = 1 case of the hierarchical sampler of the replay pass).
 * With logits = 1 the input holds log-weights (x_v), as for a bonus token from a target row. */
static int sample_final(const double *w, int logits, int V, uint64_t seed, int bid, int node, uint8_t *ex)
{
    const int C = (V + ORC_CHUNK - 1) / ORC_CHUNK;
    int bc = -1;
    double kb = -INFINITY, ks = -INFINITY, sb = 0.0, ss = 0.0;
    for (int c = 0; c < C; ++c) {
        int lo = c * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
        double A;
        if (logits) {
            A = logsumexp(w + lo, hi - lo);
        } else {
            double m = 0.0;
            for (int v = lo; v < hi; ++v) m += w[v];
            if (!(m > 0.0)) continue;
            A = log(m);
        }
        double u = orc_uniform(seed, PURPOSE_FINAL_CHUNK, bid, node, c);
        double k = A + gumbel_of(u);
        if (bc < 0 || k > kb) {
            ks = kb; ss = sb;
            bc = c; kb = k; sb = gumbel_slope(u);
        } else if (k > ks) {
            ks = k; ss = gumbel_slope(u);
        }
    }
    if (bc < 0) return -1;
    if (ex && ks > -INFINITY && near_tie_keys(kb, ks, sb > ss ? sb : ss)) *ex = 1;
    int lo = bc * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
    int best = -1;
    double eb = -INFINITY, es = -INFINITY, tb = 0.0, ts = 0.0;
    for (int v = lo; v < hi; ++v) {
        if (!logits && !(w[v] > 0.0)) continue;
        double u = orc_uniform(seed, PURPOSE_FINAL, bid, node, v);
        double k = (logits ? w[v] : log(w[v])) + gumbel_of(u);
        if (best < 0 || k > eb) {
            es = eb; ts = tb;
            best = v; eb = k; tb = gumbel_slope(u);
        } else if (k > es) {
            es = k; ts = gumbel_slope(u);
        }
    }
    if (ex && es > -INFINITY && near_tie_keys(eb, es, tb > ts ? tb : ts)) *ex = 1;
    return best;
}

/* Exact law of one node's verification for a fixed ordered child tuple (for the
 * enumeration pins): acc[i] = P(accept slot i | slots before it rejected), and the law of
 * the final token when every slot is rejected. Uses the same update as the sampler.    */
int orc_rrs_node_law(int32_t V, const double *P_in, const double *Q, int32_t m, const int32_t *y, double *acc,
                     double *final_law)
{
    double *P = (double *)malloc(sizeof(double) * V), *R = (double *)malloc(sizeof(double) * V);
    uint8_t *drawn = (uint8_t *)calloc(V, 1);
    if (!P || !R || !drawn) return -3;
    memcpy(P, P_in, sizeof(double) * V);
    double t = 1.0;
    int degenerate = 0;
    for (int i = 0; i < m; ++i) acc[i] = 0.0;
    for (int i = 0; i < m; ++i) {
        double qp = draft_ratio(Q[y[i]], t), pp = P[y[i]];
        acc[i] = qp > 0.0 ? (pp / qp < 1.0 ? pp / qp : 1.0) : (pp > 0.0 ? 1.0 : 0.0);
        double Z = rrs_residual(V, P, Q, t, drawn, R);
        if (!(Z > 0.0)) {
            /* no residual mass: fine when this slot cannot be rejected (later slots and the
             * final law are then unreachable), degenerate otherwise */
            if (acc[i] < 1.0 - 1e-12) degenerate = 1; /* beyond rounding */
            for (int v = 0; v < V; ++v) P[v] = 0.0;
            break;
        }
        for (int v = 0; v < V; ++v) P[v] = R[v] / Z;
        drawn[y[i]] = 1;
        t -= Q[y[i]];
    }
    /* after the last rejection P holds R_m / Z_m */
    for (int v = 0; v < V; ++v) final_law[v] = P[v];
    free(P); free(R); free(drawn);
    return degenerate;
}

/* The draft law of node u: softmax of its q row over the whole vocabulary, or, with pools
 * (pool_ids [B][Lp][P], row depth[u] of tree b), over the P pool tokens only (zero elsewhere). */
static void draft_law(const double *xq, int V, const int32_t *pool, int P, double *Q)
{
    if (!pool) {
        softmax(xq, V, Q);
        return;
    }
    double m = -INFINITY, s = 0.0;
    for (int j = 0; j < P; ++j)
        if (xq[pool[j]] > m) m = xq[pool[j]];
    for (int j = 0; j < P; ++j) s += exp(xq[pool[j]] - m);
    const double lse = m + log(s);
    for (int v = 0; v < V; ++v) Q[v] = 0.0;
    for (int j = 0; j < P; ++j) Q[pool[j]] = exp(xq[pool[j]] - lse);
}

static int verify_rrs_impl(const orc_logits *target, const orc_logits *q, float temperature,
                           const int32_t *qrow_of_node, int32_t N, int32_t L, const int32_t *depth,
                           const int32_t *child_off, const int32_t *child_ids, const int32_t *token, uint64_t seed,
                           const int32_t *batch_ids, const int32_t *pool_ids, int32_t Pn, int32_t Lp,
                           int32_t *out_tokens, int32_t *out_nodes, int32_t *out_len, uint8_t *exempt)
{
    if (!target || !q || N < 0 || L < 1 || !(temperature > 0.0f) || target->V != q->V || target->R < N + 1) return -1;
    const float invT = 1.0f / temperature;
    const int V = target->V, NN = N + 1;
    double *xt = (double *)malloc(sizeof(double) * V), *xq = (double *)malloc(sizeof(double) * V);
    double *P = (double *)malloc(sizeof(double) * V), *Q = (double *)malloc(sizeof(double) * V);
    double *R = (double *)malloc(sizeof(double) * V);
    uint8_t *drawn = (uint8_t *)malloc(V);
    if (!xt || !xq || !P || !Q || !R || !drawn) return -3;
    for (int b = 0; b < target->B; ++b) {
        const int64_t nb = (int64_t)b * NN;
        const int bid = batch_of(batch_ids, b);
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        int32_t *otok = out_tokens + (int64_t)b * (L + 1), *onode = out_nodes + (int64_t)b * L;
        for (int k = 0; k <= L; ++k) otok[k] = -1;
        for (int k = 0; k < L; ++k) onode[k] = -1;
        uint8_t ex = 0;
        int u = 0, nacc = 0, final_tok = -1;
        for (int step = 0; step <= L; ++step) { /* depth grows by one per accepted node */
            const int m = off[u + 1] - off[u];
            read_row(target, b, u, invT, xt);
            if (m == 0) { /* leaf: bonus token from the node's target row */
                final_tok = sample_final(xt, 1, V, seed, bid, u, &ex);
                break;
            }
            const int r = replay_row_index(qrow_of_node, depth, nb + u);
            if (r < 0 || r >= q->R) return -5;
            read_row(q, b, r, invT, xq);
            softmax(xt, V, P);
            const int pd = depth[nb + u];
            if (pool_ids && (pd < 0 || pd >= Lp)) return -5;
            draft_law(xq, V, pool_ids ? pool_ids + ((int64_t)b * Lp + pd) * Pn : NULL, Pn, Q);
            memset(drawn, 0, V);
            double t = 1.0;
            int accepted = -1;
            for (int i = 0; i < m; ++i) {
                const int c = ids[off[u] + i];
                const int y = token[nb + c];
                if (y < 0 || y >= V) return -6;
                double qp = draft_ratio(Q[y], t), pp = P[y];
                double U = orc_uniform(seed, PURPOSE_ACCEPT, bid, c, 0);
                if (qp > 0.0 && fabs(U - pp / qp) < U_BAND) ex = 1;
                if (U * qp < pp) { accepted = c; break; }
                double Z = rrs_residual(V, P, Q, t, drawn, R);
                if (!(Z > 0.0)) { /* no residual mass (rounding only): draw from the node's target row */
                    final_tok = sample_final(xt, 1, V, seed, bid, u, &ex);
                    break;
                }
                if (i == m - 1) { /* every slot rejected: draw from the last residual */
                    final_tok = sample_final(R, 0, V, seed, bid, u, &ex);
                    break;
                }
                for (int v = 0; v < V; ++v) P[v] = R[v] / Z;
                drawn[y] = 1;
                t -= Q[y];
            }
            if (accepted < 0) break;
            otok[nacc] = token[nb + accepted];
            onode[nacc] = accepted;
            ++nacc;
            u = accepted;
        }
        otok[nacc] = final_tok;
        out_len[b] = nacc + 1;
        if (exempt) exempt[b] = ex;
    }
    free(xt); free(xq); free(P); free(Q); free(R); free(drawn);
    return 0;
}

int orc_verify_rrs(const orc_logits *target, const orc_logits *q, float temperature, const int32_t *qrow_of_node,
                   int32_t N, int32_t L, const int32_t *depth, const int32_t *child_off, const int32_t *child_ids,
                   const int32_t *token, uint64_t seed, const int32_t *batch_ids, int32_t *out_tokens,
                   int32_t *out_nodes, int32_t *out_len, uint8_t *exempt)
{
    return verify_rrs_impl(target, q, temperature, qrow_of_node, N, L, depth, child_off, child_ids, token, seed,
                           batch_ids, NULL, 0, 0, out_tokens, out_nodes, out_len, exempt);
}

/* Recursive rejection sampling with pooled draft laws (Sec. 3.3: the probabilities of replayed
 * candidates are normalised within the pool; the residual stays full-vocabulary, App. B.1
 * on pools: the restriction applies to draft proposals only). pool_ids [B][Lp][P]: the pool of
 * the tokens at depth d+1 in row d, used for the children of every node at depth d. */
int orc_verify_rrs_pooled(const orc_logits *target, const orc_logits *q, float temperature,
                          const int32_t *qrow_of_node, int32_t N, int32_t L, const int32_t *depth,
                          const int32_t *child_off, const int32_t *child_ids, const int32_t *token, uint64_t seed,
                          const int32_t *batch_ids, const int32_t *pool_ids, int32_t P, int32_t Lp,
                          int32_t *out_tokens, int32_t *out_nodes, int32_t *out_len, uint8_t *exempt)
{
    if (!pool_ids || P < 1 || P > q->V || Lp < 1) return -1;
    return verify_rrs_impl(target, q, temperature, qrow_of_node, N, L, depth, child_off, child_ids, token, seed,
                           batch_ids, pool_ids, P, Lp, out_tokens, out_nodes, out_len, exempt);
}

/* ------------------------------------------------------------------------------------ */
/* BLOCK VERIFICATION of a sampled chain X_1..X_g (Sun et al. 2025, cited in Sec. 1,
 * Table 2 and App. A). With Mb_i = target law after prefix X^i (i = 0..g) and
 * Ms_i = draft law of the next token after X^i (i = 0..g-1):
 *   w_0 = 1, w_i = min(w_{i-1} Mb_{i-1}(X_i) / Ms_{i-1}(X_i), 1);
 *   h_i = S_i / (S_i + 1 - w_i) with S_i = sum_x max(w_i Mb_i(x) - Ms_i(x), 0) (i < g),
 *         h_i = 1 when the denominator is 0;  h_g = w_g;
 *   tau = max{ i in 1..g : eta_i <= h_i }, 0 if none;
 *   final token ~ Mb_g if tau = g, else ~ max(w_tau Mb_tau - Ms_tau, 0) (normalised).
 * Emits X_1..X_tau and the final token.                                                  */
static void blockv_weights(int g, int V, const double *Mb, const double *Ms, const int32_t *X, double *w, double *h,
                           double *resid /* [g*V] unnormalised, may be NULL */)
{
    w[0] = 1.0;
    for (int i = 1; i <= g; ++i) {
        double num = Mb[(int64_t)(i - 1) * V + X[i - 1]], den = Ms[(int64_t)(i - 1) * V + X[i - 1]];
        double ratio = den > 0.0 ? w[i - 1] * num / den : 1.0;
        w[i] = ratio < 1.0 ? ratio : 1.0;
    }
    for (int i = 0; i < g; ++i) {
        double S = 0.0;
        for (int v = 0; v < V; ++v) {
            double r = w[i] * Mb[(int64_t)i * V + v] - Ms[(int64_t)i * V + v];
            r = r > 0.0 ? r : 0.0;
            if (resid) resid[(int64_t)i * V + v] = r;
            S += r;
        }
        double den = S + 1.0 - w[i];
        h[i] = den > 0.0 ? S / den : 1.0;
    }
    h[g] = w[g];
}

/* Exact pieces of the block-verification law for one chain (for the enumeration pins). */
int orc_blockv_law(int32_t g, int32_t V, const double *Mb, const double *Ms, const int32_t *X, double *w, double *h,
                   double *resid)
{
    blockv_weights(g, V, Mb, Ms, X, w, h, resid);
    return 0;
}

int orc_verify_block(const orc_logits *target, const orc_logits *q, float temperature, const int32_t *qrow_of_node,
                     int32_t N, int32_t L, const int32_t *depth, const int32_t *child_off, const int32_t *child_ids,
                     const int32_t *token, uint64_t seed, const int32_t *batch_ids, int32_t *out_tokens,
                     int32_t *out_nodes, int32_t *out_len, uint8_t *exempt, int32_t *tau_out)
{
    if (!target || !q || N < 1 || N > L || !(temperature > 0.0f) || target->V != q->V || target->R < N + 1) return -1;
    const float invT = 1.0f / temperature;
    const int V = target->V, NN = N + 1, g = N;
    double *x = (double *)malloc(sizeof(double) * V);
    double *Mb = (double *)malloc(sizeof(double) * (size_t)(g + 1) * V);
    double *Ms = (double *)malloc(sizeof(double) * (size_t)g * V);
    double *resid = (double *)malloc(sizeof(double) * (size_t)g * V);
    double *w = (double *)malloc(sizeof(double) * (g + 1)), *h = (double *)malloc(sizeof(double) * (g + 1));
    int32_t *X = (int32_t *)malloc(sizeof(int32_t) * g);
    if (!x || !Mb || !Ms || !resid || !w || !h || !X) return -3;
    for (int b = 0; b < target->B; ++b) {
        const int64_t nb = (int64_t)b * NN;
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        /* the tree must be the chain 0 -> 1 -> ... -> g */
        for (int i = 0; i <= g; ++i) {
            int want = i < g ? 1 : 0;
            if (off[i + 1] - off[i] != want || (want && ids[off[i]] != i + 1)) return -7;
        }
        for (int i = 0; i <= g; ++i) {
            read_row(target, b, i, invT, x);
            softmax(x, V, Mb + (int64_t)i * V);
        }
        for (int i = 0; i < g; ++i) {
            const int r = replay_row_index(qrow_of_node, depth, nb + i);
            if (r < 0 || r >= q->R) return -5;
            read_row(q, b, r, invT, x);
            softmax(x, V, Ms + (int64_t)i * V);
            X[i] = token[nb + i + 1];
            if (X[i] < 0 || X[i] >= V) return -6;
        }
        blockv_weights(g, V, Mb, Ms, X, w, h, resid);
        const int bid = batch_of(batch_ids, b);
        uint8_t ex = 0;
        int tau = 0;
        for (int i = 1; i <= g; ++i)
            if (orc_uniform(seed, PURPOSE_BLOCK_ETA, bid, i, 0) <= h[i]) tau = i;
        for (int i = (tau > 1 ? tau : 1); i <= g; ++i) /* decisions that could move tau */
            if (fabs(orc_uniform(seed, PURPOSE_BLOCK_ETA, bid, i, 0) - h[i]) < U_BAND) ex = 1;
        int final_tok;
        if (tau == g) {
            read_row(target, b, g, invT, x);
            final_tok = sample_final(x, 1, V, seed, bid, g, &ex);
        } else {
            double S = 0.0;
            for (int v = 0; v < V; ++v) S += resid[(int64_t)tau * V + v];
            if (S > 0.0)
                final_tok = sample_final(resid + (int64_t)tau * V, 0, V, seed, bid, tau, &ex);
            else { /* cannot carry mass in exact arithmetic; draw from the target row there */
                read_row(target, b, tau, invT, x);
                final_tok = sample_final(x, 1, V, seed, bid, tau, &ex);
            }
        }
        int32_t *otok = out_tokens + (int64_t)b * (L + 1), *onode = out_nodes + (int64_t)b * L;
        for (int k = 0; k <= L; ++k) otok[k] = -1;
        for (int k = 0; k < L; ++k) onode[k] = -1;
        for (int i = 1; i <= tau; ++i) {
            otok[i - 1] = X[i - 1];
            onode[i - 1] = i;
        }
        otok[tau] = final_tok;
        out_len[b] = tau + 1;
        if (exempt) exempt[b] = ex;
        if (tau_out) tau_out[b] = tau;
    }
    free(x); free(Mb); free(Ms); free(resid); free(w); free(h); free(X);
    return 0;
}

/* ------------------------------------------------------------------------------------ */
/* TRAVERSAL VERIFICATION (Weng et al. 2025, cited in Sec. 2.3, Table 2 ("RRS with
 * sequence-level coupling", WoR candidates) and App. A; UniVer reduces to it under WoR).
 * Recursive rejection sampling lifted from tokens to sequences: a node is accepted or
 * rejected only after the whole subtree below it has been tried, deepest first.
 *
 * Every node u carries a sequence weight p_a(u), a target-side law Mb_u (initially its target
 * row's softmax P_u) and its draft law Ms_u (Q_u with the tokens of rejected children removed
 * and renormalised, t = the draft mass left). p_a(root) = 1. Entering child c of u (slot order)
 *     p_a(c) = min(p_a(u) Mb_u(y_c) / Ms_u(y_c), 1),
 * then c's children are tried first (depth first, in slot order). When every child of u has
 * been tried and rejected (or u is a leaf), u is a leaf of the remaining tree and is accepted
 * iff U[ACCEPT, u] < p_a(u); the root is accepted once its children are rejected. Accepting u
 * emits the path from the root to u and a final token: the bonus from P_u if u had no
 * children, else a draw from the last residual below. When the subtree of child c (token y) of
 * u is rejected, u is updated (the block-verification step, for trees):
 *     R(v) = max(p_a(u) Mb_u(v) - Ms_u(v), 0),  S = sum_v R(v),
 *     p_a(u) <- S / (S + 1 - p_a(u)),  Mb_u <- R / S,  y leaves Ms_u.
 * A rejected child has p_a(u) Mb_u(y) < Ms_u(y) (otherwise p_a(c) = 1 and c is accepted when
 * tried), so R(y) = 0 before y leaves the draft law. S = 0 with p_a(u) < 1 leaves p_a(u) = 0
 * (u and everything tried after it are rejected); S = 0 with p_a(u) = 1 cannot happen in exact
 * arithmetic (it needs Mb_u = Ms_u, whose child is always accepted): should rounding produce
 * it, u is accepted with its final token from its target row, as in the RRS walk.
 * On a chain this is block verification (tau = the deepest accepted position); at the root it
 * is the WoR recursive rejection sampling above.                                           */

/* p_a of a child with token y of a node in state (pa, Mb, Q with t and drawn) */
static double trav_weight(double pa, const double *Mb, const double *Q, double t, const uint8_t *drawn, int y)
{
    double qy = drawn[y] ? 0.0 : draft_ratio(Q[y], t);
    double num = pa * Mb[y];
    if (qy > 0.0) {
        double r = num / qy;
        return r < 1.0 ? r : 1.0;
    }
    return num > 0.0 ? 1.0 : 0.0;
}

/* The update after the subtree of the child with token y was rejected. R receives the
 * unnormalised residual. Returns 1 in the degenerate case (no residual mass with pa = 1). */
static int trav_reject(int V, double *pa, double *Mb, const double *Q, double *t, uint8_t *drawn, int y, double *R)
{
    double S = 0.0;
    for (int v = 0; v < V; ++v) {
        double qv = drawn[v] ? 0.0 : draft_ratio(Q[v], *t);
        double r = *pa * Mb[v] - qv;
        R[v] = r > 0.0 ? r : 0.0;
        S += R[v];
    }
    int degenerate = 0;
    if (S > 0.0) {
        *pa = S / (S + 1.0 - *pa);
        for (int v = 0; v < V; ++v) Mb[v] = R[v] / S;
    } else if (*pa < 1.0) {
        *pa = 0.0;
    } else {
        degenerate = 1;
    }
    drawn[y] = 1;
    *t -= Q[y];
    return degenerate;
}

typedef struct {
    /* inputs of one tree */
    const orc_logits *target, *q;
    float invT;
    const int32_t *qrow_of_node, *depth, *off, *ids, *token;
    int64_t nb;
    int b, bid, V;
    uint64_t seed;
    /* per stack level: Mb, Q (V doubles each), drawn (V bytes); scratch R, x */
    double *Mb, *Q, *R, *x;
    uint8_t *drawn;
    int levels;
    /* results */
    uint8_t ex;
    int err, accepted, final_tok;
} trav_walk;

/* Try node u (stack level lev) with sequence weight pa. Returns 1 if u or a node below it was
 * accepted (the walk then stops), 0 if u's whole subtree was rejected. */
static int trav_visit(trav_walk *w, int u, int lev, double pa)
{
    const int V = w->V;
    if (lev >= w->levels) { w->err = -7; return 1; }
    double *Mb = w->Mb + (int64_t)lev * V, *Q = w->Q + (int64_t)lev * V;
    uint8_t *drawn = w->drawn + (int64_t)lev * V;
    const int m = w->off[u + 1] - w->off[u];
    read_row(w->target, w->b, u, w->invT, w->x);
    softmax(w->x, V, Mb);
    double t = 1.0;
    int degenerate = 0, rejected_any = 0;
    if (m > 0) {
        const int r = replay_row_index(w->qrow_of_node, w->depth, w->nb + u);
        if (r < 0 || r >= w->q->R) { w->err = -5; return 1; }
        read_row(w->q, w->b, r, w->invT, w->x);
        softmax(w->x, V, Q);
        memset(drawn, 0, V);
    }
    for (int i = 0; i < m; ++i) {
        const int c = w->ids[w->off[u] + i];
        const int y = w->token[w->nb + c];
        if (y < 0 || y >= V) { w->err = -6; return 1; }
        if (trav_visit(w, c, lev + 1, trav_weight(pa, Mb, Q, t, drawn, y))) return 1;
        rejected_any = 1;
        if (trav_reject(V, &pa, Mb, Q, &t, drawn, y, w->R)) { degenerate = 1; break; }
    }
    int accept = 1;
    if (u != 0 && !degenerate) {
        double U = orc_uniform(w->seed, PURPOSE_ACCEPT, w->bid, u, 0);
        if (fabs(U - pa) < U_BAND) w->ex = 1;
        accept = U < pa;
    }
    if (!accept) return 0;
    w->accepted = u;
    if (!rejected_any || degenerate) { /* bonus token from the node's target row */
        read_row(w->target, w->b, u, w->invT, w->x);
        w->final_tok = sample_final(w->x, 1, V, w->seed, w->bid, u, &w->ex);
    } else { /* from the last residual (R still holds it: nothing ran since the update) */
        w->final_tok = sample_final(w->R, 0, V, w->seed, w->bid, u, &w->ex);
    }
    return 1;
}

int orc_verify_traversal(const orc_logits *target, const orc_logits *q, float temperature,
                         const int32_t *qrow_of_node, int32_t N, int32_t L, const int32_t *parent,
                         const int32_t *depth, const int32_t *child_off, const int32_t *child_ids,
                         const int32_t *token, uint64_t seed, const int32_t *batch_ids, int32_t *out_tokens,
                         int32_t *out_nodes, int32_t *out_len, uint8_t *exempt)
{
    if (!target || !q || N < 0 || L < 1 || !(temperature > 0.0f) || target->V != q->V || target->R < N + 1) return -1;
    const int V = target->V, NN = N + 1, levels = L + 2;
    trav_walk w;
    memset(&w, 0, sizeof w);
    w.target = target;
    w.q = q;
    w.invT = 1.0f / temperature;
    w.qrow_of_node = qrow_of_node;
    w.depth = depth;
    w.token = token;
    w.V = V;
    w.seed = seed;
    w.levels = levels;
    w.Mb = (double *)malloc(sizeof(double) * (size_t)levels * V);
    w.Q = (double *)malloc(sizeof(double) * (size_t)levels * V);
    w.R = (double *)malloc(sizeof(double) * V);
    w.x = (double *)malloc(sizeof(double) * V);
    w.drawn = (uint8_t *)malloc((size_t)levels * V);
    if (!w.Mb || !w.Q || !w.R || !w.x || !w.drawn) return -3;
    int rc = 0;
    for (int b = 0; b < target->B && rc == 0; ++b) {
        w.b = b;
        w.bid = batch_of(batch_ids, b);
        w.nb = (int64_t)b * NN;
        w.off = child_off + (int64_t)b * (NN + 1);
        w.ids = child_ids + (int64_t)b * N;
        w.ex = 0;
        w.err = 0;
        w.accepted = -1;
        w.final_tok = -1;
        trav_visit(&w, 0, 0, 1.0);
        if (w.err) { rc = w.err; break; }
        int32_t *otok = out_tokens + (int64_t)b * (L + 1), *onode = out_nodes + (int64_t)b * L;
        for (int k = 0; k <= L; ++k) otok[k] = -1;
        for (int k = 0; k < L; ++k) onode[k] = -1;
        const int n = depth[w.nb + w.accepted];
        if (n > L) { rc = -7; break; }
        for (int a = w.accepted, k = n - 1; k >= 0; --k, a = parent[w.nb + a]) {
            onode[k] = a;
            otok[k] = token[w.nb + a];
        }
        otok[n] = w.final_tok;
        out_len[b] = n + 1;
        if (exempt) exempt[b] = w.ex;
    }
    free(w.Mb); free(w.Q); free(w.R); free(w.x); free(w.drawn);
    return rc;
}

/* Exact law of traversal verification on one tree with explicit laws (for the enumeration
 * pins), by the same weight and update steps as the sampler: P_rows / Q_rows [NN][V] (the
 * target and draft law at every node), tokens [NN]. Writes acc[u] = P(u is the accepted node)
 * and final_law[u][V] = the law of the final token when u is accepted. Returns 1 if a
 * degenerate update was met, else 0. */
typedef struct {
    int V;
    const int32_t *off, *ids, *token;
    const double *P, *Q;
    double *Mb, *Qs, *R;
    uint8_t *drawn;
    double *acc, *law;
    int degenerate;
} trav_law_ctx;

/* Returns the probability that u's subtree is rejected, given it is entered with prob reach. */
static double trav_law_visit(trav_law_ctx *c, int u, int lev, double pa, double reach)
{
    const int V = c->V;
    double *Mb = c->Mb + (int64_t)lev * V, *Q = c->Qs + (int64_t)lev * V;
    uint8_t *drawn = c->drawn + (int64_t)lev * V;
    const int m = c->off[u + 1] - c->off[u];
    memcpy(Mb, c->P + (int64_t)u * V, sizeof(double) * V);
    memcpy(Q, c->Q + (int64_t)u * V, sizeof(double) * V);
    memset(drawn, 0, V);
    double t = 1.0, cont = reach;
    int degenerate = 0, rejected_any = 0;
    for (int i = 0; i < m; ++i) {
        const int ch = c->ids[c->off[u] + i];
        const int y = c->token[ch];
        cont = trav_law_visit(c, ch, lev + 1, trav_weight(pa, Mb, Q, t, drawn, y), cont);
        rejected_any = 1;
        if (trav_reject(V, &pa, Mb, Q, &t, drawn, y, c->R)) { degenerate = 1; break; }
    }
    if (degenerate) c->degenerate = 1;
    const double pacc = (u == 0 || degenerate) ? 1.0 : pa;
    c->acc[u] += cont * pacc;
    double *law = c->law + (int64_t)u * V;
    if (!rejected_any || degenerate) {
        memcpy(law, c->P + (int64_t)u * V, sizeof(double) * V);
    } else {
        double S = 0.0;
        for (int v = 0; v < V; ++v) S += c->R[v];
        for (int v = 0; v < V; ++v) law[v] = S > 0.0 ? c->R[v] / S : 0.0;
    }
    return cont * (1.0 - pacc);
}

int orc_traversal_law(int32_t NN, int32_t V, const int32_t *child_off, const int32_t *child_ids,
                      const int32_t *token, const double *P_rows, const double *Q_rows, double *acc, double *final_law)
{
    trav_law_ctx c;
    memset(&c, 0, sizeof c);
    c.V = V;
    c.off = child_off;
    c.ids = child_ids;
    c.token = token;
    c.P = P_rows;
    c.Q = Q_rows;
    c.Mb = (double *)malloc(sizeof(double) * (size_t)NN * V);
    c.Qs = (double *)malloc(sizeof(double) * (size_t)NN * V);
    c.R = (double *)malloc(sizeof(double) * V);
    c.drawn = (uint8_t *)malloc((size_t)NN * V);
    c.acc = acc;
    c.law = final_law;
    if (!c.Mb || !c.Qs || !c.R || !c.drawn) return -3;
    for (int u = 0; u < NN; ++u) acc[u] = 0.0;
    memset(final_law, 0, sizeof(double) * (size_t)NN * V);
    trav_law_visit(&c, 0, 0, 1.0, 1.0);
    free(c.Mb); free(c.Qs); free(c.R); free(c.drawn);
    return c.degenerate;
}

/* ------------------------------------------------------------------------------------ */
/* PLAN, expand-then-prune (the EAGLE-2-style first pass of Sec. 3.1 and App. B.3).
 * Depth by depth, the W best candidates of the newest layer (its frontier) are expanded into
 * their K children each (a node at the depth cap L gets none). Once every layer exists, the N
 * best candidates of all layers are kept and numbered in the global order
 *     (key desc, depth asc, parent's position in its layer asc, rank asc),
 * with keys as in orc_plan (key = Sx - CL[d]). Inside a layer the order is the same one
 * restricted to a depth, so a frontier is a prefix of its sorted layer and positions of
 * same-depth parents order like their node numbers. A child's key never exceeds its parent's
 * and its depth is larger, so the kept set is prefix-closed. With W >= N every node of the
 * max-heap tree stays inside the frontiers (a node with n nodes before it in the global order
 * has at most n before it in its layer) and both planners return the same tree; this is the
 * sense in which App. B.3 says a wide enough frontier recovers the heap's solution.       */
typedef struct {
    double key, sx;
    int depth, ppos, rank;
    int num; /* node number once kept, 0 otherwise */
} ept_cand;

static int ept_before(const ept_cand *a, const ept_cand *b)
{
    if (a->key != b->key) return a->key > b->key;
    if (a->depth != b->depth) return a->depth < b->depth;
    if (a->ppos != b->ppos) return a->ppos < b->ppos;
    return a->rank < b->rank;
}

static int ept_cmp(const void *pa, const void *pb)
{
    const ept_cand *a = (const ept_cand *)pa, *b = (const ept_cand *)pb;
    return ept_before(a, b) ? -1 : (ept_before(b, a) ? 1 : 0);
}

/* adjacent entries in a sorted list whose order rounding could swap (plan_band) */
static int ept_near(const ept_cand *a, const ept_cand *b, double lse_err)
{
    if (a->depth == b->depth && a->sx == b->sx) return 0; /* exact tie on every machine */
    return a->key - b->key < plan_band(a->depth, b->depth, lse_err);
}

int orc_plan_expand(const orc_logits *draft, float temperature, int32_t N, int32_t K, int32_t L, int32_t W,
                    int32_t *parent, int32_t *depth, int32_t *rank, int32_t *plan_token, double *score,
                    int32_t *child_off, int32_t *child_ids, double lse_err, uint8_t *exempt)
{
    if (!draft || N < 1 || K < 1 || L < 1 || W < 1 || K > 64 || K > draft->V || draft->R < L) return -1;
    if (!(temperature > 0.0f)) return -1;
    const float invT = 1.0f / temperature;
    const int V = draft->V, NN = N + 1;
    /* layer sizes: K at depth 1, min(W, previous) * K below */
    int64_t total = 0, prev = 0;
    int64_t *lstart = (int64_t *)malloc(sizeof(int64_t) * (L + 2));
    if (!lstart) return -3;
    for (int d = 1; d <= L; ++d) {
        int64_t n = d == 1 ? K : (prev < W ? prev : W) * (int64_t)K;
        lstart[d] = total;
        total += n;
        prev = n;
    }
    lstart[L + 1] = total;
    if (total < N) { free(lstart); return -2; }
    double *x = (double *)malloc(sizeof(double) * V);
    double *CL = (double *)malloc(sizeof(double) * (L + 1));
    int32_t *tid = (int32_t *)malloc(sizeof(int32_t) * L * K);
    double *tx = (double *)malloc(sizeof(double) * L * K);
    ept_cand *lay = (ept_cand *)malloc(sizeof(ept_cand) * (size_t)total);
    ept_cand *all = (ept_cand *)malloc(sizeof(ept_cand) * (size_t)total);
    int32_t *nchild = (int32_t *)malloc(sizeof(int32_t) * NN);
    if (!x || !CL || !tid || !tx || !lay || !all || !nchild) return -3;
    int rc = 0;
    for (int b = 0; b < draft->B && rc == 0; ++b) {
        CL[0] = 0.0;
        for (int d = 0; d < L; ++d) {
            read_row(draft, b, d, invT, x);
            CL[d + 1] = CL[d] + logsumexp(x, V);
            topk_row(x, V, K, tid + d * K, tx + d * K);
        }
        uint8_t ex = 0;
        /* 1. layers, each sorted; the frontier of depth d is the first W of layer d */
        for (int d = 1; d <= L; ++d) {
            ept_cand *cur = lay + lstart[d];
            int64_t n = 0;
            if (d == 1) {
                for (int r = 0; r < K; ++r, ++n) {
                    cur[n].sx = tx[r];
                    cur[n].ppos = 0;
                    cur[n].rank = r;
                }
            } else {
                const ept_cand *par = lay + lstart[d - 1];
                const int64_t np = lstart[d] - lstart[d - 1], nf = np < W ? np : W;
                for (int64_t f = 0; f < nf; ++f)
                    for (int r = 0; r < K; ++r, ++n) {
                        cur[n].sx = par[f].sx + tx[(d - 1) * K + r];
                        cur[n].ppos = (int)f;
                        cur[n].rank = r;
                    }
                if (np > W && ept_near(&par[W - 1], &par[W], lse_err)) ex = 1; /* frontier edge */
            }
            for (int64_t i = 0; i < n; ++i) {
                cur[i].depth = d;
                cur[i].key = cur[i].sx - CL[d];
                cur[i].num = 0;
            }
            qsort(cur, (size_t)n, sizeof(ept_cand), ept_cmp);
        }
        /* 2. the N best of all layers, numbered in the global order. Each entry remembers its
         *    layer position through (depth, index) so parents can be found after the sort. */
        for (int64_t i = 0; i < total; ++i) {
            all[i] = lay[i];
            all[i].num = (int)i; /* temporarily: index into lay[] */
        }
        qsort(all, (size_t)total, sizeof(ept_cand), ept_cmp);
        for (int64_t i = 0; i < N && i + 1 < total; ++i)
            if (ept_near(&all[i], &all[i + 1], lse_err)) ex = 1; /* numbering and the budget edge */
        int32_t *par = parent + (int64_t)b * NN, *dep = depth + (int64_t)b * NN;
        int32_t *rk = rank + (int64_t)b * NN, *tok = plan_token + (int64_t)b * NN;
        double *sc = score + (int64_t)b * NN;
        par[0] = -1; dep[0] = 0; rk[0] = -1; tok[0] = -1; sc[0] = 0.0;
        for (int i = 1; i <= N; ++i) lay[all[i - 1].num].num = i;
        for (int i = 1; i <= N; ++i) {
            const ept_cand *c = &all[i - 1];
            int p = 0;
            if (c->depth > 1) p = lay[lstart[c->depth - 1] + c->ppos].num;
            if (c->depth > 1 && (p == 0 || p >= i)) { rc = -7; break; } /* not prefix-closed */
            par[i] = p;
            dep[i] = c->depth;
            rk[i] = c->rank;
            tok[i] = tid[(c->depth - 1) * K + c->rank];
            sc[i] = c->key;
        }
        if (exempt) exempt[b] = ex;
        /* child lists (CSR); siblings are kept in rank order, so slot = rank */
        int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        for (int u = 0; u < NN; ++u) nchild[u] = 0;
        for (int i = 1; i <= N && rc == 0; ++i) nchild[par[i]]++;
        off[0] = 0;
        for (int u = 0; u < NN; ++u) off[u + 1] = off[u] + nchild[u];
        for (int i = 1; i <= N && rc == 0; ++i) {
            if (rk[i] >= nchild[par[i]]) { rc = -7; break; } /* a sibling of lower rank is missing */
            ids[off[par[i]] + rk[i]] = i;
        }
    }
    free(lstart); free(x); free(CL); free(tid); free(tx); free(lay); free(all); free(nchild);
    return rc;
}

/* ------------------------------------------------------------------------------------ */
/* REPLAY with mixed sampling (Sec. 3.2 and App. A; the greedy draft sampling of Hu et al.
 * 2025 that the paper pairs with its tree verifiers). For a parent u with m children, the
 * first m-1 child slots take the m-1 most probable tokens of q_u, by (x desc, id asc), and the
 * last slot takes one draw from q_u renormalised over the remaining tokens.
 *
 * The draw is the largest Gumbel key among the remaining tokens, with the keys of the
 * hierarchical sampler of orc_replay (chunk keys K_c, element keys shifted to their chunk's
 * maximum): the keys are jointly i.i.d. Gumbel(x_v), so the largest one over a fixed token set
 * E' has law q restricted to E' and renormalised. A chunk without excluded tokens has its
 * chunk key as its largest key, so only the chunks holding an excluded token and the best
 * clean chunks need element keys (the second-best clean chunk only to flag near ties). With
 * m = 1 nothing is excluded and the draw is orc_replay's single draw, token for token.     */
int orc_replay_mixed(const orc_logits *q, float temperature, const int32_t *qrow_of_node, int32_t N,
                     const int32_t *depth, const int32_t *child_off, const int32_t *child_ids, uint64_t seed,
                     const int32_t *batch_ids, int32_t *token, uint8_t *exempt_node)
{
    if (!q || N < 0 || !(temperature > 0.0f)) return -1;
    const float invT = 1.0f / temperature;
    const int V = q->V, C = (V + ORC_CHUNK - 1) / ORC_CHUNK, NN = N + 1;
    double *x = (double *)malloc(sizeof(double) * V);
    elem_key *ck = (elem_key *)malloc(sizeof(elem_key) * C);
    uint8_t *excl = (uint8_t *)malloc(V), *dirty = (uint8_t *)malloc(C), *expand = (uint8_t *)malloc(C);
    elem_key *ek = (elem_key *)malloc(sizeof(elem_key) * (size_t)V);
    if (!x || !ck || !excl || !dirty || !expand || !ek) return -3;
    for (int b = 0; b < q->B; ++b) {
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        const int bid = batch_of(batch_ids, b);
        token[(int64_t)b * NN + 0] = -1;
        for (int u = 0; u < NN; ++u) {
            if (exempt_node) exempt_node[(int64_t)b * NN + u] = 0;
            const int m = off[u + 1] - off[u];
            if (m == 0) continue;
            if (m > V) return -5;
            const int r = replay_row_index(qrow_of_node, depth, (int64_t)b * NN + u);
            if (r < 0 || r >= q->R) return -5;
            read_row(q, b, r, invT, x);
            /* 1. the m-1 deterministic slots: the most probable tokens in order */
            int32_t top[64];
            double topx[64];
            if (m - 1 > 64) return -5;
            if (m > 1) topk_row(x, V, m - 1, top, topx);
            memset(excl, 0, V);
            memset(dirty, 0, C);
            for (int j = 0; j < m - 1; ++j) {
                excl[top[j]] = 1;
                dirty[top[j] / ORC_CHUNK] = 1;
                token[(int64_t)b * NN + ids[off[u] + j]] = top[j];
            }
            /* 2. chunk keys; the two best clean chunks by (K desc, c asc) */
            int best1 = -1, best2 = -1;
            for (int c = 0; c < C; ++c) {
                int lo = c * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
                double uc = orc_uniform(seed, PURPOSE_REPLAY_CHUNK, bid, u, c);
                ck[c].k = logsumexp(x + lo, hi - lo) + gumbel_of(uc);
                ck[c].v = c;
                ck[c].sens = gumbel_slope(uc);
                if (dirty[c]) continue;
                if (best1 < 0 || elem_before(&ck[c], &ck[best1])) {
                    best2 = best1;
                    best1 = c;
                } else if (best2 < 0 || elem_before(&ck[c], &ck[best2])) {
                    best2 = c;
                }
            }
            for (int c = 0; c < C; ++c) expand[c] = dirty[c];
            if (best1 >= 0) expand[best1] = 1;
            if (best2 >= 0) expand[best2] = 1;
            /* 3. shifted element keys of the expanded chunks; excluded tokens drop out */
            int ne = 0;
            for (int c = 0; c < C; ++c) {
                if (!expand[c]) continue;
                const double Tc = ck[c].k, uc_slope = ck[c].sens;
                int lo = c * ORC_CHUNK, hi = lo + ORC_CHUNK < V ? lo + ORC_CHUNK : V;
                double Z = -INFINITY, umax = 0.5;
                int jmax = -1;
                double *g = (double *)malloc(sizeof(double) * (hi - lo));
                double *ug = (double *)malloc(sizeof(double) * (hi - lo));
                if (!g || !ug) return -3;
                for (int v = lo; v < hi; ++v) {
                    ug[v - lo] = orc_uniform(seed, PURPOSE_REPLAY_ELEM, bid, u, v);
                    g[v - lo] = x[v] + gumbel_of(ug[v - lo]);
                    if (g[v - lo] > Z) { Z = g[v - lo]; jmax = v; umax = ug[v - lo]; }
                }
                for (int v = lo; v < hi; ++v) {
                    if (excl[v]) continue;
                    if (v == jmax) {
                        ek[ne].k = Tc;
                        ek[ne].sens = uc_slope;
                    } else {
                        double k = shift_key(Tc, Z, g[v - lo]);
                        double s_own = gumbel_slope(ug[v - lo]) * exp(k - g[v - lo]);
                        double s_T = uc_slope * exp(k - Tc);
                        double s_Z = gumbel_slope(umax) * exp(k - Z);
                        double s = s_own > s_T ? s_own : s_T;
                        if (s_Z > s) s = s_Z;
                        ek[ne].k = k;
                        ek[ne].sens = s;
                    }
                    ek[ne].v = v;
                    ++ne;
                }
                free(g);
                free(ug);
            }
            if (ne == 0) return -5; /* cannot happen: V >= m leaves a token */
            /* 4. the best remaining key is the sampled slot */
            partial_sort(ek, ne, ne > 1 ? 2 : 1);
            uint8_t ex = (ne > 1 && near_tie(&ek[0], &ek[1])) ? 1 : 0;
            token[(int64_t)b * NN + ids[off[u] + m - 1]] = ek[0].v;
            if (exempt_node) exempt_node[(int64_t)b * NN + u] = ex;
        }
    }
    free(x); free(ck); free(excl); free(dirty); free(expand); free(ek);
    return 0;
}

/* ------------------------------------------------------------------------------------ */
/* VERIFY by target-sample matching ("Naive" in Table 2, Sec. 2.3): at the current node u a
 * token y is drawn from the target law p_u; if a child of u carries y (the first such slot),
 * that child is accepted, y is emitted and the walk continues there; otherwise y itself is
 * emitted as the final token and the walk stops. At a leaf the draw is the bonus token. Every
 * emitted token is a draw from the target law at its prefix, whatever the candidates are, so
 * the scheme is lossless for any tree and any way of filling it (deterministic first-pass
 * tokens, WoR or mixed replay); a child with token v is accepted with probability p_u(v).
 * The draw is the two-level Gumbel-max of sample_final on the target logits (purposes
 * FINAL_CHUNK and FINAL, node u), the same draw as a bonus token.                        */
int orc_verify_naive(const orc_logits *target, float temperature, int32_t N, int32_t L, const int32_t *child_off,
                     const int32_t *child_ids, const int32_t *token, uint64_t seed, const int32_t *batch_ids,
                     int32_t *out_tokens, int32_t *out_nodes, int32_t *out_len, uint8_t *exempt)
{
    if (!target || N < 0 || L < 1 || !(temperature > 0.0f) || target->R < N + 1) return -1;
    const float invT = 1.0f / temperature;
    const int V = target->V, NN = N + 1;
    double *xt = (double *)malloc(sizeof(double) * V);
    if (!xt) return -3;
    for (int b = 0; b < target->B; ++b) {
        const int64_t nb = (int64_t)b * NN;
        const int bid = batch_of(batch_ids, b);
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        int32_t *otok = out_tokens + (int64_t)b * (L + 1), *onode = out_nodes + (int64_t)b * L;
        for (int k = 0; k <= L; ++k) otok[k] = -1;
        for (int k = 0; k < L; ++k) onode[k] = -1;
        uint8_t ex = 0;
        int u = 0, nacc = 0, y = -1;
        for (;;) {
            read_row(target, b, u, invT, xt);
            y = sample_final(xt, 1, V, seed, bid, u, &ex);
            int next = -1;
            for (int i = off[u]; i < off[u + 1]; ++i) {
                const int c = ids[i];
                if (c < 1 || c > N) { free(xt); return -6; }
                if (token[nb + c] == y) { next = c; break; }
            }
            if (next < 0 || nacc >= L) break;
            otok[nacc] = y;
            onode[nacc] = next;
            ++nacc;
            u = next;
            y = -1;
        }
        otok[nacc] = y;
        out_len[b] = nacc + 1;
        if (exempt) exempt[b] = ex;
    }
    free(xt);
    return 0;
}

/* ------------------------------------------------------------------------------------ */
/* REPLAY with pooled draft laws (Sec. 3.2: q_u is restricted to the same sparse candidate
 * pools as the first pass and normalised within them). For a parent u with m children, the
 * pool is row depth[u] of pool_ids [B][Lp][P] (the P tokens of the children's position); the
 * m ordered WoR draws from q_u restricted to the pool are the top-m Gumbel keys
 * x_v + G(U[REPLAY_ELEM, u, v]) over the pool tokens (Gumbel-top-k over P tokens; the pool is
 * small, so the keys are drawn flat, with the counters the flat sampler uses).            */
int orc_replay_pooled(const orc_logits *q, float temperature, const int32_t *qrow_of_node, int32_t N,
                      const int32_t *depth, const int32_t *child_off, const int32_t *child_ids,
                      const int32_t *pool_ids, int32_t P, int32_t Lp, uint64_t seed, const int32_t *batch_ids,
                      int32_t *token, uint8_t *exempt_node)
{
    if (!q || !pool_ids || N < 0 || P < 1 || P > q->V || Lp < 1 || !(temperature > 0.0f)) return -1;
    const float invT = 1.0f / temperature;
    const int V = q->V, NN = N + 1;
    double *x = (double *)malloc(sizeof(double) * V);
    elem_key *ek = (elem_key *)malloc(sizeof(elem_key) * (size_t)P);
    if (!x || !ek) return -3;
    for (int b = 0; b < q->B; ++b) {
        const int32_t *off = child_off + (int64_t)b * (NN + 1), *ids = child_ids + (int64_t)b * N;
        const int bid = batch_of(batch_ids, b);
        token[(int64_t)b * NN] = -1;
        for (int u = 0; u < NN; ++u) {
            if (exempt_node) exempt_node[(int64_t)b * NN + u] = 0;
            const int m = off[u + 1] - off[u];
            if (m == 0) continue;
            const int d = depth[(int64_t)b * NN + u];
            const int r = replay_row_index(qrow_of_node, depth, (int64_t)b * NN + u);
            if (m > P || d < 0 || d >= Lp || r < 0 || r >= q->R) return -5;
            read_row(q, b, r, invT, x);
            const int32_t *pool = pool_ids + ((int64_t)b * Lp + d) * P;
            for (int j = 0; j < P; ++j) {
                const int v = pool[j];
                if (v < 0 || v >= V) return -6;
                const double uv = orc_uniform(seed, PURPOSE_REPLAY_ELEM, bid, u, v);
                ek[j].k = x[v] + gumbel_of(uv);
                ek[j].v = v;
                ek[j].sens = gumbel_slope(uv);
            }
            partial_sort(ek, P, m + 1 < P ? m + 1 : P);
            uint8_t ex = 0;
            for (int j = 0; j < m; ++j) {
                if (j + 1 < P && near_tie(&ek[j], &ek[j + 1])) ex = 1;
                token[(int64_t)b * NN + ids[off[u] + j]] = ek[j].v;
            }
            if (exempt_node) exempt_node[(int64_t)b * NN + u] = ex;
        }
    }
    free(x); free(ek);
    return 0;
}
