/*
 * oracle.c -- plain fp64 CPU reference of the per-step tree-verification pass
 * of Medusa/Hydra multi-token-prediction decoding (EntMTP, Sec. 2.3, 3.2, 4).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, loads or
 * calls this file; only the tests, the smoke check and the benchmark's CPU
 * baseline leg do.  It shares no code, header or table with the CUDA path.
 *
 * Every routine is the plain definition of what the verification pass
 * computes, evaluated in double precision from the same bf16 inputs that the
 * GPU sees.  No blocking, fusion or reordering beyond the definition; the only
 * parallelism is an OpenMP loop over independent outputs.
 *
 *   tree           anc(i) = {i} U anc(parent(i)), depth(root) = 0
 *                  (the precompiled tree masks / position offsets, Sec. 1, 2.3)
 *   attention      node i attends to the whole prefix [0, L) and to the tree
 *                  slots L + j of its ancestors-or-self j (tree decoding, Sec. 3.2)
 *   LM head        z = W h; greedy token argmax z (lowest index on ties);
 *                  p = softmax(z); top-1 probability max p (the p0 of Sec. 4);
 *                  entropy -sum p ln p in nats
 *   acceptance     node i is accepted when every non-root node j on its root
 *                  path carries the draft token that the target model would
 *                  emit greedily after j's parent: draft[j] == argmax[parent(j)].
 *                  The accepted path ends at the deepest accepted node (smallest
 *                  index among equally deep ones); accept_len = depth + 1 counts
 *                  the accepted drafts plus the bonus token argmax[j*]
 *                  (greedy form of the verification step, Sec. 3.2 / 5.1 tau).
 *   typical        the Medusa/Hydra typical-acceptance rule (Sec. 5.1, 5.2:
 *                  T = 0.7, eps = 0.09, alpha = 0.3): an edge is accepted when
 *                  the tempered target probability of its draft token exceeds
 *                  min(eps, alpha exp(-H)); see oracle_typical_accept.
 *
 * Pinned by tests/test_oracle_pins.py against independent references
 * (torch float64 attention, brute-force path enumeration, closed forms).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_MAX_NODES 64

static double bf16_value(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads of the OpenMP loops that follow (n >= 1); returns the previous count. */
int oracle_set_num_threads(int n)
{
    const int prev = oracle_num_threads();
#ifdef _OPENMP
    if (n >= 1)
        omp_set_num_threads(n);
#endif
    return prev;
}

/*
 * Tree bookkeeping.  in_anc[i * n + j] = 1 when j is i or an ancestor of i.
 * depth[i] = number of edges from the root.  Returns 0, or -1 when parent[]
 * is not a tree rooted at node 0 (parent[0] must be -1, every other parent in
 * [0, n), no cycles).  Nodes need not be in any particular order.
 */
int oracle_tree(const int32_t *parent, int n, int32_t *depth, uint8_t *in_anc)
{
    if (n < 1 || n > ORACLE_MAX_NODES || parent[0] != -1)
        return -1;
    for (int i = 1; i < n; ++i)
        if (parent[i] < 0 || parent[i] >= n)
            return -1;
    memset(in_anc, 0, (size_t)n * n);
    for (int i = 0; i < n; ++i) {
        int j = i, steps = 0;
        while (j != -1) {
            if (steps > n)
                return -1; /* cycle */
            in_anc[(size_t)i * n + j] = 1;
            j = (j == 0) ? -1 : parent[j];
            ++steps;
        }
        depth[i] = steps - 1;
    }
    return 0;
}

/*
 * Tree-masked attention of one layer.
 *   q    [N][Hq][d]              bf16 bits, post-rotary
 *   k, v [Hkv][head_stride] rows  bf16 bits; key slot s of kv head g starts at
 *        g * head_stride + s * d.  Slots [0, L) are the prefix, [L, L + N) the
 *        tree nodes in node order.
 *   out  [N][Hq][d]              double
 * q head h reads kv head h / (Hq / Hkv).  Softmax scale 1/sqrt(d).
 */
int oracle_tree_attention(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                          int64_t head_stride, int L, int N, int Hq, int Hkv, int d,
                          const int32_t *parent, double *out)
{
    if (Hkv < 1 || Hq % Hkv != 0 || d < 1 || L < 0)
        return -1;
    uint8_t in_anc[ORACLE_MAX_NODES * ORACLE_MAX_NODES];
    int32_t depth[ORACLE_MAX_NODES];
    if (oracle_tree(parent, N, depth, in_anc) != 0)
        return -1;
    const int group = Hq / Hkv;
    const double scale = 1.0 / sqrt((double)d);
    const int n_keys = L + N;

#pragma omp parallel
    {
        double *score = (double *)malloc(sizeof(double) * (size_t)n_keys);
        int *allowed = (int *)malloc(sizeof(int) * (size_t)n_keys);
#pragma omp for schedule(dynamic)
        for (int ih = 0; ih < N * Hq; ++ih) {
            const int i = ih / Hq, h = ih % Hq, g = h / group;
            const uint16_t *qi = q + ((size_t)i * Hq + h) * d;
            const uint16_t *kg = k + (size_t)g * head_stride;
            const uint16_t *vg = v + (size_t)g * head_stride;
            int n_allowed = 0;
            for (int s = 0; s < L; ++s)
                allowed[n_allowed++] = s;
            for (int j = 0; j < N; ++j)
                if (in_anc[(size_t)i * N + j])
                    allowed[n_allowed++] = L + j;
            double mx = -INFINITY;
            for (int a = 0; a < n_allowed; ++a) {
                const uint16_t *ks = kg + (size_t)allowed[a] * d;
                double dot = 0.0;
                for (int c = 0; c < d; ++c)
                    dot += bf16_value(qi[c]) * bf16_value(ks[c]);
                score[a] = dot * scale;
                if (score[a] > mx)
                    mx = score[a];
            }
            double denom = 0.0;
            for (int a = 0; a < n_allowed; ++a) {
                score[a] = exp(score[a] - mx);
                denom += score[a];
            }
            double *o = out + ((size_t)i * Hq + h) * d;
            for (int c = 0; c < d; ++c)
                o[c] = 0.0;
            for (int a = 0; a < n_allowed; ++a) {
                const uint16_t *vs = vg + (size_t)allowed[a] * d;
                const double w = score[a] / denom;
                for (int c = 0; c < d; ++c)
                    o[c] += w * bf16_value(vs[c]);
            }
        }
        free(score);
        free(allowed);
    }
    (void)n_keys;
    return 0;
}

/*
 * LM head and the per-row statistics of the greedy verifier.
 *   hidden [R][D], W [V][D] (nn.Linear layout), both bf16 bits.
 *   argmax[r]  first index of the largest logit
 *   top1[r]    largest softmax probability
 *   entropy[r] -sum_v p_v ln p_v (nats, temperature 1)
 *   gap[r]     largest minus second-largest logit (may be NULL)
 *   logits     [R][V] (may be NULL)
 */
int oracle_lm_head(const uint16_t *hidden, const uint16_t *W, int R, int D, int V,
                   int32_t *argmax, double *top1, double *entropy, double *gap,
                   double *logits)
{
    if (R < 0 || D < 1 || V < 1)
        return -1;
    double *z = (double *)malloc(sizeof(double) * (size_t)R * V);
    if (!z)
        return -2;
#pragma omp parallel for collapse(2) schedule(static)
    for (int r = 0; r < R; ++r)
        for (int vv = 0; vv < V; ++vv) {
            const uint16_t *h = hidden + (size_t)r * D;
            const uint16_t *w = W + (size_t)vv * D;
            double acc = 0.0;
            for (int c = 0; c < D; ++c)
                acc += bf16_value(w[c]) * bf16_value(h[c]);
            z[(size_t)r * V + vv] = acc;
        }
    for (int r = 0; r < R; ++r) {
        const double *zr = z + (size_t)r * V;
        int best = 0;
        for (int vv = 1; vv < V; ++vv)
            if (zr[vv] > zr[best])
                best = vv;
        double second = -INFINITY;
        for (int vv = 0; vv < V; ++vv)
            if (vv != best && zr[vv] > second)
                second = zr[vv];
        double denom = 0.0;
        for (int vv = 0; vv < V; ++vv)
            denom += exp(zr[vv] - zr[best]);
        double ent = 0.0, pmax = 0.0;
        for (int vv = 0; vv < V; ++vv) {
            const double p = exp(zr[vv] - zr[best]) / denom;
            if (p > 0.0)
                ent -= p * log(p);
            if (p > pmax)
                pmax = p;
        }
        argmax[r] = best;
        top1[r] = pmax;
        entropy[r] = ent;
        if (gap)
            gap[r] = zr[best] - second;
        if (logits)
            memcpy(logits + (size_t)r * V, zr, sizeof(double) * (size_t)V);
    }
    free(z);
    return 0;
}

/*
 * Greedy tree acceptance.
 *   parent[N], draft[N] (draft[0] ignored), argmax[N] (target greedy token
 *   after each node).
 * Outputs accept_len (>= 1), path[0 .. accept_len) = root .. j*, and the bonus
 * token argmax[j*].  Returns 0 or -1 for an invalid tree.
 */
int oracle_accept(const int32_t *parent, int N, const int32_t *draft,
                  const int32_t *argmax, int32_t *accept_len, int32_t *path,
                  int32_t *bonus)
{
    uint8_t in_anc[ORACLE_MAX_NODES * ORACLE_MAX_NODES];
    int32_t depth[ORACLE_MAX_NODES];
    if (oracle_tree(parent, N, depth, in_anc) != 0)
        return -1;
    int best = 0;
    for (int i = 0; i < N; ++i) {
        int ok = 1;
        for (int j = i; j != 0; j = parent[j])
            if (draft[j] != argmax[parent[j]]) {
                ok = 0;
                break;
            }
        if (ok && (depth[i] > depth[best] || (depth[i] == depth[best] && i < best)))
            best = i;
    }
    const int len = depth[best] + 1;
    for (int j = best, pos = len - 1; pos >= 0; --pos) {
        path[pos] = j;
        j = (j == 0) ? -1 : parent[j];
    }
    *accept_len = len;
    *bonus = argmax[best];
    return 0;
}

/*
 * Typical acceptance: the verification rule of Medusa/Hydra decoding that the
 * paper keeps unchanged and runs with T = 0.7, eps = 0.09, alpha = 0.3
 * (Sec. 5.1, 5.2).  The rule itself is the published Medusa one: the target
 * distribution after node u is p_u = softmax(z_u / T) with entropy
 * H_u = -sum_v p_u(v) ln p_u(v) (nats); the edge into non-root node j is
 * accepted when
 *     p_{parent(j)}(draft[j]) > min(eps, alpha * exp(-H_{parent(j)})),
 * and node i is accepted when every edge on its root path is.  Among the
 * deepest accepted nodes the one whose path has the largest log-likelihood
 * sum_{j on the path, j != root} ln p_{parent(j)}(draft[j]) wins (smallest
 * index on exact ties).  accept_len = depth + 1; the bonus token is the
 * greedy token after the last accepted node, argmax z_{j*} (lowest index on
 * ties): the first token of every step is taken greedily.
 *   logits [N][V]       z_u for every node u (double)
 *   margin[j]  (NULL ok) (p - threshold) / threshold of the edge into j; 0 for the root
 *   loglik[i]  (NULL ok) path log-likelihood of node i; 0 for the root
 *   accepted[i](NULL ok) 1 when node i is accepted
 * A draft token outside [0, V) has probability 0 and is never accepted.
 */
int oracle_typical_accept(const int32_t *parent, int N, const int32_t *draft, const double *logits, int V,
                          double temperature, double eps, double alpha, int32_t *accept_len, int32_t *path,
                          int32_t *bonus, double *margin, double *loglik, int32_t *accepted)
{
    uint8_t in_anc[ORACLE_MAX_NODES * ORACLE_MAX_NODES];
    int32_t depth[ORACLE_MAX_NODES];
    if (oracle_tree(parent, N, depth, in_anc) != 0 || V < 1 || !(temperature > 0.0))
        return -1;
    double p_edge[ORACLE_MAX_NODES], thr[ORACLE_MAX_NODES];
    int32_t amax[ORACLE_MAX_NODES];
    for (int u = 0; u < N; ++u) {
        const double *z = logits + (size_t)u * V;
        int best = 0;
        for (int v = 1; v < V; ++v)
            if (z[v] > z[best])
                best = v;
        amax[u] = best;
    }
    /* per edge: the target probability of the drafted token and the threshold */
    for (int j = 0; j < N; ++j) {
        p_edge[j] = 1.0;
        thr[j] = 0.0;
        if (j == 0)
            continue;
        const int u = parent[j];
        const double *z = logits + (size_t)u * V;
        const double m = z[amax[u]];
        double denom = 0.0;
        for (int v = 0; v < V; ++v)
            denom += exp((z[v] - m) / temperature);
        double ent = 0.0;
        for (int v = 0; v < V; ++v) {
            const double p = exp((z[v] - m) / temperature) / denom;
            if (p > 0.0)
                ent -= p * log(p);
        }
        const int tok = draft[j];
        p_edge[j] = (tok >= 0 && tok < V) ? exp((z[tok] - m) / temperature) / denom : 0.0;
        const double a = alpha * exp(-ent);
        thr[j] = eps < a ? eps : a;
    }
    /* per node: accepted when every edge of its root path is; path log-likelihood */
    int32_t ok[ORACLE_MAX_NODES];
    double ll[ORACLE_MAX_NODES];
    for (int i = 0; i < N; ++i) {
        ok[i] = 1;
        ll[i] = 0.0;
        for (int j = 0; j < N; ++j)
            if (j != 0 && in_anc[(size_t)i * N + j]) {
                if (!(p_edge[j] > thr[j]))
                    ok[i] = 0;
                ll[i] += p_edge[j] > 0.0 ? log(p_edge[j]) : -INFINITY;
            }
    }
    int best = 0;
    for (int i = 1; i < N; ++i) {
        if (!ok[i])
            continue;
        if (depth[i] > depth[best] || (depth[i] == depth[best] && ll[i] > ll[best]))
            best = i;
    }
    const int len = depth[best] + 1;
    for (int j = best, pos = len - 1; pos >= 0; --pos) {
        path[pos] = j;
        j = (j == 0) ? -1 : parent[j];
    }
    *accept_len = len;
    *bonus = amax[best];
    for (int j = 0; j < N; ++j) {
        if (margin)
            margin[j] = (j == 0 || thr[j] == 0.0) ? 0.0 : (p_edge[j] - thr[j]) / thr[j];
        if (loglik)
            loglik[j] = ll[j];
        if (accepted)
            accepted[j] = ok[j];
    }
    return 0;
}

/*
 * Statistics of the tempered target distribution p = softmax(z / T) of each
 * row (the quantities typical acceptance reads, Sec. 5.1/5.2 settings):
 *   logz[r] = ln sum_v e^(z_r[v] / T)       (log-partition)
 *   ent[r]  = -sum_v p_r(v) ln p_r(v)       (entropy, nats)
 * logits [R][V] (double).
 */
int oracle_tempered_stats(const double *logits, int R, int V, double temperature, double *logz, double *ent)
{
    if (R < 0 || V < 1 || !(temperature > 0.0))
        return -1;
    for (int r = 0; r < R; ++r) {
        const double *z = logits + (size_t)r * V;
        double m = z[0];
        for (int v = 1; v < V; ++v)
            if (z[v] > m)
                m = z[v];
        double denom = 0.0;
        for (int v = 0; v < V; ++v)
            denom += exp((z[v] - m) / temperature);
        double h = 0.0;
        for (int v = 0; v < V; ++v) {
            const double p = exp((z[v] - m) / temperature) / denom;
            if (p > 0.0)
                h -= p * log(p);
        }
        logz[r] = m / temperature + log(denom);
        ent[r] = h;
    }
    return 0;
}

static uint16_t bf16_round(double x)
{
    /* float64 -> float32 (round to nearest) -> bf16 bits (round to nearest even); finite inputs */
    float f = (float)x;
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/*
 * Rotary position embedding of the base model (Llama: frequencies
 * theta_i = base^(-2i/d), i < d/2, element i paired with element i + d/2):
 *   y_i       = x_i cos(p theta_i) - x_{i+d/2} sin(p theta_i)
 *   y_{i+d/2} = x_{i+d/2} cos(p theta_i) + x_i sin(p theta_i)
 * for row r at position pos[r].  x: bf16 bits [rows][d]; y: double [rows][d].
 */
int oracle_rope(const uint16_t *x, int rows, int d, const int32_t *pos, double base, double *y)
{
    if (rows < 0 || d < 2 || d % 2 || !(base > 0.0))
        return -1;
    const int h = d / 2;
    for (int r = 0; r < rows; ++r)
        for (int i = 0; i < h; ++i) {
            const double th = pow(base, -2.0 * i / d);
            const double a = (double)pos[r] * th;
            const double c = cos(a), s = sin(a);
            const double x1 = bf16_value(x[(size_t)r * d + i]), x2 = bf16_value(x[(size_t)r * d + i + h]);
            y[(size_t)r * d + i] = x1 * c - x2 * s;
            y[(size_t)r * d + i + h] = x2 * c + x1 * s;
        }
    return 0;
}

/*
 * Tree-masked attention with the rotary embedding applied at the tree's
 * position offsets (TopologyBank "position offsets", Sec. 1 / 2.3): node i sits
 * at position L + depth(i).  Inputs are pre-rotary for the step's tokens:
 * q [N][Hq][d] and the tree slots L + j of k; the prefix slots [0, L) of k hold
 * keys already rotated at their own positions (as a KV cache does).  The
 * rotated tree keys are stored back into the bf16 cache, so they are rounded
 * to bf16 (written to k_rot [Hkv][N][d] as bits); q stays in double.
 *   k, v  [Hkv][head_stride] rows as in oracle_tree_attention
 *   out   [N][Hq][d] double
 */
int oracle_tree_attention_rope(const uint16_t *q, const uint16_t *k, const uint16_t *v, int64_t head_stride, int L,
                               int N, int Hq, int Hkv, int d, const int32_t *parent, double base, double *out,
                               uint16_t *k_rot)
{
    if (Hkv < 1 || Hq % Hkv != 0 || d < 2 || d % 2 || L < 0 || !(base > 0.0))
        return -1;
    uint8_t in_anc[ORACLE_MAX_NODES * ORACLE_MAX_NODES];
    int32_t depth[ORACLE_MAX_NODES];
    if (oracle_tree(parent, N, depth, in_anc) != 0)
        return -1;
    int32_t pos[ORACLE_MAX_NODES];
    for (int i = 0; i < N; ++i)
        pos[i] = L + depth[i];
    /* rotated tree keys, rounded to the cache's bf16 */
    double *tmp = (double *)malloc(sizeof(double) * (size_t)N * d);
    if (!tmp)
        return -2;
    for (int g = 0; g < Hkv; ++g) {
        oracle_rope(k + (size_t)g * head_stride + (size_t)L * d, N, d, pos, base, tmp);
        for (size_t e = 0; e < (size_t)N * d; ++e)
            k_rot[(size_t)g * N * d + e] = bf16_round(tmp[e]);
    }
    free(tmp);
    const int group = Hq / Hkv;
    const double scale = 1.0 / sqrt((double)d);
#pragma omp parallel
    {
        double *score = (double *)malloc(sizeof(double) * (size_t)(L + N));
        double *qr = (double *)malloc(sizeof(double) * (size_t)d);
        const double *kp[1];
        (void)kp;
#pragma omp for schedule(dynamic)
        for (int ih = 0; ih < N * Hq; ++ih) {
            const int i = ih / Hq, h = ih % Hq, g = h / group;
            oracle_rope(q + ((size_t)i * Hq + h) * d, 1, d, &pos[i], base, qr);
            const uint16_t *kg = k + (size_t)g * head_stride;
            const uint16_t *vg = v + (size_t)g * head_stride;
            const uint16_t *kt = k_rot + (size_t)g * N * d;
            double mx = -INFINITY;
            int n = 0;
            for (int s = 0; s < L + N; ++s) {
                if (s >= L && !in_anc[(size_t)i * N + (s - L)])
                    continue;
                const uint16_t *ks = s < L ? kg + (size_t)s * d : kt + (size_t)(s - L) * d;
                double dot = 0.0;
                for (int c = 0; c < d; ++c)
                    dot += qr[c] * bf16_value(ks[c]);
                score[s] = dot * scale;
                if (score[s] > mx)
                    mx = score[s];
                ++n;
            }
            double denom = 0.0;
            for (int s = 0; s < L + N; ++s)
                if (s < L || in_anc[(size_t)i * N + (s - L)]) {
                    score[s] = exp(score[s] - mx);
                    denom += score[s];
                }
            double *o = out + ((size_t)i * Hq + h) * d;
            for (int c = 0; c < d; ++c)
                o[c] = 0.0;
            for (int s = 0; s < L + N; ++s)
                if (s < L || in_anc[(size_t)i * N + (s - L)]) {
                    const uint16_t *vs = vg + (size_t)s * d;
                    const double w = score[s] / denom;
                    for (int c = 0; c < d; ++c)
                        o[c] += w * bf16_value(vs[c]);
                }
        }
        free(score);
        free(qr);
    }
    return 0;
}

/*
 * Speculative sampling on a draft tree.  The rule of Sec. 2.1 (tokens accepted
 * left to right with probability min(1, p(t) / q(t)); at the first rejection
 * the replacement is drawn from norm(max(0, p - q))) applied at every node to
 * its children in increasing id order, the residual replacing the target after
 * each rejected sibling (the multi-candidate form of the rule):
 *   - target p_u = softmax(z_u / T) for every node u;
 *   - q_u [V]: the draft distribution the children of u were drawn from;
 *   - at node u with residual r (= p_u on arrival), child c with token t_c is
 *     accepted when unif[c] < r(t_c) / q_u(t_c) (q_u(t_c) = 0: accepted when
 *     r(t_c) > 0); the walk moves to c;
 *   - on rejection r <- max(0, r - q_u) / sum_v max(0, r(v) - q_u(v)) and the
 *     next child is tried;
 *   - when no child of u is accepted (or u is a leaf) the walk stops: the
 *     token after u is drawn from r by inverse CDF: the smallest v with
 *     sum_{w <= v} r(w) > unif[N + u].
 * accept_len = depth(u) + 1, path = root .. u, token = the drawn token.
 *   logits [N][V], q [N][V] (double); unif [2N]
 *   ratio_margin[c] (NULL ok): r(t_c) / q_u(t_c) - unif[c] for the children tried, NAN otherwise
 *   cdf_margin (NULL ok): distance of unif[N + u] to the nearest CDF value of r
 * A draft token outside [0, V) has r = 0 and is rejected.
 */
int oracle_spec_sample(const int32_t *parent, int N, const int32_t *draft, const double *logits, const double *q,
                       int V, double temperature, const double *unif, int32_t *accept_len, int32_t *path,
                       int32_t *token, double *ratio_margin, double *cdf_margin)
{
    uint8_t in_anc[ORACLE_MAX_NODES * ORACLE_MAX_NODES];
    int32_t depth[ORACLE_MAX_NODES];
    if (oracle_tree(parent, N, depth, in_anc) != 0 || V < 1 || !(temperature > 0.0))
        return -1;
    double *r = (double *)malloc(sizeof(double) * (size_t)V);
    if (!r)
        return -2;
    if (ratio_margin)
        for (int j = 0; j < N; ++j)
            ratio_margin[j] = NAN;
    int u = 0;
    for (;;) {
        /* r = p_u */
        const double *z = logits + (size_t)u * V;
        double m = z[0];
        for (int v = 1; v < V; ++v)
            if (z[v] > m)
                m = z[v];
        double s = 0.0;
        for (int v = 0; v < V; ++v) {
            r[v] = exp((z[v] - m) / temperature);
            s += r[v];
        }
        for (int v = 0; v < V; ++v)
            r[v] /= s;
        int next = -1;
        const double *qu = q + (size_t)u * V;
        for (int c = u + 1; c < N && next < 0; ++c) {
            if (parent[c] != u)
                continue;
            const int t = draft[c];
            const double rt = (t >= 0 && t < V) ? r[t] : 0.0;
            const double qt = (t >= 0 && t < V) ? qu[t] : 0.0;
            const double ratio = qt > 0.0 ? rt / qt : (rt > 0.0 ? INFINITY : 0.0);
            if (ratio_margin)
                ratio_margin[c] = ratio - unif[c];
            if (unif[c] < ratio) {
                next = c;
                break;
            }
            /* rejected: residual */
            double zr = 0.0;
            for (int v = 0; v < V; ++v) {
                r[v] = r[v] > qu[v] ? r[v] - qu[v] : 0.0;
                zr += r[v];
            }
            if (zr > 0.0)
                for (int v = 0; v < V; ++v)
                    r[v] /= zr;
        }
        if (next < 0)
            break;
        u = next;
    }
    /* inverse CDF at u */
    const double x = unif[N + u];
    double cum = 0.0, best = INFINITY;
    int tok = V - 1;
    for (int v = 0; v < V; ++v) {
        const double before = cum;
        cum += r[v];
        const double dist = fabs(cum - x);
        if (dist < best && r[v] > 0.0)
            best = dist;
        if (cum > x && before <= x) {
            tok = v;
            const double d0 = fabs(before - x);
            if (d0 < best)
                best = d0;
            break;
        }
    }
    if (cdf_margin)
        *cdf_margin = best;
    const int len = depth[u] + 1;
    for (int j = u, pos = len - 1; pos >= 0; --pos) {
        path[pos] = j;
        j = (j == 0) ? -1 : parent[j];
    }
    *accept_len = len;
    *token = tok;
    free(r);
    return 0;
}
