/*
 * oracle.c - plain fp64 CPU decoder for self-speculative decoding.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path loads this code:
 * only tests/, __graft_entry__.smoke() and the CPU-baseline leg of bench.py
 * call it.  It shares no code with the CUDA library.
 *
 * What it computes (arxiv 2309.08168, "Draft & Verify"):
 *   - the LLaMA-2 decoder forward p(x | z, x_1..x_i) of Sec. 3.2, where the
 *     sublayer mask z (one bit per attention / MLP sublayer, Sec. 3.3 Eq. 1:
 *     z in {0,1}^L with L = 2 * n_layers) makes a skipped sublayer add nothing
 *     to the residual stream; z = 0 is the original model;
 *   - greedy autoregressive decoding (Algorithm 1);
 *   - greedy self-speculative decoding (Algorithm 2): K drafts from the
 *     masked model, one verification of all of them by the full model, the
 *     longest matching prefix accepted, the first mismatch corrected, or a
 *     bonus token when every draft matches;
 *   - self-speculative sampling (Algorithm 4, App. G): drafts sampled from
 *     q = p(.|z*, ...), each accepted when r < min(1, p/q), the first
 *     rejected one replaced by a sample of norm(max(0, p - q)), and a bonus
 *     token sampled from p when all are accepted.
 * Everything is fp64; weights are the exact bf16 values widened; the KV cache
 * is kept in fp64 with no intermediate rounding.
 *
 * Readings where the paper is silent or ambiguous (each one is listed in the
 * design notes):
 *   - K drafts d_1..d_K per round; the verification runs on the K+1 rows
 *     [x_last, d_1..d_K] and gives target rows p_0..p_K; a round emits n+1
 *     tokens (n accepted drafts plus one correction or bonus token).
 *   - The draft forward attends over the committed full-model KV of earlier
 *     positions plus the KV that this round's drafts wrote, and writes KV only
 *     in the attention sublayers it runs; the verification rewrites KV for
 *     all layers; the rollback keeps the committed length len <- len + 1 + n.
 *   - The prompt's last token is the first round's x_last: the prefill runs
 *     prompt[0..P-2] and every emitted token comes from a decoding round.
 *   - The last round drafts K_eff = min(K, remaining - 1) tokens so that no
 *     token beyond n_new is produced.
 *   - Greedy ties go to the lowest token index.
 *   - Sampling distributions are softmax(logits / temperature) restricted to
 *     the nucleus {x : pi(x) >= tau*}, tau* the largest value whose upper set
 *     holds at least top_p of the mass, then renormalised; p and q both.
 *   - A residual max(0, p - q) with zero mass falls back to p.
 *   - Random numbers come from Philox4x32-10 (Salmon et al., SC'11) keyed by
 *     the 64-bit seed, counter (position, purpose, 0, 0) with purpose 0 for
 *     draft samples, 1 for acceptance uniforms, 2 for resample / bonus
 *     samples; u = (w0 + 0.5) * 2^-32.  Inverse-CDF sampling walks the tokens
 *     in ascending order and returns the first x with cumsum(x) > u * total.
 *   - RoPE pairs element i with element i + head_dim/2 (rotate-half form),
 *     frequency theta^(-2i/head_dim); GQA query head h reads KV head
 *     floor(h * n_kv_heads / n_heads).
 *   - Adaptive draft exit (Sec. 3.4, Eqs. 2-4, Algorithms 3 / 4 of App. G):
 *     the draft whose confidence falls below gamma is kept as the round's
 *     last draft (the algorithms choose x_{j+1} before the test); confidence
 *     is the largest probability of the distribution the draft was chosen
 *     from (softmax of the draft logits in greedy mode, the temperature /
 *     nucleus distribution q_j in sampling mode); AR_e = accepted / drafted
 *     of round e; gamma and AR are updated after every verification that
 *     had drafts, with beta1 = 0 at the first update; gamma starts at
 *     gamma0 for every generation.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab, max_seq;
    double rms_eps, rope_theta;
} orc_config;

/* Per-layer pointer arrays hold n_layers host pointers to bf16 bit arrays,
 * row-major [out_features][in_features]. */
typedef struct {
    const uint16_t* embed;       /* [vocab][d] */
    const uint16_t* final_norm;  /* [d] */
    const uint16_t* lm_head;     /* [vocab][d] */
    const uint16_t* const* wq;   /* [H*hd][d] */
    const uint16_t* const* wk;   /* [Hkv*hd][d] */
    const uint16_t* const* wv;   /* [Hkv*hd][d] */
    const uint16_t* const* wo;   /* [d][H*hd] */
    const uint16_t* const* attn_norm; /* [d] */
    const uint16_t* const* w_gate;    /* [F][d] */
    const uint16_t* const* w_up;      /* [F][d] */
    const uint16_t* const* w_down;    /* [d][F] */
    const uint16_t* const* mlp_norm;  /* [d] */
} orc_weights;

typedef struct {
    int rounds, drafted, accepted, emitted;
    int hist[33];
} orc_stats;

typedef struct {
    orc_config c;
    orc_weights w;
    /* copies of the per-layer pointer arrays (the caller's may go away) */
    const uint16_t** ptrs;
    double* kc; /* [L][max_seq][Hkv*hd] */
    double* vc;
} orc_model;

/* ------------------------------------------------------------------------ */
/* small helpers                                                             */
/* ------------------------------------------------------------------------ */

/* OpenMP threads of the row-parallel loops (timing runs; results do not
 * depend on it: every dot product is summed in k order by one thread). */
void orc_set_threads(int n) { omp_set_num_threads(n > 0 ? n : 1); }
int orc_get_threads(void) { return omp_get_max_threads(); }

double orc_bf16_to_f64(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

/* y[n] = sum_k W[n][k] x[k], W bf16 [N][K]; each row summed in k order. */
static void matvec(const uint16_t* W, const double* x, double* y, int N, int K) {
    #pragma omp parallel for schedule(static)
    for (int n = 0; n < N; ++n) {
        const uint16_t* row = W + (size_t)n * K;
        double acc = 0.0;
        for (int k = 0; k < K; ++k) acc += orc_bf16_to_f64(row[k]) * x[k];
        y[n] = acc;
    }
}

/* RMSNorm (LLaMA): out = x / sqrt(mean(x^2) + eps) * g */
void orc_rmsnorm(const double* x, const uint16_t* g, int d, double eps, double* out) {
    double ss = 0.0;
    for (int i = 0; i < d; ++i) ss += x[i] * x[i];
    double r = 1.0 / sqrt(ss / d + eps);
    for (int i = 0; i < d; ++i) out[i] = x[i] * r * orc_bf16_to_f64(g[i]);
}

/* Rotary position embedding, rotate-half pairing (i, i + hd/2). */
void orc_rope(double* v, int n_heads, int hd, int pos, double theta) {
    int half = hd / 2;
    for (int h = 0; h < n_heads; ++h) {
        double* x = v + (size_t)h * hd;
        for (int i = 0; i < half; ++i) {
            double freq = pow(theta, -(2.0 * i) / hd);
            double a = pos * freq;
            double c = cos(a), s = sin(a);
            double x1 = x[i], x2 = x[i + half];
            x[i] = x1 * c - x2 * s;
            x[i + half] = x2 * c + x1 * s;
        }
    }
}

static double silu(double x) { return x / (1.0 + exp(-x)); }

/* ------------------------------------------------------------------------ */
/* model object                                                              */
/* ------------------------------------------------------------------------ */

orc_model* orc_create(const orc_config* c, const orc_weights* w) {
    if (!c || !w || c->n_layers <= 0 || c->d_model <= 0 || c->n_heads <= 0 ||
        c->n_kv_heads <= 0 || c->n_heads % c->n_kv_heads || c->head_dim % 2 ||
        c->vocab <= 0 || c->max_seq <= 0)
        return NULL;
    orc_model* m = (orc_model*)calloc(1, sizeof(orc_model));
    if (!m) return NULL;
    m->c = *c;
    int L = c->n_layers;
    m->ptrs = (const uint16_t**)malloc(sizeof(void*) * 9 * (size_t)L);
    const uint16_t* const* src[9] = {w->wq, w->wk, w->wv, w->wo, w->attn_norm,
                                     w->w_gate, w->w_up, w->w_down, w->mlp_norm};
    for (int t = 0; t < 9; ++t)
        for (int l = 0; l < L; ++l) m->ptrs[t * L + l] = src[t][l];
    m->w.embed = w->embed;
    m->w.final_norm = w->final_norm;
    m->w.lm_head = w->lm_head;
    m->w.wq = m->ptrs + 0 * L;
    m->w.wk = m->ptrs + 1 * L;
    m->w.wv = m->ptrs + 2 * L;
    m->w.wo = m->ptrs + 3 * L;
    m->w.attn_norm = m->ptrs + 4 * L;
    m->w.w_gate = m->ptrs + 5 * L;
    m->w.w_up = m->ptrs + 6 * L;
    m->w.w_down = m->ptrs + 7 * L;
    m->w.mlp_norm = m->ptrs + 8 * L;
    size_t kv = (size_t)L * c->max_seq * c->n_kv_heads * c->head_dim;
    m->kc = (double*)calloc(kv, sizeof(double));
    m->vc = (double*)calloc(kv, sizeof(double));
    if (!m->kc || !m->vc) {
        free(m->kc); free(m->vc); free(m->ptrs); free(m);
        return NULL;
    }
    return m;
}

void orc_destroy(orc_model* m) {
    if (!m) return;
    free(m->kc);
    free(m->vc);
    free(m->ptrs);
    free(m);
}

/* Direct access to the fp64 KV cache (timing runs fill it at a chosen
 * context length).  which = 0 keys, 1 values; layout [L][max_seq][Hkv*hd]. */
double* orc_cache(orc_model* m, int which) { return which ? m->vc : m->kc; }

/* ------------------------------------------------------------------------ */
/* forward of one position with KV cache (Sec. 3.2: p(x | z, x_1..x_i))      */
/* ------------------------------------------------------------------------ */

/* Runs token `tok` at position `pos` through the model with sublayer mask
 * `mask` (NULL or all-zero = full model), writing K/V at `pos` in every
 * attention sublayer that runs and attending over cache positions [0, pos].
 * logits may be NULL (prefill). */
void orc_forward(orc_model* m, int tok, int pos, const uint8_t* mask, double* logits) {
    const orc_config* c = &m->c;
    int d = c->d_model, H = c->n_heads, Hkv = c->n_kv_heads, hd = c->head_dim, F = c->ffn;
    int qd = H * hd, kvd = Hkv * hd;
    double* h = (double*)malloc(sizeof(double) * d);
    double* u = (double*)malloc(sizeof(double) * d);
    double* q = (double*)malloc(sizeof(double) * qd);
    double* a = (double*)malloc(sizeof(double) * qd);
    double* o = (double*)malloc(sizeof(double) * d);
    double* g = (double*)malloc(sizeof(double) * F);
    double* up = (double*)malloc(sizeof(double) * F);
    double* sc = (double*)malloc(sizeof(double) * (size_t)(pos + 1) * H);

    for (int i = 0; i < d; ++i) h[i] = orc_bf16_to_f64(m->w.embed[(size_t)tok * d + i]);

    for (int l = 0; l < c->n_layers; ++l) {
        if (!(mask && mask[2 * l])) {
            double* kl = m->kc + ((size_t)l * c->max_seq + pos) * kvd;
            double* vl = m->vc + ((size_t)l * c->max_seq + pos) * kvd;
            orc_rmsnorm(h, m->w.attn_norm[l], d, c->rms_eps, u);
            matvec(m->w.wq[l], u, q, qd, d);
            matvec(m->w.wk[l], u, kl, kvd, d);
            matvec(m->w.wv[l], u, vl, kvd, d);
            orc_rope(q, H, hd, pos, c->rope_theta);
            orc_rope(kl, Hkv, hd, pos, c->rope_theta);
            double inv = 1.0 / sqrt((double)hd);
            #pragma omp parallel for schedule(static)
            for (int hh = 0; hh < H; ++hh) {
                int kvh = (int)(((long long)hh * Hkv) / H);
                const double* qh = q + (size_t)hh * hd;
                double* s = sc + (size_t)hh * (pos + 1);
                double mx = -INFINITY;
                for (int t = 0; t <= pos; ++t) {
                    const double* kt = m->kc + ((size_t)l * c->max_seq + t) * kvd + (size_t)kvh * hd;
                    double dot = 0.0;
                    for (int i = 0; i < hd; ++i) dot += qh[i] * kt[i];
                    s[t] = dot * inv;
                    if (s[t] > mx) mx = s[t];
                }
                double z = 0.0;
                for (int t = 0; t <= pos; ++t) { s[t] = exp(s[t] - mx); z += s[t]; }
                double* ah = a + (size_t)hh * hd;
                for (int i = 0; i < hd; ++i) ah[i] = 0.0;
                for (int t = 0; t <= pos; ++t) {
                    const double* vt = m->vc + ((size_t)l * c->max_seq + t) * kvd + (size_t)kvh * hd;
                    double w = s[t] / z;
                    for (int i = 0; i < hd; ++i) ah[i] += w * vt[i];
                }
            }
            matvec(m->w.wo[l], a, o, d, qd);
            for (int i = 0; i < d; ++i) h[i] += o[i];
        }
        if (!(mask && mask[2 * l + 1])) {
            orc_rmsnorm(h, m->w.mlp_norm[l], d, c->rms_eps, u);
            matvec(m->w.w_gate[l], u, g, F, d);
            matvec(m->w.w_up[l], u, up, F, d);
            for (int i = 0; i < F; ++i) g[i] = silu(g[i]) * up[i];
            matvec(m->w.w_down[l], g, o, d, F);
            for (int i = 0; i < d; ++i) h[i] += o[i];
        }
    }
    if (logits) {
        orc_rmsnorm(h, m->w.final_norm, d, c->rms_eps, u);
        matvec(m->w.lm_head, u, logits, c->vocab, d);
    }
    free(h); free(u); free(q); free(a); free(o); free(g); free(up); free(sc);
}

/* ------------------------------------------------------------------------ */
/* brute force: the whole sequence recomputed from scratch, no cache         */
/* ------------------------------------------------------------------------ */

/* Positions [0, n_full) run the full model; positions [n_full, n) run with
 * `mask` and attend over the full-model keys/values of [0, n_full) plus the
 * masked model's own keys/values of [n_full, p] (the draft reading).  With
 * n_full = n every position is the full model.  logits_all: [n][vocab]. */
int orc_forward_uncached(const orc_model* m, const int* toks, int n, int n_full,
                         const uint8_t* mask, double* logits_all) {
    const orc_config* c = &m->c;
    int d = c->d_model, H = c->n_heads, Hkv = c->n_kv_heads, hd = c->head_dim, F = c->ffn;
    int qd = H * hd, kvd = Hkv * hd;
    if (n <= 0 || n_full < 0 || n_full > n) return -1;
    double* hs = (double*)malloc(sizeof(double) * (size_t)n * d);
    double* Q = (double*)malloc(sizeof(double) * (size_t)n * qd);
    double* Kx = (double*)malloc(sizeof(double) * (size_t)n * kvd);
    double* Vx = (double*)malloc(sizeof(double) * (size_t)n * kvd);
    double* A = (double*)malloc(sizeof(double) * (size_t)n * qd);
    double* u = (double*)malloc(sizeof(double) * d);
    double* o = (double*)malloc(sizeof(double) * d);
    double* g = (double*)malloc(sizeof(double) * F);
    double* up = (double*)malloc(sizeof(double) * F);
    double* s = (double*)malloc(sizeof(double) * n);
    for (int p = 0; p < n; ++p)
        for (int i = 0; i < d; ++i)
            hs[(size_t)p * d + i] = orc_bf16_to_f64(m->w.embed[(size_t)toks[p] * d + i]);
    for (int l = 0; l < c->n_layers; ++l) {
        int skip_a = mask && mask[2 * l], skip_m = mask && mask[2 * l + 1];
        /* projections for every position that runs this attention sublayer */
        for (int p = 0; p < n; ++p) {
            if (p >= n_full && skip_a) continue;
            orc_rmsnorm(hs + (size_t)p * d, m->w.attn_norm[l], d, c->rms_eps, u);
            matvec(m->w.wq[l], u, Q + (size_t)p * qd, qd, d);
            matvec(m->w.wk[l], u, Kx + (size_t)p * kvd, kvd, d);
            matvec(m->w.wv[l], u, Vx + (size_t)p * kvd, kvd, d);
            orc_rope(Q + (size_t)p * qd, H, hd, p, c->rope_theta);
            orc_rope(Kx + (size_t)p * kvd, Hkv, hd, p, c->rope_theta);
        }
        for (int p = 0; p < n; ++p) {
            if (p >= n_full && skip_a) continue;
            for (int hh = 0; hh < H; ++hh) {
                int kvh = (int)(((long long)hh * Hkv) / H);
                double mx = -INFINITY, z = 0.0;
                for (int t = 0; t <= p; ++t) {
                    double dot = 0.0;
                    for (int i = 0; i < hd; ++i)
                        dot += Q[(size_t)p * qd + hh * hd + i] * Kx[(size_t)t * kvd + kvh * hd + i];
                    s[t] = dot / sqrt((double)hd);
                    if (s[t] > mx) mx = s[t];
                }
                for (int t = 0; t <= p; ++t) { s[t] = exp(s[t] - mx); z += s[t]; }
                for (int i = 0; i < hd; ++i) {
                    double acc = 0.0;
                    for (int t = 0; t <= p; ++t) acc += s[t] / z * Vx[(size_t)t * kvd + kvh * hd + i];
                    A[(size_t)p * qd + hh * hd + i] = acc;
                }
            }
        }
        for (int p = 0; p < n; ++p) {
            if (p >= n_full && skip_a) continue;
            matvec(m->w.wo[l], A + (size_t)p * qd, o, d, qd);
            for (int i = 0; i < d; ++i) hs[(size_t)p * d + i] += o[i];
        }
        for (int p = 0; p < n; ++p) {
            if (p >= n_full && skip_m) continue;
            double* hp = hs + (size_t)p * d;
            orc_rmsnorm(hp, m->w.mlp_norm[l], d, c->rms_eps, u);
            matvec(m->w.w_gate[l], u, g, F, d);
            matvec(m->w.w_up[l], u, up, F, d);
            for (int i = 0; i < F; ++i) g[i] = silu(g[i]) * up[i];
            matvec(m->w.w_down[l], g, o, d, F);
            for (int i = 0; i < d; ++i) hp[i] += o[i];
        }
    }
    for (int p = 0; p < n; ++p) {
        orc_rmsnorm(hs + (size_t)p * d, m->w.final_norm, d, c->rms_eps, u);
        matvec(m->w.lm_head, u, logits_all + (size_t)p * c->vocab, c->vocab, d);
    }
    free(hs); free(Q); free(Kx); free(Vx); free(A); free(u); free(o); free(g); free(up); free(s);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* random numbers: Philox4x32-10 (Salmon, Moraes, Dror, Shaw; SC'11)          */
/* ------------------------------------------------------------------------ */

void orc_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4]) {
    uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
        uint64_t p0 = (uint64_t)0xD2511F53u * c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t n0 = hi1 ^ c1 ^ k0;
        uint32_t n1 = lo1;
        uint32_t n2 = hi0 ^ c3 ^ k1;
        uint32_t n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* u in (0,1) for (seed, position, purpose) */
double orc_uniform(uint64_t seed, int pos, int purpose) {
    uint32_t ctr[4] = {(uint32_t)pos, (uint32_t)purpose, 0u, 0u};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t o[4];
    orc_philox4x32_10(ctr, key, o);
    return ((double)o[0] + 0.5) * (1.0 / 4294967296.0);
}

/* ------------------------------------------------------------------------ */
/* token choice                                                              */
/* ------------------------------------------------------------------------ */

int orc_argmax(const double* x, int n) {
    int best = 0;
    for (int i = 1; i < n; ++i)
        if (x[i] > x[best]) best = i;  /* strict: ties keep the lowest index */
    return best;
}

static int cmp_desc(const void* a, const void* b) {
    double x = *(const double*)a, y = *(const double*)b;
    return (x < y) - (x > y);
}

/* Sampling distribution: softmax(logits / temperature) restricted to the
 * nucleus {x : pi(x) >= tau*}, tau* = the largest value whose upper set holds
 * at least top_p of the mass, renormalised.  top_p >= 1 keeps every token. */
void orc_nucleus_probs(const double* logits, int V, double temperature, double top_p, double* out) {
    double mx = -INFINITY;
    for (int i = 0; i < V; ++i) if (logits[i] / temperature > mx) mx = logits[i] / temperature;
    double z = 0.0;
    for (int i = 0; i < V; ++i) { out[i] = exp(logits[i] / temperature - mx); z += out[i]; }
    for (int i = 0; i < V; ++i) out[i] /= z;
    if (top_p >= 1.0) return;
    double* sorted = (double*)malloc(sizeof(double) * V);
    memcpy(sorted, out, sizeof(double) * V);
    qsort(sorted, V, sizeof(double), cmp_desc);
    double cum = 0.0, tau = sorted[V - 1];
    for (int k = 0; k < V; ++k) {
        cum += sorted[k];
        if (cum >= top_p) { tau = sorted[k]; break; }
    }
    free(sorted);
    double kept = 0.0;
    for (int i = 0; i < V; ++i) {
        if (out[i] < tau) out[i] = 0.0;
        kept += out[i];
    }
    for (int i = 0; i < V; ++i) out[i] /= kept;
}

/* Inverse-CDF draw: the first x (ascending) with cumsum(x) > u * sum. */
int orc_sample(const double* probs, int V, double u) {
    double total = 0.0;
    for (int i = 0; i < V; ++i) total += probs[i];
    double target = u * total, cum = 0.0;
    int last = -1;
    for (int i = 0; i < V; ++i) {
        if (probs[i] > 0.0) last = i;
        cum += probs[i];
        if (cum > target && probs[i] > 0.0) return i;
    }
    return last < 0 ? 0 : last;
}

/* Verification of one round of speculative sampling (Algorithm 4).
 * p: (Kd+1) x V target rows p_0..p_Kd; q: Kd x V draft rows (row j-1 is q_j,
 * the distribution d_j was drawn from); r[j-1]: acceptance uniform of d_j;
 * ures[j-1]: resample uniform if d_j is rejected; ures[Kd]: bonus uniform.
 * Returns the correction / bonus token and writes the accepted count. */
int orc_spec_verify(const double* p, const double* q, const int* drafts, int Kd, int V,
                    const double* r, const double* ures, int* n_accepted) {
    double* res = (double*)malloc(sizeof(double) * V);
    int y = -1;
    int n = 0;
    for (int j = 1; j <= Kd; ++j) {
        const double* pj = p + (size_t)(j - 1) * V;
        const double* qj = q + (size_t)(j - 1) * V;
        int x = drafts[j - 1];
        double ratio = qj[x] > 0.0 ? pj[x] / qj[x] : INFINITY;
        double thr = ratio < 1.0 ? ratio : 1.0;
        if (r[j - 1] < thr) { n = j; continue; }
        double tot = 0.0;
        for (int i = 0; i < V; ++i) {
            double dlt = pj[i] - qj[i];
            res[i] = dlt > 0.0 ? dlt : 0.0;
            tot += res[i];
        }
        y = tot > 0.0 ? orc_sample(res, V, ures[j - 1]) : orc_sample(pj, V, ures[j - 1]);
        break;
    }
    if (y < 0) y = orc_sample(p + (size_t)Kd * V, V, ures[Kd]);
    free(res);
    *n_accepted = n;
    return y;
}

/* Batched form of orc_spec_verify for distribution tests: `trials` rounds
 * sharing p and q, each with its own drafts, r and ures; writes
 * out[2t] = n and out[2t + 1] = y. */
void orc_spec_verify_batch(const double* p, const double* q, int Kd, int V, int trials,
                           const int* drafts, const double* r, const double* ures, int* out) {
    #pragma omp parallel for schedule(static)
    for (int t = 0; t < trials; ++t) {
        int n;
        int y = orc_spec_verify(p, q, drafts + (size_t)t * Kd, Kd, V, r + (size_t)t * Kd,
                                ures + (size_t)t * (Kd + 1), &n);
        out[(size_t)t * 2 + 0] = n;
        out[(size_t)t * 2 + 1] = y;
    }
}

/* ------------------------------------------------------------------------ */
/* adaptive draft exit (Sec. 3.4, Eqs. 2-4)                                  */
/* ------------------------------------------------------------------------ */

typedef struct {
    int on; /* 0: Algorithm 2 / 4 without exit */
    double gamma0, alpha, eps, beta1, beta2;
} orc_exit_params;

typedef struct {
    double gamma, ar;
    int e; /* updates done */
} orc_exit_state;

/* After the verification of round e, with AR_e = accepted / drafted:
 *   AR <- beta1 AR + (1 - beta1) AR_e            (beta1 = 0 at e = 1)
 *   gamma~ = gamma + eps if AR <= alpha, else gamma - eps
 *   gamma <- beta2 gamma + (1 - beta2) gamma~ */
void orc_exit_update(orc_exit_state* s, const orc_exit_params* p, double ar_e) {
    double b1 = s->e == 0 ? 0.0 : p->beta1;
    s->ar = b1 * s->ar + (1.0 - b1) * ar_e;
    double gt = s->ar <= p->alpha ? s->gamma + p->eps : s->gamma - p->eps;
    s->gamma = p->beta2 * s->gamma + (1.0 - p->beta2) * gt;
    s->e++;
}

/* Largest probability of softmax(logits): 1 / sum_x exp(l_x - max l). */
double orc_softmax_max(const double* logits, int V) {
    double mx = logits[0];
    for (int i = 1; i < V; ++i)
        if (logits[i] > mx) mx = logits[i];
    double s = 0.0;
    for (int i = 0; i < V; ++i) s += exp(logits[i] - mx);
    return 1.0 / s;
}

/* ------------------------------------------------------------------------ */
/* decoding loops: Algorithm 1 (K = 0), Algorithm 2 / Algorithm 4 (K > 0)    */
/* ------------------------------------------------------------------------ */

/* Runs prompt[0..P-2] through the full model (len = P-1 committed positions). */
int orc_prefill(orc_model* m, const int* prompt, int n_prompt) {
    if (n_prompt < 1 || n_prompt > m->c.max_seq) return -1;
    for (int p = 0; p + 1 < n_prompt; ++p) orc_forward(m, prompt[p], p, NULL, NULL);
    return 0;
}

/* mode 0 greedy, 1 sampling.  mask: 2*n_layers bytes (the draft's z).
 * out_tokens: n_new emitted tokens.  Optional: draft_logits_out /
 * verify_logits_out receive the first round's K_eff x V draft logits and
 * (K_eff+1) x V verification logits; ex (NULL or ex->on == 0: no exit) turns
 * on the adaptive draft exit, and then keff_out / gamma_out (n_new entries
 * each, may be NULL) receive every round's draft count and its gamma after
 * the round's update.  Returns 0 or a negative error. */
int orc_generate_ex(orc_model* m, const int* prompt, int n_prompt, int n_new, int K, int mode,
                    uint64_t seed, double temperature, double top_p, const uint8_t* mask,
                    int* out_tokens, orc_stats* stats, double* draft_logits_out,
                    double* verify_logits_out, const orc_exit_params* ex, int* keff_out,
                    double* gamma_out) {
    const orc_config* c = &m->c;
    int V = c->vocab;
    if (n_new < 0 || K < 0 || K > 32 || n_prompt < 1) return -1;
    if (n_prompt + n_new + K + 1 > c->max_seq) return -2;
    if (mode == 1 && !(temperature > 0.0)) return -1;
    if (orc_prefill(m, prompt, n_prompt)) return -1;
    orc_stats st;
    memset(&st, 0, sizeof(st));
    double* logits = (double*)malloc(sizeof(double) * V);
    double* P = (double*)malloc(sizeof(double) * (size_t)(K + 1) * V);
    double* Q = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1) * V);
    int drafts[33];
    int len = n_prompt - 1;
    int x_last = prompt[n_prompt - 1];
    int emitted = 0;
    int first_round = 1;
    const int exit_on = ex && ex->on;
    orc_exit_state es = {exit_on ? ex->gamma0 : 0.0, 0.0, 0};
    while (emitted < n_new) {
        int remaining = n_new - emitted;
        int Kd = K < remaining - 1 ? K : remaining - 1;
        /* drafting stage: the masked model, one token at a time */
        for (int j = 1; j <= Kd; ++j) {
            int tin = j == 1 ? x_last : drafts[j - 2];
            orc_forward(m, tin, len + j - 1, mask, logits);
            if (first_round && draft_logits_out)
                memcpy(draft_logits_out + (size_t)(j - 1) * V, logits, sizeof(double) * V);
            double conf;
            if (mode == 0) {
                drafts[j - 1] = orc_argmax(logits, V);
                conf = exit_on ? orc_softmax_max(logits, V) : 1.0;
            } else {
                double* qj = Q + (size_t)(j - 1) * V;
                orc_nucleus_probs(logits, V, temperature, top_p, qj);
                drafts[j - 1] = orc_sample(qj, V, orc_uniform(seed, len + j, 0));
                conf = exit_on ? qj[orc_argmax(qj, V)] : 1.0;
            }
            if (exit_on && conf < es.gamma) { /* draft exit: d_j is the last draft */
                Kd = j;
                break;
            }
        }
        /* verification stage: the full model on [x_last, d_1..d_Kd] */
        for (int r = 0; r <= Kd; ++r) {
            int tin = r == 0 ? x_last : drafts[r - 1];
            double* pr = P + (size_t)r * V;
            orc_forward(m, tin, len + r, NULL, pr);
            if (first_round && verify_logits_out)
                memcpy(verify_logits_out + (size_t)r * V, pr, sizeof(double) * V);
        }
        int n = 0, y;
        if (mode == 0) {
            while (n < Kd && drafts[n] == orc_argmax(P + (size_t)n * V, V)) ++n;
            y = orc_argmax(P + (size_t)n * V, V);
        } else {
            for (int r = 0; r <= Kd; ++r) {
                double* pr = P + (size_t)r * V;
                memcpy(logits, pr, sizeof(double) * V);
                orc_nucleus_probs(logits, V, temperature, top_p, pr);
            }
            double rr[33], uu[34];
            for (int j = 1; j <= Kd; ++j) {
                rr[j - 1] = orc_uniform(seed, len + j, 1);
                uu[j - 1] = orc_uniform(seed, len + j, 2);
            }
            uu[Kd] = orc_uniform(seed, len + Kd + 1, 2);
            y = orc_spec_verify(P, Q, drafts, Kd, V, rr, uu, &n);
        }
        for (int j = 0; j < n; ++j) out_tokens[emitted++] = drafts[j];
        out_tokens[emitted++] = y;
        if (exit_on && Kd > 0) orc_exit_update(&es, ex, (double)n / Kd);
        if (keff_out) keff_out[st.rounds] = Kd;
        if (gamma_out) gamma_out[st.rounds] = es.gamma;
        st.rounds++;
        st.drafted += Kd;
        st.accepted += n;
        st.hist[n]++;
        len += n + 1;
        x_last = y;
        first_round = 0;
    }
    st.emitted = emitted;
    if (stats) *stats = st;
    free(logits); free(P); free(Q);
    return 0;
}

/* Algorithm 1 / 2 / 4 without draft exit. */
int orc_generate(orc_model* m, const int* prompt, int n_prompt, int n_new, int K, int mode,
                 uint64_t seed, double temperature, double top_p, const uint8_t* mask,
                 int* out_tokens, orc_stats* stats, double* draft_logits_out,
                 double* verify_logits_out) {
    return orc_generate_ex(m, prompt, n_prompt, n_new, K, mode, seed, temperature, top_p, mask, out_tokens,
                           stats, draft_logits_out, verify_logits_out, NULL, NULL, NULL);
}
