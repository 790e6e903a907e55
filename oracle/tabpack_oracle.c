/*
 * tabpack_oracle.c -- plain CPU fp64 oracle of the TabPack training step.
 *
 * TEST INFRASTRUCTURE ONLY (see tabpack_oracle.h).  Loops are written in the
 * order the method states them, one member at a time; the only parallelism is
 * an OpenMP loop over independent members.  Nothing here is blocked, fused or
 * reordered for speed.
 */
#include "tabpack_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Philox4x32-10, from Salmon, Moraes, Dror and Shaw, "Parallel random        */
/* numbers: as easy as 1, 2, 3" (SC'11).  One round maps the counter          */
/* (c0, c1, c2, c3) with key (k0, k1) to                                      */
/*   (hi(M1*c2) ^ c1 ^ k0,  lo(M1*c2),  hi(M0*c0) ^ c3 ^ k1,  lo(M0*c0));     */
/* the key is advanced by the Weyl increments W0 = 2^32 (golden ratio - 1)    */
/* and W1 = 2^32 (sqrt(3) - 1) between rounds.                                */
/* ------------------------------------------------------------------------ */
#define ORC_PHILOX_M0 0xD2511F53u
#define ORC_PHILOX_M1 0xCD9E8D57u
#define ORC_PHILOX_W0 0x9E3779B9u
#define ORC_PHILOX_W1 0xBB67AE85u

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += ORC_PHILOX_W0;
      k1 += ORC_PHILOX_W1;
    }
    uint64_t prod0 = (uint64_t)ORC_PHILOX_M0 * (uint64_t)c0;
    uint64_t prod1 = (uint64_t)ORC_PHILOX_M1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* Word `col & 3` of the Philox block at counter (a, col >> 2, c, d). */
static uint32_t orc_philox_word(uint64_t seed, uint32_t a, uint32_t col, uint32_t c, uint32_t d) {
  uint32_t ctr[4] = {a, col >> 2, c, d};
  uint32_t key[2] = {(uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32)};
  uint32_t out[4];
  orc_philox4x32_10(ctr, key, out);
  return out[col & 3u];
}

/* Dropout (Sec. 3.3: "sampling m dropout masks with m different rates").
 * The paper does not state the generator; reading: an element is dropped iff
 * its Philox word r satisfies r < T with T = floor(p * 2^32), so the drop
 * probability is T / 2^32 and p = 0 never drops.  Counter: (row, col >> 2,
 * step, member_id << 4 | layer), word col & 3, key = seed.                   */
static uint32_t orc_drop_threshold(float p) {
  double t = floor((double)p * 4294967296.0);
  if (t < 0.0) t = 0.0;
  if (t > 4294967295.0) t = 4294967295.0;
  return (uint32_t)t;
}

int orc_dropout_keep(uint64_t seed, uint32_t member_id, uint32_t layer, uint32_t step,
                     uint32_t row, uint32_t col, float p) {
  uint32_t T = orc_drop_threshold(p);
  if (T == 0) return 1;
  uint32_t r = orc_philox_word(seed, row, col, step, (member_id << 4) | layer);
  return r >= T ? 1 : 0;
}

/* The keep mask of rows 0..B-1 and columns 0..w-1 of one hidden layer at one
 * step (out [B, w], 1 = keep): orc_dropout_keep element by element.        */
void orc_dropout_mask(uint64_t seed, uint32_t member_id, uint32_t layer, uint32_t step,
                      int32_t B, int32_t w, float p, uint8_t* out) {
  const uint32_t T = orc_drop_threshold(p);
  #pragma omp parallel for schedule(static)
  for (int32_t r = 0; r < B; ++r)
    for (int32_t c4 = 0; c4 < w; c4 += 4) {   /* one counter gives columns c4 .. c4 + 3 */
      const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
      const uint32_t ctr[4] = {(uint32_t)r, (uint32_t)c4 >> 2, step, (member_id << 4) | layer};
      uint32_t word[4];
      orc_philox4x32_10(ctr, key, word);
      for (int32_t k = 0; k < 4 && c4 + k < w; ++k)
        out[(int64_t)r * w + c4 + k] = (uint8_t)(T == 0 || word[k] >= T);
    }
}

/* bfloat16 storage rounding.  A value stored in bf16 is first an fp32 value
 * (the GPU computes in fp32), so x is rounded to fp32 and then to bf16: 8
 * significant bits, fp32 exponent range, subnormal ulp 2^-133, round to
 * nearest with ties to even at both steps.                                   */
double orc_round_bf16(double x) {
  x = (double)(float)x;
  if (x == 0.0 || isnan(x) || isinf(x)) return x;
  int e;
  frexp(x, &e);                 /* x = f * 2^e, 0.5 <= |f| < 1 */
  int ulp_exp = e - 8;
  if (ulp_exp < -133) ulp_exp = -133;
  double q = nearbyint(ldexp(x, -ulp_exp)); /* default mode: nearest, ties even */
  double r = ldexp(q, ulp_exp);
  const double bf16_max = ldexp(255.0, 120); /* (2 - 2^-7) * 2^127 */
  if (fabs(r) > bf16_max) return x > 0 ? INFINITY : -INFINITY;
  return r;
}

/* Initialisation (not stated in the paper; reading: the default of a PyTorch
 * Linear layer, U(-1/sqrt(fan_in), 1/sqrt(fan_in)) for weights and biases).
 * Element e of a layer (weights row-major, then biases) draws the Philox word
 * at counter (e >> 2, 0, 0, 1 << 28 | member_id << 4 | layer), word e & 3;
 * u = ((r >> 8) + 1/2) 2^-24 and the value is (2u - 1) / sqrt(fan_in),
 * rounded to fp32 (the GPU keeps fp32 master weights).                       */
double orc_init_value(uint64_t seed, uint32_t member_id, uint32_t layer, uint32_t e, int32_t fan_in) {
  uint32_t r = orc_philox_word(seed, e >> 2, e & 3u, 0u, (1u << 28) | (member_id << 4) | layer);
  double u = ((double)(r >> 8) + 0.5) * ldexp(1.0, -24);
  double bound = 1.0 / sqrt((double)fan_in);
  return (double)(float)((2.0 * u - 1.0) * bound);
}

/* ------------------------------------------------------------------------ */
/* Pack state                                                                 */
/* ------------------------------------------------------------------------ */
typedef struct {
  int32_t L, w, id;
  float p, lr, wd;
  int64_t t;          /* optimizer steps taken by this member */
  int32_t active;
  int32_t *in_dim, *out_dim;                 /* [L + 1]; layer L is the head */
  double **W, **b, **gW, **gb, **mW, **vW, **mb, **vb;
  /* last step */
  int32_t B;
  double **Hin;       /* [L + 1]: input of layer l, B x in_dim[l]          */
  double **Z;         /* [L]: pre-activations, B x w                       */
  uint8_t **keep;     /* [L]: dropout keep decisions, B x w                */
  double *logits;     /* B x d_out                                          */
  double margin;      /* min |Z| / rms(Z) of the last forward               */
  double lr_muon;     /* Muon learning rate (when the pack uses Muon)       */
  double **dir;       /* [L]: the last Muon direction O of each hidden W    */
  /* periodic feature embeddings (App. "Feature Embeddings"; d_emb 0: none):
   * emb = [w: d_in x (d_emb - 1)] [b: d_in x (d_emb - 1)] [alpha: d_in x
   * d_emb] [beta: d_in x d_emb]; feature j becomes
   * alpha_j * [x_j, cos(w_j x_j + b_j)] + beta_j, layer 1 reads the d_in
   * embeddings side by side (in_dim[0] = d_in d_emb).                      */
  int32_t d_emb;
  int64_t n_emb;
  double *emb, *gemb, *memb, *vemb;
  double *xraw;       /* the last batch's inputs, B x d_in                  */
} orc_member;

struct orc_pack {
  orc_config cfg;
  orc_member* mem;
  int32_t muon;       /* 1: hidden-layer weights take Muon steps (Sec. 3.4) */
  double momentum;    /* Muon momentum mu                                   */
  int32_t ns_steps;   /* Newton-Schulz iterations                           */
};

static double* orc_zeros(int64_t n) { return (double*)calloc((size_t)(n > 0 ? n : 1), sizeof(double)); }

/* Column-major copy t[c * rows + r] = a[r * cols + c] of a row-major
 * [rows, cols] matrix: a sum over r then reads consecutive memory.  Only the
 * memory layout changes; every product and the order of every sum stay those
 * of the plain loops over the row-major matrix.                              */
static double* orc_transpose(const double* a, int64_t rows, int64_t cols) {
  double* t = orc_zeros(rows * cols);
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t c = 0; c < cols; ++c) t[c * rows + r] = a[r * cols + c];
  return t;
}

static void orc_free_cache(orc_member* M) {
  free(M->xraw);
  M->xraw = NULL;
  if (M->Hin) for (int l = 0; l <= M->L; ++l) free(M->Hin[l]);
  if (M->Z) for (int l = 0; l < M->L; ++l) free(M->Z[l]);
  if (M->keep) for (int l = 0; l < M->L; ++l) free(M->keep[l]);
  free(M->Hin); free(M->Z); free(M->keep); free(M->logits);
  M->Hin = NULL; M->Z = NULL; M->keep = NULL; M->logits = NULL; M->B = 0;
}

static void orc_alloc_cache(orc_member* M, int32_t B, int32_t d_out) {
  if (M->B == B && M->Hin) return;
  orc_free_cache(M);
  M->B = B;
  M->Hin = (double**)calloc((size_t)M->L + 1, sizeof(double*));
  M->Z = (double**)calloc((size_t)M->L + 1, sizeof(double*));
  M->keep = (uint8_t**)calloc((size_t)M->L + 1, sizeof(uint8_t*));
  for (int l = 0; l <= M->L; ++l) M->Hin[l] = orc_zeros((int64_t)B * M->in_dim[l]);
  for (int l = 0; l < M->L; ++l) {
    M->Z[l] = orc_zeros((int64_t)B * M->w);
    M->keep[l] = (uint8_t*)calloc((size_t)B * M->w + 1, 1);
  }
  M->logits = orc_zeros((int64_t)B * d_out);
  M->xraw = orc_zeros((int64_t)B * (M->d_emb ? M->in_dim[0] / M->d_emb : M->in_dim[0]));
}

void orc_destroy(orc_pack* h) {
  if (!h) return;
  for (int i = 0; i < h->cfg.m; ++i) {
    orc_member* M = &h->mem[i];
    orc_free_cache(M);
    for (int l = 0; l <= M->L; ++l) {
      free(M->W[l]); free(M->b[l]); free(M->gW[l]); free(M->gb[l]);
      free(M->mW[l]); free(M->vW[l]); free(M->mb[l]); free(M->vb[l]);
    }
    free(M->W); free(M->b); free(M->gW); free(M->gb);
    free(M->mW); free(M->vW); free(M->mb); free(M->vb);
    if (M->dir) {
      for (int l = 0; l < M->L; ++l) free(M->dir[l]);
      free(M->dir);
    }
    free(M->emb); free(M->gemb); free(M->memb); free(M->vemb);
    free(M->in_dim); free(M->out_dim);
  }
  free(h->mem);
  free(h);
}

orc_pack* orc_create_emb(const orc_config* cfg, const int32_t* depth, const int32_t* width,
                         const float* dropout, const float* lr, const float* wd,
                         const int32_t* member_id, const int32_t* d_emb, const double* freq) {
  if (!cfg || cfg->m <= 0 || cfg->d_in <= 0 || cfg->d_out <= 0) return NULL;
  if (cfg->task < 0 || cfg->task > 2) return NULL;
  if (cfg->task != ORC_MULTICLASS && cfg->d_out != 1) return NULL;
  if (cfg->task == ORC_MULTICLASS && cfg->d_out < 2) return NULL;
  for (int i = 0; i < cfg->m; ++i) {
    if (depth[i] < 1 || depth[i] > 14 || width[i] < 1) return NULL;
    if (!(dropout[i] >= 0.0f && dropout[i] < 1.0f)) return NULL;
    if (!(lr[i] >= 0.0f) || !(wd[i] >= 0.0f)) return NULL;
  }
  orc_pack* h = (orc_pack*)calloc(1, sizeof(orc_pack));
  h->cfg = *cfg;
  h->mem = (orc_member*)calloc((size_t)cfg->m, sizeof(orc_member));
  for (int i = 0; i < cfg->m; ++i) {
    orc_member* M = &h->mem[i];
    M->L = depth[i];
    M->w = width[i];
    M->p = dropout[i];
    M->lr = lr[i];
    M->wd = wd[i];
    M->id = member_id ? member_id[i] : i;
    M->active = 1;
    M->in_dim = (int32_t*)calloc((size_t)M->L + 1, sizeof(int32_t));
    M->out_dim = (int32_t*)calloc((size_t)M->L + 1, sizeof(int32_t));
    M->d_emb = d_emb ? d_emb[i] : 0;
    for (int l = 0; l <= M->L; ++l) {
      M->in_dim[l] = (l == 0) ? cfg->d_in * (M->d_emb ? M->d_emb : 1) : M->w;
      M->out_dim[l] = (l == M->L) ? cfg->d_out : M->w;
    }
    if (M->d_emb > 0) {  /* frequencies from the caller, phases and scales zero */
      M->n_emb = (int64_t)cfg->d_in * (4 * M->d_emb - 2);
      M->emb = orc_zeros(M->n_emb);
      M->gemb = orc_zeros(M->n_emb);
      M->memb = orc_zeros(M->n_emb);
      M->vemb = orc_zeros(M->n_emb);
      const int64_t nf = (int64_t)cfg->d_in * (M->d_emb - 1);
      for (int64_t e = 0; e < nf; ++e) M->emb[e] = *freq++;
    }
    int nl = M->L + 1;
    M->W = (double**)calloc((size_t)nl, sizeof(double*));
    M->b = (double**)calloc((size_t)nl, sizeof(double*));
    M->gW = (double**)calloc((size_t)nl, sizeof(double*));
    M->gb = (double**)calloc((size_t)nl, sizeof(double*));
    M->mW = (double**)calloc((size_t)nl, sizeof(double*));
    M->vW = (double**)calloc((size_t)nl, sizeof(double*));
    M->mb = (double**)calloc((size_t)nl, sizeof(double*));
    M->vb = (double**)calloc((size_t)nl, sizeof(double*));
    for (int l = 0; l <= M->L; ++l) {
      int64_t nw = (int64_t)M->out_dim[l] * M->in_dim[l], nb = M->out_dim[l];
      M->W[l] = orc_zeros(nw); M->b[l] = orc_zeros(nb);
      M->gW[l] = orc_zeros(nw); M->gb[l] = orc_zeros(nb);
      M->mW[l] = orc_zeros(nw); M->vW[l] = orc_zeros(nw);
      M->mb[l] = orc_zeros(nb); M->vb[l] = orc_zeros(nb);
      for (int64_t e = 0; e < nw; ++e)
        M->W[l][e] = orc_init_value(cfg->seed, (uint32_t)M->id, (uint32_t)l, (uint32_t)e, M->in_dim[l]);
      for (int64_t e = 0; e < nb; ++e)
        M->b[l][e] = orc_init_value(cfg->seed, (uint32_t)M->id, (uint32_t)l, (uint32_t)(nw + e), M->in_dim[l]);
    }
    M->margin = INFINITY;
  }
  return h;
}

orc_pack* orc_create(const orc_config* cfg, const int32_t* depth, const int32_t* width,
                     const float* dropout, const float* lr, const float* wd,
                     const int32_t* member_id) {
  return orc_create_emb(cfg, depth, width, dropout, lr, wd, member_id, NULL, NULL);
}

int orc_get_emb(const orc_pack* h, int32_t member, int32_t grads, double* out) {
  if (!h || member < 0 || member >= h->cfg.m || !h->mem[member].d_emb) return 1;
  const orc_member* M = &h->mem[member];
  memcpy(out, grads ? M->gemb : M->emb, sizeof(double) * (size_t)M->n_emb);
  return 0;
}

int orc_set_emb(orc_pack* h, int32_t member, const double* in) {
  if (!h || member < 0 || member >= h->cfg.m || !h->mem[member].d_emb) return 1;
  orc_member* M = &h->mem[member];
  memcpy(M->emb, in, sizeof(double) * (size_t)M->n_emb);
  return 0;
}

/* value as stored between kernels: bf16 in bf16 mode, exact otherwise */
static double orc_st(const orc_pack* h, double x) { return h->cfg.bf16_storage ? orc_round_bf16(x) : x; }

/* ------------------------------------------------------------------------ */
/* Forward (Sec. 3.3): H_0 = x; for each of the member's L blocks             */
/* Z = H W^T + b, H = Dropout_p(ReLU(Z)) with inverted scaling 1 / (1 - p);   */
/* logits = H_L W_head^T + b_head.  Only the member's own L layers are        */
/* applied (shallower members skip the deeper layers).                        */
/* ------------------------------------------------------------------------ */
static void orc_member_forward(const orc_pack* h, orc_member* M, const float* X, const int32_t* idx,
                               int32_t B, uint32_t step, int train) {
  const int d_in = h->cfg.d_in, d_out = h->cfg.d_out;
  for (int b = 0; b < B; ++b) {
    int64_t row = idx ? idx[b] : b;
    for (int k = 0; k < d_in; ++k) M->xraw[(int64_t)b * d_in + k] = (double)X[row * d_in + k];
  }
  if (M->d_emb == 0) {
    for (int64_t e = 0; e < (int64_t)B * d_in; ++e) M->Hin[0][e] = orc_st(h, M->xraw[e]);
  } else {  /* periodic embeddings */
    const int d = M->d_emb, in0 = d_in * d;
    const double *ew = M->emb, *eb = ew + (int64_t)d_in * (d - 1), *ea = eb + (int64_t)d_in * (d - 1),
                 *ebt = ea + (int64_t)d_in * d;
    for (int b = 0; b < B; ++b)
      for (int j = 0; j < d_in; ++j) {
        const double x = M->xraw[(int64_t)b * d_in + j];
        for (int k = 0; k < d; ++k) {
          const double f = k == 0 ? x : cos(ew[(int64_t)j * (d - 1) + k - 1] * x + eb[(int64_t)j * (d - 1) + k - 1]);
          M->Hin[0][(int64_t)b * in0 + j * d + k] =
              orc_st(h, ea[(int64_t)j * d + k] * f + ebt[(int64_t)j * d + k]);
        }
      }
  }
  double margin = INFINITY;
  for (int l = 0; l < M->L; ++l) {
    const int in = M->in_dim[l], w = M->w;
    /* the matrix-product operand: the bf16 weight copy in bf16 mode */
    double* Weff = orc_zeros((int64_t)w * in);
    for (int64_t e = 0; e < (int64_t)w * in; ++e) Weff[e] = orc_st(h, M->W[l][e]);
    double ss = 0.0;
    for (int b = 0; b < B; ++b) {
      for (int j = 0; j < w; ++j) {
        double z = 0.0;
        for (int k = 0; k < in; ++k) z += M->Hin[l][(int64_t)b * in + k] * Weff[(int64_t)j * in + k];
        z += M->b[l][j];
        M->Z[l][(int64_t)b * w + j] = z;
        ss += z * z;
        double a = z > 0.0 ? z : 0.0;
        int keep = train ? orc_dropout_keep(h->cfg.seed, (uint32_t)M->id, (uint32_t)l, step,
                                            (uint32_t)b, (uint32_t)j, M->p)
                         : 1;
        M->keep[l][(int64_t)b * w + j] = (uint8_t)keep;
        double hval = keep ? (train ? a / (1.0 - (double)M->p) : a) : 0.0;
        M->Hin[l + 1][(int64_t)b * w + j] = orc_st(h, hval);
      }
    }
    double rms = sqrt(ss / ((double)B * w));
    if (rms > 0.0)
      for (int64_t e = 0; e < (int64_t)B * w; ++e) {
        double r = fabs(M->Z[l][e]) / rms;
        if (r < margin) margin = r;
      }
    free(Weff);
  }
  M->margin = margin;
  const int L = M->L, w = M->w;
  for (int b = 0; b < B; ++b)
    for (int c = 0; c < d_out; ++c) {
      double z = 0.0;
      for (int j = 0; j < w; ++j) z += M->Hin[L][(int64_t)b * w + j] * M->W[L][(int64_t)c * w + j];
      M->logits[(int64_t)b * d_out + c] = z + M->b[L][c];
    }
}

/* Per-row loss and d(loss_row)/d(logits) (Appendix F.1: cross-entropy for
 * classification, MSE for regression; binary tasks use one logit with the
 * logistic loss -- a reading, the paper does not say how binary heads look). */
static double orc_row_loss(int task, int d_out, const double* z, int32_t yi, float yf, double* dz) {
  if (task == ORC_MULTICLASS) {
    double mx = z[0];
    for (int c = 1; c < d_out; ++c) if (z[c] > mx) mx = z[c];
    double s = 0.0;
    for (int c = 0; c < d_out; ++c) s += exp(z[c] - mx);
    double lse = mx + log(s);
    for (int c = 0; c < d_out; ++c) dz[c] = exp(z[c] - lse) - (c == yi ? 1.0 : 0.0);
    return lse - z[yi];
  } else if (task == ORC_BINARY) {
    double x = z[0], y = (double)yi;
    double sig = 1.0 / (1.0 + exp(-x));
    dz[0] = sig - y;
    return (x > 0.0 ? x : 0.0) - x * y + log1p(exp(-fabs(x)));
  } else {
    double d = z[0] - (double)yf;
    dz[0] = 2.0 * d;
    return d * d;
  }
}

/* Loss (Sec. 3.6: members are trained independently; losses are aggregated,
 * so each member's gradient is its own loss's gradient) and the exact
 * backward pass.  Returns the member's mean loss over the B rows.            */
static double orc_member_backward(const orc_pack* h, orc_member* M, const int32_t* idx,
                                  const int32_t* y_int, const float* y_float, int32_t B) {
  const int d_out = h->cfg.d_out, L = M->L, w = M->w;
  double* dlog = orc_zeros((int64_t)B * d_out);
  double loss = 0.0;
  for (int b = 0; b < B; ++b) {
    int64_t row = idx ? idx[b] : b;
    int32_t yi = y_int ? y_int[row] : 0;
    float yf = y_float ? y_float[row] : 0.0f;
    loss += orc_row_loss(h->cfg.task, d_out, &M->logits[(int64_t)b * d_out], yi, yf, &dlog[(int64_t)b * d_out]);
  }
  loss /= (double)B;
  for (int64_t e = 0; e < (int64_t)B * d_out; ++e) dlog[e] /= (double)B;

  /* head: dW_h[c, j] = sum_b dlogits[b, c] H_L[b, j] (b increasing) */
  double* dlogT = orc_transpose(dlog, B, d_out);
  double* HT = orc_transpose(M->Hin[L], B, w);
  for (int c = 0; c < d_out; ++c) {
    for (int j = 0; j < w; ++j) {
      double g = 0.0;
      for (int b = 0; b < B; ++b) g += dlogT[(int64_t)c * B + b] * HT[(int64_t)j * B + b];
      M->gW[L][(int64_t)c * w + j] = g;
    }
    double gb = 0.0;
    for (int b = 0; b < B; ++b) gb += dlog[(int64_t)b * d_out + c];
    M->gb[L][c] = gb;
  }
  free(dlogT);
  free(HT);
  double* dH = orc_zeros((int64_t)B * w);
  for (int b = 0; b < B; ++b)
    for (int j = 0; j < w; ++j) {
      double s = 0.0;
      for (int c = 0; c < d_out; ++c) s += dlog[(int64_t)b * d_out + c] * M->W[L][(int64_t)c * w + j];
      dH[(int64_t)b * w + j] = s;
    }
  free(dlog);

  /* hidden blocks, last to first */
  for (int l = L - 1; l >= 0; --l) {
    const int in = M->in_dim[l];
    double* dZ = orc_zeros((int64_t)B * w);
    for (int64_t e = 0; e < (int64_t)B * w; ++e) {
      double g = (M->keep[l][e] && M->Z[l][e] > 0.0) ? dH[e] / (1.0 - (double)M->p) : 0.0;
      dZ[e] = orc_st(h, g);
    }
    /* dW[j, k] = sum_b dZ[b, j] H_l[b, k], db[j] = sum_b dZ[b, j] (b increasing) */
    double* dZT = orc_transpose(dZ, B, w);
    double* HT_l = orc_transpose(M->Hin[l], B, in);
    for (int j = 0; j < w; ++j) {
      for (int k = 0; k < in; ++k) {
        double g = 0.0;
        for (int b = 0; b < B; ++b) g += dZT[(int64_t)j * B + b] * HT_l[(int64_t)k * B + b];
        M->gW[l][(int64_t)j * in + k] = g;
      }
      double gb = 0.0;
      for (int b = 0; b < B; ++b) gb += dZT[(int64_t)j * B + b];
      M->gb[l][j] = gb;
    }
    free(dZT);
    free(HT_l);
    free(dH);
    dH = NULL;
    if (l == 0 && M->d_emb > 0) {
      /* dE[b, q] = sum_j dZ[b, j] W_0[j, q] (W as stored; dE stored like dZ),
       * then the embedding parameters' gradients, rows b increasing */
      const int d = M->d_emb, d_in = h->cfg.d_in;
      double* dE = orc_zeros((int64_t)B * in);
      for (int b = 0; b < B; ++b)
        for (int q = 0; q < in; ++q) {
          double s = 0.0;
          for (int j = 0; j < w; ++j) s += dZ[(int64_t)b * w + j] * orc_st(h, M->W[0][(int64_t)j * in + q]);
          dE[(int64_t)b * in + q] = orc_st(h, s);
        }
      const double *ew = M->emb, *eb = ew + (int64_t)d_in * (d - 1), *ea = eb + (int64_t)d_in * (d - 1);
      double *gw = M->gemb, *gbb = gw + (int64_t)d_in * (d - 1), *ga = gbb + (int64_t)d_in * (d - 1),
             *gbt = ga + (int64_t)d_in * d;
      for (int j = 0; j < d_in; ++j)
        for (int k = 0; k < d; ++k) {
          double sa = 0.0, sbt = 0.0, sw = 0.0, sb = 0.0;
          const double a = ea[(int64_t)j * d + k];
          for (int b = 0; b < B; ++b) {
            const double g = dE[(int64_t)b * in + j * d + k], x = M->xraw[(int64_t)b * d_in + j];
            sbt += g;
            if (k == 0) {
              sa += g * x;
            } else {
              const double u = ew[(int64_t)j * (d - 1) + k - 1] * x + eb[(int64_t)j * (d - 1) + k - 1];
              sa += g * cos(u);
              sw += g * a * (-sin(u)) * x;
              sb += g * a * (-sin(u));
            }
          }
          ga[(int64_t)j * d + k] = sa;
          gbt[(int64_t)j * d + k] = sbt;
          if (k > 0) {
            gw[(int64_t)j * (d - 1) + k - 1] = sw;
            gbb[(int64_t)j * (d - 1) + k - 1] = sb;
          }
        }
      free(dE);
    }
    if (l > 0) {
      /* dH_l[b, k] = sum_j dZ[b, j] W_l[j, k] (j increasing), W as stored */
      double* WT = orc_zeros((int64_t)in * w);
      for (int j = 0; j < w; ++j)
        for (int k = 0; k < in; ++k) WT[(int64_t)k * w + j] = orc_st(h, M->W[l][(int64_t)j * in + k]);
      dH = orc_zeros((int64_t)B * in);
      for (int b = 0; b < B; ++b)
        for (int k = 0; k < in; ++k) {
          double s = 0.0;
          for (int j = 0; j < w; ++j) s += dZ[(int64_t)b * w + j] * WT[(int64_t)k * w + j];
          dH[(int64_t)b * in + k] = s;
        }
      free(WT);
    }
    free(dZ);
  }
  free(dH);
  return loss;
}

/* AdamW (Loshchilov & Hutter; Sec. 3.4 packs one optimizer per member with
 * its own learning rate and weight decay).  PyTorch semantics: decoupled
 * decay p <- p - lr wd p, then the bias-corrected Adam step.                 */
void orc_adamw_apply(double* p, double* m, double* v, const double* g, int64_t n, int64_t t, double lr,
                     double wd, double b1, double b2, double eps) {
  const double bc1 = 1.0 - pow(b1, (double)t);
  const double bc2 = 1.0 - pow(b2, (double)t);
  for (int64_t e = 0; e < n; ++e) {
    p[e] = p[e] - lr * wd * p[e];
    m[e] = b1 * m[e] + (1.0 - b1) * g[e];
    v[e] = b2 * v[e] + (1.0 - b2) * g[e] * g[e];
    double mhat = m[e] / bc1;
    double vhat = v[e] / bc2;
    p[e] = p[e] - lr * mhat / (sqrt(vhat) + eps);
  }
}

static void orc_adamw(const orc_pack* h, const orc_member* M, double* p, double* m, double* v,
                      const double* g, int64_t n, int is_bias) {
  const double wd = (is_bias && !h->cfg.wd_on_bias) ? 0.0 : (double)M->wd;
  orc_adamw_apply(p, m, v, g, n, M->t, (double)M->lr, wd, h->cfg.beta1, h->cfg.beta2, h->cfg.eps);
}

/* ------------------------------------------------------------------------ */
/* Muon (Sec. 3.4 and App. F.1: Muon for the weight matrices of the hidden  */
/* layers, AdamW for biases and the head), after Jordan et al. (2024):       */
/*   M <- mu M + (1 - mu) G;  U = (1 - mu) G + mu M (Nesterov);              */
/*   X = U / max(||U||_F, 1e-7), taken transposed when U has more rows than  */
/*   columns;                                                                */
/*   ns_steps times: A = X X^T, Bm = b A + c A A, X = a X + Bm X with        */
/*   (a, b, c) = (3.4445, -4.7750, 2.0315);  O = X (transposed back);        */
/*   W <- W - lr wd W;  W <- W - lr max(1, rows / cols)^(1/2) O.             */
/* In bf16-storage mode X, A and Bm are rounded to bf16 where the GPU       */
/* stores them.                                                              */
/* ------------------------------------------------------------------------ */
static const double ORC_NS_A = 3.4445, ORC_NS_B = -4.7750, ORC_NS_C = 2.0315;

/* The orthogonalized direction O [rows, cols] of U [rows, cols].            */
void orc_newton_schulz(const double* U, int32_t rows, int32_t cols, int32_t steps, int32_t bf16, double* O) {
  const int tr = rows > cols;
  const int r = tr ? cols : rows, c = tr ? rows : cols;
  double* X = orc_zeros((int64_t)r * c);
  double* A = orc_zeros((int64_t)r * r);
  double* Bm = orc_zeros((int64_t)r * r);
  double* Xn = orc_zeros((int64_t)r * c);
  double nrm = 0.0;
  for (int64_t e = 0; e < (int64_t)rows * cols; ++e) nrm += U[e] * U[e];
  nrm = sqrt(nrm);
  if (nrm < 1e-7) nrm = 1e-7;
  for (int i = 0; i < rows; ++i)
    for (int j = 0; j < cols; ++j) {
      const double x = U[(int64_t)i * cols + j] / nrm;
      X[tr ? (int64_t)j * c + i : (int64_t)i * c + j] = bf16 ? orc_round_bf16(x) : x;
    }
  for (int it = 0; it < steps; ++it) {
    for (int i = 0; i < r; ++i)          /* A = X X^T */
      for (int j = 0; j < r; ++j) {
        double s = 0.0;
        for (int k = 0; k < c; ++k) s += X[(int64_t)i * c + k] * X[(int64_t)j * c + k];
        A[(int64_t)i * r + j] = bf16 ? orc_round_bf16(s) : s;
      }
    for (int i = 0; i < r; ++i)          /* Bm = b A + c A A */
      for (int j = 0; j < r; ++j) {
        double s = 0.0;
        for (int k = 0; k < r; ++k) s += A[(int64_t)i * r + k] * A[(int64_t)k * r + j];
        const double v = ORC_NS_B * A[(int64_t)i * r + j] + ORC_NS_C * s;
        Bm[(int64_t)i * r + j] = bf16 ? orc_round_bf16(v) : v;
      }
    for (int i = 0; i < r; ++i)          /* X = a X + Bm X */
      for (int j = 0; j < c; ++j) {
        double s = 0.0;
        for (int k = 0; k < r; ++k) s += Bm[(int64_t)i * r + k] * X[(int64_t)k * c + j];
        const double v = ORC_NS_A * X[(int64_t)i * c + j] + s;
        Xn[(int64_t)i * c + j] = bf16 ? orc_round_bf16(v) : v;
      }
    double* t = X;
    X = Xn;
    Xn = t;
  }
  for (int i = 0; i < rows; ++i)
    for (int j = 0; j < cols; ++j) O[(int64_t)i * cols + j] = X[tr ? (int64_t)j * c + i : (int64_t)i * c + j];
  free(X); free(A); free(Bm); free(Xn);
}

static void orc_muon(const orc_pack* h, orc_member* M, int l) {
  const int rows = M->out_dim[l], cols = M->in_dim[l];
  const int64_t n = (int64_t)rows * cols;
  double* U = orc_zeros(n);
  const double mu = h->momentum;
  for (int64_t e = 0; e < n; ++e) {
    M->mW[l][e] = mu * M->mW[l][e] + (1.0 - mu) * M->gW[l][e];
    U[e] = (1.0 - mu) * M->gW[l][e] + mu * M->mW[l][e];
  }
  if (!M->dir[l]) M->dir[l] = orc_zeros(n);
  orc_newton_schulz(U, rows, cols, h->ns_steps, h->cfg.bf16_storage, M->dir[l]);
  const double lr = M->lr_muon, wd = (double)M->wd;
  const double scale = sqrt(rows > cols ? (double)rows / (double)cols : 1.0);
  for (int64_t e = 0; e < n; ++e) {
    M->W[l][e] = M->W[l][e] - lr * wd * M->W[l][e];
    M->W[l][e] = M->W[l][e] - lr * scale * M->dir[l][e];
  }
  free(U);
}

int orc_set_muon(orc_pack* h, const double* lr_muon, double momentum, int32_t ns_steps) {
  if (!h || !lr_muon || !(momentum >= 0.0 && momentum < 1.0) || ns_steps < 1) return 1;
  for (int i = 0; i < h->cfg.m; ++i) if (!(lr_muon[i] >= 0.0)) return 1;
  h->muon = 1;
  h->momentum = momentum;
  h->ns_steps = ns_steps;
  for (int i = 0; i < h->cfg.m; ++i) {
    orc_member* M = &h->mem[i];
    M->lr_muon = lr_muon[i];
    if (!M->dir) M->dir = (double**)calloc((size_t)M->L, sizeof(double*));
  }
  return 0;
}

int orc_get_muon_dir(const orc_pack* h, int32_t member, int32_t layer, double* out) {
  if (!h || !h->muon || member < 0 || member >= h->cfg.m) return 1;
  const orc_member* M = &h->mem[member];
  if (layer < 0 || layer >= M->L || !M->dir[layer]) return 1;
  memcpy(out, M->dir[layer], sizeof(double) * (size_t)M->out_dim[layer] * (size_t)M->in_dim[layer]);
  return 0;
}

/* One step of every active member; member i reads its batch rows from
 * idx + i * idx_stride (idx_stride 0: one batch shared by all members;
 * idx_stride B: the stacked per-member batches of Sec. 3.6).               */
static int orc_step(orc_pack* h, const float* X, int64_t N, const int32_t* idx, int64_t idx_stride,
                    const int32_t* y_int, const float* y_float, int32_t B,
                    uint32_t step, int32_t update, double* loss_out) {
  if (!h || !X || !idx || B <= 0) return 1;
  if (h->cfg.task == ORC_REGRESSION ? !y_float : !y_int) return 1;
  const int n_rows = idx_stride ? h->cfg.m : 1;
  for (int i = 0; i < n_rows; ++i)
    for (int b = 0; b < B; ++b) {
      const int32_t r = idx[(int64_t)i * idx_stride + b];
      if (r < 0 || r >= N) return 1;
    }
  int status = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int i = 0; i < h->cfg.m; ++i) {
    orc_member* M = &h->mem[i];
    if (!M->active) {
      if (loss_out) loss_out[i] = NAN;
      continue;
    }
    const int32_t* idx_i = idx + (int64_t)i * idx_stride;
    orc_alloc_cache(M, B, h->cfg.d_out);
    orc_member_forward(h, M, X, idx_i, B, step, 1);
    double loss = orc_member_backward(h, M, idx_i, y_int, y_float, B);
    if (loss_out) loss_out[i] = loss;
    if (update) {
      M->t += 1;
      for (int l = 0; l <= M->L; ++l) {
        if (h->muon && l < M->L) orc_muon(h, M, l);
        else orc_adamw(h, M, M->W[l], M->mW[l], M->vW[l], M->gW[l], (int64_t)M->out_dim[l] * M->in_dim[l], 0);
        orc_adamw(h, M, M->b[l], M->mb[l], M->vb[l], M->gb[l], M->out_dim[l], 1);
      }
      if (M->d_emb > 0) orc_adamw(h, M, M->emb, M->memb, M->vemb, M->gemb, M->n_emb, 1);
    }
  }
  return status;
}

int orc_train_step(orc_pack* h, const float* X, int64_t N, const int32_t* idx,
                   const int32_t* y_int, const float* y_float, int32_t B,
                   uint32_t step, int32_t update, double* loss_out) {
  return orc_step(h, X, N, idx, 0, y_int, y_float, B, step, update, loss_out);
}

int orc_train_step_stacked(orc_pack* h, const float* X, int64_t N, const int32_t* idx,
                           const int32_t* y_int, const float* y_float, int32_t B,
                           uint32_t step, int32_t update, double* loss_out) {
  return orc_step(h, X, N, idx, B, y_int, y_float, B, step, update, loss_out);
}

/* Per-member validation predictions (Sec. 3.5 "Online ensemble": the pool is
 * rebuilt from the members' latest states once per epoch): forward without
 * dropout; softmax probabilities, sigmoid probability or the value.          */
int orc_predict(orc_pack* h, const float* X, int64_t N, double* out) {
  if (!h || !X || !out || N <= 0) return 1;
  const int d_out = h->cfg.d_out;
#pragma omp parallel for schedule(dynamic, 1)
  for (int i = 0; i < h->cfg.m; ++i) {
    orc_member* M = &h->mem[i];
    if (!M->active) continue;
    /* a private cache sized for the validation rows */
    orc_member V = *M;
    V.Hin = NULL; V.Z = NULL; V.keep = NULL; V.logits = NULL; V.xraw = NULL; V.B = 0;
    orc_alloc_cache(&V, (int32_t)N, d_out);
    orc_member_forward(h, &V, X, NULL, (int32_t)N, 0u, 0);
    for (int64_t b = 0; b < N; ++b) {
      const double* z = &V.logits[b * d_out];
      double* o = &out[((int64_t)i * N + b) * d_out];
      if (h->cfg.task == ORC_MULTICLASS) {
        double mx = z[0];
        for (int c = 1; c < d_out; ++c) if (z[c] > mx) mx = z[c];
        double s = 0.0;
        for (int c = 0; c < d_out; ++c) s += exp(z[c] - mx);
        for (int c = 0; c < d_out; ++c) o[c] = exp(z[c] - mx) / s;
      } else if (h->cfg.task == ORC_BINARY) {
        o[0] = 1.0 / (1.0 + exp(-z[0]));
      } else {
        o[0] = z[0];
      }
    }
    orc_free_cache(&V);
  }
  return 0;
}

int orc_set_active(orc_pack* h, const uint8_t* active) {
  if (!h || !active) return 1;
  for (int i = 0; i < h->cfg.m; ++i) h->mem[i].active = active[i] ? 1 : 0;
  return 0;
}

static int orc_check_ml(const orc_pack* h, int32_t member, int32_t layer) {
  if (!h || member < 0 || member >= h->cfg.m) return 1;
  if (layer < 0 || layer > h->mem[member].L) return 1;
  return 0;
}

int orc_get_params(const orc_pack* h, int32_t member, int32_t layer, double* W, double* b) {
  if (orc_check_ml(h, member, layer)) return 1;
  const orc_member* M = &h->mem[member];
  int64_t nw = (int64_t)M->out_dim[layer] * M->in_dim[layer];
  if (W) memcpy(W, M->W[layer], (size_t)nw * sizeof(double));
  if (b) memcpy(b, M->b[layer], (size_t)M->out_dim[layer] * sizeof(double));
  return 0;
}

int orc_set_params(orc_pack* h, int32_t member, int32_t layer, const double* W, const double* b) {
  if (orc_check_ml(h, member, layer)) return 1;
  orc_member* M = &h->mem[member];
  int64_t nw = (int64_t)M->out_dim[layer] * M->in_dim[layer];
  if (W) memcpy(M->W[layer], W, (size_t)nw * sizeof(double));
  if (b) memcpy(M->b[layer], b, (size_t)M->out_dim[layer] * sizeof(double));
  return 0;
}

int orc_get_grads(const orc_pack* h, int32_t member, int32_t layer, double* W, double* b) {
  if (orc_check_ml(h, member, layer)) return 1;
  const orc_member* M = &h->mem[member];
  int64_t nw = (int64_t)M->out_dim[layer] * M->in_dim[layer];
  if (W) memcpy(W, M->gW[layer], (size_t)nw * sizeof(double));
  if (b) memcpy(b, M->gb[layer], (size_t)M->out_dim[layer] * sizeof(double));
  return 0;
}

int orc_get_adam_state(const orc_pack* h, int32_t member, int32_t layer,
                       double* mW, double* vW, double* mb, double* vb) {
  if (orc_check_ml(h, member, layer)) return 1;
  const orc_member* M = &h->mem[member];
  int64_t nw = (int64_t)M->out_dim[layer] * M->in_dim[layer];
  if (mW) memcpy(mW, M->mW[layer], (size_t)nw * sizeof(double));
  if (vW) memcpy(vW, M->vW[layer], (size_t)nw * sizeof(double));
  if (mb) memcpy(mb, M->mb[layer], (size_t)M->out_dim[layer] * sizeof(double));
  if (vb) memcpy(vb, M->vb[layer], (size_t)M->out_dim[layer] * sizeof(double));
  return 0;
}

int orc_get_logits(const orc_pack* h, int32_t member, double* out) {
  if (orc_check_ml(h, member, 0) || !h->mem[member].logits) return 1;
  const orc_member* M = &h->mem[member];
  memcpy(out, M->logits, (size_t)M->B * h->cfg.d_out * sizeof(double));
  return 0;
}

int orc_get_keep(const orc_pack* h, int32_t member, int32_t layer, uint8_t* out) {
  if (orc_check_ml(h, member, layer) || layer >= h->mem[member].L || !h->mem[member].keep) return 1;
  const orc_member* M = &h->mem[member];
  memcpy(out, M->keep[layer], (size_t)M->B * M->w);
  return 0;
}

int orc_get_preact(const orc_pack* h, int32_t member, int32_t layer, double* out) {
  if (orc_check_ml(h, member, layer) || layer >= h->mem[member].L || !h->mem[member].Z) return 1;
  const orc_member* M = &h->mem[member];
  memcpy(out, M->Z[layer], (size_t)M->B * M->w * sizeof(double));
  return 0;
}

double orc_get_margin(const orc_pack* h, int32_t member) {
  if (orc_check_ml(h, member, 0)) return NAN;
  return h->mem[member].margin;
}

int64_t orc_member_steps(const orc_pack* h, int32_t member) {
  if (orc_check_ml(h, member, 0)) return -1;
  return h->mem[member].t;
}

/* ------------------------------------------------------------------------ */
/* Greedy ensembling (Sec. 3.5).  The ensemble's prediction is the mean of its */
/* members' predictions (probabilities for classification -- a reading).      */
/* Scores are "lower is better": the loss, minus the accuracy, or the RMSE.   */
/* Start from the best single candidate; then repeatedly add the candidate,   */
/* not yet used, whose addition gives the best ensemble score; stop at m_ens  */
/* members or when the best addition does not strictly improve the score.     */
/* Ties go to the lowest candidate index.                                     */
/* ------------------------------------------------------------------------ */
#define ORC_CLIP_LO 1e-7
#define ORC_CLIP_HI (1.0 - 1e-7)

/* plain fp64 score of the ensemble whose row predictions are ens[N, d_out] */
typedef struct { float key; int32_t y; } orc_ranked;
static int orc_cmp_ranked(const void* a, const void* b) {
  const float x = ((const orc_ranked*)a)->key, z = ((const orc_ranked*)b)->key;
  return x < z ? -1 : (x > z ? 1 : 0);
}

double orc_auc(const double* e, const int32_t* y, int64_t N) {
  orc_ranked* v = (orc_ranked*)malloc(sizeof(orc_ranked) * (size_t)(N > 0 ? N : 1));
  int64_t n_pos = 0;
  for (int64_t b = 0; b < N; ++b) {
    v[b].key = (float)e[b];
    v[b].y = y[b] == 1;
    n_pos += v[b].y;
  }
  const int64_t n_neg = N - n_pos;
  if (n_pos == 0 || n_neg == 0) {
    free(v);
    return NAN;
  }
  qsort(v, (size_t)N, sizeof(orc_ranked), orc_cmp_ranked);
  double rank_sum = 0.0;  /* ranks 1..N; a tie group [i, j) shares (i + 1 + j) / 2 */
  for (int64_t i = 0; i < N;) {
    int64_t j = i + 1;
    while (j < N && v[j].key == v[i].key) ++j;
    int64_t pos = 0;
    for (int64_t k = i; k < j; ++k) pos += v[k].y;
    rank_sum += (double)pos * 0.5 * (double)(i + 1 + j);
    i = j;
  }
  free(v);
  return (rank_sum - 0.5 * (double)n_pos * (double)(n_pos + 1)) / ((double)n_pos * (double)n_neg);
}

static double orc_score_rows(const double* ens, int64_t N, int32_t d_out, const int32_t* y_int,
                             const float* y_float, int32_t task, int32_t score) {
  if (score == ORC_SCORE_AUC) return -orc_auc(ens, y_int, N);
  double acc = 0.0;
  for (int64_t b = 0; b < N; ++b) {
    const double* e = &ens[b * d_out];
    if (score == ORC_SCORE_ACCURACY) {
      int pred;
      if (task == ORC_MULTICLASS) {
        pred = 0;
        for (int c = 1; c < d_out; ++c) if (e[c] > e[pred]) pred = c;
      } else {
        pred = e[0] > 0.5 ? 1 : 0;
      }
      acc += (pred == y_int[b]) ? 1.0 : 0.0;
    } else if (task == ORC_REGRESSION) {
      double d = e[0] - (double)y_float[b];
      acc += d * d;
    } else {
      double q = task == ORC_MULTICLASS ? e[y_int[b]] : e[0];
      q = q < ORC_CLIP_LO ? ORC_CLIP_LO : (q > ORC_CLIP_HI ? ORC_CLIP_HI : q);
      if (task == ORC_MULTICLASS || y_int[b] == 1) acc += -log(q);
      else acc += -log(1.0 - q);
    }
  }
  double mean = acc / (double)N;
  if (score == ORC_SCORE_ACCURACY) return -mean;
  if (score == ORC_SCORE_RMSE) return sqrt(mean);
  return mean;
}

/* fp32-term score of the ensemble (S + p) / (n + 1): the ensemble value is
 * formed in fp64 as (S + p) * (1 / (n + 1)); each row's term is then taken
 * in fp32 (loss terms) or from the fp64 values (accuracy), and terms are
 * summed in fp64.                                                            */
static double orc_score_fp32_terms(const double* S, const float* p, int32_t n, int64_t N, int32_t d_out,
                                   const int32_t* y_int, const float* y_float, int32_t task, int32_t score) {
  const double inv = 1.0 / (double)(n + 1);
  if (score == ORC_SCORE_AUC) {  /* the fp64 ensemble values; orc_auc ranks them in fp32 */
    double* e = orc_zeros(N);
    for (int64_t b = 0; b < N; ++b) e[b] = (S[b] + (double)p[b]) * inv;
    const double r = -orc_auc(e, y_int, N);
    free(e);
    return r;
  }
  double acc = 0.0;
  for (int64_t b = 0; b < N; ++b) {
    const double* s = &S[b * d_out];
    const float* q = &p[b * d_out];
    if (score == ORC_SCORE_ACCURACY) {
      int pred;
      if (task == ORC_MULTICLASS) {
        pred = 0;
        double best = (s[0] + (double)q[0]) * inv;
        for (int c = 1; c < d_out; ++c) {
          double e = (s[c] + (double)q[c]) * inv;
          if (e > best) { best = e; pred = c; }
        }
      } else {
        pred = (s[0] + (double)q[0]) * inv > 0.5 ? 1 : 0;
      }
      acc += (pred == y_int[b]) ? 1.0 : 0.0;
    } else if (task == ORC_REGRESSION) {
      float e = (float)((s[0] + (double)q[0]) * inv);
      float d = e - y_float[b];
      acc += (double)(d * d);
    } else {
      int k = task == ORC_MULTICLASS ? y_int[b] : 0;
      float e = (float)((s[k] + (double)q[k]) * inv);
      e = e < 1e-7f ? 1e-7f : (e > 1.0f - 1e-7f ? 1.0f - 1e-7f : e);
      float t = (task == ORC_MULTICLASS || y_int[b] == 1) ? -logf(e) : -logf(1.0f - e);
      acc += (double)t;
    }
  }
  double mean = acc / (double)N;
  if (score == ORC_SCORE_ACCURACY) return -mean;
  if (score == ORC_SCORE_RMSE) return sqrt(mean);
  return mean;
}

static int orc_score_valid(int32_t task, int32_t score, int32_t d_out) {
  if (score < 0 || score > 3) return 0;
  if (score == ORC_SCORE_AUC && task != ORC_BINARY) return 0;
  if (score == ORC_SCORE_ACCURACY && task == ORC_REGRESSION) return 0;
  if (score == ORC_SCORE_RMSE && task != ORC_REGRESSION) return 0;
  if (task != ORC_MULTICLASS && d_out != 1) return 0;
  return 1;
}

double orc_ensemble_score(const float* preds, const int32_t* subset, int32_t n_subset,
                          int64_t N, int32_t d_out, const int32_t* y_int, const float* y_float,
                          int32_t task, int32_t score) {
  if (!orc_score_valid(task, score, d_out) || n_subset <= 0) return NAN;
  double* ens = orc_zeros(N * d_out);
  for (int s = 0; s < n_subset; ++s)
    for (int64_t e = 0; e < N * d_out; ++e) ens[e] += (double)preds[(int64_t)subset[s] * N * d_out + e];
  for (int64_t e = 0; e < N * d_out; ++e) ens[e] /= (double)n_subset;
  double r = orc_score_rows(ens, N, d_out, y_int, y_float, task, score);
  free(ens);
  return r;
}

int orc_greedy(const float* preds, int32_t P, int64_t N, int32_t d_out,
               const int32_t* y_int, const float* y_float, int32_t task, int32_t score,
               int32_t m_ens, int32_t fp32_terms,
               int32_t* selected, int32_t* n_selected, double* final_score,
               double* step_best, double* step_gap) {
  if (!preds || P <= 0 || N <= 0 || m_ens <= 0 || !selected || !n_selected) return 1;
  if (!orc_score_valid(task, score, d_out)) return 1;
  if (task == ORC_REGRESSION ? !y_float : !y_int) return 1;
  const int64_t R = N * d_out;
  double* S = orc_zeros(R);      /* sum of the selected members' predictions */
  double* ens = orc_zeros(R);
  uint8_t* used = (uint8_t*)calloc((size_t)P, 1);
  int32_t n = 0;
  double cur = INFINITY;
  for (int32_t it = 0; it < m_ens; ++it) {
    double best = INFINITY, second = INFINITY;
    int32_t bc = -1;
    for (int32_t c = 0; c < P; ++c) {
      if (used[c]) continue;
      const float* pc = &preds[(int64_t)c * R];
      double s;
      if (fp32_terms) {
        s = orc_score_fp32_terms(S, pc, n, N, d_out, y_int, y_float, task, score);
      } else {
        for (int64_t e = 0; e < R; ++e) ens[e] = (S[e] + (double)pc[e]) / (double)(n + 1);
        s = orc_score_rows(ens, N, d_out, y_int, y_float, task, score);
      }
      if (s < best) { second = best; best = s; bc = c; }
      else if (s < second) second = s;
    }
    if (bc < 0) break;
    if (n > 0 && !(best < cur)) break;
    for (int64_t e = 0; e < R; ++e) S[e] += (double)preds[(int64_t)bc * R + e];
    used[bc] = 1;
    selected[n++] = bc;
    cur = best;
    if (step_best) step_best[it] = best;
    if (step_gap) step_gap[it] = second - best;
  }
  *n_selected = n;
  if (final_score) *final_score = cur;
  free(S); free(ens); free(used);
  return 0;
}
