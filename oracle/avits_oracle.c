/*
 * avits_oracle.c — plain, slow, CPU reference of the AViTS transition.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call this: it is
 * used by the tests, by __graft_entry__.smoke() and by bench.py's CPU
 * baseline arm.  It shares no code, header, table or helper with the CUDA
 * library; both read the same seeded inputs and nothing else.
 *
 * Each function follows the paper's definition in the paper's order:
 *   spatial   Sec. 3.3.1, Eq. 3 (head mean of text attention mass) with the
 *             joint-attention extraction of Eq. 4-5 (softmax of Q K^T/sqrt(d)
 *             over the concatenated [text; image] keys, image rows, text cols)
 *   attention Eq. 4-5, the block's joint attention O = softmax(Q K^T/sqrt(d)) V
 *             with the logsumexp over all and over the text keys and Eq. 3
 *   temporal  Sec. 3.3.2 — the relative two-snapshot change used by this
 *             build, and Eq. 6-7 (unbiased step variance, channel mean)
 *   fuse      Sec. 3.3.3, min-max normalisation and Eq. 8
 *   top-K     Eq. 9, K tokens of largest S, ties to the lower index
 *   upsample  Sec. 3.2 Stage 2, selected tokens 2x upsampled, the rest kept,
 *             packed in token order
 *   merge     Sec. 3.2 Stage 3, every token expanded to full resolution and
 *             laid out in spatial order
 * Floating point is fp64 except the fuse/top-K step, which works in fp32 with
 * a fixed operation order (the selection is an integer decision and is taken
 * in the precision the kernel takes it in), and the resampling arithmetic,
 * which is fp32 as the library's outputs are.  Build with -ffp-contract=off.
 *
 * Parity pins (tests/test_oracle_pins.py): brute-force NumPy softmax and a
 * full sort on small inputs, torch's CPU scaled_dot_product_attention in
 * fp64, closed forms (Q = 0, one hot logit, h_t = c h_prev,
 * two-snapshot variance), invariants (mass in [0,1], |S| = k, N_out = M + 3k,
 * exact tiling), the hand-worked 4x4 example in tests/golden/, and torch's
 * bilinear / nearest resize on dense grids.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_BAD_ARG 1
#define OR_COVERAGE 6

/* element access: dtype 0 = fp32, 1 = bf16 (bit pattern in uint16) */
static double get_elem(const void* base, int dtype, int64_t idx) {
  if (dtype == 0) return (double)((const float*)base)[idx];
  uint32_t bits = ((uint32_t)((const uint16_t*)base)[idx]) << 16;
  float f;
  memcpy(&f, &bits, 4);
  return (double)f;
}

static float get_f32(const void* base, int dtype, int64_t idx) {
  return (float)get_elem(base, dtype, idx);
}

/* fp32 -> bf16, round to nearest, ties to even (the IEEE default rounding). */
static uint16_t f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return 0x7FC0; /* NaN */
  uint32_t lsb = (u >> 16) & 1u;
  uint32_t r = u + 0x7FFFu + lsb;
  return (uint16_t)(r >> 16);
}

static void put_elem(void* base, int dtype, int64_t idx, float v) {
  if (dtype == 0) ((float*)base)[idx] = v;
  else ((uint16_t*)base)[idx] = f32_to_bf16(v);
}

/* ---------------------------------------------------------------------------
 * Spatial importance, Eq. 3 / Eq. 5.
 *
 * For every image query i of batch b and head h the full joint-attention row
 * P_ij = scale * q_i . k_j over all Nk keys is formed, softmax-normalised
 * (alpha_ij, Eq. 5; the row maximum is subtracted first, which does not change
 * the softmax) and its first L entries — the text columns — are summed.  A_i
 * is the mean of that text mass over the heads (Eq. 3), times `weight`, added
 * to A_i when `accumulate` (aggregation over blocks and collection steps,
 * end of Sec. 3.3.1).  `l2norm` applies the literal reading of the sentence
 * after Eq. 5 (unit-norm q and k rows before the product).
 *
 * rows: NULL for all B*M queries, else `nrows` flat indices b*M + i.
 * mass_out [B,H,M] and lse_out [B,H,M,2] are optional (fp64).
 * text_mask: NULL (the text keys are the first L), else [B,Nk] bytes, key j
 * of element b is a text key iff text_mask[b*Nk + j] != 0 (the unified
 * sequences of MLLM-conditioned models, where text and image tokens
 * interleave; Sec. 3.3.1).  L is then ignored.
 * ------------------------------------------------------------------------- */
int avits_oracle_score_spatial(const void* q, const void* k, int dtype, int B, int H, int M,
                               int Nk, int L, int d, int64_t q_sb, int64_t q_sh, int64_t q_sn,
                               int64_t k_sb, int64_t k_sh, int64_t k_sn, double scale,
                               double weight, int accumulate, int l2norm, const int32_t* rows,
                               int nrows, const uint8_t* text_mask, float* A, double* mass_out,
                               double* lse_out) {
  if (B <= 0 || H <= 0 || M <= 0 || Nk <= 0 || d <= 0 || L < 0 || L > Nk) return OR_BAD_ARG;
  int n = rows ? nrows : B * M;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int r = 0; r < n; ++r) {
    int flat = rows ? rows[r] : r;
    if (flat < 0 || flat >= B * M) { bad = 1; continue; }
    int b = flat / M, i = flat % M;
    double* P = (double*)malloc(sizeof(double) * (size_t)Nk);
    double* qv = (double*)malloc(sizeof(double) * (size_t)d);
    double head_sum = 0.0;
    for (int h = 0; h < H; ++h) {
      const int64_t qoff = (int64_t)b * q_sb + (int64_t)h * q_sh + (int64_t)i * q_sn;
      double qn = 0.0;
      for (int c = 0; c < d; ++c) { qv[c] = get_elem(q, dtype, qoff + c); qn += qv[c] * qv[c]; }
      if (l2norm) { qn = sqrt(qn); for (int c = 0; c < d; ++c) qv[c] = qn > 0 ? qv[c] / qn : 0.0; }
      /* joint attention logits, Eq. 5 before the softmax */
      for (int j = 0; j < Nk; ++j) {
        const int64_t koff = (int64_t)b * k_sb + (int64_t)h * k_sh + (int64_t)j * k_sn;
        double dot = 0.0, kn = 0.0;
        for (int c = 0; c < d; ++c) {
          double kv = get_elem(k, dtype, koff + c);
          dot += qv[c] * kv;
          kn += kv * kv;
        }
        if (l2norm) { kn = sqrt(kn); dot = kn > 0 ? dot / kn : 0.0; }
        P[j] = scale * dot;
      }
      /* softmax over all keys */
      double mx = -INFINITY;
      for (int j = 0; j < Nk; ++j) if (P[j] > mx) mx = P[j];
      double z = 0.0;
      for (int j = 0; j < Nk; ++j) { P[j] = exp(P[j] - mx); z += P[j]; }
      double mass = 0.0, ztxt = 0.0;
      for (int j = 0; j < Nk; ++j) {                                      /* image->text block */
        const int is_text = text_mask ? text_mask[(int64_t)b * Nk + j] != 0 : j < L;
        if (is_text) { mass += P[j] / z; ztxt += P[j]; }
      }
      head_sum += mass;
      if (mass_out) mass_out[((int64_t)b * H + h) * M + i] = mass;
      if (lse_out) {
        lse_out[(((int64_t)b * H + h) * M + i) * 2 + 0] = mx + log(z);
        lse_out[(((int64_t)b * H + h) * M + i) * 2 + 1] = ztxt > 0 ? mx + log(ztxt) : -INFINITY;
      }
    }
    double a = weight * (head_sum / (double)H);   /* Eq. 3: mean over heads */
    if (A) A[flat] = accumulate ? (float)((double)A[flat] + a) : (float)a;
    free(P);
    free(qv);
  }
  return bad ? OR_BAD_ARG : OR_OK;
}

/* ---------------------------------------------------------------------------
 * Joint-attention forward of a double-stream block, Eq. 4-5 (Sec. 3.3.1):
 * the block's own attention over the concatenated [text; image] sequence,
 *   O_i = sum_j softmax_j(scale * q_i . k_j) v_j,
 * with, from the same softmax row, the logsumexp over all keys, the
 * logsumexp over the text keys (the first L) and the text mass that Eq. 5
 * extracts; A_i is the mean of that mass over the heads (Eq. 3), times
 * `weight`, added to A_i when `accumulate`.  Query rows are whatever the
 * caller passes (text and image rows of the joint sequence alike); A is
 * given for every row.
 *
 * q [B,H,Mq,d], k and v [B,H,Nk,d], all contiguous.
 * rows: NULL for all B*Mq rows, else `nrows` flat indices b*Mq + i.
 * o_out [B,H,Mq,d] fp64, lse_out [B,H,Mq,2] fp64 (all, text; -inf when the
 * row has no text key), mass_out [B,H,Mq] fp64, A [B,Mq] fp32; each may be
 * NULL.
 * ------------------------------------------------------------------------- */
int avits_oracle_attention(const void* q, const void* k, const void* v, int dtype, int B, int H,
                           int Mq, int Nk, int L, int d, double scale, double weight,
                           int accumulate, const int32_t* rows, int nrows, double* o_out,
                           double* lse_out, double* mass_out, float* A) {
  if (B <= 0 || H <= 0 || Mq <= 0 || Nk <= 0 || d <= 0 || L < 0 || L > Nk) return OR_BAD_ARG;
  int n = rows ? nrows : B * Mq;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int r = 0; r < n; ++r) {
    int flat = rows ? rows[r] : r;
    if (flat < 0 || flat >= B * Mq) { bad = 1; continue; }
    int b = flat / Mq, i = flat % Mq;
    double* w = (double*)malloc(sizeof(double) * (size_t)Nk);
    double* ov = (double*)malloc(sizeof(double) * (size_t)d);
    double head_sum = 0.0;
    for (int h = 0; h < H; ++h) {
      const int64_t qoff = (((int64_t)b * H + h) * Mq + i) * d;
      const int64_t kv0 = ((int64_t)b * H + h) * (int64_t)Nk * d;
      /* logits P = scale * Q K^T (the row of query i) */
      for (int j = 0; j < Nk; ++j) {
        double dot = 0.0;
        for (int c = 0; c < d; ++c)
          dot += get_elem(q, dtype, qoff + c) * get_elem(k, dtype, kv0 + (int64_t)j * d + c);
        w[j] = scale * dot;
      }
      /* softmax over all keys (the row maximum subtracted first) */
      double mx = -INFINITY;
      for (int j = 0; j < Nk; ++j) if (w[j] > mx) mx = w[j];
      double z = 0.0, ztxt = 0.0;
      for (int j = 0; j < Nk; ++j) {
        w[j] = exp(w[j] - mx);
        z += w[j];
        if (j < L) ztxt += w[j];
      }
      /* O = softmax(P) V */
      for (int c = 0; c < d; ++c) ov[c] = 0.0;
      for (int j = 0; j < Nk; ++j) {
        const double a = w[j] / z;
        for (int c = 0; c < d; ++c) ov[c] += a * get_elem(v, dtype, kv0 + (int64_t)j * d + c);
      }
      const double mass = ztxt / z;   /* Eq. 5: this row's text columns of the softmax */
      head_sum += mass;
      const int64_t row = ((int64_t)b * H + h) * Mq + i;
      if (o_out) for (int c = 0; c < d; ++c) o_out[row * d + c] = ov[c];
      if (lse_out) {
        lse_out[row * 2 + 0] = mx + log(z);
        lse_out[row * 2 + 1] = ztxt > 0 ? mx + log(ztxt) : -INFINITY;
      }
      if (mass_out) mass_out[row] = mass;
    }
    double a = weight * (head_sum / (double)H);   /* Eq. 3: mean over heads */
    if (A) A[flat] = accumulate ? (float)((double)A[flat] + a) : (float)a;
    free(w);
    free(ov);
  }
  return bad ? OR_BAD_ARG : OR_OK;
}

/* ---------------------------------------------------------------------------
 * Temporal importance from the two latest snapshots:
 *   V = ||h_t - h_prev||_2 / (||h_prev||_2 + eps), per token, fp64 sums.
 * ------------------------------------------------------------------------- */
int avits_oracle_score_temporal(const void* ht, const void* hp, int dtype, int B, int N, int D,
                                double eps, float* V) {
  if (B <= 0 || N <= 0 || D <= 0) return OR_BAD_ARG;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < (int64_t)B * N; ++t) {
    double dd = 0.0, pp = 0.0;
    for (int c = 0; c < D; ++c) {
      double a = get_elem(ht, dtype, t * D + c), p = get_elem(hp, dtype, t * D + c);
      dd += (a - p) * (a - p);
      pp += p * p;
    }
    V[t] = (float)(sqrt(dd) / (sqrt(pp) + eps));
  }
  return OR_OK;
}

/* ---------------------------------------------------------------------------
 * Temporal importance, Eq. 6-7: temporal mean per channel over the N_T
 * snapshots, unbiased variance per channel, mean over channels.  fp64.
 * snaps: n_t pointers to [B,N,D] arrays, oldest first.
 * ------------------------------------------------------------------------- */
int avits_oracle_score_temporal_var(const void* const* snaps, int n_t, int dtype, int B, int N,
                                    int D, float* V) {
  if (n_t < 2 || B <= 0 || N <= 0 || D <= 0) return OR_BAD_ARG;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < (int64_t)B * N; ++t) {
    double acc = 0.0;
    for (int c = 0; c < D; ++c) {
      double mean = 0.0;                                    /* Eq. 6 */
      for (int s = 0; s < n_t; ++s) mean += get_elem(snaps[s], dtype, t * D + c);
      mean /= (double)n_t;
      double ss = 0.0;
      for (int s = 0; s < n_t; ++s) {
        double dv = get_elem(snaps[s], dtype, t * D + c) - mean;
        ss += dv * dv;
      }
      acc += ss / (double)(n_t - 1);                        /* Eq. 7, inner */
    }
    V[t] = (float)(acc / (double)D);                        /* Eq. 7, channel mean */
  }
  return OR_OK;
}

/* ---------------------------------------------------------------------------
 * Joint score, Sec. 3.3.3 + Eq. 8, in fp32 with this exact order:
 *   mn = min, mx = max (NaN entries ignored), den = (mx - mn) + eps,
 *   A^ = (A - mn) / den, V^ likewise, S = (alpha * A^) + ((1 - alpha) * V^).
 * ------------------------------------------------------------------------- */
static void minmax_f32(const float* x, int M, float* mn, float* mx) {
  float lo = NAN, hi = NAN;
  for (int i = 0; i < M; ++i) {
    float v = x[i];
    if (isnan(v)) continue;
    if (isnan(lo) || v < lo) lo = v;
    if (isnan(hi) || v > hi) hi = v;
  }
  *mn = lo;
  *mx = hi;
}

/* perturb (NULL or [B,M]): the paper's tie-breaking noise, Eq. 9 (Sec.
 * 3.3.3), supplied by the caller and added to S as one more rounded fp32
 * addition: S' = S + perturb. */
int avits_oracle_fuse(const float* A, const float* V, int B, int M, float alpha, float eps,
                      const float* perturb, float* S) {
  if (B <= 0 || M <= 0) return OR_BAD_ARG;
  for (int b = 0; b < B; ++b) {
    const float* a = A + (int64_t)b * M;
    const float* v = V + (int64_t)b * M;
    float amn, amx, vmn, vmx;
    minmax_f32(a, M, &amn, &amx);
    minmax_f32(v, M, &vmn, &vmx);
    volatile float aden = (amx - amn);
    aden = aden + eps;
    volatile float vden = (vmx - vmn);
    vden = vden + eps;
    volatile float one_m = 1.0f - alpha;
    for (int i = 0; i < M; ++i) {
      volatile float an = a[i] - amn;
      an = an / aden;
      volatile float vn = v[i] - vmn;
      vn = vn / vden;
      volatile float t1 = alpha * an;
      volatile float t2 = one_m * vn;
      volatile float sc = t1 + t2;
      if (perturb) sc = sc + perturb[(int64_t)b * M + i];
      S[(int64_t)b * M + i] = sc;
    }
  }
  return OR_OK;
}

/* ---------------------------------------------------------------------------
 * TopK, Eq. 9: order tokens by S descending (NaN last, -0 == +0), ties by
 * ascending index; keep the first k; report them in ascending index order.
 * tok_offset_i = i + 3 * #(selected j < i)  (start of token i in the packed
 * mixed sequence: each selected token becomes 4 tokens).
 * ------------------------------------------------------------------------- */
typedef struct { float s; int i; } sk_t;

static int cmp_sk(const void* pa, const void* pb) {
  const sk_t* a = (const sk_t*)pa;
  const sk_t* b = (const sk_t*)pb;
  int an = isnan(a->s), bn = isnan(b->s);
  if (an != bn) return an ? 1 : -1;                  /* NaN ranks lowest */
  if (!an && a->s != b->s) return a->s > b->s ? -1 : 1;
  return (a->i > b->i) - (a->i < b->i);              /* lower index first */
}

int avits_oracle_topk(const float* S, int B, int M, int k, int32_t* sel_idx, uint8_t* mask,
                      int32_t* tok_offset) {
  if (B <= 0 || M <= 0 || k < 0 || k > M) return OR_BAD_ARG;
  sk_t* buf = (sk_t*)malloc(sizeof(sk_t) * (size_t)M);
  uint8_t* m = (uint8_t*)malloc((size_t)M);
  for (int b = 0; b < B; ++b) {
    for (int i = 0; i < M; ++i) { buf[i].s = S[(int64_t)b * M + i]; buf[i].i = i; }
    qsort(buf, (size_t)M, sizeof(sk_t), cmp_sk);
    memset(m, 0, (size_t)M);
    for (int r = 0; r < k; ++r) m[buf[r].i] = 1;
    int c = 0;
    for (int i = 0; i < M; ++i) {
      if (tok_offset) tok_offset[(int64_t)b * M + i] = i + 3 * c;
      if (m[i]) { if (sel_idx) sel_idx[(int64_t)b * k + c] = i; ++c; }
      if (mask) mask[(int64_t)b * M + i] = m[i];
    }
  }
  free(buf);
  free(m);
  return OR_OK;
}

/* ---------------------------------------------------------------------------
 * 2x resize weights of a half-pixel-centred bilinear upsample (the usual
 * align_corners=False convention) along one axis: output pixel P of a
 * 2n-pixel axis reads source pixels r0, r1 (clamped to [0, n-1]) with weights
 * w0, w1: even P = 2m -> (m-1: 0.25, m: 0.75); odd P = 2m+1 -> (m: 0.75,
 * m+1: 0.25).
 * ------------------------------------------------------------------------- */
static void bil_axis(int P, int n, int* r0, int* r1, float* w0, float* w1) {
  int m = P >> 1;
  if ((P & 1) == 0) { *r0 = m - 1; *r1 = m; *w0 = 0.25f; *w1 = 0.75f; }
  else { *r0 = m; *r1 = m + 1; *w0 = 0.75f; *w1 = 0.25f; }
  if (*r0 < 0) *r0 = 0;
  if (*r1 > n - 1) *r1 = n - 1;
}

/* out = wy0*(wx0*p00 + wx1*p01) + wy1*(wx0*p10 + wx1*p11), fp32, this order */
static float bil_combine(float p00, float p01, float p10, float p11, float wy0, float wy1,
                         float wx0, float wx1) {
  volatile float a = wx0 * p00;
  volatile float b2 = wx1 * p01;
  volatile float top = a + b2;
  volatile float c = wx0 * p10;
  volatile float d = wx1 * p11;
  volatile float bot = c + d;
  volatile float t = wy0 * top;
  volatile float u = wy1 * bot;
  return t + u;
}

/* ---------------------------------------------------------------------------
 * Multi-level bilinear resampling (the reading of "orthogonal upsampling" for
 * frames that hold tokens of several spans, Sec. 3.2 Stages 2-3).
 *
 * A frame of fh x fw cells is tiled by tokens of span s (a power of two, the
 * token at a multiple of s); its pixel image E (2fh x 2fw) repeats each of a
 * token's 2x2 pixels over the s x s full pixels it stands for.  The pyramid:
 * P_0 = E and P_l = the 2x2 average pool of P_(l-1), ((a + b) + (c + d)) *
 * 0.25 over (2R,2Q), (2R,2Q+1), (2R+1,2Q), (2R+1,2Q+1), except that a level-l
 * pixel lying inside one token pixel (the token's span >= 2^l) is that pixel
 * itself.  A selected token of span 2^l is upsampled by the half-pixel-
 * centred 2x bilinear resize of P_l (Stage 2); the merge refines every token
 * coarser than level l from level l + 1 the same way, coarsest level first
 * (Stage 3).  With spans 1 and 2 only this is the single-level rule: P_0 is
 * the dense latent image, P_1 the rebuilt half-resolution image.
 * ------------------------------------------------------------------------- */
typedef struct {
  const void* mixed;      /* token values of one element, [N, T] */
  int dtype, T;
  const int32_t* pos;     /* [N, 2] */
  const int32_t* span;    /* [N] */
  const int32_t* owner;   /* [fh * fw] cell -> covering token */
  int fh, fw;
} frame_t;

static int is_pow2(int s) { return s > 0 && (s & (s - 1)) == 0; }
static int log2i(int s) { int l = 0; while ((1 << l) < s) ++l; return l; }

/* owner map of one element's tokens; OR_COVERAGE unless they tile the frame
 * exactly with power-of-two spans at multiples of their span */
static int frame_owner(const int32_t* pos, const int32_t* span, int N, int fh, int fw,
                       int32_t* owner, int32_t* count) {
  int rc = OR_OK;
  for (int64_t c = 0; c < (int64_t)fh * fw; ++c) { owner[c] = -1; count[c] = 0; }
  for (int t = 0; t < N; ++t) {
    const int y = pos[t * 2], x = pos[t * 2 + 1], s = span[t];
    if (!is_pow2(s) || y % s || x % s) { rc = OR_COVERAGE; continue; }
    for (int u = 0; u < s; ++u)
      for (int v = 0; v < s; ++v) {
        const int Y = y + u, X = x + v;
        if (Y < 0 || Y >= fh || X < 0 || X >= fw) { rc = OR_COVERAGE; continue; }
        count[(int64_t)Y * fw + X]++;
        owner[(int64_t)Y * fw + X] = t;
      }
  }
  for (int64_t c = 0; c < (int64_t)fh * fw; ++c)
    if (count[c] != 1) rc = OR_COVERAGE;
  return rc;
}

/* P_l(R, Q), channel ch */
static float pyr_pixel(const frame_t* f, int ch, int l, int R, int Q) {
  const int Y = R << l, X = Q << l;   /* the block's first full pixel */
  const int t = f->owner[(int64_t)(Y >> 1) * f->fw + (X >> 1)];
  const int s = f->span[t];
  if (s >= (1 << l)) {
    const int ty = (Y - 2 * f->pos[t * 2]) / s, tx = (X - 2 * f->pos[t * 2 + 1]) / s;
    return get_f32(f->mixed, f->dtype, (int64_t)t * f->T + ch * 4 + ty * 2 + tx);
  }
  volatile float a = pyr_pixel(f, ch, l - 1, 2 * R, 2 * Q);
  volatile float b = pyr_pixel(f, ch, l - 1, 2 * R, 2 * Q + 1);
  volatile float c = pyr_pixel(f, ch, l - 1, 2 * R + 1, 2 * Q);
  volatile float d = pyr_pixel(f, ch, l - 1, 2 * R + 1, 2 * Q + 1);
  volatile float top = a + b;
  volatile float bot = c + d;
  volatile float sum = top + bot;
  return sum * 0.25f;
}

/* Stage 3 value of level-l pixel (R, Q): U_L = P_L; below it, a pixel of a
 * token coarser than 2^l is the 2x bilinear resize of U_(l+1), any other the
 * frame's own P_l */
static float cascade_pixel(const frame_t* f, int ch, int l, int L, int R, int Q) {
  if (l >= L) return pyr_pixel(f, ch, l, R, Q);
  const int Y = R << l, X = Q << l;
  const int s = f->span[f->owner[(int64_t)(Y >> 1) * f->fw + (X >> 1)]];
  if (s <= (1 << l)) return pyr_pixel(f, ch, l, R, Q);
  const int nh = (2 * f->fh) >> (l + 1), nw = (2 * f->fw) >> (l + 1);
  int r0, r1, c0, c1;
  float wy0, wy1, wx0, wx1;
  bil_axis(R, nh, &r0, &r1, &wy0, &wy1);
  bil_axis(Q, nw, &c0, &c1, &wx0, &wx1);
  return bil_combine(cascade_pixel(f, ch, l + 1, L, r0, c0), cascade_pixel(f, ch, l + 1, L, r0, c1),
                     cascade_pixel(f, ch, l + 1, L, r1, c0), cascade_pixel(f, ch, l + 1, L, r1, c1),
                     wy0, wy1, wx0, wx1);
}

/* ---------------------------------------------------------------------------
 * Selective upsampling, Sec. 3.2 Stage 2, p = 2, tokens of C*4 values in
 * (channel, patch row, patch col) order.  Tokens are visited in index order;
 * a selected token at (y,x) with span s becomes 4 children (a,b) at
 * (2y + a*s, 2x + b*s) with span s, child (a,b) being the 2x upsample of the
 * parent's pixel (a,b); a deferred token is copied to (2y, 2x) with span 2s.
 * Nearest: each child pixel equals the parent pixel.  Bilinear: the children
 * of a selected token of span 2^l are its pixels in the half-pixel-centred 2x
 * bilinear resize of level l of the input frame's pyramid (see above; for a
 * dense grid, level 0 is the latent image itself).  A mixed input (pos_in)
 * must tile the gh x gw frame; bilinear then also needs gh, gw even.
 * Returns the number of emitted tokens in *n_out.
 * ------------------------------------------------------------------------- */
int avits_oracle_selective_upsample(const void* latent, int dtype, int B, int M, int gh, int gw,
                                    int C, const int32_t* pos_in, const int32_t* span_in,
                                    const uint8_t* mask, int mode, void* out, int32_t* pos,
                                    int32_t* span, int32_t* src_tok, int8_t* src_sub,
                                    int* n_out) {
  if (B <= 0 || M <= 0 || C <= 0 || gh <= 0 || gw <= 0) return OR_BAD_ARG;
  if (!pos_in && M != gh * gw) return OR_BAD_ARG;
  if (mode == 1 && pos_in && ((gh & 1) || (gw & 1))) return OR_BAD_ARG;
  const int T = C * 4;
  int k = 0;
  for (int i = 0; i < M; ++i) k += mask[i] ? 1 : 0;
  const int64_t NO = (int64_t)M + 3 * (int64_t)k;
  /* bilinear: the input frame (its owner map; a dense grid is the frame of
   * span-1 tokens in raster order) */
  int32_t *owner = NULL, *cnt = NULL, *dpos = NULL, *dspan = NULL;
  if (mode == 1) {
    owner = (int32_t*)malloc(sizeof(int32_t) * (size_t)gh * gw);
    cnt = (int32_t*)malloc(sizeof(int32_t) * (size_t)gh * gw);
    if (!pos_in) {
      dpos = (int32_t*)malloc(sizeof(int32_t) * 2 * (size_t)M);
      dspan = (int32_t*)malloc(sizeof(int32_t) * (size_t)M);
      for (int i = 0; i < M; ++i) { dpos[2 * i] = i / gw; dpos[2 * i + 1] = i % gw; dspan[i] = 1; }
    }
  }
  int rc = OR_OK;
  for (int b = 0; b < B && rc == OR_OK; ++b) {
    int kb = 0;
    for (int i = 0; i < M; ++i) kb += mask[(int64_t)b * M + i] ? 1 : 0;
    if (kb != k) { rc = OR_BAD_ARG; break; }      /* one k per call */
    const int64_t lbase = (int64_t)b * M * T;
    frame_t fr;
    if (mode == 1) {
      fr.mixed = (const char*)latent + lbase * (dtype == 0 ? 4 : 2);
      fr.dtype = dtype;
      fr.T = T;
      fr.pos = pos_in ? pos_in + (int64_t)b * M * 2 : dpos;
      fr.span = pos_in ? span_in + (int64_t)b * M : dspan;
      fr.owner = owner;
      fr.fh = gh;
      fr.fw = gw;
      if (frame_owner(fr.pos, fr.span, M, gh, gw, owner, cnt) != OR_OK) { rc = OR_BAD_ARG; break; }
    }
    int64_t o = 0;
    for (int i = 0; i < M; ++i) {
      int y, x, s;
      if (pos_in) {
        y = pos_in[((int64_t)b * M + i) * 2];
        x = pos_in[((int64_t)b * M + i) * 2 + 1];
        s = span_in[(int64_t)b * M + i];
      } else { y = i / gw; x = i % gw; s = 1; }
      if (mask[(int64_t)b * M + i]) {
        for (int a = 0; a < 2; ++a)
          for (int bb = 0; bb < 2; ++bb) {
            const int64_t ot = (int64_t)b * NO + o;
            for (int c = 0; c < C; ++c)
              for (int ph = 0; ph < 2; ++ph)
                for (int pw = 0; pw < 2; ++pw) {
                  float v;
                  if (mode == 0) {
                    v = get_f32(latent, dtype, lbase + (int64_t)i * T + c * 4 + a * 2 + bb);
                  } else {
                    /* the parent covers level-l pixels (2y/s + {0,1}, 2x/s + {0,1});
                     * child (a,b) pixel (ph,pw) is pixel (2(2y/s) + 2a + ph, ...) of
                     * the 2x resize of P_l ((2gh >> l) x (2gw >> l) pixels) */
                    const int l = log2i(s);
                    int r0, r1, c0, c1;
                    float wy0, wy1, wx0, wx1;
                    bil_axis(2 * ((2 * y) >> l) + 2 * a + ph, (2 * gh) >> l, &r0, &r1, &wy0, &wy1);
                    bil_axis(2 * ((2 * x) >> l) + 2 * bb + pw, (2 * gw) >> l, &c0, &c1, &wx0, &wx1);
                    v = bil_combine(pyr_pixel(&fr, c, l, r0, c0), pyr_pixel(&fr, c, l, r0, c1),
                                    pyr_pixel(&fr, c, l, r1, c0), pyr_pixel(&fr, c, l, r1, c1),
                                    wy0, wy1, wx0, wx1);
                  }
                  put_elem(out, dtype, ot * T + c * 4 + ph * 2 + pw, v);
                }
            pos[ot * 2] = 2 * y + a * s;
            pos[ot * 2 + 1] = 2 * x + bb * s;
            span[ot] = s;
            src_tok[ot] = i;
            src_sub[ot] = (int8_t)(2 * a + bb);
            ++o;
          }
      } else {
        const int64_t ot = (int64_t)b * NO + o;
        for (int e = 0; e < T; ++e)
          put_elem(out, dtype, ot * T + e, get_f32(latent, dtype, lbase + (int64_t)i * T + e));
        pos[ot * 2] = 2 * y;
        pos[ot * 2 + 1] = 2 * x;
        span[ot] = 2 * s;
        src_tok[ot] = i;
        src_sub[ot] = -1;
        ++o;
      }
    }
    if (o != NO) { rc = OR_BAD_ARG; break; }
  }
  free(owner);
  free(cnt);
  free(dpos);
  free(dspan);
  if (n_out) *n_out = (int)NO;
  return rc;
}

/* ---------------------------------------------------------------------------
 * Final merge, Sec. 3.2 Stage 3.  Every token (y,x,span s) covers the cells
 * [y,y+s) x [x,x+s) of the fh x fw frame; the cover must be exact
 * (cover_count, optional [B,fh*fw], receives the per-cell count; any count
 * != 1 returns OR_COVERAGE).  Output is in raster order of the frame.
 * Nearest: full-res pixel (Y,X) (Y in [2y, 2y+2s)) takes the token pixel
 * ((Y-2y)/s, (X-2x)/s).  Bilinear (power-of-two spans at multiples of their
 * span, fh and fw even, 2fh and 2fw multiples of the largest span): span-1
 * tokens are copied; every other pixel is the coarse-to-fine cascade of the
 * multi-level resampling above.  With spans 1 and 2 it is: the
 * half-resolution latent image is rebuilt (a span-2 token gives its own
 * pixels, each 2x2 block of span-1 tokens gives the 2x2 average of its
 * child's pixels: pooled (a,b) = ((p00 + p01) + (p10 + p11)) * 0.25 of child
 * (a,b)) and span-2 cells take its 2x bilinear resize (weights as above).
 * ------------------------------------------------------------------------- */
int avits_oracle_merge_final(const void* mixed, int dtype, int B, int N, const int32_t* pos,
                             const int32_t* span, int fh, int fw, int C, int mode, void* out,
                             int32_t* cover_count) {
  if (B <= 0 || N <= 0 || fh <= 0 || fw <= 0 || C <= 0) return OR_BAD_ARG;
  const int T = C * 4;
  const int64_t F = (int64_t)fh * fw;
  int32_t* owner = (int32_t*)malloc(sizeof(int32_t) * (size_t)F);
  int32_t* cnt = (int32_t*)malloc(sizeof(int32_t) * (size_t)F);
  int rc = OR_OK;
  for (int b = 0; b < B && rc == OR_OK; ++b) {
    for (int64_t c = 0; c < F; ++c) { owner[c] = -1; cnt[c] = 0; }
    for (int t = 0; t < N; ++t) {
      int y = pos[((int64_t)b * N + t) * 2], x = pos[((int64_t)b * N + t) * 2 + 1];
      int s = span[(int64_t)b * N + t];
      for (int u = 0; u < s; ++u)
        for (int v = 0; v < s; ++v) {
          int Y = y + u, X = x + v;
          if (Y < 0 || Y >= fh || X < 0 || X >= fw) { rc = OR_COVERAGE; continue; }
          cnt[(int64_t)Y * fw + X]++;
          owner[(int64_t)Y * fw + X] = t;
        }
    }
    for (int64_t c = 0; c < F; ++c) {
      if (cnt[c] != 1) rc = OR_COVERAGE;
      if (cover_count) cover_count[(int64_t)b * F + c] = cnt[c];
    }
    if (rc != OR_OK) break;
    const int64_t mb = (int64_t)b * N * T;
    const int64_t ob = (int64_t)b * F * T;
    if (mode == 0) {
      for (int Y = 0; Y < fh; ++Y)
        for (int X = 0; X < fw; ++X) {
          int t = owner[(int64_t)Y * fw + X];
          int y = pos[((int64_t)b * N + t) * 2], x = pos[((int64_t)b * N + t) * 2 + 1];
          int s = span[(int64_t)b * N + t];
          for (int c = 0; c < C; ++c)
            for (int ph = 0; ph < 2; ++ph)
              for (int pw = 0; pw < 2; ++pw) {
                int ty = (2 * Y + ph - 2 * y) / s, tx = (2 * X + pw - 2 * x) / s;
                float v = get_f32(mixed, dtype, mb + (int64_t)t * T + c * 4 + ty * 2 + tx);
                put_elem(out, dtype, ob + ((int64_t)Y * fw + X) * T + c * 4 + ph * 2 + pw, v);
              }
        }
    } else {
      /* bilinear: every token coarser than a level is refined from the level
       * above, coarsest first (see the multi-level resampling above) */
      if ((fh & 1) || (fw & 1)) { rc = OR_BAD_ARG; break; }
      int smax = 1;
      for (int t = 0; t < N; ++t) {
        const int s = span[(int64_t)b * N + t];
        if (!is_pow2(s) || pos[((int64_t)b * N + t) * 2] % s || pos[((int64_t)b * N + t) * 2 + 1] % s) {
          rc = OR_BAD_ARG;
          break;
        }
        if (s > smax) smax = s;
      }
      if (rc != OR_OK) break;
      const int L = log2i(smax);
      if (((2 * fh) >> L) << L != 2 * fh || ((2 * fw) >> L) << L != 2 * fw) { rc = OR_BAD_ARG; break; }
      frame_t fr;
      fr.mixed = (const char*)mixed + mb * (dtype == 0 ? 4 : 2);
      fr.dtype = dtype;
      fr.T = T;
      fr.pos = pos + (int64_t)b * N * 2;
      fr.span = span + (int64_t)b * N;
      fr.owner = owner;
      fr.fh = fh;
      fr.fw = fw;
      for (int Y = 0; Y < fh; ++Y)
        for (int X = 0; X < fw; ++X)
          for (int c = 0; c < C; ++c)
            for (int ph = 0; ph < 2; ++ph)
              for (int pw = 0; pw < 2; ++pw)
                put_elem(out, dtype, ob + ((int64_t)Y * fw + X) * T + c * 4 + ph * 2 + pw,
                         cascade_pixel(&fr, c, 0, L, 2 * Y + ph, 2 * X + pw));
    }
  }
  free(owner);
  free(cnt);
  return rc;
}
