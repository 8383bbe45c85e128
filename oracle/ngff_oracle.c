/*
 * ORACLE for Novelty-Guided Frame Filtering (NGFF), CoFiE Section 3.2.
 *
 * Test infrastructure only. This is a plain, slow, single-threaded
 * restatement of the method, used to check the GPU library. Only the test
 * suite, the smoke check and the benchmark's CPU-baseline leg may load it;
 * the library never calls it and shares no code, header or table with it.
 *
 * What it computes, step by step in the paper's order:
 *   1. Grayscale (Sec. 3.2, the histogram novelty paragraph): the paper
 *      does not give the conversion. Reading used here: ITU-R BT.601 luma
 *      with integer weights and round-half-up,
 *          Y = floor((wR*R + wG*G + wB*B + floor(den/2)) / den),
 *      default (wR, wG, wB, den) = (299, 587, 114, 1000); wR+wG+wB = den so
 *      Y is in [0, 255].
 *   2. Normalised B-bin histogram over the normalised intensity range
 *      (Sec. 3.2; B = 32 in App. A). Reading: B equal-width bins over the
 *      intensity range [0, 256), bin = floor(Y * B / 256), the convention
 *      of common histogram routines; for every B that divides 256 (B = 32
 *      included) it equals cutting Y/255 in [0, 1] into B equal bins with
 *      the last bin closed. Counts are kept as integers;
 *      h_t[b] = count_t[b] / N with N = W*H, so sum_b h_t[b] = 1.
 *   3. Total-variation distance d(h_i, h_j) = 1/2 ||h_i - h_j||_1 (Eq. 2),
 *      evaluated in double precision.
 *   4. s_adj = d(h_t, h_{t-1}), s_ref = d(h_t, h_{r(t)}) (Eq. 3), with r(t)
 *      the most recent retained frame before t; s = max(s_adj, s_ref) (Eq. 4).
 *   5. Retention (Eq. 5 and the safeguards before it): the first frame is
 *      always retained; frame t > 0 is retained when s >= tau_h or
 *      t - r(t) >= L_max (L_max = 0, a value the paper does not use, is read
 *      as no forced retention). The keep decision is taken in fp32, the precision
 *      the GPU library decides in: d32 = fp32(sum_b |c_i[b] - c_j[b]|) /
 *      fp32(2N), one correctly rounded fp32 division.
 *   6. Finalisation (safeguards of Sec. 3.2): add the last frame T-1; if
 *      fewer than M_min candidates remain, add the uniformly spaced frames
 *      round(i (T-1) / (M_min-1)), i = 0..M_min-1 (round half up).
 *
 * Keep codes written to keep_out: 0 drop, 1 novelty (s >= tau_h), 2 gap
 * (t - r(t) >= L_max and not novelty), 3 first frame. Any nonzero code
 * means the frame is retained and becomes r for later frames.
 *
 * Indexing is 0-based: the paper's 1-based frames 1 < t < T are 0 < t < T-1
 * here; the rule is applied to every frame t >= 1 as frames arrive, and the
 * last frame is added at finalisation because in a stream the last frame is
 * only known when the prefix is closed.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  uint32_t width, height;
  uint32_t bins;       /* B */
  uint32_t l_max;      /* L_max; 0 turns the forced-retention term of Eq. 5 off */
  uint32_t m_min;      /* M_min */
  float tau;           /* tau_h */
  uint32_t luma_w[3];  /* wR, wG, wB */
  uint32_t luma_den;   /* den = wR + wG + wB */
} ngff_oracle_params;

enum { KEEP_DROP = 0, KEEP_NOVELTY = 1, KEEP_GAP = 2, KEEP_FIRST = 3 };

static int params_ok(const ngff_oracle_params* p) {
  if (!p || p->width == 0 || p->height == 0) return 0;
  if (p->bins < 1 || p->bins > 256) return 0;
  if (p->luma_den == 0 || p->luma_w[0] + p->luma_w[1] + p->luma_w[2] != p->luma_den) return 0;
  if (p->tau != p->tau) return 0; /* NaN */
  return 1;
}

/* Step 1: grayscale intensity of one RGB pixel. */
uint32_t ngff_oracle_luma(uint32_t r, uint32_t g, uint32_t b, const ngff_oracle_params* p) {
  uint64_t num = (uint64_t)p->luma_w[0] * r + (uint64_t)p->luma_w[1] * g + (uint64_t)p->luma_w[2] * b;
  return (uint32_t)((num + p->luma_den / 2) / p->luma_den);
}

/* Step 1 over n pixels (uint8 RGB triples): y_out[i] = intensity of pixel i. */
void ngff_oracle_luma_map(const uint8_t* px, uint64_t n, const ngff_oracle_params* p, uint8_t* y_out) {
  for (uint64_t i = 0; i < n; ++i) y_out[i] = (uint8_t)ngff_oracle_luma(px[3 * i], px[3 * i + 1], px[3 * i + 2], p);
}

/* Step 2: bin of an intensity Y in [0, 255] among B equal bins of [0, 256). */
uint32_t ngff_oracle_bin(uint32_t y, uint32_t bins) { return (y * bins) / 256u; }

/* Step 2: integer histogram of one frame (uint8 RGB, HWC). counts[bins]. */
void ngff_oracle_histogram(const uint8_t* frame, const ngff_oracle_params* p, uint32_t* counts) {
  for (uint32_t b = 0; b < p->bins; ++b) counts[b] = 0;
  for (uint32_t y = 0; y < p->height; ++y) {
    for (uint32_t x = 0; x < p->width; ++x) {
      const uint8_t* px = frame + ((size_t)y * p->width + x) * 3;
      uint32_t lum = ngff_oracle_luma(px[0], px[1], px[2], p);
      counts[ngff_oracle_bin(lum, p->bins)] += 1;
    }
  }
}

/* Eq. 2: d(h_i, h_j) = 1/2 sum_b |h_i[b] - h_j[b]|, with h = counts / N. */
double ngff_oracle_tv(const uint32_t* ci, const uint32_t* cj, uint32_t bins, uint64_t npix) {
  double acc = 0.0;
  for (uint32_t b = 0; b < bins; ++b) {
    double hi = (double)ci[b] / (double)npix;
    double hj = (double)cj[b] / (double)npix;
    acc += hi > hj ? hi - hj : hj - hi;
  }
  return 0.5 * acc;
}

/* The same distance as the fp32 value the keep decision compares with tau. */
float ngff_oracle_tv32(const uint32_t* ci, const uint32_t* cj, uint32_t bins, uint64_t npix) {
  uint64_t l1 = 0;
  for (uint32_t b = 0; b < bins; ++b) l1 += ci[b] > cj[b] ? ci[b] - cj[b] : cj[b] - ci[b];
  volatile float num = (float)l1;
  volatile float den = (float)(2 * npix);
  return num / den;
}

/*
 * Steps 4-5 on given histograms hist[T][bins] of a stream's frames 0..T-1.
 * score_out[t] = max(s_adj, s_ref) in double (0 for the first frame);
 * keep_out[t] = keep code. Either output may be NULL. Returns 0, or -1 on
 * bad parameters.
 */
int ngff_oracle_select(const uint32_t* hist, uint32_t T, const ngff_oracle_params* p,
                       double* score_out, uint8_t* keep_out) {
  if (!params_ok(p)) return -1;
  const uint32_t B = p->bins;
  const uint64_t N = (uint64_t)p->width * p->height;
  uint32_t r = 0; /* r(t): most recent retained frame */
  for (uint32_t t = 0; t < T; ++t) {
    double score = 0.0;
    uint8_t keep;
    if (t == 0) {
      keep = KEEP_FIRST; /* the first sampled frame is always retained */
    } else {
      const uint32_t* ht = hist + (size_t)t * B;
      double s_adj = ngff_oracle_tv(ht, hist + (size_t)(t - 1) * B, B, N); /* Eq. 3 */
      double s_ref = ngff_oracle_tv(ht, hist + (size_t)r * B, B, N);       /* Eq. 3 */
      score = s_adj > s_ref ? s_adj : s_ref;                               /* Eq. 4 */
      float d_adj = ngff_oracle_tv32(ht, hist + (size_t)(t - 1) * B, B, N);
      float d_ref = ngff_oracle_tv32(ht, hist + (size_t)r * B, B, N);
      float s32 = d_adj > d_ref ? d_adj : d_ref;
      int novelty = s32 >= p->tau;                                         /* Eq. 5 */
      int gap = p->l_max > 0 && (t - r) >= p->l_max;                       /* Eq. 5 */
      keep = novelty ? KEEP_NOVELTY : (gap ? KEEP_GAP : KEEP_DROP);
    }
    if (keep != KEEP_DROP) r = t;
    if (score_out) score_out[t] = score;
    if (keep_out) keep_out[t] = keep;
  }
  return 0;
}

/*
 * Steps 1-5 over a whole stream: frames is T frames of W*H*3 bytes back to
 * back. hist_out (T*bins), score_out (T) and keep_out (T) may each be NULL.
 */
int ngff_oracle_run(const uint8_t* frames, uint32_t T, const ngff_oracle_params* p,
                    uint32_t* hist_out, double* score_out, uint8_t* keep_out) {
  if (!params_ok(p)) return -1;
  const size_t fb = (size_t)p->width * p->height * 3;
  uint32_t* hist = hist_out ? hist_out : (uint32_t*)calloc((size_t)(T ? T : 1) * p->bins, sizeof(uint32_t));
  if (!hist) return -2;
  for (uint32_t t = 0; t < T; ++t) ngff_oracle_histogram(frames + (size_t)t * fb, p, hist + (size_t)t * p->bins);
  int rc = ngff_oracle_select(hist, T, p, score_out, keep_out);
  if (!hist_out) free(hist);
  return rc;
}

/*
 * Step 6: the candidate set S_c of a closed prefix of T frames, given the
 * keep codes of steps 1-5. Writes the sorted frame indices to idx_out
 * (capacity T) and their count to *m. Returns 0, or -1 on bad arguments.
 */
int ngff_oracle_candidates(const uint8_t* keep, uint32_t T, uint32_t m_min, uint32_t* idx_out, uint32_t* m) {
  if (!m) return -1;
  *m = 0;
  if (T == 0) return 0;
  if (!keep || !idx_out) return -1;
  uint8_t* in = (uint8_t*)calloc(T, 1);
  if (!in) return -2;
  uint32_t count = 0;
  for (uint32_t t = 0; t < T; ++t) in[t] = keep[t] != KEEP_DROP;
  in[T - 1] = 1; /* the last sampled frame is always retained */
  for (uint32_t t = 0; t < T; ++t) count += in[t];
  if (count < m_min) {
    /* uniformly spaced frames round(i (T-1) / (M_min - 1)), round half up */
    if (m_min == 1) {
      in[0] = 1;
    } else {
      for (uint32_t i = 0; i < m_min; ++i) {
        uint64_t num = 2ull * i * (T - 1) + (m_min - 1);
        uint64_t den = 2ull * (m_min - 1);
        in[num / den] = 1;
      }
    }
  }
  for (uint32_t t = 0; t < T; ++t)
    if (in[t]) idx_out[(*m)++] = t;
  free(in);
  return 0;
}
