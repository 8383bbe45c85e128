/*
 * Seeded synthetic video streams: uint8 RGB frames, HWC, frames back to back.
 *
 * This file is input generation only. It holds none of the filtering
 * method's arithmetic (no grayscale conversion, no histogram, no distance):
 * it writes raw colour frames and the ground-truth scene-cut and event
 * indices that the tests and the benchmark use. Both the oracle and the GPU
 * path read the bytes it writes.
 *
 * Everything that decides a pixel value is integer arithmetic, so a seed
 * gives the same bytes on x86_64 and aarch64:
 *   - Random numbers: SplitMix64 (Steele, Lea & Flood, OOPSLA 2014) used as a
 *     counter-based generator, out(key, i) = mix64(key + (i + 1) * gamma).
 *   - Gaussian pixel noise of standard deviation sigma: a centred binomial,
 *     popcount of 4*sigma^2 random bits minus 2*sigma^2 (variance sigma^2).
 *   - Geometric scene lengths: 1 + the number of failed Bernoulli(1/mean)
 *     trials, each trial an integer comparison (mean length = mean).
 *
 * Recipes (frame streams the paper's workloads stand in for):
 *   SYNTH_UNIFORM_SCENES  fixed-length scenes, each a uniform-random base
 *                         image plus per-frame noise.
 *   SYNTH_GRADIENT_DRIFT  geometric scene lengths; each scene a bilinear
 *                         gradient between four random corner colours with a
 *                         +-1 per-frame global brightness drift, plus noise;
 *                         optional injected rectangle events.
 *   SYNTH_TEXTURE_WALK    geometric scene lengths; each scene a two-octave
 *                         value-noise texture with its own mean and contrast,
 *                         translated with wrap-around by a +-2 px/frame
 *                         random walk, plus noise.
 *   SYNTH_BANDED_SCENES   fixed-length scenes whose base channels are uniform
 *                         in the disjoint band [64 s, 64 s + 63], so that the
 *                         intensity distributions of consecutive scenes do
 *                         not overlap.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <pthread.h>

#define SYNTH_UNIFORM_SCENES 1
#define SYNTH_GRADIENT_DRIFT 2
#define SYNTH_TEXTURE_WALK 3
#define SYNTH_BANDED_SCENES 4

typedef struct {
  int32_t recipe;
  uint32_t width, height, frames;
  uint64_t seed;
  uint32_t sigma;            /* noise standard deviation, 0..4 */
  uint32_t scene_len;        /* fixed scene length (recipes 1 and 4) */
  uint32_t mean_scene_len;   /* geometric mean scene length (recipes 2 and 3) */
  uint32_t n_events;         /* injected rectangle events (recipe 2) */
} synth_spec;

/* ---------------------------------------------------------------- RNG -- */

static const uint64_t GAMMA = 0x9E3779B97F4A7C15ull;

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* out(key, i): the i-th output of a SplitMix64 stream whose state starts at key. */
uint64_t synth_u64(uint64_t key, uint64_t i) { return mix64(key + (i + 1) * GAMMA); }

/* A sub-stream key: hashes (key, tag) into a new, unrelated key. */
static inline uint64_t subkey(uint64_t key, uint64_t tag) {
  return synth_u64(key ^ 0xA0761D6478BD642Full, tag);
}

/* Uniform integer in [lo, hi] (inclusive) by multiply-shift of 32 bits. */
static inline int64_t uniform_int(uint64_t r, int64_t lo, int64_t hi) {
  uint64_t span = (uint64_t)(hi - lo + 1);
  return lo + (int64_t)(((r >> 32) * span) >> 32);
}

static inline int noise_value(uint64_t r, uint32_t sigma) {
  /* centred binomial with 4 sigma^2 fair bits: variance sigma^2 */
  if (sigma == 0) return 0;
  uint32_t nbits = 4u * sigma * sigma; /* <= 64 */
  uint64_t mask = nbits >= 64 ? ~0ull : ((1ull << nbits) - 1ull);
  return __builtin_popcountll(r & mask) - (int)(nbits / 2);
}

static inline uint8_t clamp_u8(int v) { return (uint8_t)(v < 0 ? 0 : (v > 255 ? 255 : v)); }

/* ------------------------------------------------------------- scenes -- */

enum { TAG_SCENES = 1, TAG_SCENE = 2, TAG_NOISE = 3, TAG_EVENTS = 4, TAG_WALK = 5 };

typedef struct {
  uint32_t start, len;
  uint64_t key;
} scene_t;

/* Scene list covering [0, frames). Returns the count; *out is malloc'd. */
static uint32_t plan_scenes(const synth_spec* s, scene_t** out) {
  uint32_t cap = 16, n = 0;
  scene_t* sc = (scene_t*)malloc(cap * sizeof(scene_t));
  uint64_t kscenes = subkey(s->seed, TAG_SCENES);
  uint64_t ctr = 0;
  uint32_t t = 0;
  while (t < s->frames) {
    uint32_t len;
    if (s->recipe == SYNTH_GRADIENT_DRIFT || s->recipe == SYNTH_TEXTURE_WALK) {
      /* 1 + Geometric(p = 1/mean): failures before the first success */
      uint64_t thresh = ((1ull << 53) + s->mean_scene_len / 2) / (s->mean_scene_len ? s->mean_scene_len : 1);
      len = 1;
      while ((synth_u64(kscenes, ctr++) >> 11) >= thresh) ++len;
    } else {
      len = s->scene_len ? s->scene_len : s->frames;
    }
    if (len > s->frames - t) len = s->frames - t;
    if (n == cap) { cap *= 2; sc = (scene_t*)realloc(sc, cap * sizeof(scene_t)); }
    sc[n].start = t;
    sc[n].len = len;
    sc[n].key = subkey(s->seed, ((uint64_t)TAG_SCENE << 32) | n);
    ++n;
    t += len;
  }
  *out = sc;
  return n;
}

int synth_scene_starts(const synth_spec* s, uint32_t* out, uint32_t cap, uint32_t* count) {
  scene_t* sc;
  uint32_t n = plan_scenes(s, &sc);
  for (uint32_t i = 0; i < n && i < cap; ++i) out[i] = sc[i].start;
  *count = n;
  free(sc);
  return n <= cap ? 0 : 1;
}

/* ------------------------------------------------------------- events -- */

typedef struct {
  uint32_t frame, len;             /* frames [frame, frame + len) */
  uint32_t x0, y0, w, h;           /* rectangle */
  int32_t off[3];                  /* per-channel colour offset */
} event_t;

static uint32_t isqrt64(uint64_t v) {
  uint64_t r = 0, bit = 1ull << 62;
  while (bit > v) bit >>= 2;
  while (bit) {
    if (v >= r + bit) { v -= r + bit; r = (r >> 1) + bit; } else r >>= 1;
    bit >>= 2;
  }
  return (uint32_t)r;
}

static uint32_t plan_events(const synth_spec* s, event_t** out) {
  uint32_t n = (s->recipe == SYNTH_GRADIENT_DRIFT) ? s->n_events : 0;
  event_t* ev = (event_t*)calloc(n ? n : 1, sizeof(event_t));
  uint64_t k = subkey(s->seed, TAG_EVENTS);
  uint64_t c = 0;
  uint64_t area_total = (uint64_t)s->width * s->height;
  for (uint32_t i = 0; i < n; ++i) {
    event_t* e = &ev[i];
    e->len = (uint32_t)uniform_int(synth_u64(k, c++), 1, 3);
    int64_t last = (int64_t)s->frames - (int64_t)e->len;
    e->frame = (uint32_t)uniform_int(synth_u64(k, c++), 0, last < 0 ? 0 : last);
    if (e->frame + e->len > s->frames) e->len = s->frames - e->frame;
    /* area fraction in [5%, 30%] (per mille), aspect ratio q/8 with q in [4, 16] */
    uint64_t permille = (uint64_t)uniform_int(synth_u64(k, c++), 50, 300);
    uint64_t q = (uint64_t)uniform_int(synth_u64(k, c++), 4, 16);
    uint64_t area = area_total * permille / 1000;
    uint32_t w = isqrt64(area * q / 8);
    if (w < 1) w = 1;
    if (w > s->width) w = s->width;
    uint32_t h = (uint32_t)(area / w);
    if (h < 1) h = 1;
    if (h > s->height) h = s->height;
    e->w = w;
    e->h = h;
    e->x0 = (uint32_t)uniform_int(synth_u64(k, c++), 0, s->width - w);
    e->y0 = (uint32_t)uniform_int(synth_u64(k, c++), 0, s->height - h);
    for (int ch = 0; ch < 3; ++ch) {
      int32_t mag = (int32_t)uniform_int(synth_u64(k, c++), 64, 160);
      e->off[ch] = (synth_u64(k, c++) >> 63) ? mag : -mag;
    }
  }
  *out = ev;
  return n;
}

/* mask[t] = 1 for every frame an event touches. */
int synth_event_frames(const synth_spec* s, uint8_t* mask) {
  event_t* ev;
  uint32_t n = plan_events(s, &ev);
  memset(mask, 0, s->frames);
  for (uint32_t i = 0; i < n; ++i)
    for (uint32_t f = ev[i].frame; f < ev[i].frame + ev[i].len; ++f) mask[f] = 1;
  free(ev);
  return 0;
}

/* ------------------------------------------------------- scene bases -- */

/* Base image of one scene, uint8 HWC. Returns malloc'd buffer or NULL. */
static uint8_t* make_base(const synth_spec* s, const scene_t* sc, uint32_t scene_index) {
  const uint32_t W = s->width, H = s->height;
  uint8_t* b = (uint8_t*)malloc((size_t)W * H * 3);
  if (!b) return NULL;
  uint64_t k = sc->key;
  if (s->recipe == SYNTH_UNIFORM_SCENES || s->recipe == SYNTH_BANDED_SCENES) {
    int lo = 0, span = 256;
    if (s->recipe == SYNTH_BANDED_SCENES) { lo = 64 * (int)(scene_index % 4); span = 64; }
    size_t nbytes = (size_t)W * H * 3;
    for (size_t i = 0; i < nbytes; i += 8) {
      uint64_t r = synth_u64(k, i / 8);
      for (size_t j = 0; j < 8 && i + j < nbytes; ++j)
        b[i + j] = (uint8_t)(lo + (int)((((r >> (8 * j)) & 0xFF) * (uint64_t)span) >> 8));
    }
  } else if (s->recipe == SYNTH_GRADIENT_DRIFT) {
    /* bilinear blend of four random corner colours, 16.16 fixed point */
    int corner[4][3];
    for (int c = 0; c < 4; ++c)
      for (int ch = 0; ch < 3; ++ch) corner[c][ch] = (int)(synth_u64(k, 1 + c * 3 + ch) >> 56);
    for (uint32_t y = 0; y < H; ++y) {
      uint64_t fy = H > 1 ? ((uint64_t)y << 16) / (H - 1) : 0;
      for (uint32_t x = 0; x < W; ++x) {
        uint64_t fx = W > 1 ? ((uint64_t)x << 16) / (W - 1) : 0;
        for (int ch = 0; ch < 3; ++ch) {
          uint64_t top = (uint64_t)corner[0][ch] * (65536 - fx) + (uint64_t)corner[1][ch] * fx;
          uint64_t bot = (uint64_t)corner[2][ch] * (65536 - fx) + (uint64_t)corner[3][ch] * fx;
          uint64_t v = (top * (65536 - fy) + bot * fy + (1ull << 31)) >> 32;
          b[((size_t)y * W + x) * 3 + ch] = (uint8_t)v;
        }
      }
    }
  } else { /* SYNTH_TEXTURE_WALK: two octaves of value noise */
    int mean[3], contrast = (int)uniform_int(synth_u64(k, 1), 24, 110);
    for (int ch = 0; ch < 3; ++ch) mean[ch] = (int)uniform_int(synth_u64(k, 2 + ch), 40, 215);
    uint32_t cell[2];
    cell[0] = (uint32_t)uniform_int(synth_u64(k, 5), 64, 192);
    cell[1] = (uint32_t)uniform_int(synth_u64(k, 6), 8, 32);
    uint64_t kl[2] = {subkey(k, 101), subkey(k, 102)};
    uint32_t gw[2], gh[2];
    for (int o = 0; o < 2; ++o) { gw[o] = W / cell[o] + 2; gh[o] = H / cell[o] + 2; }
    for (uint32_t y = 0; y < H; ++y) {
      for (uint32_t x = 0; x < W; ++x) {
        for (int ch = 0; ch < 3; ++ch) {
          int64_t acc = 0; /* sum of octaves, each in [-256, 256] << 16 */
          for (int o = 0; o < 2; ++o) {
            uint32_t cx = x / cell[o], cy = y / cell[o];
            uint64_t fx = ((uint64_t)(x % cell[o]) << 16) / cell[o];
            uint64_t fy = ((uint64_t)(y % cell[o]) << 16) / cell[o];
            int64_t v[4];
            for (int c = 0; c < 4; ++c) {
              uint64_t idx = ((uint64_t)(cy + (c >> 1)) * gw[o] + (cx + (c & 1))) * 3 + ch;
              v[c] = (int64_t)(synth_u64(kl[o], idx) >> 55) - 256; /* [-256, 255] */
            }
            (void)gh;
            int64_t top = v[0] * (int64_t)(65536 - fx) + v[1] * (int64_t)fx;
            int64_t bot = v[2] * (int64_t)(65536 - fx) + v[3] * (int64_t)fx;
            int64_t val = (top * (int64_t)(65536 - fy) + bot * (int64_t)fy) >> 16; /* << 16 */
            acc += (o == 0) ? val * 2 : val; /* low octave weighted 2:1 */
          }
          /* acc / (3 * 256 << 16) in [-1, 1]; scale by contrast around the mean */
          int64_t pix = mean[ch] + (acc * contrast) / (3ll * 256 * 65536);
          b[((size_t)y * W + x) * 3 + ch] = clamp_u8((int)pix);
        }
      }
    }
  }
  return b;
}

/* ------------------------------------------------------------ frames -- */

typedef struct {
  const synth_spec* s;
  const scene_t* scenes;
  uint32_t n_scenes;
  uint8_t** bases;          /* per scene, NULL if not needed */
  const int32_t* walk;      /* per frame (dx, dy), recipe 3 */
  const event_t* events;
  uint32_t n_events;
  uint32_t f0, f1;
  uint8_t* out;
  uint32_t next;            /* work counter, atomically advanced */
  uint32_t base_next;
  const uint32_t* needed;   /* scene indices whose base is needed */
  uint32_t n_needed;
} gen_ctx;

static uint32_t scene_of(const gen_ctx* g, uint32_t f) {
  uint32_t lo = 0, hi = g->n_scenes; /* last scene with start <= f */
  while (hi - lo > 1) {
    uint32_t mid = (lo + hi) / 2;
    if (g->scenes[mid].start <= f) lo = mid; else hi = mid;
  }
  return lo;
}

static void gen_frame(const gen_ctx* g, uint32_t f) {
  const synth_spec* s = g->s;
  const uint32_t W = s->width, H = s->height;
  const size_t fb = (size_t)W * H * 3;
  uint32_t si = scene_of(g, f);
  const scene_t* sc = &g->scenes[si];
  const uint8_t* base = g->bases[si];
  uint8_t* o = g->out + (size_t)(f - g->f0) * fb;
  uint64_t kn = subkey(s->seed, ((uint64_t)TAG_NOISE << 40) | f);
  const uint32_t sigma = s->sigma;
  /* noise words: sigma <= 2 packs 4 values per 64-bit draw, else 1 */
  const int per = (sigma <= 2) ? 4 : 1;
  const int shift = 64 / per;

  int drift = 0;
  if (s->recipe == SYNTH_GRADIENT_DRIFT) {
    int sign = (synth_u64(sc->key, 0) >> 63) ? 1 : -1;
    drift = sign * (int)(f - sc->start);
  }
  uint32_t dx = 0, dy = 0;
  if (s->recipe == SYNTH_TEXTURE_WALK) { dx = (uint32_t)g->walk[2 * f]; dy = (uint32_t)g->walk[2 * f + 1]; }

  size_t i = 0;
  uint64_t word = 0;
  for (uint32_t y = 0; y < H; ++y) {
    uint32_t yy = y + dy;
    if (yy >= H) yy -= H;
    const uint8_t* row = base + (size_t)yy * W * 3;
    for (uint32_t x = 0; x < W; ++x) {
      uint32_t xx = x + dx;
      if (xx >= W) xx -= W;
      const uint8_t* px = row + (size_t)xx * 3;
      for (int ch = 0; ch < 3; ++ch, ++i) {
        uint64_t r;
        if (per == 4) {
          if ((i & 3) == 0) word = synth_u64(kn, i >> 2);
          r = word >> (shift * (int)(i & 3));
        } else {
          r = synth_u64(kn, i);
        }
        o[i] = clamp_u8((int)px[ch] + drift + noise_value(r, sigma));
      }
    }
  }
  for (uint32_t e = 0; e < g->n_events; ++e) {
    const event_t* ev = &g->events[e];
    if (f < ev->frame || f >= ev->frame + ev->len) continue;
    for (uint32_t y = ev->y0; y < ev->y0 + ev->h; ++y)
      for (uint32_t x = ev->x0; x < ev->x0 + ev->w; ++x)
        for (int ch = 0; ch < 3; ++ch) {
          uint8_t* p = o + ((size_t)y * W + x) * 3 + ch;
          *p = clamp_u8((int)*p + ev->off[ch]);
        }
  }
}

static void* base_worker(void* arg) {
  gen_ctx* g = (gen_ctx*)arg;
  for (;;) {
    uint32_t j = __atomic_fetch_add(&g->base_next, 1, __ATOMIC_RELAXED);
    if (j >= g->n_needed) break;
    uint32_t si = g->needed[j];
    g->bases[si] = make_base(g->s, &g->scenes[si], si);
  }
  return NULL;
}

static void* frame_worker(void* arg) {
  gen_ctx* g = (gen_ctx*)arg;
  for (;;) {
    uint32_t f = __atomic_fetch_add(&g->next, 1, __ATOMIC_RELAXED);
    if (f >= g->f1 - g->f0) break;
    gen_frame(g, g->f0 + f);
  }
  return NULL;
}

static void run_threads(void* (*fn)(void*), gen_ctx* g, int nthreads) {
  if (nthreads <= 1) { fn(g); return; }
  pthread_t* th = (pthread_t*)malloc(sizeof(pthread_t) * (size_t)nthreads);
  int started = 0;
  for (int i = 0; i < nthreads; ++i)
    if (pthread_create(&th[i], NULL, fn, g) == 0) ++started;
  if (started == 0) fn(g);
  for (int i = 0; i < started; ++i) pthread_join(th[i], NULL);
  free(th);
}

/*
 * Writes frames [f0, f1) of the stream into out (uint8, (f1 - f0) * H * W * 3
 * bytes). Returns 0 on success, nonzero on bad arguments or allocation failure.
 */
int synth_generate(const synth_spec* s, uint32_t f0, uint32_t f1, uint8_t* out, int nthreads) {
  if (!s || !out || f0 > f1 || f1 > s->frames || s->width == 0 || s->height == 0) return 1;
  if (s->sigma > 4) return 1;
  if (f0 == f1) return 0;
  gen_ctx g;
  memset(&g, 0, sizeof g);
  g.s = s;
  g.n_scenes = plan_scenes(s, (scene_t**)&g.scenes);
  g.n_events = plan_events(s, (event_t**)&g.events);
  g.f0 = f0;
  g.f1 = f1;
  g.out = out;
  g.bases = (uint8_t**)calloc(g.n_scenes, sizeof(uint8_t*));
  uint32_t* needed = (uint32_t*)malloc(sizeof(uint32_t) * g.n_scenes);
  uint32_t nn = 0;
  uint32_t s_lo = scene_of(&g, f0), s_hi = scene_of(&g, f1 - 1);
  for (uint32_t i = s_lo; i <= s_hi; ++i) needed[nn++] = i;
  g.needed = needed;
  g.n_needed = nn;
  int32_t* walk = NULL;
  if (s->recipe == SYNTH_TEXTURE_WALK) {
    /* per scene: random start offset, then a +-2 px/frame walk per axis */
    walk = (int32_t*)malloc(sizeof(int32_t) * 2 * (size_t)s->frames);
    for (uint32_t si = 0; si < g.n_scenes; ++si) {
      const scene_t* sc = &g.scenes[si];
      uint64_t kw = subkey(sc->key, TAG_WALK);
      int64_t x = uniform_int(synth_u64(kw, 0), 0, (int64_t)s->width - 1);
      int64_t y = uniform_int(synth_u64(kw, 1), 0, (int64_t)s->height - 1);
      for (uint32_t j = 0; j < sc->len; ++j) {
        if (j > 0) {
          x += uniform_int(synth_u64(kw, 2 + 2 * (uint64_t)j), -2, 2);
          y += uniform_int(synth_u64(kw, 3 + 2 * (uint64_t)j), -2, 2);
          x = ((x % (int64_t)s->width) + s->width) % s->width;
          y = ((y % (int64_t)s->height) + s->height) % s->height;
        }
        walk[2 * (size_t)(sc->start + j)] = (int32_t)x;
        walk[2 * (size_t)(sc->start + j) + 1] = (int32_t)y;
      }
    }
  }
  g.walk = walk;
  int nt = nthreads < 1 ? 1 : nthreads;
  run_threads(base_worker, &g, nt < (int)nn ? nt : (int)nn);
  int rc = 0;
  for (uint32_t j = 0; j < nn; ++j)
    if (!g.bases[needed[j]]) rc = 2;
  if (rc == 0) run_threads(frame_worker, &g, nt);
  for (uint32_t i = 0; i < g.n_scenes; ++i) free(g.bases[i]);
  free(g.bases);
  free(needed);
  free(walk);
  free((void*)g.scenes);
  free((void*)g.events);
  return rc;
}
