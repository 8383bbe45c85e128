/* A plain C client of libcofie_ngff.so (no CUDA runtime, no Python): reads
 * frames from a file, pushes them from pageable host memory in pieces of the
 * given sizes, closing the stream after every piece (its candidate set S_c,
 * into host memory), and writes every frame's score and keep code (host
 * outputs) and each piece's candidate set to an output file.
 * Usage: ngff_client IN OUT WIDTH HEIGHT FRAMES TAU L_MAX PIECE...
 * IN holds FRAMES * WIDTH * HEIGHT * 3 bytes; OUT receives FRAMES floats,
 * FRAMES keep bytes, then per piece: the prefix length T (uint32), |S_c|
 * (uint32) and |S_c| uint32 indices. It then pushes the same frames as two
 * streams of one handle through cofie_ngff_push_batch in the same pieces
 * and checks that both equal the single-stream results (exit status 7 if
 * not). Exit status 0 on success; a failing call prints the library's
 * message. */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include "cofie_ngff.h"

static int check(int rc, cofie_ngff_t* h, const char* what) {
  if (rc != COFIE_OK) {
    fprintf(stderr, "%s failed (%d): %s\n", what, rc, h ? cofie_ngff_last_error(h) : cofie_ngff_global_error());
    return 1;
  }
  return 0;
}

int main(int argc, char** argv) {
  if (argc < 9) {
    fprintf(stderr, "usage: %s IN OUT WIDTH HEIGHT FRAMES TAU L_MAX PIECE...\n", argv[0]);
    return 2;
  }
  const uint32_t W = (uint32_t)strtoul(argv[3], NULL, 10), H = (uint32_t)strtoul(argv[4], NULL, 10);
  const uint32_t T = (uint32_t)strtoul(argv[5], NULL, 10);
  const size_t frame_bytes = (size_t)W * H * 3;
  uint8_t* frames = malloc(frame_bytes * T);
  float* scores = malloc(sizeof(float) * T);
  uint8_t* keep = malloc(T);
  uint32_t* idx = malloc(sizeof(uint32_t) * (T ? T : 1));
  if (!frames || !scores || !keep || !idx) return 3;
  FILE* in = fopen(argv[1], "rb");
  if (!in || fread(frames, 1, frame_bytes * T, in) != frame_bytes * T) return 4;
  fclose(in);

  cofie_ngff_params p;
  cofie_ngff_default_params(&p, W, H);
  p.tau = strtof(argv[6], NULL);
  p.l_max = (uint32_t)strtoul(argv[7], NULL, 10);
  p.max_frames_per_push = T ? T : 1;
  cofie_ngff_t* h = NULL;
  if (check(cofie_ngff_create(&p, &h), NULL, "cofie_ngff_create")) return 1;

  FILE* out = fopen(argv[2], "wb");
  if (!out) return 5;
  fseek(out, (long)(T * (sizeof(float) + 1)), SEEK_SET); /* the candidate sets follow scores and keep codes */
  uint32_t off = 0;
  for (int a = 8; a < argc && off < T; ++a) {
    uint32_t n = (uint32_t)strtoul(argv[a], NULL, 10);
    if (n > T - off) n = T - off;
    if (check(cofie_ngff_push(h, 0, frames + (size_t)off * frame_bytes, n, scores + off, keep + off, NULL), h,
              "cofie_ngff_push"))
      return 1;
    off += n;
    uint32_t m = 0;
    if (check(cofie_ngff_candidates(h, 0, idx, T, &m, NULL), h, "cofie_ngff_candidates")) return 1;
    if (m > off) return 6;
    fwrite(&off, sizeof off, 1, out);
    fwrite(&m, sizeof m, 1, out);
    fwrite(idx, sizeof(uint32_t), m, out);
  }
  if (off != T) {
    fprintf(stderr, "pieces cover %u of %u frames\n", off, T);
    return 2;
  }
  if (check(cofie_ngff_status(h, NULL), h, "cofie_ngff_status")) return 1;
  cofie_ngff_destroy(h);

  /* The same frames as two streams of one handle through the batched call,
   * in the same pieces, from pageable host memory into host outputs: each
   * stream's scores and keep codes must equal the single-stream run's. */
  p.max_streams = 2;
  p.max_frames_per_push = 2 * (T ? T : 1);
  cofie_ngff_t* hb = NULL;
  if (check(cofie_ngff_create(&p, &hb), NULL, "cofie_ngff_create (batch)")) return 1;
  float* bs = malloc(sizeof(float) * 2 * (T ? T : 1));
  uint8_t* bk = malloc(2 * (T ? T : 1));
  if (!bs || !bk) return 3;
  off = 0;
  for (int a = 8; a < argc && off < T; ++a) {
    uint32_t n = (uint32_t)strtoul(argv[a], NULL, 10);
    if (n > T - off) n = T - off;
    cofie_ngff_push_desc d[2];
    for (uint32_t s = 0; s < 2; ++s) {
      d[s].stream = s;
      d[s].n = n;
      d[s].frames = frames + (size_t)off * frame_bytes;
      d[s].scores_out = bs + (size_t)s * T + off;
      d[s].keep_out = bk + (size_t)s * T + off;
    }
    if (check(cofie_ngff_push_batch(hb, d, 2, NULL), hb, "cofie_ngff_push_batch")) return 1;
    off += n;
  }
  if (check(cofie_ngff_status(hb, NULL), hb, "cofie_ngff_status (batch)")) return 1;
  cofie_ngff_destroy(hb);
  for (uint32_t s = 0; s < 2; ++s)
    for (uint32_t t = 0; t < T; ++t)
      if (bk[(size_t)s * T + t] != keep[t] || bs[(size_t)s * T + t] != scores[t]) {
        fprintf(stderr, "batched stream %u differs from the single-stream run at frame %u\n", s, t);
        return 7;
      }
  free(bs);
  free(bk);

  fseek(out, 0, SEEK_SET);
  fwrite(scores, sizeof(float), T, out);
  fwrite(keep, 1, T, out);
  fclose(out);
  free(frames);
  free(scores);
  free(keep);
  free(idx);
  return 0;
}
