/*
 * cofie_ngff.h -- C ABI of libcofie_ngff.so, a GB300 (sm_103a) implementation
 * of Novelty-Guided Frame Filtering (NGFF), the coarse, pre-encoder stage of
 * CoFiE (Sec. 3.2, Eqs. 2-5; hyperparameters from App. A and App. B.2).
 *
 * What the library computes for every frame I_t of a stream, in order:
 *   1. grayscale Y of every pixel: ITU-R BT.601 luma with integer weights,
 *      Y = floor((wR R + wG G + wB B + floor(den/2)) / den), default
 *      (299, 587, 114) / 1000 (the paper names no conversion; Sec. 3.2);
 *   2. the B-bin histogram h_t over the intensity range, bin = floor(Y B / 256),
 *      kept as integer counts c_t (h_t = c_t / N, N = W H; Sec. 3.2, App. A);
 *   3. the total-variation distances (Eq. 2) to the previous frame, s_adj,
 *      and to the most recent retained frame r(t), s_ref (Eq. 3), and the
 *      novelty score s = max(s_adj, s_ref) (Eq. 4), each distance evaluated
 *      in fp32 as sum_b |c_i[b] - c_j[b]| / (2N) (one IEEE division);
 *   4. the retention decision (Eq. 5 and the first-frame safeguard): the
 *      stream's first frame is kept; frame t > 0 is kept when s >= tau_h or
 *      t - r(t) >= L_max.
 * Decisions are causal and final when a push completes; the closing
 * safeguards of Sec. 3.2 that need the end of the prefix (the last frame, the
 * M_min uniform fill) are applied by cofie_ngff_candidates, which reads the
 * stream's retention record (the library notes every retained frame of every
 * stream on the device as it decides it).
 *
 * Conventions for every entry point:
 *   - All calls are asynchronous on `cuda_stream` (a cudaStream_t passed as
 *     void*; NULL means the legacy default stream) unless stated otherwise.
 *     Buffers passed in must stay valid until that stream has passed the call.
 *   - Frame data is uint8 RGB, height x width x 3 (HWC), frames back to back
 *     (3 W H bytes per frame), in device memory or in host memory (pinned
 *     host memory is copied asynchronously; pageable host memory works but
 *     the copy is synchronous with the host).
 *   - Output buffers may be device or host memory; the library detects which.
 *   - A nonzero return is an error code below and cofie_ngff_last_error()
 *     describes it. Argument errors (COFIE_EINVAL) are found before anything
 *     is enqueued, so they leave the stream state unchanged; a COFIE_ECUDA
 *     from a failed launch may leave earlier pieces of the call enqueued.
 *   - A handle is not thread-safe: calls on one handle must be serialised.
 *     Its device scratch is shared by all of its calls, so work it enqueues
 *     on different CUDA streams must also be ordered on the device (one
 *     stream per handle, or events between the streams); otherwise it races.
 *     The same holds for a QER handle (cofie_qer_*).
 *   - Nothing aborts, traps or prints. Device-side waits are bounded; a wait
 *     that runs out sets an error word that cofie_ngff_status() reports.
 */
#ifndef COFIE_NGFF_H
#define COFIE_NGFF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define COFIE_NGFF_ABI_VERSION 5

/* Return codes. */
#define COFIE_OK 0
#define COFIE_EINVAL 1   /* bad argument: null pointer, size, stream index, parameter */
#define COFIE_ENOMEM 2   /* a device or pinned-host allocation failed */
#define COFIE_ECUDA 3    /* a CUDA runtime call failed */
#define COFIE_ETIMEOUT 4 /* a device-side bounded wait ran out (cofie_ngff_status) */
#define COFIE_EDEVICE 5  /* a device-side check failed: a gather index outside the frames, candidates of a
                            stream that ran past its retention record, or in a build with
                            -DCOFIE_DEBUG_CHECKS=1 an index or layout check (cofie_ngff_status, cofie_qer_status) */

/* Keep codes written to keep_out. Nonzero means retained (a candidate). */
#define COFIE_KEEP_DROP 0
#define COFIE_KEEP_NOVELTY 1 /* s >= tau_h (Eq. 5, first term) */
#define COFIE_KEEP_GAP 2     /* t - r(t) >= L_max and not novelty (Eq. 5, second term) */
#define COFIE_KEEP_FIRST 3   /* the stream's first frame (Sec. 3.2 safeguard) */
#define COFIE_KEEP_SCENE 4   /* a scene change (signal COFIE_SIGNAL_SCD only), not novelty */

/* Novelty signals (the distance d inside Eqs. 3-5). */
#define COFIE_SIGNAL_HISTOGRAM 0 /* TV distance of B-bin grayscale histograms (Sec. 3.2, the paper's signal) */
#define COFIE_SIGNAL_LOWRES 1    /* mean |difference| of 16 x 16-cell block-averaged grayscale frames */
#define COFIE_SIGNAL_DHASH 2     /* Hamming distance / 64 of 9 x 8-cell difference hashes */
#define COFIE_SIGNAL_SCD 3       /* the histogram rule plus twin-comparison scene changes */

/* Limits. */
#define COFIE_NGFF_MAX_BINS 256
#define COFIE_NGFF_MAX_LMAX 256
#define COFIE_NGFF_MAX_BATCH 64 /* descriptors per cofie_ngff_push_batch call */

typedef struct cofie_ngff cofie_ngff_t;

/*
 * Parameters of a handle. Fill with cofie_ngff_default_params() and override.
 *   width, height     frame size in pixels, >= 1 each.
 *   bins              B, 1..256; default 32 (App. A).
 *   l_max             L_max in sampled-frame indices, 0..256; default 30 (App. B.2).
 *                     0 turns the forced retention (Eq. 5's second term) off:
 *                     frames are then kept only as first, novelty or scene
 *                     change, the rule is walked in frame order (by windows
 *                     of 32 frames between keeps, one warp per stream), and
 *                     the stream cannot be sharded.
 *   m_min             M_min, used by cofie_ngff_candidates only; default 4 (App. B.2).
 *   tau               tau_h, any non-NaN float; default 0.30f (App. B.2).
 *   luma_w, luma_den  grayscale weights (wR, wG, wB) / den; each weight <= 65535,
 *                     wR + wG + wB == den; default (299, 587, 114) / 1000.
 *   max_streams       number of independent streams the handle holds, >= 1.
 *   max_frames_per_push
 *                     sizes the device scratch; larger pushes are processed in
 *                     pieces of this many frames (results are identical).
 *   device            CUDA device ordinal, or -1 for the calling thread's current device.
 *   host_stage_bytes  size of each of the two device staging buffers used when
 *                     frames come from host memory; 0 picks 256 MiB (at least one frame).
 *   signal            COFIE_SIGNAL_*: the distance in the retention rule. The
 *                     alternatives are the lightweight signals of the paper's
 *                     signal ablation (Table "hdiff-signal"), defined here as:
 *                     low-res: cells (floor(y 16 / H), floor(x 16 / W)), S_c the
 *                       cell's grayscale sum, d = sum_c |S_c - S'_c| / (255 W H)
 *                       (W, H >= 16, W H <= 16,777,216);
 *                     dHash: 8 rows x 9 columns of cells, bit (r, c) = cell mean
 *                       (r, c) > cell mean (r, c+1), d = Hamming distance / 64
 *                       (W >= 9, H >= 8).
 *                     scene change detection + H-diff: the histogram rule
 *                       unchanged, and a frame is also kept (code
 *                       COFIE_KEEP_SCENE, moving r(t)) at a scene change found
 *                       by twin comparison of the adjacent histogram
 *                       differences SD_t = d(c_t, c_{t-1}): a cut when
 *                       SD_t >= scd_cut; frames with scd_gradual <= SD_t <
 *                       scd_cut form a run whose summed SD is a gradual
 *                       transition at the frame where the sum first reaches
 *                       scd_cut; a cut or SD_t < scd_gradual ends the run.
 *                       Comparisons are fp32(L1 numerator) / fp32(2 W H).
 *                       Streams of this signal cannot be sharded.
 *                     hist_out of cofie_ngff_push_ex then receives the signal's
 *                     feature rows (cofie_ngff_feature_words uint32 per frame).
 *   scd_cut, scd_gradual
 *                     the twin-comparison thresholds T_b, T_s of the scene
 *                     change signal (non-NaN); defaults 0.30f and 0.10f.
 *   max_stream_frames frames per stream that the retention record covers
 *                     (cofie_ngff_candidates), rounded up to a multiple of 32;
 *                     0 picks the default, 1048576 (9.7 h at 30 frames/s). The
 *                     record takes ceil(max_stream_frames / 32) * 4 bytes of
 *                     device memory per stream (128 KiB at the default).
 */
typedef struct {
  uint32_t width, height;
  uint32_t bins;
  uint32_t l_max;
  uint32_t m_min;
  float tau;
  uint32_t luma_w[3];
  uint32_t luma_den;
  uint32_t max_streams;
  uint32_t max_frames_per_push;
  int32_t device;
  uint64_t host_stage_bytes;
  uint32_t signal;
  float scd_cut;
  float scd_gradual;
  uint32_t max_stream_frames;
} cofie_ngff_params;

/* One stream's frames in a batched push (see cofie_ngff_push_batch). */
typedef struct {
  uint32_t stream;        /* stream index, < max_streams; distinct within one batch */
  uint32_t n;             /* number of frames, may be 0 */
  const uint8_t* frames;  /* n frames: device memory (16-byte aligned) or host memory */
  float* scores_out;      /* n floats, device or host memory, or NULL */
  uint8_t* keep_out;      /* n keep codes, device or host memory, or NULL */
} cofie_ngff_push_desc;

/* uint32 words per frame of the handle's signal features (bins for the histogram). */
uint32_t cofie_ngff_feature_words(const cofie_ngff_t* h);

/* Fills *p with the paper's defaults for a width x height stream. */
void cofie_ngff_default_params(cofie_ngff_params* p, uint32_t width, uint32_t height);

/*
 * Creates a handle: validates *p and allocates the device state of
 * max_streams streams (a ring of the last L_max histograms each) and the
 * scratch for max_frames_per_push frames. Synchronous. On success *out owns
 * the allocations until cofie_ngff_destroy. Errors: COFIE_EINVAL (bad
 * parameter; *out untouched), COFIE_ENOMEM, COFIE_ECUDA.
 */
int cofie_ngff_create(const cofie_ngff_params* p, cofie_ngff_t** out);

/* Frees everything the handle owns (after synchronising its device). NULL is a no-op. */
void cofie_ngff_destroy(cofie_ngff_t* h);

/*
 * Pushes n new frames of stream `stream` (Sec. 3.2: the next frames of the
 * sampled prefix V_{1:T}) and decides each one.
 *   frames      n frames (3 W H bytes each), device or host memory.
 *   scores_out  n floats or NULL: s = max(s_adj, s_ref) per frame (Eq. 4);
 *               0 for the stream's first frame.
 *   keep_out    n bytes or NULL: keep code per frame (COFIE_KEEP_*).
 * n == 0 is a no-op. Splitting a stream into pushes of any sizes gives the
 * same results as one push. Errors: COFIE_EINVAL (null handle or frames with
 * n > 0, stream out of range), COFIE_ECUDA.
 *
 * CUDA graphs: a push whose frames and outputs are all device memory (or
 * NULL outputs) may be enqueued on a stream that is capturing into a CUDA
 * graph; each launch of the graph then decides the next n frames of the
 * stream, reading the frames and writing the outputs at the addresses given
 * at capture, exactly as an ordinary push at that point would. Every push
 * leaves the library's scratch as it found it, so captured and ordinary
 * pushes may be interleaved on one handle. Host memory while capturing is
 * COFIE_EINVAL. Frames decided by graph launches are not counted by
 * cofie_ngff_frames_seen, and kernel timing (cofie_ngff_profile_reset) skips
 * captured pushes.
 */
int cofie_ngff_push(cofie_ngff_t* h, uint32_t stream, const uint8_t* frames, uint32_t n,
                    float* scores_out, uint8_t* keep_out, void* cuda_stream);

/*
 * cofie_ngff_push, and also writes the integer histograms c_t of the n frames
 * to hist_out (n * bins uint32, row-major, device or host memory; NULL skips).
 * sum_b c_t[b] = W H for every frame.
 */
int cofie_ngff_push_ex(cofie_ngff_t* h, uint32_t stream, const uint8_t* frames, uint32_t n,
                       float* scores_out, uint8_t* keep_out, uint32_t* hist_out, void* cuda_stream);

/*
 * Pushes frames of several streams in one set of launches (serving many
 * concurrent streams). desc[i] is as in cofie_ngff_push for stream
 * desc[i].stream; streams distinct within the call; nd <=
 * COFIE_NGFF_MAX_BATCH and the total frame count <= max_frames_per_push.
 * Frames and outputs may be device or host memory, descriptor by descriptor:
 * the host frames of one call are copied (one copy per descriptor, on the
 * handle's copy stream) into one of the two staging buffers, so together
 * they must fit host_stage_bytes (COFIE_EINVAL otherwise); host outputs are
 * copied back on cuda_stream after the selection. Equivalent to one
 * cofie_ngff_push per descriptor. With device frames and outputs only, the
 * call is capturable into a CUDA graph as cofie_ngff_push is (host memory
 * while capturing is COFIE_EINVAL). Errors: COFIE_EINVAL, COFIE_ENOMEM (the
 * staging buffers, allocated on first use), COFIE_ECUDA.
 */
int cofie_ngff_push_batch(cofie_ngff_t* h, const cofie_ngff_push_desc* desc, uint32_t nd, void* cuda_stream);

/*
 * Closes stream `stream` at the frames pushed so far (Sec. 3.2, the
 * retention safeguards that need the end of the prefix) and
 * writes its candidate set S_c as ascending frame indices. With T the number
 * of frames the stream has been pushed when the call runs on cuda_stream
 * (read on the device, so the call may be captured into a CUDA graph after
 * the pushes it closes), S_c holds every frame t < T-1 that was retained
 * (nonzero keep code), the last frame T-1, and -- when that leaves fewer
 * than M_min frames -- the uniformly spaced frames
 * round(i (T-1) / (M_min - 1)), i = 0..M_min-1, rounded half up.
 * The frames come from the stream's retention record: one bit per frame,
 * set on the device by every push (and shard commit) as it decides the
 * frame, so the caller needs to keep no keep codes. The stream is not
 * changed: pushes may continue and a later call closes a longer prefix.
 *   idx_out  room for `cap` uint32 indices (NULL when cap == 0): device
 *            memory, or host memory together with a host m_out (the first
 *            such call allocates a device buffer of max_stream_frames
 *            indices, kept until cofie_ngff_destroy). Only the first
 *            min(|S_c|, cap) indices are written.
 *   m_out    |S_c| (also when it exceeds cap): device memory (asynchronous)
 *            or host memory (the call then synchronises cuda_stream; not
 *            while capturing).
 * T == 0 gives |S_c| = 0. A stream that has been pushed more than
 * max_stream_frames frames has no complete record: COFIE_EINVAL when the
 * handle knows it on the host, otherwise m_out = 0 and cofie_ngff_status
 * reports COFIE_EDEVICE. After cofie_ngff_reset the record starts empty;
 * cofie_ngff_state_save/load carry it; after cofie_ngff_shard_commit it holds
 * the committed shard's frames only (close a sharded stream with
 * cofie_ngff_candidates_from_keep over the shards' keep codes). M_min is the
 * handle's m_min. Errors: COFIE_EINVAL, COFIE_ENOMEM, COFIE_ECUDA.
 */
int cofie_ngff_candidates(cofie_ngff_t* h, uint32_t stream, uint32_t* idx_out, uint32_t cap, uint32_t* m_out,
                          void* cuda_stream);

/*
 * The same candidate set S_c for a prefix of T frames given as keep codes
 * (Sec. 3.2): every frame t < T-1 with a nonzero keep code, the last frame
 * T-1, and the M_min uniform fill as above.
 *   keep     T keep codes of frames 0..T-1 (for example the concatenated
 *            keep_out of a stream's pushes, or of a sharded stream's
 *            shards), device memory.
 *   idx_out  room for T uint32 indices, device memory.
 *   m_out    |S_c|, device memory (asynchronous) or host memory (the call then
 *            synchronises cuda_stream).
 * T == 0 gives |S_c| = 0. Errors: COFIE_EINVAL, COFIE_ECUDA.
 */
int cofie_ngff_candidates_from_keep(cofie_ngff_t* h, const uint8_t* keep, uint32_t T, uint32_t* idx_out,
                                    uint32_t* m_out, void* cuda_stream);

/*
 * Copies the m frames idx[0..m) of `frames` back to back into `out`: the
 * frames S_c that go on to the vision encoder (Sec. 3.2: the encoder
 * sees the candidate frames and no others).
 *   frames   n_frames frames of 3 W H bytes: device memory, or pinned host
 *            memory (read by the kernel over the host link through the
 *            device's mapping of it; pageable host memory is COFIE_EINVAL).
 *   idx      m frame indices, device memory (for example the idx_out of cofie_ngff_candidates).
 *   out      m * 3 W H bytes, device memory, not overlapping frames.
 * An index >= n_frames is skipped and reported as COFIE_EDEVICE by
 * cofie_ngff_status. Errors: COFIE_EINVAL, COFIE_ECUDA.
 */
int cofie_ngff_gather(cofie_ngff_t* h, const uint8_t* frames, uint32_t n_frames, const uint32_t* idx, uint32_t m,
                      uint8_t* out, void* cuda_stream);

/*
 * Checkpoint and resume of one stream. The saved state is everything a later
 * push depends on (Sec. 3.2: r(t) enters only through the gap t - r(t), and
 * distances reach back at most L_max frames), and the retention record that
 * cofie_ngff_candidates reads: a 64-byte header (format tag "NGFS", version 3,
 * width, height, bins, l_max, signal, frames seen t, current gap g, the
 * scene-change signal's open run sum, the record's word count) followed by
 * the ring of the last l_max feature rows (l_max * cofie_ngff_feature_words
 * uint32, slot i holds the frame t' with t' mod l_max == i; for l_max == 0
 * two rows, the previous frame's and the current reference frame's), then
 * the record (ceil(max_stream_frames / 32) uint32, bit t of word t / 32 set
 * when frame t was retained).
 *   cofie_ngff_state_bytes   the size of that buffer.
 *   cofie_ngff_state_save    writes stream `stream`'s state to buf (device or
 *                            host memory; host memory synchronises cuda_stream).
 *   cofie_ngff_state_load    restores a saved state into stream `stream` of a
 *                            handle with the same width, height, bins, l_max,
 *                            signal and max_stream_frames (COFIE_EINVAL otherwise);
 *                            pushes and candidate sets that follow behave exactly
 *                            as if the saved stream had continued.
 */
size_t cofie_ngff_state_bytes(const cofie_ngff_t* h);
int cofie_ngff_state_save(cofie_ngff_t* h, uint32_t stream, void* buf, void* cuda_stream);
int cofie_ngff_state_load(cofie_ngff_t* h, uint32_t stream, const void* buf, void* cuda_stream);

/*
 * Sharding one stream across GPUs or machines. The decision of frame t
 * depends on the past only through the gap g = t - r(t), which lies in
 * [1, L_max], and through the histograms of the L_max frames before t
 * (Sec. 3.2, Eqs. 3-5). So contiguous shards of one stream can be prepared
 * independently, in any order or in parallel, and decided afterwards:
 *   1. cofie_ngff_shard_prepare(h, stream, frames, n_halo, n, t0, map_out):
 *      `frames` holds the halo (the n_halo = min(t0, L_max) frames just before
 *      the shard) followed by the shard's n frames (device memory); t0 is the
 *      stream index of the shard's first frame. Computes the shard's
 *      histograms, distances and keep bits and writes its gap map: map_out[g-1]
 *      (L_max uint16, device or host memory) is the gap after the shard's last
 *      frame when the shard is entered with gap g. For t0 == 0 all entries are
 *      equal (frame 0 is a first frame).
 *   2. The caller chains the maps in stream order: the entry gap of the next
 *      shard is map[entry - 1] of the previous one (any entry for t0 == 0).
 *   3. cofie_ngff_shard_commit(h, stream, entry_gap, scores_out, keep_out):
 *      emits the shard's scores and keep codes (n each, device or host memory)
 *      and leaves the stream as after pushing frames [0, t0 + n).
 * Steps 1 and 3 of one shard use the same handle and stream, with no other
 * call on that handle between them; n_halo + n <= max_frames_per_push.
 * Errors: COFIE_EINVAL, COFIE_ECUDA.
 */
int cofie_ngff_shard_prepare(cofie_ngff_t* h, uint32_t stream, const uint8_t* frames, uint32_t n_halo, uint32_t n,
                             uint64_t t0, uint16_t* map_out, void* cuda_stream);
int cofie_ngff_shard_commit(cofie_ngff_t* h, uint32_t stream, uint32_t entry_gap, float* scores_out, uint8_t* keep_out,
                            void* cuda_stream);

/* Restarts stream `stream` at t = 0 (its next frame is a first frame) and
 * empties its retention record (one small kernel on cuda_stream). */
int cofie_ngff_reset(cofie_ngff_t* h, uint32_t stream, void* cuda_stream);

/*
 * Synchronises cuda_stream and reports device-side failures of earlier
 * calls on the handle: COFIE_ETIMEOUT if a bounded wait inside a kernel ran
 * out (the affected results are invalid), COFIE_EDEVICE if a gather index
 * was outside its frames or a candidate set was asked of a stream that had
 * run past its retention record, COFIE_ECUDA on a CUDA error, COFIE_OK
 * otherwise.
 * Clears the device error word.
 */
int cofie_ngff_status(cofie_ngff_t* h, void* cuda_stream);

/*
 * Number of frames stream `stream` has been pushed since creation or its
 * last reset, as enqueued (host-side count, no synchronisation; launches of
 * a CUDA graph that holds captured pushes are not counted).
 */
int cofie_ngff_frames_seen(const cofie_ngff_t* h, uint32_t stream, uint64_t* t_out);

/*
 * Test hooks for the failure paths (no counterpart in the paper). Neither
 * faults, traps or hangs a GPU.
 *   cofie_ngff_debug_fail_alloc  after >= 0: that many further device
 *                                allocations of the library succeed and the
 *                                next one fails (cofie_ngff_create then returns
 *                                COFIE_ENOMEM and frees what it had taken; a
 *                                push from host memory whose staging buffer
 *                                fails returns COFIE_ENOMEM); the hook then
 *                                switches itself off. after < 0 switches it off.
 *                                Process-wide, not thread-safe against creates.
 *   cofie_ngff_debug_wait        enqueues a one-thread kernel that waits, with
 *                                the streaming kernel's bounded mbarrier wait,
 *                                for a phase nothing completes; after
 *                                timeout_ns (<= 1 s, else COFIE_EINVAL) it sets
 *                                the same error bit a stalled consumer sets and
 *                                returns, so cofie_ngff_status then reports
 *                                COFIE_ETIMEOUT and clears it; the context and
 *                                the handle stay usable.
 */
void cofie_ngff_debug_fail_alloc(int32_t after);

/* 1 if this library is the checked build (compiled with -DCOFIE_DEBUG_CHECKS=1):
 * its kernels check computed indices against their launch arguments, skip an
 * access that fails, and cofie_ngff_status then reports COFIE_EDEVICE (error
 * bit 16). It stands in for a memory checker; normal builds return 0 and
 * carry no checks. */
int cofie_ngff_checked_build(void);
int cofie_ngff_debug_wait(cofie_ngff_t* h, uint64_t timeout_ns, void* cuda_stream);

/*
 * Diagnostic: applies the fast histogram kernel's own per-pixel grayscale and
 * bin functions to n_pixels RGB triples (device memory, 3 * n_pixels bytes,
 * n_pixels a multiple of 4) and writes one bin index per pixel to bins_out
 * (device memory, n_pixels bytes). Lets tests check the device binning of
 * every RGB triple. COFIE_EINVAL if the handle's parameters only run the
 * generic kernel.
 */
int cofie_ngff_debug_bins(cofie_ngff_t* h, const uint8_t* pixels, uint64_t n_pixels, uint8_t* bins_out,
                          void* cuda_stream);

/*
 * Launch counters and kernel timing (a tracing aid). Counters run always;
 * with timing on, every launch of the histogram kernel, and every pair of
 * distance + scan launches, is bracketed by two CUDA events recorded on the
 * stream it is launched on.
 */
typedef struct {
  uint64_t hist_launches;   /* histogram-kernel launches since the last reset */
  uint64_t select_launches; /* distance + scan kernel launches since the last reset */
  uint64_t hist_bytes;      /* algorithmic bytes of those histogram launches: frame bytes read + counts written */
  uint64_t hist_timed;      /* histogram launches that were event-timed */
  double hist_ms;           /* summed event-timed histogram-kernel durations, milliseconds */
  uint64_t select_timed;    /* distance + scan launch pairs that were event-timed */
  double select_ms;         /* summed event-timed durations of those pairs, milliseconds */
  uint64_t other_launches;  /* launches of the stream-reset, candidate and gather kernels */
} cofie_ngff_profile;

/* Zeroes the counters; time_kernels != 0 turns event timing on, 0 off. */
int cofie_ngff_profile_reset(cofie_ngff_t* h, int time_kernels);

/* Waits for the timed launches and writes the counters to *out. */
int cofie_ngff_profile_read(cofie_ngff_t* h, cofie_ngff_profile* out);

/*
 * Selection without device allocation (the paper has no counterpart: this is
 * an interface for callers that may not allocate device memory, such as a
 * process whose device memory belongs to another framework's pooling
 * allocator under a hard cap, a media or ingest plugin that is handed buffers
 * but may not allocate, or a latency-bound pipeline that fixes its memory at
 * start-up because cudaMalloc can synchronise the device).
 *
 * Decides the first n frames of a fresh stream from their integer histograms
 * and writes the same scores and keep codes cofie_ngff_push_ex gives on a new
 * stream of the histogram signal (no scene changes). Needs no handle and
 * allocates nothing: its working tables live in a static device array of
 * 1048576 32-bit words (4 MiB) that every GPU loading the library holds until
 * the process exits. Two launches on cuda_stream: a grid computes every
 * frame's windowed distances, then one CTA scans them (0.22 ms at the
 * largest n for L_max = 30 on GB300).
 *   p           width, height, bins, l_max and tau are used; signal must be
 *               COFIE_SIGNAL_HISTOGRAM (else COFIE_EINVAL); the rest is ignored.
 *   hist        n * bins uint32 counts, row-major, device memory on the
 *               current device (for example hist_out of cofie_ngff_push_ex).
 *   n           frames; n * (l_max + ceil(l_max / 32)) must not exceed
 *               1048576 (33825 frames at l_max = 30), else COFIE_EINVAL.
 *   scores_out, keep_out
 *               n floats / n bytes in device memory on the current device, or NULL.
 *   err, err_cap  optional buffer that receives the error text (may be NULL).
 * Runs on the calling thread's current device, asynchronously on cuda_stream.
 * The first call on a device looks up the array's device address and sets
 * the kernel's shared-memory limit (no allocation); make that first call
 * before any stream capture. All calls share the array and it keeps the
 * previous call's contents (each call overwrites every entry it reads), so
 * calls that overlap on the GPU race: serialise them.
 * Errors: COFIE_EINVAL, COFIE_ECUDA.
 */
int cofie_ngff_select_static(const cofie_ngff_params* p, const uint32_t* hist, uint32_t n, float* scores_out,
                             uint8_t* keep_out, char* err, size_t err_cap, void* cuda_stream);

/* ------------------------------------------------------------------------
 * Query-specific evidence refinement (QER, CoFiE Sec. 3.3, Eqs. 6-8): the
 * fine stage that ranks the NGFF candidates by text-to-vision attention.
 *
 *   a_ij = (1/H) sum_h <q_i^h, k_j^h> / sqrt(d_h)        (Eq. 6)
 *   w_f  = mean over the frame's tokens of max_i a_ij    (Eq. 7)
 *   S_e  = the max(1, round(rho m)) best frames by w_f   (Eq. 8)
 *
 * Query head h reads key head h / (H / H_kv) (grouped key/value heads, as in
 * the attention). The query heads of each group are summed in fp32 and
 * rounded to bf16; the contraction runs on the tensor cores in bf16 with fp32
 * accumulation. round() rounds half to even; equal scores rank by lower
 * frame index; S_e is returned in time order. A query of more than 256 text
 * tokens is split into ceil(n_text / 256) equal blocks scored in successive
 * passes over the keys, each pass keeping the running max of Eq. 7's inner
 * max (the keys are read once per pass).
 * ------------------------------------------------------------------------ */
typedef struct cofie_qer cofie_qer_t;

typedef struct {
  uint32_t n_text;           /* text tokens |Q|, 1..4096 (scored in passes of at most 256) */
  uint32_t n_heads;          /* H query heads */
  uint32_t n_kv_heads;       /* H_kv key heads, divides H */
  uint32_t head_dim;         /* d_h; H_kv * d_h a multiple of 64, at most 16384 */
  uint32_t max_frames;       /* largest |S_c| per call */
  uint32_t tokens_per_frame; /* |V_f|, the same for every frame */
  float rho;                 /* keep ratio, [0, 1] */
  int32_t device;            /* CUDA device ordinal, or -1 for the current device */
  uint32_t kernel;           /* scoring kernel: COFIE_QER_KERNEL_* */
} cofie_qer_params;

/* Scoring kernels: the paired-SM one (clusters of two CTAs, one M = 256 MMA
 * per pair) needs the text block (n_text, or for n_text > 256 its blocks,
 * which are padded to 32) rounded up to 16 to be a multiple of 32; AUTO takes
 * it when it applies and the 256-token tiles of a run either fit one per
 * co-resident pair (76 on GB300) or exceed one wave of the one-SM kernel (one
 * per SM). The results of the two agree up to the order of fp32 accumulation
 * inside the tensor cores. */
#define COFIE_QER_KERNEL_AUTO 0
#define COFIE_QER_KERNEL_ONE_SM 1
#define COFIE_QER_KERNEL_PAIR 2

/* Validates *p and allocates the scratch (group-summed queries, per-token
 * maxima, frame scores). Synchronous. Errors: COFIE_EINVAL, COFIE_ENOMEM, COFIE_ECUDA. */
int cofie_qer_create(const cofie_qer_params* p, cofie_qer_t** out);

void cofie_qer_destroy(cofie_qer_t* h);

/* COFIE_QER_KERNEL_PAIR if the handle can run the paired-SM kernel (AUTO
 * then picks it per run as described above; PAIR always), else
 * COFIE_QER_KERNEL_ONE_SM (0 for NULL). */
uint32_t cofie_qer_kernel_in_use(const cofie_qer_t* h);

/*
 * Ranks n_frames candidate frames (Eqs. 6-8).
 *   q        bf16 [n_text][H][d_h], device memory.
 *   k        bf16 [n_frames * tokens_per_frame][H_kv][d_h], device memory,
 *            16-byte aligned; frame f owns tokens [f T, (f+1) T).
 *   w_out    n_frames floats (w_f), device memory, or NULL.
 *   sel_out  room for n_frames uint32 frame indices (S_e, ascending), device memory.
 *   k_out    |S_e|: device memory (asynchronous) or host memory (synchronises).
 * With k_out in device memory the call may be captured into a CUDA graph;
 * each launch of the graph ranks the q and k then at the captured addresses
 * (kernel timing skips captured calls; a host k_out while capturing is
 * COFIE_EINVAL). Errors: COFIE_EINVAL, COFIE_ECUDA; device-side waits are
 * reported by cofie_qer_status.
 */
int cofie_qer_run(cofie_qer_t* h, const uint16_t* q, const uint16_t* k, uint32_t n_frames, float* w_out,
                  uint32_t* sel_out, uint32_t* k_out, void* cuda_stream);

/* Synchronises cuda_stream; COFIE_ETIMEOUT if a bounded device wait ran out;
 * in a build with -DCOFIE_DEBUG_CHECKS=1, COFIE_EDEVICE if a kernel found its
 * shared-memory rings or TMEM accumulators outside what the launch gave it
 * (it then ran no tile). */
int cofie_qer_status(cofie_qer_t* h, void* cuda_stream);

/* Launch counter and CUDA-event timing of the scoring (tensor-core) kernel:
 * reset zeroes the counters (time_kernels != 0 brackets every launch with two
 * events on its stream); read waits for the timed launches and reports the
 * launches, the timed launches, their summed milliseconds, the contraction's
 * FLOPs (2 N n_visual D, N the padded text count) and the key bytes read. */
int cofie_qer_profile_reset(cofie_qer_t* h, int time_kernels);
int cofie_qer_profile_read(cofie_qer_t* h, uint64_t* launches, uint64_t* timed, double* score_ms, double* flops,
                           double* key_bytes);

/* Last error of h, or of the last failed cofie_qer_create when h is NULL. Never NULL. */
const char* cofie_qer_last_error(const cofie_qer_t* h);

/* Text of the last error on this handle (empty string if none). Never NULL. */
const char* cofie_ngff_last_error(const cofie_ngff_t* h);

/* Text of the last error from a call that had no valid handle (create). Never NULL. */
const char* cofie_ngff_global_error(void);

#ifdef __cplusplus
}
#endif

#endif /* COFIE_NGFF_H */
