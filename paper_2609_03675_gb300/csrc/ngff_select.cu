// K2 and K3: novelty scores and the keep/drop decisions (CoFiE Sec. 3.2,
// Eqs. 2-5).
//
// The decision for frame t depends on r(t), the most recent retained frame,
// through the gap g = t - r(t). Because the gap rule (Eq. 5, second term)
// retains a frame whenever g reaches L_max, g always lies in [1, L_max], so
// every distance the rule can need is one of the L_max windowed distances
// d(h_t, h_{t-k}), k = 1..L_max. That turns the sequential rule into:
//
// K2 (one warp per frame, lane = lag): L1[t][k-1] = sum_b |c_t[b] - c_{t-k}[b]|
//    for every k (Eq. 2 up to the factor 1/(2N)), reading h_{t-k} from this
//    push's histograms or from the stream's ring of the last L_max
//    histograms, and the keep decision for every possible gap g as one bit:
//    keep_t(g) = fp32(max(L1[t][0], L1[t][g-1])) / fp32(2N) >= tau_h
//                (Eqs. 3-4: s = max(s_adj, s_ref))
//                or g >= L_max (Eq. 5).
//
// K3 (one 1024-thread CTA per stream): the frame-to-frame gap update
//    g' = keep_t(g) ? 1 : g + 1 is a map on [1, L_max]. Each warp composes
//    the maps of a contiguous run of frames for all entry gaps at once (lane
//    = entry gap), thread 0 chains the 32 run maps, each warp replays its run
//    from the resolved entry gap, and all threads then emit score and keep
//    code per frame. The stream state (frames seen, current gap, ring of the
//    last L_max histograms) is updated at the end, and the push's histogram
//    rows are zeroed for the next push unless the caller asked for them.
//
// Small pushes (at most kSmallMax frames per stream) run K2 and K3 as one
// kernel: the same CTA first computes its stream's distances, then scans.
// With at most kWalkMaxFrames frames per stream and L_max <= kWalkMaxLmax the
// push is smaller still and a lighter kernel decides it (select_walk_kernel):
// one 256-thread CTA per stream stages the stream's ring and the push's rows
// in shared memory, keeps the distances and keep bits there, and walks the
// rule in frame order from the stream's gap, which for so few frames is
// shorter than composing gap maps.
#include "ngff_common.cuh"

namespace cofie {
namespace {

constexpr int kWinWarps = 8;
constexpr int kScanThreads = 1024;
constexpr int kScanWarps = kScanThreads / 32;
constexpr uint32_t kScanTile = 4096;  // frames per shared-memory tile
constexpr uint32_t kSmallMax = 64;    // frames per stream segment for the fused small-push kernel
constexpr int kWalkThreads = 256;
constexpr uint32_t kWalkMaxFrames = 64;
constexpr uint32_t kWalkMaxLmax = 64;
constexpr size_t kWalkStageBudget = 48 * 1024;  // shared memory a walk CTA takes without opting in

__device__ __forceinline__ uint32_t absdiff(uint32_t a, uint32_t b) { return a > b ? a - b : b - a; }

// K2's work for one frame (row of the push), done by one warp. Lane k-1 sums
// |c_t - c_{t-k}| over all bins of row t-k (16-byte loads when B % 4 == 0),
// so the warp's loads are independent and in flight together; the keep bit
// for gap g = k is decided in the same lane.
template <bool kVec4>
__device__ __forceinline__ void window_row(uint32_t row, uint32_t lane, const Segment& sg, const SelectArgs& a,
                                           const uint32_t* __restrict__ hist, const uint32_t* __restrict__ ring,
                                           unsigned long long t0, uint32_t* __restrict__ l1,
                                           uint32_t* __restrict__ mask) {
  const uint32_t stream = sg.stream;
  const uint32_t j = row - sg.row0;
  const unsigned long long t = t0 + j;
  const uint32_t B = a.bins, L = a.l_max;
  const uint32_t* ct = hist + static_cast<uint64_t>(row) * B;
  uint32_t l_adj = 0;
  for (uint32_t w = 0; w < a.mask_words; ++w) {
    const uint32_t k = 32 * w + lane + 1;  // this lane's lag, and the gap it decides
    const bool valid = k <= L && k <= t;
    const uint32_t* src = ct;
    if (valid)
      src = (k <= j + sg.halo) ? (COFIE_BOUND(k <= row) ? hist + static_cast<uint64_t>(row - k) * B : ct)
                               : ring + (static_cast<uint64_t>(stream) * L + (t - k) % L) * B;
    uint32_t d = 0;
    if (kVec4) {
      const uint4* c4 = reinterpret_cast<const uint4*>(ct);
      const uint4* s4 = reinterpret_cast<const uint4*>(src);
#pragma unroll 8
      for (uint32_t q = 0; q < B / 4; ++q) {
        const uint4 x = c4[q], y = s4[q];
        d += absdiff(x.x, y.x) + absdiff(x.y, y.y) + absdiff(x.z, y.z) + absdiff(x.w, y.w);
      }
    } else if (a.dist_kind == 1) {  // Hamming distance of bit vectors (dHash)
      for (uint32_t b = 0; b < B; ++b) d += __popc(ct[b] ^ src[b]);
    } else {
#pragma unroll 4
      for (uint32_t b = 0; b < B; ++b) d += absdiff(ct[b], src[b]);
    }
    if (!valid) d = 0;
    if (w == 0) l_adj = __shfl_sync(0xffffffffu, d, 0);  // lag 1
    if (k <= L) l1[static_cast<uint64_t>(row) * L + k - 1] = d;
    bool keep = false;
    if (k <= L) {
      const float s = __fdiv_rn(static_cast<float>(max(l_adj, d)), a.two_n);
      keep = (s >= a.tau) || (k >= L);
    }
    const uint32_t m = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) mask[static_cast<uint64_t>(row) * a.mask_words + w] = m;
  }
}

template <bool kVec4>
__global__ void __launch_bounds__(kWinWarps * 32) window_kernel(SegTable segs, SelectArgs a,
                                                                const uint32_t* __restrict__ hist,
                                                                const uint32_t* __restrict__ ring,
                                                                const StreamState* __restrict__ state,
                                                                uint32_t* __restrict__ l1, uint32_t* __restrict__ mask) {
  pdl_trigger();
  pdl_wait();  // the histograms of the first-stage kernel before it
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t row = blockIdx.x * kWinWarps + warp;
  if (row >= segs.rows) return;
  uint32_t seg = 0;
  while (seg + 1 < segs.count && row >= segs.s[seg + 1].row0) ++seg;
  const Segment sg = segs.s[seg];
  if (row < sg.row0) return;  // halo rows: history only, no decision
  window_row<kVec4>(row, lane, sg, a, hist, ring, state[sg.stream].t, l1, mask);
}

template <bool kOneWord>
__device__ __forceinline__ uint32_t step_gap(const uint32_t* m, uint32_t g) {
  const uint32_t word = kOneWord ? m[0] : m[(g - 1) >> 5];
  return ((word >> ((g - 1) & 31)) & 1u) ? 1u : g + 1u;
}

// (reset, sum) pairs of the twin comparison's run accumulator over a span of
// frames: "reset" marks that the run ended inside the span, "sum" is the L1
// numerator summed since the last end. Spans combine left to right:
static_assert(kScanTile == 4 * kScanThreads, "scd_tile: four frames per thread");

struct RunSum {
  uint32_t reset;
  unsigned long long sum;
};
__device__ __forceinline__ RunSum run_cat(RunSum a, RunSum b) {
  return RunSum{a.reset | b.reset, b.reset ? b.sum : a.sum + b.sum};
}
__device__ __forceinline__ RunSum run_shfl_up(RunSum v, uint32_t off) {
  return RunSum{__shfl_up_sync(0xffffffffu, v.reset, off), __shfl_up_sync(0xffffffffu, v.sum, off)};
}

// Scene changes (signal SCD) of the m <= 4 kScanThreads frames of one tile:
// twin comparison of the adjacent differences SD_t = L1[t][lag 1] / 2N. A cut
// (SD >= T_b) and a low difference (SD < T_s) end the run; a middle
// difference adds to it; a gradual transition is found where the run's sum
// first reaches T_b. The run sums are a block-wide segmented prefix sum
// (thread: 4 consecutive frames; warps and the block by shuffles and shared
// memory) entered with the sum carry_in open before the tile. A scene-change
// frame gets every keep bit of its mask row and its bit in sflag. Returns the
// sum open after the tile (the same in every thread).
__device__ __forceinline__ unsigned long long scd_tile(const uint32_t* __restrict__ l1, uint64_t row_first,
                                                       uint32_t m, const SelectArgs& a, uint32_t* smask,
                                                       uint32_t* sflag, unsigned long long carry_in) {
  __shared__ uint32_t wreset[kScanWarps + 1];
  __shared__ unsigned long long wsum[kScanWarps + 1];
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t W = a.mask_words, L = a.l_max;
  uint32_t adj[4], cls[4];  // cls: 2 cut, 1 middle, 0 low (or past the tile)
  RunSum loc[4];
  RunSum acc{0u, 0ull};
#pragma unroll
  for (uint32_t k = 0; k < 4; ++k) {
    const uint32_t f = 4 * tid + k;
    adj[k] = f < m ? l1[(row_first + f) * L] : 0u;
    const float sd = __fdiv_rn(static_cast<float>(adj[k]), a.two_n);
    cls[k] = f >= m ? 0u : (sd >= a.scd_cut ? 2u : (sd >= a.scd_grad ? 1u : 0u));
    const RunSum e = f >= m ? RunSum{0u, 0ull}                                    // past the tile: identity
                            : (cls[k] == 1u ? RunSum{0u, adj[k]} : RunSum{1u, 0ull});  // joins / ends the run
    acc = run_cat(acc, e);
    loc[k] = acc;
  }
  RunSum incl = acc;  // inclusive over this warp's threads
#pragma unroll
  for (uint32_t off = 1; off < 32; off <<= 1) {
    const RunSum o = run_shfl_up(incl, off);
    if (lane >= off) incl = run_cat(o, incl);
  }
  if (lane == 31) {
    wreset[warp] = incl.reset;
    wsum[warp] = incl.sum;
  }
  __syncthreads();
  if (warp == 0) {  // exclusive scan of the warp totals; slot kScanWarps = the whole tile
    RunSum w{wreset[lane], wsum[lane]};
#pragma unroll
    for (uint32_t off = 1; off < 32; off <<= 1) {
      const RunSum o = run_shfl_up(w, off);
      if (lane >= off) w = run_cat(o, w);
    }
    const RunSum before = run_shfl_up(w, 1);
    __syncwarp();
    wreset[lane] = lane ? before.reset : 0u;
    wsum[lane] = lane ? before.sum : 0ull;
    if (lane == 31) {
      wreset[kScanWarps] = w.reset;
      wsum[kScanWarps] = w.sum;
    }
  }
  __syncthreads();
  RunSum ex = run_shfl_up(incl, 1);
  if (lane == 0) ex = RunSum{0u, 0ull};
  ex = run_cat(RunSum{wreset[warp], wsum[warp]}, ex);  // everything before this thread's frames
  const auto reaches = [&](unsigned long long x) { return __fdiv_rn(__ull2float_rn(x), a.two_n) >= a.scd_cut; };
#pragma unroll
  for (uint32_t k = 0; k < 4; ++k) {
    const uint32_t f = 4 * tid + k;
    if (f >= m) break;
    const RunSum pre = run_cat(ex, loc[k]);
    const unsigned long long run = pre.reset ? pre.sum : carry_in + pre.sum;  // the run's sum at f
    const bool scene = cls[k] == 2u || (cls[k] == 1u && reaches(run) && !reaches(run - adj[k]));
    if (scene) {
      for (uint32_t w = 0; w < W; ++w) smask[f * W + w] = 0xffffffffu;
      atomicOr(&sflag[f >> 5], 1u << (f & 31));
    }
  }
  return wreset[kScanWarps] ? wsum[kScanWarps] : carry_in + wsum[kScanWarps];
}

// K3's work for one stream segment, done by a whole 1024-thread CTA. sseg,
// t0, g0 and acc0 are the segment and its stream's state on entry (shared
// memory).
template <bool kOneWord>
__device__ __forceinline__ void scan_segment(const Segment& sseg, unsigned long long t0, uint32_t g0,
                                             unsigned long long acc0, const SelectArgs& a, const uint32_t* __restrict__ l1,
                                             const uint32_t* __restrict__ mask, uint32_t* __restrict__ hist,
                                             uint32_t* __restrict__ ring, StreamState* __restrict__ state,
                                             uint32_t* ssm, uint32_t* entry) {
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t W = a.mask_words, L = a.l_max, B = a.bins;
  uint32_t* smask = ssm;                                                // [kScanTile][W]
  uint16_t* sgap = reinterpret_cast<uint16_t*>(smask + kScanTile * W);  // [kScanTile]
  uint16_t* sexit = sgap + kScanTile;                                   // [kScanWarps][L]
  const uint32_t n = sseg.n, row0 = sseg.row0, stream = sseg.stream;
  if (n == 0) return;
  const uint32_t j_start = (t0 == 0) ? 1u : 0u;  // the stream's first frame is decided below
  uint32_t g_entry = (t0 == 0) ? 1u : g0;
  unsigned long long acc = (t0 == 0) ? 0ull : acc0;  // the scene-change run open before the segment
  __shared__ uint32_t sflag[kScanTile / 32];
  if (g_entry < 1u || g_entry > L) g_entry = L;  // the state only ever holds [1, L]

  for (uint32_t tile0 = j_start; tile0 < n; tile0 += kScanTile) {
    const uint32_t m = min(kScanTile, n - tile0);
    for (uint32_t i = tid; i < m * W; i += kScanThreads)
      smask[i] = mask[static_cast<uint64_t>(row0 + tile0) * W + i];
    if (a.scd)
      for (uint32_t i = tid; i < kScanTile / 32; i += kScanThreads) sflag[i] = 0;
    __syncthreads();
    if (a.scd) {
      acc = scd_tile(l1, static_cast<uint64_t>(row0 + tile0), m, a, smask, sflag, acc);
      __syncthreads();
    }
    const uint32_t run = (m + kScanWarps - 1) / kScanWarps;
    const uint32_t f0 = min(warp * run, m), f1 = min(f0 + run, m);
    // compose this warp's run of gap maps for every entry gap
    for (uint32_t gin = lane + 1; gin <= L; gin += 32) {
      uint32_t g = gin;
#pragma unroll 4
      for (uint32_t f = f0; f < f1; ++f) g = step_gap<kOneWord>(smask + f * W, g);
      (void)COFIE_BOUND(g >= 1 && g <= L);  // a gap stays in [1, L_max]
      sexit[warp * L + gin - 1] = static_cast<uint16_t>(g);
    }
    __syncthreads();
    if (tid == 0) {
      uint32_t g = g_entry;
      for (uint32_t w = 0; w < kScanWarps; ++w) {
        entry[w] = g;
        if (min(w * run, m) < min(w * run + run, m)) g = sexit[w * L + g - 1];
      }
      entry[kScanWarps] = g;
    }
    __syncthreads();
    if (lane == 0) {
      uint32_t g = entry[warp];
#pragma unroll 4
      for (uint32_t f = f0; f < f1; ++f) {
        sgap[f] = static_cast<uint16_t>(g);
        g = step_gap<kOneWord>(smask + f * W, g);
      }
    }
    __syncthreads();
    for (uint32_t base = 0; base < m; base += kScanThreads) {  // warps stay whole: the record takes a ballot
      const uint32_t f = base + tid;
      const uint32_t jj = tile0 + f;
      bool kept = false;
      if (f < m) {
        uint32_t g = sgap[f];
        if (!COFIE_BOUND(g >= 1 && g <= L)) g = 1;  // checked build: keep the L1 read in its row
        const uint64_t r = static_cast<uint64_t>(row0 + jj) * L;
        const uint32_t lm = max(l1[r], l1[r + g - 1]);
        const float s = __fdiv_rn(static_cast<float>(lm), a.two_n);
        const bool nov = s >= a.tau;
        const bool scene = a.scd && ((sflag[f >> 5] >> (f & 31)) & 1u);
        const uint8_t code = nov ? 1 : (scene ? 4 : (g >= L ? 2 : 0));
        if (sseg.scores) sseg.scores[jj] = s;
        if (sseg.keep) sseg.keep[jj] = code;
        kept = code != 0;
      }
      const uint32_t bits = __ballot_sync(0xffffffffu, kept);
      if (lane == 0 && a.record)
        record_bits(a.record + static_cast<uint64_t>(stream) * a.rec_words, a.rec_words, t0 + jj, bits);
    }
    g_entry = entry[kScanWarps];
    __syncthreads();
  }

  if (tid == 0) {
    if (t0 == 0) {  // first frame of the stream: always retained, score 0
      if (sseg.scores) sseg.scores[0] = 0.0f;
      if (sseg.keep) sseg.keep[0] = 3;
      if (a.record) record_bits(a.record + static_cast<uint64_t>(stream) * a.rec_words, a.rec_words, 0ull, 1u);
    }
    state[stream].t = t0 + n;
    state[stream].g = g_entry;
    state[stream].acc = acc;
  }
  // ring: histograms of the last min(n, L) frames of the push
  const uint32_t keep_n = min(n, L);
  for (uint32_t i = tid; i < keep_n * B; i += kScanThreads) {
    const uint32_t jj = n - keep_n + i / B, b = i % B;
    const uint64_t slot = (t0 + jj) % L;
    ring[(static_cast<uint64_t>(stream) * L + slot) * B + b] = hist[static_cast<uint64_t>(row0 + jj) * B + b];
  }
  if (a.zero_hist) {  // leave the push's histogram rows zeroed for the next push
    __syncthreads();
    for (uint64_t i = tid; i < static_cast<uint64_t>(n) * B; i += kScanThreads)
      hist[static_cast<uint64_t>(row0) * B + i] = 0;
  }
}

template <bool kOneWord>
__global__ void __launch_bounds__(kScanThreads) scan_kernel(SegTable segs, SelectArgs a,
                                                            const uint32_t* __restrict__ l1,
                                                            const uint32_t* __restrict__ mask,
                                                            uint32_t* __restrict__ hist, uint32_t* __restrict__ ring,
                                                            StreamState* __restrict__ state) {
  extern __shared__ __align__(16) uint32_t ssm[];
  __shared__ Segment sseg;
  __shared__ uint32_t entry[kScanWarps + 1];
  __shared__ unsigned long long s_t0, s_acc;
  __shared__ uint32_t s_g;
  pdl_wait();  // the distance and mask rows of the window kernel before it
  if (threadIdx.x == 0) {
    sseg = segs.s[blockIdx.x];
    s_t0 = state[sseg.stream].t;
    s_g = state[sseg.stream].g;
    s_acc = state[sseg.stream].acc;
  }
  __syncthreads();
  scan_segment<kOneWord>(sseg, s_t0, s_g, s_acc, a, l1, mask, hist, ring, state, ssm, entry);
}

// Small pushes: one CTA per stream segment computes the segment's windowed
// distances (one warp per frame) and then scans them.
template <bool kVec4, bool kOneWord>
__global__ void __launch_bounds__(kScanThreads) select_small_kernel(SegTable segs, SelectArgs a,
                                                                    uint32_t* __restrict__ hist,
                                                                    uint32_t* __restrict__ ring,
                                                                    StreamState* __restrict__ state,
                                                                    uint32_t* __restrict__ l1,
                                                                    uint32_t* __restrict__ mask) {
  extern __shared__ __align__(16) uint32_t ssm[];
  __shared__ Segment sseg;
  __shared__ uint32_t entry[kScanWarps + 1];
  __shared__ unsigned long long s_t0, s_acc;
  __shared__ uint32_t s_g;
  pdl_trigger();  // the next push's first-stage kernel may be scheduled; it waits for this grid before its work
  // Every read of device memory follows the wait: the histograms of the
  // first-stage kernel before this one, and the stream's state, which the
  // previous push's selection may still have been writing when that kernel
  // was scheduled.
  pdl_wait();
  if (threadIdx.x == 0) {
    sseg = segs.s[blockIdx.x];
    s_t0 = state[sseg.stream].t;
    s_g = state[sseg.stream].g;
    s_acc = state[sseg.stream].acc;
  }
  __syncthreads();
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (uint32_t j = warp; j < sseg.n; j += kScanWarps)
    window_row<kVec4>(sseg.row0 + j, lane, sseg, a, hist, ring, s_t0, l1, mask);
  __syncthreads();  // this CTA's distance and mask rows are visible to all its threads
  scan_segment<kOneWord>(sseg, s_t0, s_g, s_acc, a, l1, mask, hist, ring, state, ssm, entry);
}

// Small pushes, one 256-thread CTA per stream segment (n <= kWalkMaxFrames,
// L_max <= kWalkMaxLmax), in the order the rule states it:
//   0. (kStaged) the stream's ring of the last L_max rows and the push's own
//      rows are copied into shared memory in one coalesced pass, alongside
//      the read of the stream's state, so that everything after it reads
//      shared memory only;
//   1. windowed distances, a warp per frame, lane = lag k (the Eq. 2
//      numerators L1[j][k-1] = sum_b |c_t - c_{t-k}|), each lane starting at
//      a column rotated by its lane so a warp's 16-byte reads of different
//      rows fall in different banks, and the keep bit of every possible gap g
//      (Eqs. 3-5: fp32(max(L1[j][0], L1[j][g-1])) / fp32(2N) >= tau_h, or
//      g >= L_max), into shared memory;
//   2. one thread walks the frames in order from the stream's gap: frame j is
//      kept when its bit for the current gap is set (or, with scene changes,
//      when twin comparison of the adjacent differences finds one, with the
//      numerator thresholds that equal the fp32 decisions), and the gap
//      becomes 1 on a keep and g + 1 otherwise;
//   3. all threads emit scores and keep codes, note retained frames in the
//      stream's retention record, store the last L_max rows in the ring,
//      update the stream state and zero the push's rows for the next push.
// Without kStaged (rows too wide for the staging budget) the same steps read
// the rows from global memory.
template <bool kVec4, bool kStaged>
__global__ void __launch_bounds__(kWalkThreads) select_walk_kernel(SegTable segs, SelectArgs a,
                                                                   uint32_t* __restrict__ hist,
                                                                   uint32_t* __restrict__ ring,
                                                                   StreamState* __restrict__ state) {
  constexpr uint32_t kWarps = kWalkThreads / 32;
  extern __shared__ __align__(16) uint32_t wsm[];
  __shared__ unsigned long long s_t0, s_acc;
  __shared__ uint32_t s_g, s_slot0;
  pdl_trigger();  // the next push's first-stage kernel may be scheduled; it waits for this grid before its work
  pdl_wait();     // every device read follows: the histograms before it, and the state the last push left
  const Segment sg = segs.s[blockIdx.x];
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t n = sg.n, row0 = sg.row0, stream = sg.stream;
  const uint32_t B = a.bins, L = a.l_max, W = a.mask_words;
  if (n == 0) return;
  uint32_t* srows = wsm;                                   // kStaged: [L + n][B], ring slots then the push
  uint32_t* sl1 = wsm + (kStaged ? (L + n) * B : 0u);      // [n][L]
  uint32_t* smask = sl1 + n * L;                           // [n][W]
  uint32_t* sgap = smask + n * W;                          // [n]: gap, bit 31 a scene change
  const uint32_t* ring_s = ring + static_cast<uint64_t>(stream) * L * B;
  const uint32_t* hist_s = hist + static_cast<uint64_t>(row0) * B;
  if (tid == 0) {
    s_t0 = state[stream].t;
    s_acc = state[stream].acc;
    s_g = state[stream].g;
    s_slot0 = static_cast<uint32_t>(s_t0 % L);  // the ring slot of the push's first frame (one 64-bit division)
  }
  if (kStaged) {
    if (kVec4) {
      const uint32_t rq = L * B / 4, hq = n * B / 4;
      for (uint32_t i = tid; i < rq + hq; i += kWalkThreads)
        reinterpret_cast<uint4*>(srows)[i] =
            i < rq ? reinterpret_cast<const uint4*>(ring_s)[i] : reinterpret_cast<const uint4*>(hist_s)[i - rq];
    } else {
      for (uint32_t i = tid; i < (L + n) * B; i += kWalkThreads)
        srows[i] = i < L * B ? ring_s[i] : hist_s[i - L * B];
    }
  }
  __syncthreads();
  const unsigned long long t0 = s_t0;
  const int slot0 = static_cast<int>(s_slot0), Li = static_cast<int>(L);
  const uint32_t nq = B / 4, rot = kStaged && kVec4 ? lane % max(nq, 1u) : 0u;

  // 1. distances and keep bits
  for (uint32_t j = warp; j < n; j += kWarps) {
    const unsigned long long t = t0 + j;
    const uint32_t* ct = kStaged ? srows + (L + j) * B : hist_s + static_cast<uint64_t>(j) * B;
    uint32_t l_adj = 0;
    for (uint32_t w = 0; w < W; ++w) {
      const uint32_t k = 32 * w + lane + 1;
      const bool valid = k <= L && k <= t;
      const uint32_t* src = ct;
      if (valid) {
        if (k <= j) src = ct - static_cast<uint64_t>(k) * B;
        else {  // ring slot of frame t - k: (slot0 + j - k) mod L, with |j - k| < 2^7
          int slot = (slot0 + static_cast<int>(j) - static_cast<int>(k)) % Li;
          if (slot < 0) slot += Li;
          src = (kStaged ? srows : ring_s) + static_cast<uint32_t>(slot) * B;
        }
      }
      uint32_t d = 0;
      if (kVec4) {
        const uint4* c4 = reinterpret_cast<const uint4*>(ct);
        const uint4* s4 = reinterpret_cast<const uint4*>(src);
        uint32_t q = rot;
#pragma unroll 8
        for (uint32_t i = 0; i < nq; ++i) {
          const uint4 x = c4[q], y = s4[q];
          d += absdiff(x.x, y.x) + absdiff(x.y, y.y) + absdiff(x.z, y.z) + absdiff(x.w, y.w);
          if (++q == nq) q = 0;
        }
      } else if (a.dist_kind == 1) {  // Hamming distance of bit vectors (dHash)
        for (uint32_t b = 0; b < B; ++b) d += __popc(ct[b] ^ src[b]);
      } else {
#pragma unroll 4
        for (uint32_t b = 0; b < B; ++b) d += absdiff(ct[b], src[b]);
      }
      if (!valid) d = 0;
      if (w == 0) l_adj = __shfl_sync(0xffffffffu, d, 0);  // lag 1
      if (k <= L) sl1[j * L + k - 1] = d;
      bool keep = false;
      // fp32(max) / 2N >= tau exactly when max >= x_tau (the smallest such numerator)
      if (k <= L) keep = max(l_adj, d) >= a.x_tau || k >= L;
      const uint32_t m = __ballot_sync(0xffffffffu, keep);
      if (lane == 0) smask[j * W + w] = m;
    }
  }
  __syncthreads();

  // 2. the rule in frame order
  if (tid == 0) {
    uint32_t g = s_g;
    if (g < 1 || g > L) g = L;  // the state only ever holds [1, L]
    unsigned long long acc = t0 == 0 ? 0ull : s_acc;
    for (uint32_t j = 0; j < n; ++j) {
      if (t0 + j == 0) {  // the stream's first frame: kept, the gap restarts
        sgap[j] = 1;
        g = 1;
        continue;
      }
      bool scene = false;
      if (a.scd) {
        const unsigned long long adj = sl1[j * L];
        if (adj >= a.x_cut) {  // a cut ends the run
          scene = true;
          acc = 0;
        } else if (adj >= a.x_grad) {  // joins the run: a gradual change where its sum first reaches T_b
          acc += adj;
          scene = acc >= a.x_cut && acc - adj < a.x_cut;
        } else {  // a low difference ends the run
          acc = 0;
        }
      }
      const bool keep = ((smask[j * W + ((g - 1) >> 5)] >> ((g - 1) & 31)) & 1u) || scene;
      sgap[j] = g | (scene ? 0x80000000u : 0u);
      g = keep ? 1u : g + 1u;
    }
    s_acc = acc;
    s_g = g;
  }
  __syncthreads();

  // 3. outputs, the retention record, ring, state, and the rows cleared
  uint32_t* rec = a.record ? a.record + static_cast<uint64_t>(stream) * a.rec_words : nullptr;
  for (uint32_t base = 0; base < n; base += kWalkThreads) {
    const uint32_t j = base + tid;
    bool kept = false;
    if (j < n) {
      float s = 0.0f;
      uint8_t code = 3;
      if (t0 + j != 0) {
        uint32_t g = sgap[j] & 0x7fffffffu;
        if (!COFIE_BOUND(g >= 1 && g <= L)) g = 1;
        s = __fdiv_rn(static_cast<float>(max(sl1[j * L], sl1[j * L + g - 1])), a.two_n);
        const bool nov = s >= a.tau, scene = sgap[j] >> 31;
        code = nov ? 1 : (scene ? 4 : (g >= L ? 2 : 0));
      }
      if (sg.scores) sg.scores[j] = s;
      if (sg.keep) sg.keep[j] = code;
      kept = code != 0;
    }
    const uint32_t bits = __ballot_sync(0xffffffffu, kept);
    if (lane == 0 && rec) record_bits(rec, a.rec_words, t0 + base + 32 * warp, bits);
  }
  const uint32_t keep_n = min(n, L);
  uint32_t* ring_w = ring + static_cast<uint64_t>(stream) * L * B;
  for (uint32_t i = tid; i < keep_n * B; i += kWalkThreads) {
    const uint32_t jj = n - keep_n + i / B, b = i % B;
    ring_w[((s_slot0 + jj) % L) * B + b] = kStaged ? srows[(L + jj) * B + b] : hist_s[static_cast<uint64_t>(jj) * B + b];
  }
  if (tid == 0) {
    state[stream].t = t0 + n;
    state[stream].g = s_g;
    state[stream].acc = s_acc;
  }
  if (a.zero_hist) {
    if (!kStaged) __syncthreads();  // the ring copies above have read the rows
    for (uint32_t i = tid; i < n * B; i += kWalkThreads) hist[static_cast<uint64_t>(row0) * B + i] = 0;
  }
}

size_t walk_smem_bytes(uint32_t n, uint32_t l_max, uint32_t mask_words, uint32_t bins, bool staged) {
  return (static_cast<size_t>(n) * (l_max + mask_words + 1) + (staged ? static_cast<size_t>(l_max + n) * bins : 0)) * 4;
}

// The gap map of one stream segment: map[g-1] = the gap after its last frame
// when its first frame is entered with gap g (for a stream's first segment,
// frame 0 is a first frame and every entry gives the same result). One CTA:
// each warp composes the maps of a run of frames for all entry gaps (lane =
// entry gap), then lanes chain the 32 run maps; tiles of kScanTile frames are
// chained the same way.
template <bool kOneWord>
__global__ void __launch_bounds__(kScanThreads) gap_map_kernel(Segment sg, SelectArgs a, unsigned long long t0,
                                                               const uint32_t* __restrict__ mask,
                                                               uint16_t* __restrict__ map_out) {
  extern __shared__ __align__(16) uint32_t ssm[];
  __shared__ uint16_t smap[kMaxLmax];
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t W = a.mask_words, L = a.l_max;
  uint32_t* smask = ssm;
  uint16_t* sexit = reinterpret_cast<uint16_t*>(smask + kScanTile * W) + kScanTile;  // [kScanWarps][L]
  for (uint32_t g = tid; g < L; g += kScanThreads) smap[g] = static_cast<uint16_t>(g + 1);  // identity
  const uint32_t j_start = (t0 == 0) ? 1u : 0u;  // frame 0 of a stream is a first frame: gap 1 after it
  if (t0 == 0 && sg.n > 0)
    for (uint32_t g = tid; g < L; g += kScanThreads) smap[g] = 1;
  __syncthreads();
  for (uint32_t tile0 = j_start; tile0 < sg.n; tile0 += kScanTile) {
    const uint32_t m = min(kScanTile, sg.n - tile0);
    for (uint32_t i = tid; i < m * W; i += kScanThreads)
      smask[i] = mask[static_cast<uint64_t>(sg.row0 + tile0) * W + i];
    __syncthreads();
    const uint32_t run = (m + kScanWarps - 1) / kScanWarps;
    const uint32_t f0 = min(warp * run, m), f1 = min(f0 + run, m);
    for (uint32_t gin = lane + 1; gin <= L; gin += 32) {
      uint32_t g = gin;
      for (uint32_t f = f0; f < f1; ++f) g = step_gap<kOneWord>(smask + f * W, g);
      (void)COFIE_BOUND(g >= 1 && g <= L);  // a gap stays in [1, L_max]
      sexit[warp * L + gin - 1] = static_cast<uint16_t>(g);
    }
    __syncthreads();
    // compose: the map so far, then the 32 runs of this tile in order
    for (uint32_t e = tid; e < L; e += kScanThreads) {
      uint32_t g = smap[e];
      for (uint32_t w = 0; w < kScanWarps; ++w)
        if (min(w * run, m) < min(w * run + run, m)) g = sexit[w * L + g - 1];
      smap[e] = static_cast<uint16_t>(g);
    }
    __syncthreads();
  }
  for (uint32_t g = tid; g < L; g += kScanThreads) map_out[g] = smap[g];
}

// ring[(t_first + i) mod L] = hist row i, for rows [0, rows) of a stream.
__global__ void ring_store_kernel(const uint32_t* __restrict__ hist, uint32_t rows, unsigned long long t_first,
                                  uint32_t stream, SelectArgs a, uint32_t* __restrict__ ring) {
  const uint32_t B = a.bins, L = a.l_max;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < rows * B; i += gridDim.x * blockDim.x) {
    const uint32_t r = i / B, b = i % B;
    ring[(static_cast<uint64_t>(stream) * L + (t_first + r) % L) * B + b] = hist[static_cast<uint64_t>(r) * B + b];
  }
}

size_t scan_smem_bytes(uint32_t mask_words, uint32_t l_max) {
  return static_cast<size_t>(kScanTile) * mask_words * 4 + kScanTile * 2 + static_cast<size_t>(kScanWarps) * l_max * 2;
}

}  // namespace

uint32_t select_small_max() { return kSmallMax; }
uint32_t select_walk_max_frames() { return kWalkMaxFrames; }
uint32_t select_walk_max_lmax() { return kWalkMaxLmax; }

cudaError_t launch_select_walk(const SegTable& segs, const SelectArgs& a, uint32_t* hist, uint32_t* ring,
                               StreamState* state, cudaStream_t st, bool pdl) {
  uint32_t longest = 0;
  for (uint32_t i = 0; i < segs.count; ++i) longest = max(longest, segs.s[i].n);
  // rows staged in shared memory when they fit the default 48 KiB with the tables
  const bool staged = walk_smem_bytes(longest, a.l_max, a.mask_words, a.bins, true) <= kWalkStageBudget;
  const size_t smem = walk_smem_bytes(longest, a.l_max, a.mask_words, a.bins, staged);  // <= 48 KiB
  const bool vec = a.bins % 4 == 0 && a.dist_kind == 0;
  const auto kernel = vec ? (staged ? select_walk_kernel<true, true> : select_walk_kernel<true, false>)
                          : (staged ? select_walk_kernel<false, true> : select_walk_kernel<false, false>);
  const cudaError_t e =
      launch_dependent(pdl, kernel, dim3(segs.count), dim3(kWalkThreads), smem, st, segs, a, hist, ring, state);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_gap_map(const Segment& seg, const SelectArgs& a, unsigned long long t0, const uint32_t* mask,
                           uint16_t* map_out, cudaStream_t st) {
  const size_t smem = scan_smem_bytes(a.mask_words, a.l_max);
  cudaError_t e;
  if (a.mask_words == 1) {
    e = cudaFuncSetAttribute(gap_map_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e == cudaSuccess) gap_map_kernel<true><<<1, kScanThreads, smem, st>>>(seg, a, t0, mask, map_out);
  } else {
    e = cudaFuncSetAttribute(gap_map_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e == cudaSuccess) gap_map_kernel<false><<<1, kScanThreads, smem, st>>>(seg, a, t0, mask, map_out);
  }
  return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_ring_store(const uint32_t* hist, uint32_t rows, unsigned long long t_first, uint32_t stream,
                              const SelectArgs& a, uint32_t* ring, cudaStream_t st) {
  if (rows == 0) return cudaSuccess;
  ring_store_kernel<<<(rows * a.bins + 255) / 256, 256, 0, st>>>(hist, rows, t_first, stream, a, ring);
  return cudaGetLastError();
}

cudaError_t scan_prepare(uint32_t mask_words, uint32_t l_max) {
  const int smem = static_cast<int>(scan_smem_bytes(mask_words, l_max));
  cudaError_t e;
  if (mask_words == 1) {
    e = cudaFuncSetAttribute(scan_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(select_small_kernel<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(select_small_kernel<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  } else {
    e = cudaFuncSetAttribute(scan_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(select_small_kernel<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(select_small_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  }
  return e;
}

cudaError_t launch_window(const SegTable& segs, const SelectArgs& a, const uint32_t* hist, const uint32_t* ring,
                          const StreamState* state, uint32_t* l1, uint32_t* mask, cudaStream_t st, bool pdl) {
  const uint32_t grid = (segs.rows + kWinWarps - 1) / kWinWarps;
  const cudaError_t e =
      (a.bins % 4 == 0 && a.dist_kind == 0)
          ? launch_dependent(pdl, window_kernel<true>, dim3(grid), dim3(kWinWarps * 32), 0, st, segs, a, hist, ring,
                             state, l1, mask)
          : launch_dependent(pdl, window_kernel<false>, dim3(grid), dim3(kWinWarps * 32), 0, st, segs, a, hist, ring,
                             state, l1, mask);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_scan(const SegTable& segs, const SelectArgs& a, const uint32_t* l1, const uint32_t* mask,
                        uint32_t* hist, uint32_t* ring, StreamState* state, cudaStream_t st, bool pdl) {
  const size_t smem = scan_smem_bytes(a.mask_words, a.l_max);
  const cudaError_t e =
      a.mask_words == 1
          ? launch_dependent(pdl, scan_kernel<true>, dim3(segs.count), dim3(kScanThreads), smem, st, segs, a, l1, mask,
                             hist, ring, state)
          : launch_dependent(pdl, scan_kernel<false>, dim3(segs.count), dim3(kScanThreads), smem, st, segs, a, l1,
                             mask, hist, ring, state);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_select_small(const SegTable& segs, const SelectArgs& a, uint32_t* hist, uint32_t* ring,
                                StreamState* state, uint32_t* l1, uint32_t* mask, cudaStream_t st, bool pdl) {
  const size_t smem = scan_smem_bytes(a.mask_words, a.l_max);
  const bool vec = a.bins % 4 == 0 && a.dist_kind == 0, one = a.mask_words == 1;
  const auto kernel = vec ? (one ? select_small_kernel<true, true> : select_small_kernel<true, false>)
                          : (one ? select_small_kernel<false, true> : select_small_kernel<false, false>);
  const cudaError_t e =
      launch_dependent(pdl, kernel, dim3(segs.count), dim3(kScanThreads), smem, st, segs, a, hist, ring, state, l1, mask);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

uint32_t take_bounds_errors_select() { return take_local_bounds_errors(); }

}  // namespace cofie
