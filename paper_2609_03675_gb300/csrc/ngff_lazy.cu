// The retention rule without forced retention (L_max = 0, Eq. 5's second
// term off). With no bound on t - r(t) the reference frame can lie any
// distance back, so the windowed distances of K2/K3 do not apply; the rule
// is walked in frame order instead, computing d(c_t, c_{r(t)}) on the fly.
//
// One CTA per stream segment. Warp 0 walks the frames of a tile of feature
// rows in shared memory while the other warps stage the next tile from the
// (L2-resident) feature rows into the other buffer with asynchronous copies.
// The walk goes by windows: the reference stays fixed until the next keep,
// so lane l scores frame f + l against it (the whole row, read from a
// per-lane rotated word so the lanes hit distinct banks); one ballot finds
// the first keep in the window, the frames up to it stand, it becomes the
// reference, and the next window starts after it. With a keep every few
// frames this replaces a warp reduction per frame by a fraction of one.
// Scene changes (twin comparison) depend only on the adjacent differences,
// not on the reference, so a tile's scene flags are found first, by a scan,
// and enter the walk as keeps.
// The stream's state between pushes is {t, the open scene-change run} and
// two ring rows: slot 0 holds c_{t-1}, slot 1 holds c_{r(t)}.
#include "ngff_common.cuh"

namespace cofie {
namespace {

constexpr int kLazyThreads = 256;
constexpr uint32_t kLazyTileWords = 8192;  // 32 KiB per buffer, two buffers
constexpr uint32_t kLazyMaxRows = kLazyTileWords / 2;  // rows per tile at the smallest width (dHash, 2 words)

__device__ __forceinline__ uint32_t word_dist(uint32_t x, uint32_t y, uint32_t kind) {
  return kind == 1 ? static_cast<uint32_t>(__popc(x ^ y)) : (x > y ? x - y : y - x);
}

// The same for B = 4 kQ (kQ a power of two), fully unrolled: every load's
// address is known up front, so all 2 kQ 16-byte loads are in flight at once.
template <uint32_t kQ>
__device__ __forceinline__ uint32_t row_dist_q(const uint32_t* x, const uint32_t* y, uint32_t start, uint32_t kind) {
  static_assert((kQ & (kQ - 1)) == 0, "kQ must be a power of two");
  const uint4* x4 = reinterpret_cast<const uint4*>(x);
  const uint4* y4 = reinterpret_cast<const uint4*>(y);
  uint32_t s0 = 0, s1 = 0, s2 = 0, s3 = 0;
#pragma unroll
  for (uint32_t i = 0; i < kQ; ++i) {
    const uint32_t q = (start + i) & (kQ - 1);
    const uint4 u = x4[q], v = y4[q];
    s0 += word_dist(u.x, v.x, kind);
    s1 += word_dist(u.y, v.y, kind);
    s2 += word_dist(u.z, v.z, kind);
    s3 += word_dist(u.w, v.w, kind);
  }
  return (s0 + s1) + (s2 + s3);
}

// The distance numerator between two feature rows of B words in shared
// memory, taken by one thread. With B % 4 == 0, 16-byte words starting at
// the rotated word `start` (lanes that read rows B words apart then touch
// distinct banks), four independent sums so the loads of four words are in
// flight together; otherwise word by word from `start`.
__device__ __forceinline__ uint32_t row_dist(const uint32_t* x, const uint32_t* y, uint32_t B, uint32_t start,
                                             uint32_t kind) {
  if (B == 32) return row_dist_q<8>(x, y, start, kind);   // the paper's B
  if (B == 64) return row_dist_q<16>(x, y, start, kind);
  if (B % 4 == 0) {
    const uint32_t Q = B / 4;
    const uint4* x4 = reinterpret_cast<const uint4*>(x);
    const uint4* y4 = reinterpret_cast<const uint4*>(y);
    uint32_t q = start % Q, s0 = 0, s1 = 0, s2 = 0, s3 = 0;
#pragma unroll 4
    for (uint32_t i = 0; i < Q; ++i) {
      const uint4 u = x4[q], v = y4[q];
      s0 += word_dist(u.x, v.x, kind);
      s1 += word_dist(u.y, v.y, kind);
      s2 += word_dist(u.z, v.z, kind);
      s3 += word_dist(u.w, v.w, kind);
      q = (q + 1 == Q) ? 0u : q + 1;
    }
    return (s0 + s1) + (s2 + s3);
  }
  uint32_t b = start % B, sum = 0;
  for (uint32_t i = 0; i < B; ++i) {
    sum += word_dist(x[b], y[b], kind);
    b = (b + 1 == B) ? 0u : b + 1;
  }
  return sum;
}

// The twin comparison's run as a monoid: a frame ends the open run (reset,
// the run restarts at sum 0 after it) or adds its adjacent numerator to it.
struct LzRun {
  uint32_t reset;
  unsigned long long sum;
};
__device__ __forceinline__ LzRun lz_cat(LzRun x, LzRun y) { return y.reset ? y : LzRun{x.reset, x.sum + y.sum}; }
__device__ __forceinline__ LzRun lz_shfl_up(LzRun v, uint32_t off) {
  return LzRun{__shfl_up_sync(0xffffffffu, v.reset, off), __shfl_up_sync(0xffffffffu, v.sum, off)};
}

// Per tile of feature rows (shared memory, double-buffered):
//   all warps  adjacent distances d_adj[f] = |c_f - c_{f-1}| of the tile (a
//              thread per row for B <= 64, else a warp per row);
//   warp 0     with scene changes, the tile's scene flags first (a scan of
//              the run monoid: a lane takes a run of consecutive frames, the
//              runs are scanned across the warp, each lane replays its run
//              from its prefix), then the windowed walk: d_ref = |c_f - c_r|,
//              the decision as an integer compare against the host-computed
//              thresholds (the smallest numerators whose fp32 quotient by 2N
//              reaches tau_h, T_b, T_s; exact since that quotient never
//              decreases as the numerator grows), and the reference update;
//              meanwhile the other warps stage the next tile with
//              asynchronous copies;
//   all warps  the tile's fp32 scores and keep codes to global memory.
__global__ void __launch_bounds__(kLazyThreads) lazy_select_kernel(SegTable segs, SelectArgs a,
                                                                   const uint32_t* __restrict__ feat,
                                                                   uint32_t* __restrict__ ring,
                                                                   StreamState* __restrict__ state) {
  extern __shared__ __align__(16) uint32_t smem[];
  uint32_t* tiles = smem;                            // [2][kLazyTileWords]
  uint32_t* sadj = tiles + 2 * kLazyTileWords;       // [rows_per_tile] adjacent numerators
  uint32_t* sd = sadj + kLazyMaxRows;                // [rows_per_tile] max(d_adj, d_ref)
  uint8_t* scode = reinterpret_cast<uint8_t*>(sd + kLazyMaxRows);  // [rows_per_tile]
  uint8_t* sscene = scode + kLazyMaxRows;                          // [rows_per_tile] scene-change flags
  uint32_t* sprev = reinterpret_cast<uint32_t*>(sscene + kLazyMaxRows);  // [B] the row before the tile
  uint32_t* sref = sprev + kMaxBins;                                     // [B] the reference row
  const Segment sg = segs.s[blockIdx.x];
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t B = a.bins, n = sg.n;
  const uint32_t rows_per_tile = kLazyTileWords / B;
  const uint32_t n_tiles = (n + rows_per_tile - 1) / rows_per_tile;
  // Every read of device memory follows the wait: the first-stage kernel
  // before this one may itself have been scheduled before the previous
  // push's selection finished writing the stream's state and ring.
  pdl_wait();
  const unsigned long long t0 = state[sg.stream].t;
  uint32_t* sring = ring + static_cast<uint64_t>(sg.stream) * 2 * B;
  if (n == 0) return;

  // asynchronous copies (all of a thread's copies in flight at once), 16
  // bytes when B % 4 == 0 (the rows of the tile are then 16-byte aligned:
  // the feature array and the tile buffers are), else 4; waited for by the
  // staging threads before the block barrier
  const bool vec16 = B % 4 == 0;
  auto stage = [&](uint32_t tile, uint32_t first_thread, uint32_t threads) {
    const uint32_t j0 = tile * rows_per_tile, m = min(rows_per_tile, n - j0);
    uint32_t* dst = tiles + (tile & 1) * kLazyTileWords;
    const uint32_t* src = feat + static_cast<uint64_t>(sg.row0 + j0) * B;
    if (vec16) {
      for (uint32_t i = 4 * (tid - first_thread); i < m * B; i += 4 * threads)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                         static_cast<uint32_t>(__cvta_generic_to_shared(dst + i))),
                     "l"(src + i)
                     : "memory");
    } else {
      for (uint32_t i = tid - first_thread; i < m * B; i += threads)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                         static_cast<uint32_t>(__cvta_generic_to_shared(dst + i))),
                     "l"(src + i)
                     : "memory");
    }
    asm volatile("cp.async.commit_group;\ncp.async.wait_all;" ::: "memory");
  };
  // adjacent numerators of a staged tile: for B <= 64 a thread per row
  // (row_dist), else warp w takes rows w, w + 8, ... (a warp reduction each)
  auto adjacent = [&](uint32_t tile) {
    const uint32_t j0 = tile * rows_per_tile, m = min(rows_per_tile, n - j0);
    const uint32_t* buf = tiles + (tile & 1) * kLazyTileWords;
    if (B <= 64) {
      for (uint32_t f = tid; f < m; f += kLazyThreads) {
        const uint32_t* c = buf + f * B;
        const uint32_t d = row_dist(c, f ? c - B : sprev, B, lane, a.dist_kind);
        if (COFIE_BOUND(f < kLazyMaxRows)) sadj[f] = d;
      }
      return;
    }
    for (uint32_t f = warp; f < m; f += kLazyThreads / 32) {
      const uint32_t* c = buf + f * B;
      const uint32_t* p = f ? c - B : sprev;
      uint32_t part = 0;
      for (uint32_t b = lane; b < B; b += 32) part += word_dist(c[b], p[b], a.dist_kind);
      part = __reduce_add_sync(0xffffffffu, part);
      if (lane == 0 && COFIE_BOUND(f < kLazyMaxRows)) sadj[f] = part;
    }
  };

  unsigned long long acc = t0 > 0 ? state[sg.stream].acc : 0ull;  // warp 0: the scene-change run open so far
  for (uint32_t b = tid; b < B; b += kLazyThreads) {
    sref[b] = t0 > 0 ? sring[B + b] : 0u;
    sprev[b] = t0 > 0 ? sring[b] : 0u;
  }
  stage(0, 0, kLazyThreads);
  __syncthreads();
  adjacent(0);
  __syncthreads();
  for (uint32_t tile = 0; tile < n_tiles; ++tile) {
    const uint32_t j0 = tile * rows_per_tile, m = min(rows_per_tile, n - j0);
    const uint32_t* buf = tiles + (tile & 1) * kLazyTileWords;
    if (warp != 0) {
      if (tile + 1 < n_tiles) stage(tile + 1, 32, kLazyThreads - 32);
    } else {
      if (a.scd) {
        // scene flags: frame f cuts (d_adj >= T_b: a scene change that ends
        // the run), joins the run (T_s <= d_adj < T_b: a scene change when
        // the run's sum first reaches T_b) or ends it; the stream's first
        // frame is neither (the identity)
        const uint32_t per = (m + 31) / 32, f0 = min(lane * per, m), f1 = min(f0 + per, m);
        auto elem = [&](uint32_t f) {
          const uint32_t d = sadj[f];
          if (t0 + j0 + f == 0) return LzRun{0u, 0ull};
          return (d >= a.x_cut || d < a.x_grad) ? LzRun{1u, 0ull} : LzRun{0u, d};
        };
        LzRun run{0u, 0ull};
        for (uint32_t f = f0; f < f1; ++f) run = lz_cat(run, elem(f));
        LzRun incl = run;
#pragma unroll
        for (uint32_t off = 1; off < 32; off <<= 1) {
          const LzRun o = lz_shfl_up(incl, off);
          if (lane >= off) incl = lz_cat(o, incl);
        }
        LzRun pre = lz_shfl_up(incl, 1);
        if (lane == 0) pre = LzRun{0u, 0ull};
        for (uint32_t f = f0; f < f1; ++f) {
          const uint32_t d = sadj[f];
          pre = lz_cat(pre, elem(f));
          const unsigned long long r = pre.reset ? pre.sum : acc + pre.sum;  // the run's sum at f
          const bool first = t0 + j0 + f == 0;
          const bool scene = !first && (d >= a.x_cut || (d >= a.x_grad && r >= a.x_cut && r - d < a.x_cut));
          if (COFIE_BOUND(f < kLazyMaxRows)) sscene[f] = scene ? 1 : 0;
        }
        const LzRun total{__shfl_sync(0xffffffffu, incl.reset, 31), __shfl_sync(0xffffffffu, incl.sum, 31)};
        acc = total.reset ? total.sum : acc + total.sum;
        __syncwarp();
      }
      // the windowed walk
      for (uint32_t f = 0; f < m;) {
        const uint32_t fl = f + lane;
        const uint32_t dref = fl < m ? row_dist(buf + fl * B, sref, B, lane, a.dist_kind) : 0u;
        const uint32_t d = fl < m ? max(sadj[fl], dref) : 0u;
        const bool first = t0 + j0 + fl == 0;
        const bool nov = d >= a.x_tau, scene = a.scd && fl < m && sscene[fl];
        const bool keep = fl < m && (first || nov || scene);
        const uint32_t bal = __ballot_sync(0xffffffffu, keep);
        const uint32_t upto = bal ? static_cast<uint32_t>(__ffs(bal)) - 1 : 31u;  // the last lane whose result stands
        if (lane <= upto && fl < m && COFIE_BOUND(fl < kLazyMaxRows)) {
          sd[fl] = d;
          scode[fl] = first ? 3 : (nov ? 1 : (scene ? 4 : 0));
        }
        if (bal) {  // frame f + upto is kept: it becomes the reference
          __syncwarp();
          const uint32_t* krow = buf + (f + upto) * B;
          for (uint32_t bb = lane; bb < B; bb += 32) sref[bb] = krow[bb];
          __syncwarp();
        }
        f += upto + 1;
      }
    }
    __syncthreads();
    for (uint32_t base = 0; base < m; base += kLazyThreads) {  // warps stay whole: the record takes a ballot
      const uint32_t f = base + tid;
      bool kept = false;
      if (f < m) {
        const bool first = t0 + j0 + f == 0;
        if (sg.scores) sg.scores[j0 + f] = first ? 0.0f : __fdiv_rn(static_cast<float>(sd[f]), a.two_n);
        if (sg.keep) sg.keep[j0 + f] = scode[f];
        kept = scode[f] != 0;
      }
      const uint32_t bits = __ballot_sync(0xffffffffu, kept);
      if (lane == 0 && a.record)
        record_bits(a.record + static_cast<uint64_t>(sg.stream) * a.rec_words, a.rec_words, t0 + j0 + f, bits);
    }
    if (tile + 1 < n_tiles) {
      for (uint32_t b = tid; b < B; b += kLazyThreads) sprev[b] = buf[(m - 1) * B + b];
      __syncthreads();
      adjacent(tile + 1);
    }
    __syncthreads();
  }
  // the ring: slot 0 the last frame's row, slot 1 the reference's
  const uint32_t last = (n - 1) - (n_tiles - 1) * rows_per_tile;
  const uint32_t* lbuf = tiles + ((n_tiles - 1) & 1) * kLazyTileWords;
  for (uint32_t b = tid; b < B; b += kLazyThreads) {
    sring[b] = lbuf[last * B + b];
    sring[B + b] = sref[b];
  }
  if (tid == 0) {
    state[sg.stream].t = t0 + n;
    state[sg.stream].g = 1;
    state[sg.stream].acc = acc;
  }
}

}  // namespace

cudaError_t launch_lazy_select(const SegTable& segs, const SelectArgs& a, const uint32_t* feat, uint32_t* ring,
                               StreamState* state, cudaStream_t st, bool pdl) {
  const size_t smem = 2 * kLazyTileWords * 4 + kLazyMaxRows * (4 + 4 + 1 + 1) + 2 * kMaxBins * 4;
  cudaError_t e = cudaFuncSetAttribute(lazy_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  e = launch_dependent(pdl, lazy_select_kernel, dim3(segs.count), dim3(kLazyThreads), smem, st, segs, a, feat, ring,
                       state);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

uint32_t take_bounds_errors_lazy() { return take_local_bounds_errors(); }

}  // namespace cofie
