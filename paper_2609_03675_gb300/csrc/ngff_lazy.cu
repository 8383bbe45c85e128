// The retention rule without forced retention (L_max = 0, Eq. 5's second
// term off). With no bound on t - r(t) the reference frame can lie any
// distance back, so the windowed distances of K2/K3 do not apply; the rule
// is walked in frame order instead, computing d(c_t, c_{r(t)}) on the fly.
//
// One CTA per stream segment. Warp 0 holds c_{t-1} and c_{r(t)} of its
// stream in registers (lane l: feature words l, l + 32, ...) and walks the
// frames of a tile of feature rows in shared memory: both distances with one
// warp reduction each, the fp32 decision, and the reference update. The
// other warps meanwhile stage the next tile from the (L2-resident) feature
// rows into the other shared-memory buffer. The stream's state between
// pushes is {t, the open scene-change run} and two ring rows: slot 0 holds
// c_{t-1}, slot 1 holds c_{r(t)}.
#include "ngff_common.cuh"

namespace cofie {
namespace {

constexpr int kLazyThreads = 256;
constexpr uint32_t kLazyTileWords = 8192;  // 32 KiB per buffer, two buffers
constexpr uint32_t kPer = kMaxBins / 32;   // feature words per lane, at most

__device__ __forceinline__ uint32_t word_dist(uint32_t x, uint32_t y, uint32_t kind) {
  return kind == 1 ? static_cast<uint32_t>(__popc(x ^ y)) : (x > y ? x - y : y - x);
}

__global__ void __launch_bounds__(kLazyThreads) lazy_select_kernel(SegTable segs, SelectArgs a,
                                                                   const uint32_t* __restrict__ feat,
                                                                   uint32_t* __restrict__ ring,
                                                                   StreamState* __restrict__ state) {
  extern __shared__ __align__(16) uint32_t tiles[];  // [2][kLazyTileWords]
  const Segment sg = segs.s[blockIdx.x];
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t B = a.bins, n = sg.n;
  const uint32_t rows_per_tile = kLazyTileWords / B;
  const uint32_t n_tiles = (n + rows_per_tile - 1) / rows_per_tile;
  const unsigned long long t0 = state[sg.stream].t;
  uint32_t* sring = ring + static_cast<uint64_t>(sg.stream) * 2 * B;

  auto stage = [&](uint32_t tile, uint32_t first_thread, uint32_t threads) {
    const uint32_t j0 = tile * rows_per_tile, m = min(rows_per_tile, n - j0);
    uint32_t* dst = tiles + (tile & 1) * kLazyTileWords;
    const uint32_t* src = feat + static_cast<uint64_t>(sg.row0 + j0) * B;
    for (uint32_t i = tid - first_thread; i < m * B; i += threads) dst[i] = src[i];
  };

  // warp 0's registers: previous frame, reference frame, and the run sum
  uint32_t prev[kPer], ref[kPer];
  unsigned long long acc = 0;
  if (warp == 0) {
#pragma unroll
    for (uint32_t q = 0; q < kPer; ++q) {
      const uint32_t b = lane + 32 * q;
      prev[q] = (t0 > 0 && b < B) ? sring[b] : 0u;
      ref[q] = (t0 > 0 && b < B) ? sring[B + b] : 0u;
    }
    acc = t0 > 0 ? state[sg.stream].acc : 0ull;
  }
  if (n_tiles > 0) stage(0, 0, kLazyThreads);
  __syncthreads();
  for (uint32_t tile = 0; tile < n_tiles; ++tile) {
    if (warp != 0) {
      if (tile + 1 < n_tiles) stage(tile + 1, 32, kLazyThreads - 32);
    } else {
      const uint32_t j0 = tile * rows_per_tile, m = min(rows_per_tile, n - j0);
      const uint32_t* buf = tiles + (tile & 1) * kLazyTileWords;
      for (uint32_t f = 0; f < m; ++f) {
        const uint32_t j = j0 + f;
        const unsigned long long t = t0 + j;
        uint32_t cur[kPer];
        uint32_t pa = 0, pr = 0;
#pragma unroll
        for (uint32_t q = 0; q < kPer; ++q) {
          const uint32_t b = lane + 32 * q;
          cur[q] = b < B ? buf[f * B + b] : 0u;
          pa += word_dist(cur[q], prev[q], a.dist_kind);
          pr += word_dist(cur[q], ref[q], a.dist_kind);
        }
        const uint32_t d_adj = __reduce_add_sync(0xffffffffu, pa);
        const uint32_t d_ref = __reduce_add_sync(0xffffffffu, pr);
        float s = 0.0f;
        uint8_t code;
        if (t == 0) {
          code = 3;  // the stream's first frame
        } else {
          s = __fdiv_rn(static_cast<float>(max(d_adj, d_ref)), a.two_n);
          bool scene = false;
          if (a.scd) {  // twin comparison on the adjacent difference
            const float sd = __fdiv_rn(static_cast<float>(d_adj), a.two_n);
            if (sd >= a.scd_cut) {
              scene = true;
              acc = 0;
            } else if (sd >= a.scd_grad) {
              const unsigned long long before = acc;
              acc += d_adj;
              scene = __fdiv_rn(__ull2float_rn(acc), a.two_n) >= a.scd_cut &&
                      !(__fdiv_rn(__ull2float_rn(before), a.two_n) >= a.scd_cut);
            } else {
              acc = 0;
            }
          }
          code = s >= a.tau ? 1 : (scene ? 4 : 0);
        }
        if (lane == 0) {
          if (sg.scores) sg.scores[j] = s;
          if (sg.keep) sg.keep[j] = code;
        }
#pragma unroll
        for (uint32_t q = 0; q < kPer; ++q) {
          if (code) ref[q] = cur[q];
          prev[q] = cur[q];
        }
      }
    }
    __syncthreads();
  }
  if (warp == 0 && n > 0) {
#pragma unroll
    for (uint32_t q = 0; q < kPer; ++q) {
      const uint32_t b = lane + 32 * q;
      if (b < B) {
        sring[b] = prev[q];
        sring[B + b] = ref[q];
      }
    }
    if (lane == 0) {
      state[sg.stream].t = t0 + n;
      state[sg.stream].g = 1;
      state[sg.stream].acc = acc;
    }
  }
}

}  // namespace

cudaError_t launch_lazy_select(const SegTable& segs, const SelectArgs& a, const uint32_t* feat, uint32_t* ring,
                               StreamState* state, cudaStream_t st) {
  const size_t smem = 2 * kLazyTileWords * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(lazy_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  lazy_select_kernel<<<segs.count, kLazyThreads, smem, st>>>(segs, a, feat, ring, state);
  return cudaGetLastError();
}

}  // namespace cofie
