// K1: per-frame grayscale histograms (CoFiE Sec. 3.2 "Lightweight
// histogram-based novelty"; B = 32 bins per App. A).
//
// Per pixel: Y = floor((wR R + wG G + wB B + floor(den/2)) / den) (BT.601
// reading), bin = floor(Y B / 256), count[bin] += 1. Integer arithmetic only,
// so the histogram is independent of summation order and bit-exact.
//
// Fast kernel (frames of a multiple of 16 pixels, 16-byte aligned):
//   - a persistent grid; each CTA owns a contiguous range of 24 KiB chunks of
//     the push (a chunk never crosses a frame boundary);
//   - one producer thread streams chunks HBM -> shared memory with 1-D bulk
//     async copies (cp.async.bulk, the TMA engine) into a 4-stage ring
//     guarded by mbarriers (full: transaction bytes, empty: consumer warps);
//   - 4 consumer warps read 48-byte groups (16 RGB pixels) with three 128-bit
//     shared loads at a 48-byte stride (conflict-free), form the luma sums
//     with two dp2a per pixel, bin them with one multiply-high, and count
//     into lane-private shared counters cnt[bin][lane] (bank = lane, so a
//     warp's 32 increments never collide) with red.shared.add;
//   - when the chunk sequence moves to the next frame, the consumers reduce
//     the 32 lane columns per bin and add them to hist[row][bin] with one
//     global atomic per bin.
// Every mbarrier wait is bounded (globaltimer); a wait that runs out sets a
// bit in the error word, stops issuing work and returns without leaving bulk
// copies in flight.
#include "ngff_common.cuh"

namespace cofie {
namespace {

// Tuning constants (compile-time overridable for sweeps). Measured on GB300
// over the 1080p stream: 4 consumer warps (one per SM sub-partition) with two
// CTAs per SM stream at ~7.59 TB/s; 3 or 5 warps (uneven over the
// sub-partitions) lose 8-20 %, 8 warps lose 8 %, and any shape that leaves
// one CTA per SM loses 25-40 %. The L2 evict-first hint makes no measurable
// difference; the default policy is kept.
#ifndef COFIE_K1_CONSUMER_WARPS
#define COFIE_K1_CONSUMER_WARPS 4
#endif
#ifndef COFIE_K1_STAGES
#define COFIE_K1_STAGES 4
#endif
#ifndef COFIE_K1_CHUNK_GROUPS
#define COFIE_K1_CHUNK_GROUPS 512
#endif
#ifndef COFIE_K1_EVICT_FIRST
#define COFIE_K1_EVICT_FIRST 0
#endif

constexpr int kConsumerWarps = COFIE_K1_CONSUMER_WARPS;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;  // + one producer warp
constexpr int kStages = COFIE_K1_STAGES;
constexpr int kGroupBytes = 48;            // 16 RGB pixels
constexpr int kChunkGroups = COFIE_K1_CHUNK_GROUPS;
constexpr int kChunkBytes = kChunkGroups * kGroupBytes;  // 24 KiB by default

struct SegLite {
  const uint8_t* frames;
  uint32_t n;
  uint32_t row0;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase of parity `parity` to complete; false after timeout_ns.
__device__ __noinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > timeout_ns) return false;
  }
}

__device__ __forceinline__ uint64_t l2_read_policy() {
  uint64_t pol;
#if COFIE_K1_EVICT_FIRST
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
#else
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
#endif
  return pol;
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(pol)
      : "memory");
}

__device__ __forceinline__ void red_add_shared(uint32_t addr) {
  asm volatile("red.shared.add.u32 [%0], 1;" ::"r"(addr) : "memory");
}

__device__ __forceinline__ void consumer_bar() { asm volatile("bar.sync 1, %0;" ::"n"(kConsumers) : "memory"); }

// Luma sums v = wR R + wG G + wB B + half of the four pixels packed in three
// little-endian words (bytes R0 G0 B0 R1 | G1 B1 R2 G2 | B2 R3 G3 B3).
__device__ __forceinline__ void luma4(uint32_t w0, uint32_t w1, uint32_t w2, const LumaConsts& L, uint32_t& v0,
                                      uint32_t& v1, uint32_t& v2, uint32_t& v3) {
  v0 = __dp2a_hi(L.w_b0, w0, __dp2a_lo(L.w_rg, w0, L.half));  // R0 G0 | B0
  v1 = __dp2a_lo(L.w_gb, w1, __dp2a_hi(L.w_0r, w0, L.half));  // R1 | G1 B1
  v2 = __dp2a_lo(L.w_b0, w2, __dp2a_hi(L.w_rg, w1, L.half));  // R2 G2 | B2
  v3 = __dp2a_hi(L.w_gb, w2, __dp2a_lo(L.w_0r, w2, L.half));  // R3 | G3 B3
}

template <int kBin>
__device__ __forceinline__ uint32_t bin_of(uint32_t v, const LumaConsts& L) {
  if (kBin == kBinFast) return __umulhi(v, L.magic);  // floor(v / (den * 256 / B)), host-verified
  const uint32_t y = __umulhi(v, L.magic_y);          // floor(v / den), host-verified
  return (y * L.bins) >> 8;
}

template <int kBin>
__device__ __forceinline__ void count4(uint32_t w0, uint32_t w1, uint32_t w2, const LumaConsts& L, uint32_t cnt_lane) {
  uint32_t v0, v1, v2, v3;
  luma4(w0, w1, w2, L, v0, v1, v2, v3);
  red_add_shared(cnt_lane + (bin_of<kBin>(v0, L) << 7));
  red_add_shared(cnt_lane + (bin_of<kBin>(v1, L) << 7));
  red_add_shared(cnt_lane + (bin_of<kBin>(v2, L) << 7));
  red_add_shared(cnt_lane + (bin_of<kBin>(v3, L) << 7));
}

// Walks the chunk sequence of a push: chunk c is chunk k of frame row.
struct ChunkCursor {
  uint32_t row, k, seg;

  __device__ void init(uint64_t c, uint32_t cpf, const SegLite* segs, uint32_t nseg) {
    row = static_cast<uint32_t>(c / cpf);
    k = static_cast<uint32_t>(c % cpf);
    seg = 0;
    while (seg + 1 < nseg && row >= segs[seg + 1].row0) ++seg;
  }
  __device__ void advance(uint32_t cpf, const SegLite* segs, uint32_t nseg) {
    if (++k == cpf) {
      k = 0;
      ++row;
      while (seg + 1 < nseg && row >= segs[seg + 1].row0) ++seg;
    }
  }
  __device__ const uint8_t* src(const SegLite* segs, uint64_t frame_bytes) const {
    return segs[seg].frames + static_cast<uint64_t>(row - segs[seg].row0) * frame_bytes +
           static_cast<uint64_t>(k) * kChunkBytes;
  }
  __device__ uint32_t groups(uint32_t gpf) const {
    const uint32_t left = gpf - k * kChunkGroups;
    return left < kChunkGroups ? left : kChunkGroups;
  }
};

template <int kBin>
__global__ void __launch_bounds__(kThreads) hist_fast_kernel(SegTable segs, HistArgs a, LumaConsts L,
                                                             uint32_t* __restrict__ hist, uint32_t* __restrict__ err) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SegLite sseg[kMaxSegs];
  uint8_t* ring = smem;
  uint32_t* cnt = reinterpret_cast<uint32_t*>(smem + kStages * kChunkBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(cnt + L.bins * 32);

  const uint64_t total = static_cast<uint64_t>(segs.rows) * a.chunks_per_frame;
  const uint64_t c0 = total * blockIdx.x / gridDim.x;
  const uint64_t c1 = total * (blockIdx.x + 1) / gridDim.x;
  if (c0 >= c1) return;  // uniform across the CTA

  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);
  for (uint32_t i = tid; i < segs.count; i += kThreads) {
    sseg[i].frames = segs.s[i].frames;
    sseg[i].n = segs.s[i].n;
    sseg[i].row0 = segs.s[i].row0;
  }
  for (uint32_t i = tid; i < L.bins * 32; i += kThreads) cnt[i] = 0;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kConsumerWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  const uint32_t nseg = segs.count, cpf = a.chunks_per_frame, gpf = a.groups_per_frame;

  if (warp == kConsumerWarps) {
    // ---------------------------------------------------------- producer --
    if (lane != 0) return;
    const uint64_t pol = l2_read_policy();
    const uint32_t ring0 = smem_u32(ring);
    ChunkCursor cur;
    cur.init(c0, cpf, sseg, nseg);
    uint32_t issued = 0;
    for (uint64_t c = c0; c < c1; ++c) {
      const uint32_t slot = issued % kStages, use = issued / kStages;
      if (use > 0 && !mbar_wait_bounded(empty0 + 8 * slot, (use - 1) & 1, a.timeout_ns)) {
        atomicOr(err, kErrProducerTimeout);
        break;
      }
      const uint32_t bytes = cur.groups(gpf) * kGroupBytes;
      mbar_arrive_expect_tx(full0 + 8 * slot, bytes);
      bulk_load(ring0 + slot * kChunkBytes, cur.src(sseg, a.frame_bytes), bytes, full0 + 8 * slot, pol);
      cur.advance(cpf, sseg, nseg);
      ++issued;
    }
    // No copy may still be writing shared memory when the CTA exits.
    const uint32_t first = issued > kStages ? issued - kStages : 0;
    for (uint32_t j = first; j < issued; ++j)
      if (!mbar_wait_bounded(full0 + 8 * (j % kStages), (j / kStages) & 1, a.timeout_ns))
        atomicOr(err, kErrDrainTimeout);
    return;
  }

  // ------------------------------------------------------------ consumers --
  const uint32_t cnt_lane = smem_u32(cnt) + lane * 4;
  ChunkCursor cur;
  cur.init(c0, cpf, sseg, nseg);
  uint32_t row = cur.row;
  bool ok = true;
  uint32_t i = 0;
  for (uint64_t c = c0; c < c1; ++c, ++i) {
    const uint32_t slot = i % kStages, use = i / kStages;
    if (ok && !mbar_wait_bounded(full0 + 8 * slot, use & 1, a.timeout_ns)) {
      atomicOr(err, kErrConsumerTimeout);
      ok = false;  // keep walking the sequence so every CTA barrier is still reached
    }
    if (ok) {
      const uint32_t groups = cur.groups(gpf);
      const uint8_t* buf = ring + slot * kChunkBytes;
#pragma unroll 2
      for (uint32_t g = tid; g < groups; g += kConsumers) {
        const uint4* p = reinterpret_cast<const uint4*>(buf + g * kGroupBytes);
        const uint4 x = p[0], y = p[1], z = p[2];
        count4<kBin>(x.x, x.y, x.z, L, cnt_lane);
        count4<kBin>(x.w, y.x, y.y, L, cnt_lane);
        count4<kBin>(y.z, y.w, z.x, L, cnt_lane);
        count4<kBin>(z.y, z.z, z.w, L, cnt_lane);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * slot);
    }
    cur.advance(cpf, sseg, nseg);
    if (c + 1 == c1 || cur.row != row) {
      // frame done for this CTA: fold the 32 lane columns of every bin
      consumer_bar();
      for (uint32_t b = tid; b < L.bins; b += kConsumers) {
        uint32_t sum = 0;
        uint32_t* rowp = cnt + b * 32;
#pragma unroll 8
        for (uint32_t l = 0; l < 32; ++l) {
          const uint32_t idx = (l + b) & 31;  // rotate: conflict-free across the warp
          sum += rowp[idx];
          rowp[idx] = 0;
        }
        if (sum && ok) atomicAdd(hist + static_cast<uint64_t>(row) * L.bins + b, sum);
      }
      consumer_bar();
      row = cur.row;
    }
  }
}

// Generic kernel: any frame size or alignment. One CTA per (frame, slice of
// kGenericPixels pixels); byte loads; block-shared counters with atomics.
constexpr int kGenericThreads = 256;
constexpr uint32_t kGenericPixels = 16384;

__global__ void __launch_bounds__(kGenericThreads) hist_generic_kernel(SegTable segs, HistArgs a, LumaConsts L,
                                                                      uint32_t* __restrict__ hist) {
  __shared__ uint32_t cnt[kMaxBins];
  const uint32_t row = blockIdx.y;
  uint32_t seg = 0;
  while (seg + 1 < segs.count && row >= segs.s[seg + 1].row0) ++seg;
  const uint8_t* frame = segs.s[seg].frames + static_cast<uint64_t>(row - segs.s[seg].row0) * a.frame_bytes;
  for (uint32_t b = threadIdx.x; b < L.bins; b += blockDim.x) cnt[b] = 0;
  __syncthreads();
  const uint64_t p0 = static_cast<uint64_t>(blockIdx.x) * kGenericPixels;
  const uint64_t p1 = min(p0 + kGenericPixels, static_cast<uint64_t>(a.npix));
  for (uint64_t p = p0 + threadIdx.x; p < p1; p += blockDim.x) {
    const uint8_t* px = frame + 3 * p;
    const uint32_t v = L.w[0] * px[0] + L.w[1] * px[1] + L.w[2] * px[2] + L.half;
    const uint32_t y = v / L.den;
    atomicAdd(&cnt[(y * L.bins) >> 8], 1u);
  }
  __syncthreads();
  for (uint32_t b = threadIdx.x; b < L.bins; b += blockDim.x)
    if (cnt[b]) atomicAdd(hist + static_cast<uint64_t>(row) * L.bins + b, cnt[b]);
}

// Diagnostic: the fast kernel's per-pixel luma and bin functions applied to
// 4-pixel groups (12 bytes each), one bin index per pixel.
template <int kBin>
__global__ void debug_bins_kernel(const uint8_t* __restrict__ px, uint64_t n_groups, LumaConsts L,
                                  uint8_t* __restrict__ out) {
  for (uint64_t g = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; g < n_groups;
       g += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint8_t* q = px + 12 * g;
    uint32_t w[3];
#pragma unroll
    for (int k = 0; k < 3; ++k)
      w[k] = q[4 * k] | (q[4 * k + 1] << 8) | (q[4 * k + 2] << 16) | (static_cast<uint32_t>(q[4 * k + 3]) << 24);
    uint32_t v0, v1, v2, v3;
    luma4(w[0], w[1], w[2], L, v0, v1, v2, v3);
    out[4 * g + 0] = static_cast<uint8_t>(bin_of<kBin>(v0, L));
    out[4 * g + 1] = static_cast<uint8_t>(bin_of<kBin>(v1, L));
    out[4 * g + 2] = static_cast<uint8_t>(bin_of<kBin>(v2, L));
    out[4 * g + 3] = static_cast<uint8_t>(bin_of<kBin>(v3, L));
  }
}

}  // namespace

size_t hist_smem_bytes(uint32_t bins) {
  return static_cast<size_t>(kStages) * kChunkBytes + static_cast<size_t>(bins) * 32 * 4 + 2 * kStages * 8;
}

static int configure(int bin_path, uint32_t bins) {
  const size_t smem = hist_smem_bytes(bins);
  cudaError_t e = (bin_path == kBinFast)
                      ? cudaFuncSetAttribute(hist_fast_kernel<kBinFast>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem))
                      : cudaFuncSetAttribute(hist_fast_kernel<kBinTwoStep>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  return e == cudaSuccess ? 0 : -1;
}

int hist_blocks_per_sm(int bin_path, uint32_t bins) {
  if (configure(bin_path, bins) != 0) return -1;
  int n = 0;
  const size_t smem = hist_smem_bytes(bins);
  cudaError_t e = (bin_path == kBinFast)
                      ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, hist_fast_kernel<kBinFast>, kThreads, smem)
                      : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, hist_fast_kernel<kBinTwoStep>, kThreads, smem);
  return e == cudaSuccess ? n : -1;
}

uint32_t hist_chunk_groups() { return kChunkGroups; }

cudaError_t launch_hist_fast(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, int bin_path,
                             uint32_t* hist, uint32_t* err, int grid, cudaStream_t st) {
  const size_t smem = hist_smem_bytes(lc.bins);
  if (bin_path == kBinFast)
    hist_fast_kernel<kBinFast><<<grid, kThreads, smem, st>>>(segs, a, lc, hist, err);
  else
    hist_fast_kernel<kBinTwoStep><<<grid, kThreads, smem, st>>>(segs, a, lc, hist, err);
  return cudaGetLastError();
}

cudaError_t launch_hist_generic(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, uint32_t* hist,
                                cudaStream_t st) {
  dim3 grid((a.npix + kGenericPixels - 1) / kGenericPixels, segs.rows);
  hist_generic_kernel<<<grid, kGenericThreads, 0, st>>>(segs, a, lc, hist);
  return cudaGetLastError();
}

cudaError_t launch_debug_bins(const uint8_t* px, uint64_t n_groups, const LumaConsts& lc, int bin_path,
                              uint8_t* bins_out, cudaStream_t st) {
  const int threads = 256;
  const uint64_t want = (n_groups + threads - 1) / threads;
  const int grid = static_cast<int>(want < 4096 ? (want ? want : 1) : 4096);
  if (bin_path == kBinFast)
    debug_bins_kernel<kBinFast><<<grid, threads, 0, st>>>(px, n_groups, lc, bins_out);
  else
    debug_bins_kernel<kBinTwoStep><<<grid, threads, 0, st>>>(px, n_groups, lc, bins_out);
  return cudaGetLastError();
}

}  // namespace cofie
