// K1: per-frame grayscale histograms (CoFiE Sec. 3.2, the histogram
// novelty paragraph; B = 32 bins per App. A).
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
// The same kernel, instantiated for kCells, serves the spatial signals: the
// consumers add each 16-pixel group's grayscale to its cell of the grid (one
// shared atomic per cell the group touches), and the fold adds the CTA's cell
// sums to the frame's row.
// Every mbarrier wait is bounded (globaltimer); a wait that runs out sets a
// bit in the error word, stops issuing work and returns without leaving bulk
// copies in flight.
#include "ngff_device.cuh"

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
// The spatial signals' shape (consumer warps, ring stages), from a sweep on
// GB300 over the 1080p stream: 4 warps and a 2-stage ring (4 CTAs per SM)
// stream fastest.
#ifndef COFIE_CELL_WARPS
#define COFIE_CELL_WARPS 4
#endif
#ifndef COFIE_CELL_STAGES
#define COFIE_CELL_STAGES 2
#endif
constexpr int kCellWarps = COFIE_CELL_WARPS;
template <int kBin>
struct Shape {
  static constexpr int warps = kBin == kCells ? kCellWarps : kConsumerWarps;
  static constexpr int consumers = warps * 32;
  static constexpr int threads = consumers + 32;
  static constexpr int stages = kBin == kCells ? COFIE_CELL_STAGES : COFIE_K1_STAGES;
};
constexpr int kStages = COFIE_K1_STAGES;
constexpr int kGroupBytes = 48;            // 16 RGB pixels
constexpr int kChunkGroups = COFIE_K1_CHUNK_GROUPS;
constexpr int kChunkBytes = kChunkGroups * kGroupBytes;  // 24 KiB by default

struct SegLite {
  const uint8_t* frames;
  uint32_t n;
  uint32_t row0;
};

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

template <int kN>
__device__ __forceinline__ void consumer_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(kN) : "memory");
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

// One chunk of 16-pixel groups for the spatial signals: group j of the chunk
// is group g0 + j of its frame (row-major, width a multiple of 16, so a group
// never spans two image rows). Each run of a group's pixels that lies in one
// cell is added to that cell with one shared atomic (lanes of a warp that hit
// the same cell serialise; that costs less than reducing across the warp).
template <int kN>
__device__ __forceinline__ void cells_chunk(const uint8_t* buf, uint32_t groups, uint32_t g0, const HistArgs& a,
                                            const LumaConsts& L, uint32_t* cells, uint32_t tid) {
  const uint32_t W = a.width, gh = a.grid_h, gw = a.grid_w;
  for (uint32_t j = tid; j < groups; j += kN) {
    const uint4* p = reinterpret_cast<const uint4*>(buf + j * kGroupBytes);
    const uint4 x = p[0], y = p[1], z = p[2];
    uint32_t v[16];
    luma4(x.x, x.y, x.z, L, v[0], v[1], v[2], v[3]);
    luma4(x.w, y.x, y.y, L, v[4], v[5], v[6], v[7]);
    luma4(y.z, y.w, z.x, L, v[8], v[9], v[10], v[11]);
    luma4(z.y, z.z, z.w, L, v[12], v[13], v[14], v[15]);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __umulhi(v[i], L.magic_y);  // Y = floor(v / den), host-verified
    // divisions by multiply-high, each host-verified over its whole range:
    // image row r = gi / gpr, cell column floor(xg gw / gpr) of the first
    // pixel (x0 = 16 xg, W = 16 gpr), cell row floor(r gh / H)
    const uint32_t gi = g0 + j, r = __umulhi(gi, a.m_gpr), xg = gi - r * a.gpr, x0 = xg << 4;
    const uint32_t crow = __umulhi(r * gh, a.m_h) * gw;
    uint32_t cx = __umulhi(xg * gw, a.m_gpr);
    uint32_t edge = (cx + 1) * W;  // pixel x lies past cell column cx iff x gw >= edge
    if (a.wide) {
      // cell columns of 16 pixels or more: a group spans one or two cells.
      // Prefix sums P of the group's grayscale; the first s pixels lie in
      // cell cx, s = (first x of the next cell column) - x0, capped at 16;
      // P[s - 1] is picked by a 4-level select tree on the bits of s - 1.
      uint32_t P[16];
      P[0] = v[0];
#pragma unroll
      for (int i = 1; i < 16; ++i) P[i] = P[i - 1] + v[i];
      const uint32_t nx = __umulhi(edge + gw - 1, a.m_gw);  // ceil(edge / gw), host-verified
      const uint32_t i = min(nx - x0, 16u) - 1;
      uint32_t q[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) q[k] = (i & 1) ? P[2 * k + 1] : P[2 * k];
#pragma unroll
      for (int k = 0; k < 4; ++k) q[k] = (i & 2) ? q[2 * k + 1] : q[2 * k];
#pragma unroll
      for (int k = 0; k < 2; ++k) q[k] = (i & 4) ? q[2 * k + 1] : q[2 * k];
      const uint32_t lo = (i & 8) ? q[1] : q[0];
      if (COFIE_BOUND(crow + cx < gh * gw)) atomicAdd(&cells[crow + cx], lo);
      if (i < 15 && COFIE_BOUND(crow + cx + 1 < gh * gw)) atomicAdd(&cells[crow + cx + 1], P[15] - lo);
    } else {
      uint32_t acc = 0;
#pragma unroll
      for (uint32_t i = 0; i < 16; ++i) {
        if ((x0 + i) * gw >= edge) {
          if (COFIE_BOUND(crow + cx < gh * gw)) atomicAdd(&cells[crow + cx], acc);
          acc = 0;
          ++cx;
          edge += W;
        }
        acc += v[i];
      }
      if (COFIE_BOUND(crow + cx < gh * gw)) atomicAdd(&cells[crow + cx], acc);
    }
  }
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
__global__ void __launch_bounds__(Shape<kBin>::threads) hist_fast_kernel(SegTable segs, HistArgs a, LumaConsts L,
                                                                         uint32_t* __restrict__ hist,
                                                                         uint32_t* __restrict__ err) {
  constexpr int kCW = Shape<kBin>::warps, kNC = Shape<kBin>::consumers, kNT = Shape<kBin>::threads;
  constexpr int kS = Shape<kBin>::stages;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ SegLite sseg[kMaxSegs];
  uint8_t* ring = smem;
  uint32_t* cnt = reinterpret_cast<uint32_t*>(smem + kS * kChunkBytes);
  const uint32_t n_cnt = kBin == kCells ? a.grid_h * a.grid_w : L.bins * 32;
  uint64_t* bars = reinterpret_cast<uint64_t*>(cnt + (kBin == kCells ? kMaxBins : L.bins * 32));

  pdl_trigger();  // the push's selection kernels may be scheduled; they wait for this grid before reading it
  const uint64_t total = static_cast<uint64_t>(segs.rows) * a.chunks_per_frame;
  const uint64_t c0 = total * blockIdx.x / gridDim.x;
  const uint64_t c1 = total * (blockIdx.x + 1) / gridDim.x;
  if (c0 >= c1) return;  // uniform across the CTA

  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kS);
  for (uint32_t i = tid; i < segs.count; i += kNT) {
    sseg[i].frames = segs.s[i].frames;
    sseg[i].n = segs.s[i].n;
    sseg[i].row0 = segs.s[i].row0;
  }
  for (uint32_t i = tid; i < n_cnt; i += kNT) cnt[i] = 0;
  if (tid == 0) {
    for (int s = 0; s < kS; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kCW);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  const uint32_t nseg = segs.count, cpf = a.chunks_per_frame, gpf = a.groups_per_frame;

  if (warp == kCW) {
    // ---------------------------------------------------------- producer --
    if (lane != 0) return;
    // Launched as a programmatic dependent of the kernel before it, this CTA
    // has set up while that kernel ran; no frame is read and no row written
    // until that kernel has completed and its memory is visible.
    pdl_wait();
    const uint64_t pol = l2_read_policy();
    const uint32_t ring0 = smem_u32(ring);
    ChunkCursor cur;
    cur.init(c0, cpf, sseg, nseg);
    uint32_t issued = 0;
    for (uint64_t c = c0; c < c1; ++c) {
      const uint32_t slot = issued % kS, use = issued / kS;
      if (use > 0 && !mbar_wait_bounded(empty0 + 8 * slot, (use - 1) & 1, a.timeout_ns)) {
        atomicOr(err, kErrProducerTimeout);
        break;
      }
      const uint32_t bytes = cur.groups(gpf) * kGroupBytes;
      // checked build: a chunk outside the push stops the producer (the
      // consumers' bounded waits then end the launch with an error)
      if (!COFIE_BOUND(cur.row < segs.rows && cur.k < cpf && bytes <= kChunkBytes)) break;
      mbar_arrive_expect_tx(full0 + 8 * slot, bytes);
      bulk_load(ring0 + slot * kChunkBytes, cur.src(sseg, a.frame_bytes), bytes, full0 + 8 * slot, pol);
      cur.advance(cpf, sseg, nseg);
      ++issued;
    }
    // No copy may still be writing shared memory when the CTA exits.
    const uint32_t first = issued > kS ? issued - kS : 0;
    for (uint32_t j = first; j < issued; ++j)
      if (!mbar_wait_bounded(full0 + 8 * (j % kS), (j / kS) & 1, a.timeout_ns))
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
    const uint32_t slot = i % kS, use = i / kS;
    if (ok && !mbar_wait_bounded(full0 + 8 * slot, use & 1, a.timeout_ns)) {
      atomicOr(err, kErrConsumerTimeout);
      ok = false;  // keep walking the sequence so every CTA barrier is still reached
    }
    if constexpr (kBin == kCells) {
      if (ok) cells_chunk<kNC>(ring + slot * kChunkBytes, cur.groups(gpf), cur.k * kChunkGroups, a, L, cnt, tid);
    } else if (ok) {
      const uint32_t groups = cur.groups(gpf);
      const uint8_t* buf = ring + slot * kChunkBytes;
#pragma unroll 2
      for (uint32_t g = tid; g < groups; g += kNC) {
        const uint4* p = reinterpret_cast<const uint4*>(buf + g * kGroupBytes);
        const uint4 x = p[0], y = p[1], z = p[2];
        count4<kBin>(x.x, x.y, x.z, L, cnt_lane);
        count4<kBin>(x.w, y.x, y.y, L, cnt_lane);
        count4<kBin>(y.z, y.w, z.x, L, cnt_lane);
        count4<kBin>(z.y, z.z, z.w, L, cnt_lane);
      }
    }
    if (ok) {
      __syncwarp();
      if (lane == 0) mbar_arrive(empty0 + 8 * slot);
    }
    cur.advance(cpf, sseg, nseg);
    if (c + 1 == c1 || cur.row != row) {
      // frame done for this CTA: fold the 32 lane columns of every bin (or
      // hand over the cell sums)
      consumer_bar<kNC>();
      if (kBin == kCells) {
        for (uint32_t b = tid; b < n_cnt; b += kNC) {
          const uint32_t sum = cnt[b];
          cnt[b] = 0;
          if (sum && ok && COFIE_BOUND(row < segs.rows))
            atomicAdd(hist + static_cast<uint64_t>(row) * n_cnt + b, sum);
        }
      } else {
        for (uint32_t b = tid; b < L.bins; b += kNC) {
          uint32_t sum = 0;
          uint32_t* rowp = cnt + b * 32;
#pragma unroll 8
          for (uint32_t l = 0; l < 32; ++l) {
            const uint32_t idx = (l + b) & 31;  // rotate: conflict-free across the warp
            sum += rowp[idx];
            rowp[idx] = 0;
          }
          if (sum && ok && COFIE_BOUND(row < segs.rows))
            atomicAdd(hist + static_cast<uint64_t>(row) * L.bins + b, sum);
        }
      }
      consumer_bar<kNC>();
      row = cur.row;
    }
  }
}

// Generic kernel: any frame size or alignment (frames whose pixel count is
// not a multiple of 16, or that do not start on a 16-byte boundary). Grid
// (slices, rows): CTA x of row r counts slice x of frame r. A frame's pixels
// split into a prologue of p_a < 16 pixels, an interior of whole 16-pixel
// groups that each start on a 16-byte boundary (p_a is the first pixel whose
// address is 16-byte aligned: frame + 3 p_a = 0 mod 16), and an epilogue of
// fewer than 16 pixels. Interior groups are loaded with three 128-bit loads
// and binned as in the fast kernel (two dp2a per pixel, a multiply-high
// verified on the host); prologue and epilogue pixels with byte loads. Counts
// go to lane-private shared counters cnt[bin][lane] (bank = lane), folded
// into the frame's row with one global atomic per bin per CTA.
constexpr int kGenericThreads = 256;
constexpr uint32_t kGenericGroupsPerCta = 2048;  // 32768 pixels per CTA, unless the launch asks for fewer
constexpr int kGenericDiv = 3;                   // no verified multiply-high: Y = v / den

template <int kBin>
__device__ __forceinline__ uint32_t generic_bin(uint32_t v, const LumaConsts& L) {
  if constexpr (kBin == kGenericDiv) return ((v / L.den) * L.bins) >> 8;
  else return bin_of<kBin>(v, L);
}

template <int kBin>
__global__ void __launch_bounds__(kGenericThreads) hist_generic_kernel(SegTable segs, HistArgs a, LumaConsts L,
                                                                      uint32_t* __restrict__ hist) {
  extern __shared__ __align__(16) uint32_t gcnt[];  // [B][32]
  pdl_trigger();
  const uint32_t row = blockIdx.y, tid = threadIdx.x, lane = tid & 31;
  uint32_t seg = 0;
  while (seg + 1 < segs.count && row >= segs.s[seg + 1].row0) ++seg;
  const uint8_t* frame = segs.s[seg].frames + static_cast<uint64_t>(row - segs.s[seg].row0) * a.frame_bytes;
  for (uint32_t i = tid; i < L.bins * 32; i += kGenericThreads) gcnt[i] = 0;
  // Launched as a programmatic dependent of the kernel before it (small
  // launches), this CTA has set up while that kernel ran; no frame is read
  // and no row written until that kernel has completed and its memory is
  // visible. A no-op for an ordinary launch.
  pdl_wait();
  __syncthreads();
  const uint32_t cnt_lane = static_cast<uint32_t>(__cvta_generic_to_shared(gcnt)) + lane * 4;
  const uint32_t npix = a.npix;
  // first 16-byte aligned pixel: 3 p = -(frame mod 16) mod 16, and 3 * 11 = 1 mod 16
  const uint32_t mis = static_cast<uint32_t>(reinterpret_cast<uintptr_t>(frame) & 15u);
  const uint32_t p_a = min(((16u - mis) * 11u) & 15u, npix);
  const uint32_t G = (npix - p_a) / 16;
  const uint32_t spc = a.slice_groups;
  const uint32_t g0 = blockIdx.x * spc, g1 = min(g0 + spc, G);
  const uint8_t* base = frame + 3ull * p_a;
#pragma unroll 2
  for (uint32_t g = g0 + tid; g < g1; g += kGenericThreads) {
    const uint4* p = reinterpret_cast<const uint4*>(base + 48ull * g);
    const uint4 x = __ldcs(p), y = __ldcs(p + 1), z = __ldcs(p + 2);
    uint32_t v[16];
    luma4(x.x, x.y, x.z, L, v[0], v[1], v[2], v[3]);
    luma4(x.w, y.x, y.y, L, v[4], v[5], v[6], v[7]);
    luma4(y.z, y.w, z.x, L, v[8], v[9], v[10], v[11]);
    luma4(z.y, z.z, z.w, L, v[12], v[13], v[14], v[15]);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t b = generic_bin<kBin>(v[i], L);
      if (COFIE_BOUND(b < L.bins)) red_add_shared(cnt_lane + (b << 7));
    }
  }
  // the ragged edges: prologue (first CTA of the row) and epilogue (last CTA)
  const auto scalar = [&](uint32_t q) {
    const uint8_t* px = frame + 3ull * q;
    const uint32_t v = L.w[0] * px[0] + L.w[1] * px[1] + L.w[2] * px[2] + L.half;
    const uint32_t b = generic_bin<kBin>(v, L);
    if (COFIE_BOUND(b < L.bins)) red_add_shared(cnt_lane + (b << 7));
  };
  if (blockIdx.x == 0)
    for (uint32_t q = tid; q < p_a; q += kGenericThreads) scalar(q);
  if (blockIdx.x == gridDim.x - 1)
    for (uint32_t q = p_a + 16 * G + tid; q < npix; q += kGenericThreads) scalar(q);
  __syncthreads();
  for (uint32_t b = tid; b < L.bins; b += kGenericThreads) {
    uint32_t sum = 0;
#pragma unroll 8
    for (uint32_t l = 0; l < 32; ++l) sum += gcnt[b * 32 + ((l + b) & 31)];  // rotated: conflict-free
    if (sum && COFIE_BOUND(row < segs.rows)) atomicAdd(hist + static_cast<uint64_t>(row) * L.bins + b, sum);
  }
}

}  // namespace

size_t hist_smem_bytes(uint32_t bins) {
  return static_cast<size_t>(kStages) * kChunkBytes + static_cast<size_t>(bins) * 32 * 4 + 2 * kStages * 8;
}

static size_t cells_smem_bytes() {
  constexpr int kS = Shape<kCells>::stages;
  return static_cast<size_t>(kS) * kChunkBytes + static_cast<size_t>(kMaxBins) * 4 + 2 * kS * 8;
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

int cells_blocks_per_sm() {
  const size_t smem = cells_smem_bytes();
  if (cudaFuncSetAttribute(hist_fast_kernel<kCells>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return -1;
  int n = 0;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, hist_fast_kernel<kCells>, Shape<kCells>::threads, smem) ==
                 cudaSuccess
             ? n
             : -1;
}

cudaError_t launch_cells_fast(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, uint32_t* cells,
                              uint32_t* err, int grid, cudaStream_t st, bool pdl) {
  const cudaError_t e = launch_dependent(pdl, hist_fast_kernel<kCells>, dim3(grid), dim3(Shape<kCells>::threads),
                                         cells_smem_bytes(), st, segs, a, lc, cells, err);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_hist_fast(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, int bin_path,
                             uint32_t* hist, uint32_t* err, int grid, cudaStream_t st, bool pdl) {
  const size_t smem = hist_smem_bytes(lc.bins);
  const cudaError_t e =
      bin_path == kBinFast
          ? launch_dependent(pdl, hist_fast_kernel<kBinFast>, dim3(grid), dim3(kThreads), smem, st, segs, a, lc, hist,
                             err)
          : launch_dependent(pdl, hist_fast_kernel<kBinTwoStep>, dim3(grid), dim3(kThreads), smem, st, segs, a, lc,
                             hist, err);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

uint32_t hist_generic_slices(uint32_t npix, uint32_t slice_groups) {
  const uint32_t spc = slice_groups ? slice_groups : kGenericGroupsPerCta;
  const uint32_t groups = npix / 16;  // at least the interior's groups, whatever the alignment
  return groups ? (groups + spc - 1) / spc : 1;
}

int hist_generic_blocks_per_sm(int bin_path, uint32_t bins) {
  int n = 0;
  const size_t smem = static_cast<size_t>(bins) * 32 * 4;
  const cudaError_t e =
      bin_path == kBinFast
          ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, hist_generic_kernel<kBinFast>, kGenericThreads, smem)
      : bin_path == kBinTwoStep
          ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, hist_generic_kernel<kBinTwoStep>, kGenericThreads, smem)
          : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, hist_generic_kernel<kGenericDiv>, kGenericThreads, smem);
  return e == cudaSuccess ? n : -1;
}

cudaError_t launch_hist_generic(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, int bin_path,
                                uint32_t* hist, cudaStream_t st, uint32_t slice_groups, bool pdl) {
  HistArgs b = a;
  b.slice_groups = slice_groups ? slice_groups : kGenericGroupsPerCta;
  const dim3 grid(hist_generic_slices(a.npix, b.slice_groups), segs.rows);
  const size_t smem = static_cast<size_t>(lc.bins) * 32 * 4;
  const auto kernel = bin_path == kBinFast      ? hist_generic_kernel<kBinFast>
                      : bin_path == kBinTwoStep ? hist_generic_kernel<kBinTwoStep>
                                                : hist_generic_kernel<kGenericDiv>;
  const cudaError_t e = launch_dependent(pdl, kernel, grid, dim3(kGenericThreads), smem, st, segs, b, lc, hist);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

uint32_t take_bounds_errors_hist() { return take_local_bounds_errors(); }

}  // namespace cofie
