// Per-frame kernels around K1: the spatial signals where the streaming
// kernel does not apply, the dHash bits from cell sums, the bounded-wait
// probe of the failure path, and the bin check over arbitrary pixels. They
// share K1's grayscale and bin functions (ngff_device.cuh).
#include "ngff_device.cuh"

namespace cofie {
namespace {

// The spatial signals (low-res difference, dHash) where the TMA kernel does
// not apply (width not a multiple of 16, unaligned frames, or no verified
// multiply-high for the grayscale division): one CTA per frame sums the
// grayscale of each cell of a grid_h x grid_w grid in shared memory. Fast path
// (width a multiple of 16, aligned frames): 16-pixel groups, the same dp2a
// luma as the histogram kernel, runs of pixels of one cell added in registers
// and flushed with one shared atomic per run. Then low-res writes the cell
// sums, dHash the 64 bits [mean(r, c) > mean(r, c + 1)] compared exactly by
// cross-multiplying sums and pixel counts.
constexpr int kFeatThreads = 512;

__global__ void __launch_bounds__(kFeatThreads) features_kernel(SegTable segs, FeatArgs fa, LumaConsts L,
                                                                uint32_t* __restrict__ feat, uint32_t fw) {
  __shared__ uint32_t cell[256];
  pdl_trigger();
  const uint32_t row = blockIdx.x, tid = threadIdx.x;
  uint32_t seg = 0;
  while (seg + 1 < segs.count && row >= segs.s[seg + 1].row0) ++seg;
  const uint8_t* frame = segs.s[seg].frames + static_cast<uint64_t>(row - segs.s[seg].row0) * fa.frame_bytes;
  const uint32_t gh = fa.grid_h, gw = fa.grid_w, W = fa.width, H = fa.height;
  for (uint32_t i = tid; i < gh * gw; i += kFeatThreads) cell[i] = 0;
  __syncthreads();
  const bool fast = (W % 16 == 0) && (reinterpret_cast<uintptr_t>(frame) % 16 == 0) && (fa.frame_bytes % 16 == 0);
  if (fast) {
    const uint32_t gpr = W / 16, groups = fa.npix / 16;
    for (uint32_t g = tid; g < groups; g += kFeatThreads) {
      const uint32_t y = g / gpr, x0 = (g - y * gpr) * 16;
      const uint32_t cy = y * gh / H;
      const uint4* p4 = reinterpret_cast<const uint4*>(frame + static_cast<uint64_t>(g) * 48);
      const uint4 a = p4[0], b = p4[1], c = p4[2];
      uint32_t v[16];
      luma4(a.x, a.y, a.z, L, v[0], v[1], v[2], v[3]);
      luma4(a.w, b.x, b.y, L, v[4], v[5], v[6], v[7]);
      luma4(b.z, b.w, c.x, L, v[8], v[9], v[10], v[11]);
      luma4(c.y, c.z, c.w, L, v[12], v[13], v[14], v[15]);
      uint32_t cx = x0 * gw / W;
      uint32_t next = ((cx + 1) * W + gw - 1) / gw;  // first x of the next cell column
      uint32_t acc = 0;
#pragma unroll
      for (uint32_t i = 0; i < 16; ++i) {
        const uint32_t yv = fa.use_magic ? __umulhi(v[i], L.magic_y) : v[i] / L.den;
        if (x0 + i >= next) {
          if (COFIE_BOUND(cy * gw + cx < gh * gw)) atomicAdd(&cell[cy * gw + cx], acc);
          acc = 0;
          ++cx;
          next = ((cx + 1) * W + gw - 1) / gw;
        }
        acc += yv;
      }
      if (COFIE_BOUND(cy * gw + cx < gh * gw)) atomicAdd(&cell[cy * gw + cx], acc);
    }
  } else {
    for (uint32_t p = tid; p < fa.npix; p += kFeatThreads) {
      const uint8_t* px = frame + 3ull * p;
      const uint32_t yv = (L.w[0] * px[0] + L.w[1] * px[1] + L.w[2] * px[2] + L.half) / L.den;
      const uint32_t y = p / W, x = p - y * W;
      const uint32_t ci = (y * gh / H) * gw + x * gw / W;
      if (COFIE_BOUND(ci < gh * gw)) atomicAdd(&cell[ci], yv);
    }
  }
  __syncthreads();
  uint32_t* out = feat + static_cast<uint64_t>(row) * fw;
  if (fa.kind == 1) {
    for (uint32_t i = tid; i < gh * gw; i += kFeatThreads) out[i] = cell[i];
  } else if (tid < 64) {  // warps 0 and 1: bit (r, c) of the 8 x 8 hash
    const uint32_t r = tid / 8, c = tid % 8;
    const uint64_t sa = cell[r * gw + c], sb = cell[r * gw + c + 1];
    const uint64_t na = static_cast<uint64_t>(fa.row_h[r]) * fa.col_w[c];
    const uint64_t nb = static_cast<uint64_t>(fa.row_h[r]) * fa.col_w[c + 1];
    const uint32_t word = __ballot_sync(0xffffffffu, sa * nb > sb * na);
    if ((tid & 31) == 0) out[tid >> 5] = word;
  }
}

// dHash from the 8 x 9 cell sums the fast kernel accumulated (row-major, 72
// per frame): bit (r, c) = [S(r, c) n(r, c + 1) > S(r, c + 1) n(r, c)], the
// comparison of the two cell means without division. The cell row is zeroed
// for the next push once read.
__global__ void __launch_bounds__(96) dhash_finish_kernel(uint32_t* __restrict__ cells, FeatArgs fa,
                                                          uint32_t* __restrict__ bits) {
  pdl_trigger();
  pdl_wait();  // the cell sums of the streaming kernel before it
  const uint32_t row = blockIdx.x, tid = threadIdx.x;
  uint32_t* c = cells + static_cast<uint64_t>(row) * 72;
  if (tid < 64) {
    const uint32_t r = tid / 8, k = tid % 8;
    const uint64_t sa = c[r * 9 + k], sb = c[r * 9 + k + 1];
    const uint64_t na = static_cast<uint64_t>(fa.row_h[r]) * fa.col_w[k];
    const uint64_t nb = static_cast<uint64_t>(fa.row_h[r]) * fa.col_w[k + 1];
    const uint32_t word = __ballot_sync(0xffffffffu, sa * nb > sb * na);
    if ((tid & 31) == 0) bits[static_cast<uint64_t>(row) * 2 + (tid >> 5)] = word;
  }
  __syncthreads();
  if (tid < 72) c[tid] = 0;
}

// Failure-path probe: one thread waits, with the pipeline's bounded wait, for
// an mbarrier phase that nothing completes; when the bound runs out it sets
// the consumer-timeout bit, exactly as a stalled K1 consumer would, and the
// kernel returns normally.
__global__ void wait_probe_kernel(uint64_t timeout_ns, uint32_t* __restrict__ err) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_u32(&bar);
  mbar_init(b, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  if (!mbar_wait_bounded(b, 0, timeout_ns)) atomicOr(err, kErrConsumerTimeout);
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

cudaError_t launch_dhash_finish(uint32_t* cells, uint32_t rows, const FeatArgs& fa, uint32_t* bits, cudaStream_t st,
                                bool pdl) {
  const cudaError_t e = launch_dependent(pdl, dhash_finish_kernel, dim3(rows), dim3(96), 0, st, cells, fa, bits);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

cudaError_t launch_features(const SegTable& segs, const FeatArgs& fa, const LumaConsts& lc, uint32_t* feat, uint32_t fw,
                            cudaStream_t st) {
  features_kernel<<<segs.rows, kFeatThreads, 0, st>>>(segs, fa, lc, feat, fw);
  return cudaGetLastError();
}

cudaError_t launch_wait_probe(uint64_t timeout_ns, uint32_t* err, cudaStream_t st) {
  wait_probe_kernel<<<1, 1, 0, st>>>(timeout_ns, err);
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

uint32_t take_bounds_errors_features() { return take_local_bounds_errors(); }

}  // namespace cofie
