// cofie_ngff_select_static: the selection step for callers that cannot
// allocate device memory.
//
// Some callers may not call cudaMalloc at all: processes whose device memory
// is owned by another framework's pooling allocator under a hard cap, media
// and ingest plugins that are given buffers but no right to allocate, and
// latency-bound pipelines that fix their memory at start-up because
// cudaMalloc can synchronise the device. This entry point serves them: the
// caller passes the inputs (the integer histograms of a stream's first n
// frames) and the outputs (scores and keep codes), and the working tables
// live in a file-scope static device array of a fixed size, so the call
// allocates nothing.
//
// It is a variant of the library's window and scan kernels: a grid of warps
// (one per frame, lane = lag, 16-byte loads when the rows allow them) writes
// the windowed L1 distances and the per-gap keep bits of every frame into the
// static array, then one 1024-thread CTA runs the same gap-map scan over
// them. Decisions and scores equal those of cofie_ngff_push_ex on a fresh
// stream of the histogram signal without scene changes (other signals are
// refused).
//
// The array holds kStaticScratchWords 32-bit words (4 MiB) on every GPU that
// loads the library, until the process exits. Every call shares it and it
// keeps the last call's contents; each call writes every entry it later
// reads, so nothing needs clearing, but calls that overlap on the GPU (on
// different streams, or from different threads) race on it.
#include <cstring>
#include <mutex>

#include "cofie_ngff.h"
#include "ngff_common.cuh"

namespace cofie {
namespace {

constexpr uint32_t kStaticScratchWords = 1u << 20;  // 4 MiB
constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr uint32_t kTile = 2048;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint32_t g_select_scratch[kStaticScratchWords];

__device__ __forceinline__ uint32_t absdiff(uint32_t a, uint32_t b) { return a > b ? a - b : b - a; }

__device__ __forceinline__ uint32_t next_gap(const uint32_t* m, uint32_t g) {
  return ((m[(g - 1) >> 5] >> ((g - 1) & 31)) & 1u) ? 1u : g + 1u;
}

constexpr int kWinThreads = 256;  // the distance kernel: 8 frames per CTA

// Phase 1: windowed distances and per-gap keep bits of every frame (warp per
// frame, lane = lag k: the lane sums |c_t - c_{t-k}| over all bins, so the
// warp's loads are independent and in flight together).
template <bool kVec4>
__global__ void __launch_bounds__(kWinThreads) static_window_kernel(const uint32_t* __restrict__ hist, uint32_t n,
                                                                    SelectArgs a, uint32_t* __restrict__ scratch) {
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t B = a.bins, L = a.l_max, W = a.mask_words;
  uint32_t* l1 = scratch;                                   // [n][L]
  uint32_t* mask = scratch + static_cast<uint64_t>(n) * L;  // [n][W]
  const uint32_t warps = gridDim.x * (kWinThreads / 32);
  for (uint32_t t = blockIdx.x * (kWinThreads / 32) + (threadIdx.x >> 5); t < n; t += warps) {
    const uint32_t* ct = hist + static_cast<uint64_t>(t) * B;
    uint32_t l_adj = 0;
    for (uint32_t w = 0; w < W; ++w) {
      const uint32_t k = 32 * w + lane + 1;
      const bool valid = k <= L && k <= t;
      const uint32_t* cs = valid ? ct - static_cast<uint64_t>(k) * B : ct;
      uint32_t d = 0;
      if (kVec4) {
        const uint4* c4 = reinterpret_cast<const uint4*>(ct);
        const uint4* s4 = reinterpret_cast<const uint4*>(cs);
#pragma unroll 8
        for (uint32_t q = 0; q < B / 4; ++q) {
          const uint4 x = c4[q], y = s4[q];
          d += absdiff(x.x, y.x) + absdiff(x.y, y.y) + absdiff(x.z, y.z) + absdiff(x.w, y.w);
        }
      } else {
#pragma unroll 4
        for (uint32_t b = 0; b < B; ++b) d += absdiff(ct[b], cs[b]);
      }
      if (!valid) d = 0;
      if (w == 0) l_adj = __shfl_sync(0xffffffffu, d, 0);  // lag 1
      if (k <= L) l1[static_cast<uint64_t>(t) * L + k - 1] = d;
      bool kp = false;
      if (k <= L) kp = __fdiv_rn(static_cast<float>(max(l_adj, d)), a.two_n) >= a.tau || k >= L;
      const uint32_t m = __ballot_sync(0xffffffffu, kp);
      if (lane == 0) mask[static_cast<uint64_t>(t) * W + w] = m;
    }
  }
}

// Phase 2: gap-map scan from a fresh stream (frame 0 is the first frame), one
// CTA, over the distances and keep bits the kernel before it wrote.
__global__ void __launch_bounds__(kThreads) select_static_kernel(uint32_t n, SelectArgs a,
                                                                 const uint32_t* __restrict__ scratch,
                                                                 float* __restrict__ scores,
                                                                 uint8_t* __restrict__ keep) {
  extern __shared__ __align__(16) uint32_t sm[];
  __shared__ uint32_t entry[kWarps + 1];
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t L = a.l_max, W = a.mask_words;
  const uint32_t* l1 = scratch;                                   // [n][L]
  const uint32_t* mask = scratch + static_cast<uint64_t>(n) * L;  // [n][W]
  uint32_t* smask = sm;                                              // [kTile][W]
  uint16_t* sgap = reinterpret_cast<uint16_t*>(smask + kTile * W);   // [kTile]
  uint16_t* sexit = sgap + kTile;                                    // [kWarps][L]
  uint32_t g_entry = 1;
  for (uint32_t tile0 = 1; tile0 < n; tile0 += kTile) {
    const uint32_t m = min(kTile, n - tile0);
    for (uint32_t i = tid; i < m * W; i += kThreads) smask[i] = mask[static_cast<uint64_t>(tile0) * W + i];
    __syncthreads();
    const uint32_t run = (m + kWarps - 1) / kWarps;
    const uint32_t f0 = min(warp * run, m), f1 = min(f0 + run, m);
    for (uint32_t gin = lane + 1; gin <= L; gin += 32) {
      uint32_t g = gin;
      for (uint32_t f = f0; f < f1; ++f) g = next_gap(smask + f * W, g);
      sexit[warp * L + gin - 1] = static_cast<uint16_t>(g);
    }
    __syncthreads();
    if (tid == 0) {
      uint32_t g = g_entry;
      for (uint32_t w = 0; w < kWarps; ++w) {
        entry[w] = g;
        if (min(w * run, m) < min(w * run + run, m)) g = sexit[w * L + g - 1];
      }
      entry[kWarps] = g;
    }
    __syncthreads();
    if (lane == 0) {
      uint32_t g = entry[warp];
      for (uint32_t f = f0; f < f1; ++f) {
        sgap[f] = static_cast<uint16_t>(g);
        g = next_gap(smask + f * W, g);
      }
    }
    __syncthreads();
    for (uint32_t f = tid; f < m; f += kThreads) {
      const uint32_t t = tile0 + f, g = sgap[f];
      const uint64_t r = static_cast<uint64_t>(t) * L;
      const float s = __fdiv_rn(static_cast<float>(max(l1[r], l1[r + g - 1])), a.two_n);
      const bool nov = s >= a.tau;
      if (scores) scores[t] = s;
      if (keep) keep[t] = nov ? 1 : (g >= L ? 2 : 0);
    }
    g_entry = entry[kWarps];
    __syncthreads();
  }
  if (tid == 0) {
    if (scores) scores[0] = 0.0f;
    if (keep) keep[0] = 3;
  }
}

size_t static_smem_bytes(uint32_t l_max, uint32_t mask_words) {
  return static_cast<size_t>(kTile) * mask_words * 4 + kTile * 2 + static_cast<size_t>(kWarps) * l_max * 2;
}

// Per-device set-up: the device address of the static array, and the kernel's
// shared-memory limit raised to the largest size it can need.
std::mutex g_setup_mu;
uint32_t* g_scratch_ptr[kMaxDevices] = {};

cudaError_t setup_device(int dev, uint32_t** out) {
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_ptr[dev]) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_select_scratch);
    if (e != cudaSuccess) return e;
    const int smem = static_cast<int>(static_smem_bytes(kMaxLmax, (kMaxLmax + 31) / 32));
    e = cudaFuncSetAttribute(select_static_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = static_cast<uint32_t*>(ptr);
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

// Copies msg into the caller's buffer (if any); allocates nothing.
int fail(int code, const char* msg, char* err, size_t cap) {
  if (err && cap) {
    size_t i = 0;
    for (; msg[i] && i + 1 < cap; ++i) err[i] = msg[i];
    err[i] = 0;
  }
  return code;
}

bool on_device(const void* p, int dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) && a.device == dev;
}

}  // namespace
}  // namespace cofie

using namespace cofie;

extern "C" {

int cofie_ngff_select_static(const cofie_ngff_params* p, const uint32_t* hist, uint32_t n, float* scores_out,
                             uint8_t* keep_out, char* err, size_t err_cap, void* cuda_stream) {
  if (err && err_cap) err[0] = 0;
  if (!p) return fail(COFIE_EINVAL, "params is NULL", err, err_cap);
  if (p->width == 0 || p->height == 0 || static_cast<uint64_t>(p->width) * p->height > 0x7fffffffull)
    return fail(COFIE_EINVAL, "width * height must be in [1, 2^31)", err, err_cap);
  if (p->bins < 1 || p->bins > COFIE_NGFF_MAX_BINS) return fail(COFIE_EINVAL, "bins must be in [1, 256]", err, err_cap);
  if (p->l_max < 1 || p->l_max > COFIE_NGFF_MAX_LMAX)
    return fail(COFIE_EINVAL, "l_max must be in [1, 256]", err, err_cap);
  if (p->tau != p->tau) return fail(COFIE_EINVAL, "tau is NaN", err, err_cap);
  if (p->signal != COFIE_SIGNAL_HISTOGRAM)
    return fail(COFIE_EINVAL, "only the histogram signal (COFIE_SIGNAL_HISTOGRAM, no scene changes) is supported",
                err, err_cap);
  if (n == 0) return COFIE_OK;
  const uint32_t W = (p->l_max + 31) / 32;
  if (static_cast<uint64_t>(n) * (p->l_max + W) > kStaticScratchWords)
    return fail(COFIE_EINVAL,
                "n * (l_max + ceil(l_max / 32)) exceeds the static scratch of 1048576 words "
                "(at most 33825 frames for l_max = 30)",
                err, err_cap);
  if (!hist) return fail(COFIE_EINVAL, "hist is NULL", err, err_cap);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return fail(COFIE_ECUDA, "no usable current CUDA device", err, err_cap);
  if (!on_device(hist, dev) || (scores_out && !on_device(scores_out, dev)) || (keep_out && !on_device(keep_out, dev)))
    return fail(COFIE_EINVAL, "hist and the outputs must be device memory on the current device", err, err_cap);
  uint32_t* scratch = nullptr;
  cudaError_t e = setup_device(dev, &scratch);
  if (e != cudaSuccess) return fail(COFIE_ECUDA, cudaGetErrorString(e), err, err_cap);
  SelectArgs a{};
  a.bins = p->bins;
  a.l_max = p->l_max;
  a.mask_words = W;
  a.tau = p->tau;
  a.two_n = static_cast<float>(2ull * p->width * p->height);
  const size_t smem = static_smem_bytes(p->l_max, W);
  const cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const uint32_t win_grid = (n + kWinThreads / 32 - 1) / (kWinThreads / 32);
  if (p->bins % 4 == 0 && reinterpret_cast<uintptr_t>(hist) % 16 == 0)
    static_window_kernel<true><<<win_grid, kWinThreads, 0, st>>>(hist, n, a, scratch);
  else
    static_window_kernel<false><<<win_grid, kWinThreads, 0, st>>>(hist, n, a, scratch);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(COFIE_ECUDA, cudaGetErrorString(e), err, err_cap);
  select_static_kernel<<<1, kThreads, smem, st>>>(n, a, scratch, scores_out, keep_out);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(COFIE_ECUDA, cudaGetErrorString(e), err, err_cap);
  return COFIE_OK;
}

}  // extern "C"
