// K4 finalize and K5 gather: closing a stream prefix (CoFiE Sec. 3.2, the
// safeguards stated before Eq. 5) and handing the selected frames on.
//
// K4 (one 1024-thread CTA): the candidate set of a closed prefix of T frames,
//   S_c = {t : keep[t] != 0} U {T-1}, and, when |S_c| < M_min, also the
//   uniformly spaced frames round(i (T-1) / (M_min-1)), i = 0..M_min-1 (round
//   half up) -- written as sorted indices by a block-wide stream compaction
//   (ballot + popcount within warps, a scan of the 32 warp totals across them),
//   one 1024-frame tile at a time.
// K5 (2-D grid: frame x slice): copies the m selected frames of a stream back
//   to back into one buffer (the vision encoder's input), 16 bytes per thread
//   per step, streaming stores.
#include "ngff_common.cuh"

namespace cofie {
namespace {

constexpr int kFinThreads = 1024;
constexpr int kFinWarps = kFinThreads / 32;
constexpr int kGatherThreads = 256;
constexpr uint32_t kGatherVecPerThread = 4;

// t is one of round(i (T-1) / (M-1)), i = 0..M-1 (round half up)?
__device__ __forceinline__ bool in_uniform(uint64_t t, uint64_t T, uint64_t M) {
  if (M == 0) return false;
  if (M == 1 || T == 1) return t == 0;
  // smallest i whose rounded position is >= t, then test that position
  const uint64_t i = (t == 0) ? 0 : ((2 * t - 1) * (M - 1) + 2 * (T - 1) - 1) / (2 * (T - 1));
  if (i > M - 1) return false;
  return (2 * i * (T - 1) + (M - 1)) / (2 * (M - 1)) == t;
}

__global__ void __launch_bounds__(kFinThreads) candidates_kernel(const uint8_t* __restrict__ keep, uint32_t T,
                                                                 uint32_t m_min, uint32_t* __restrict__ idx,
                                                                 uint32_t* __restrict__ m_out) {
  __shared__ uint32_t wsum[kFinWarps];
  __shared__ uint32_t s_total;
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // retained frames before T-1, plus T-1 itself
  uint32_t c = 0;
  for (uint32_t t = tid; t + 1 < T; t += kFinThreads) c += keep[t] != 0;
  c = __reduce_add_sync(0xffffffffu, c);
  if (lane == 0) wsum[warp] = c;
  __syncthreads();
  if (warp == 0) {
    const uint32_t v = __reduce_add_sync(0xffffffffu, wsum[lane]);
    if (lane == 0) s_total = v + 1;
  }
  __syncthreads();
  const bool fill = s_total < m_min;
  __syncthreads();

  uint32_t base = 0;
  for (uint32_t t0 = 0; t0 < T; t0 += kFinThreads) {
    const uint32_t t = t0 + tid;
    const bool in = t < T && (keep[t] != 0 || t == T - 1 || (fill && in_uniform(t, T, m_min)));
    const uint32_t bal = __ballot_sync(0xffffffffu, in);
    const uint32_t before = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) wsum[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {  // exclusive scan of the warp totals
      const uint32_t v = wsum[lane];
      uint32_t x = v;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, d);
        if (lane >= static_cast<uint32_t>(d)) x += y;
      }
      wsum[lane] = x - v;
      if (lane == 31) s_total = x;
    }
    __syncthreads();
    if (in && COFIE_BOUND(base + wsum[warp] + before < T)) idx[base + wsum[warp] + before] = t;
    base += s_total;
    __syncthreads();
  }
  if (tid == 0) *m_out = base;
}

template <bool kVec>
__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const uint8_t* __restrict__ frames, uint32_t n_frames,
                                                                uint64_t frame_bytes, const uint32_t* __restrict__ idx,
                                                                uint32_t m, uint8_t* __restrict__ out,
                                                                uint32_t* __restrict__ err) {
  for (uint32_t f = blockIdx.y; f < m; f += gridDim.y) {
    const uint32_t sel = idx[f];
    if (sel >= n_frames) {  // an index outside the frame buffer: skip it and report
      if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(err, kErrBadIndex);
      continue;
    }
    const uint8_t* src = frames + static_cast<uint64_t>(sel) * frame_bytes;
    uint8_t* dst = out + static_cast<uint64_t>(f) * frame_bytes;
    if (kVec) {
      const uint64_t n16 = frame_bytes / 16;
      const uint4* s4 = reinterpret_cast<const uint4*>(src);
      uint4* d4 = reinterpret_cast<uint4*>(dst);
      const uint64_t i0 = static_cast<uint64_t>(blockIdx.x) * kGatherThreads * kGatherVecPerThread + threadIdx.x;
      uint4 v[kGatherVecPerThread];
#pragma unroll
      for (uint32_t u = 0; u < kGatherVecPerThread; ++u) {
        const uint64_t i = i0 + u * kGatherThreads;
        if (i < n16) v[u] = __ldg(s4 + i);
      }
#pragma unroll
      for (uint32_t u = 0; u < kGatherVecPerThread; ++u) {
        const uint64_t i = i0 + u * kGatherThreads;
        if (i < n16) __stcs(d4 + i, v[u]);
      }
    } else {
      for (uint64_t i = static_cast<uint64_t>(blockIdx.x) * kGatherThreads + threadIdx.x; i < frame_bytes;
           i += static_cast<uint64_t>(gridDim.x) * kGatherThreads)
        dst[i] = src[i];
    }
  }
}

}  // namespace

cudaError_t launch_candidates(const uint8_t* keep, uint32_t T, uint32_t m_min, uint32_t* idx, uint32_t* m_out,
                              cudaStream_t st) {
  candidates_kernel<<<1, kFinThreads, 0, st>>>(keep, T, m_min, idx, m_out);
  return cudaGetLastError();
}

cudaError_t launch_gather(const uint8_t* frames, uint32_t n_frames, uint64_t frame_bytes, const uint32_t* idx, uint32_t m,
                          uint8_t* out, uint32_t* err, cudaStream_t st) {
  const bool vec = frame_bytes % 16 == 0 && reinterpret_cast<uintptr_t>(frames) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(out) % 16 == 0;
  const uint32_t gy = m < 65535u ? m : 65535u;
  if (vec) {
    const uint64_t per_block = static_cast<uint64_t>(kGatherThreads) * kGatherVecPerThread;
    dim3 grid(static_cast<uint32_t>((frame_bytes / 16 + per_block - 1) / per_block), gy);
    gather_kernel<true><<<grid, kGatherThreads, 0, st>>>(frames, n_frames, frame_bytes, idx, m, out, err);
  } else {
    const uint64_t want = (frame_bytes + kGatherThreads - 1) / kGatherThreads;
    dim3 grid(static_cast<uint32_t>(want < 1024 ? want : 1024), gy);
    gather_kernel<false><<<grid, kGatherThreads, 0, st>>>(frames, n_frames, frame_bytes, idx, m, out, err);
  }
  return cudaGetLastError();
}

uint32_t take_bounds_errors_finalize() { return take_local_bounds_errors(); }

}  // namespace cofie
