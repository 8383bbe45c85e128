// K4 finalize and K5 gather: closing a stream prefix (CoFiE Sec. 3.2, the
// safeguards stated before Eq. 5) and handing the selected frames on.
//
// K4 (one 1024-thread CTA): the candidate set of a closed prefix of T frames,
//   S_c = {t : keep[t] != 0} U {T-1}, and, when |S_c| < M_min, also the
//   uniformly spaced frames round(i (T-1) / (M_min-1)), i = 0..M_min-1 (round
//   half up) -- written as sorted indices by a block-wide stream compaction
//   (ballot + popcount within warps, a scan of the 32 warp totals across them),
//   one 1024-frame tile at a time.
// K4 on a stream's retention record (one 1024-thread CTA): the same set for
//   the prefix a stream has been pushed so far, T read from the stream's
//   state on the device, the retained frames read from its record (one bit
//   per frame, written by the selection kernels), one word per thread per
//   step: popcounts, a block-wide exclusive scan, then each thread writes the
//   indices of its word's set bits.
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

// Exclusive block-wide prefix sum of one value per thread (kFinThreads
// threads); *total receives the sum. Uses wsum[kFinWarps] and ends with a
// barrier, so the caller may reuse both right away.
__device__ __forceinline__ uint32_t block_exclusive_sum(uint32_t v, uint32_t* wsum, uint32_t* total) {
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint32_t x = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, d);
    if (lane >= static_cast<uint32_t>(d)) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = wsum[lane];
    uint32_t z = w;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, z, d);
      if (lane >= static_cast<uint32_t>(d)) z += y;
    }
    wsum[lane] = z - w;
    if (lane == 31) *total = z;
  }
  __syncthreads();
  const uint32_t r = wsum[warp] + x - v;
  __syncthreads();
  return r;
}

// Bits of record word w of a prefix of T frames that belong to S_c: retained
// frames before T-1, the last frame T-1, and with `fill` the uniformly spaced
// frames.
__device__ __forceinline__ uint32_t candidate_bits(const uint32_t* rec, uint64_t w, uint64_t T, uint32_t m_min,
                                                   bool fill) {
  const uint64_t t0 = 32 * w;
  uint32_t bits = 0;
  if (t0 < T - 1) {
    bits = __ldcg(rec + w);
    if (T - 1 - t0 < 32) bits &= (1u << (T - 1 - t0)) - 1u;
  }
  if (T - 1 >= t0 && T - 1 < t0 + 32) bits |= 1u << (T - 1 - t0);
  if (fill)
    for (uint32_t i = 0; i < 32 && t0 + i < T; ++i)
      if (in_uniform(t0 + i, T, m_min)) bits |= 1u << i;
  return bits;
}

__global__ void __launch_bounds__(kFinThreads) stream_candidates_kernel(const uint32_t* __restrict__ rec,
                                                                        uint32_t rec_words,
                                                                        const StreamState* __restrict__ state,
                                                                        uint32_t m_min, uint32_t* __restrict__ idx,
                                                                        uint32_t cap, uint32_t* __restrict__ m_out,
                                                                        uint32_t* __restrict__ err) {
  __shared__ uint32_t wsum[kFinWarps];
  __shared__ uint32_t s_total;
  const uint32_t tid = threadIdx.x;
  const uint64_t T = __ldcg(&state->t);
  if (T > 32ull * rec_words) {  // the stream has run past its record: no candidate set
    if (tid == 0) {
      atomicOr(err, kErrRecord);
      *m_out = 0;
    }
    return;
  }
  if (T == 0) {
    if (tid == 0) *m_out = 0;
    return;
  }
  const uint64_t words = (T + 31) / 32;
  // |S| before the fill: retained frames before T-1, plus T-1
  uint32_t c = 0;
  for (uint64_t w = tid; w < words; w += kFinThreads) c += __popc(candidate_bits(rec, w, T, m_min, false));
  block_exclusive_sum(c, wsum, &s_total);
  const bool fill = s_total < m_min;
  uint32_t base = 0;
  for (uint64_t w0 = 0; w0 < words; w0 += kFinThreads) {
    const uint64_t w = w0 + tid;
    uint32_t bits = w < words ? candidate_bits(rec, w, T, m_min, fill) : 0u;
    const uint32_t off = base + block_exclusive_sum(__popc(bits), wsum, &s_total);
    for (uint32_t k = 0; bits; ++k, bits &= bits - 1) {
      const uint32_t pos = off + k;
      if (pos < cap) idx[pos] = static_cast<uint32_t>(32 * w) + (__ffs(bits) - 1);
    }
    base += s_total;
    __syncthreads();
  }
  if (tid == 0) *m_out = base;
}

// A stream restarts at t = 0: the record bits of the frames it has seen are
// cleared (bits are set only below t) and its state zeroed.
__global__ void stream_reset_kernel(StreamState* __restrict__ state, uint32_t* __restrict__ rec, uint32_t rec_words) {
  const uint64_t t = __ldcg(&state->t);
  const uint64_t words = min((t + 31) / 32, static_cast<uint64_t>(rec_words));
  for (uint64_t w = threadIdx.x; w < words; w += blockDim.x) rec[w] = 0;
  __syncthreads();
  if (threadIdx.x == 0) *state = StreamState{0ull, 0u, 0u, 0ull};
}

// kHostSrc: the frames are pinned host memory read through the device's
// mapping of it (plain loads; the read-only path is kept for device frames).
template <bool kVec, bool kHostSrc>
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
        if (i < n16) v[u] = kHostSrc ? s4[i] : __ldg(s4 + i);
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

cudaError_t launch_stream_candidates(const uint32_t* rec, uint32_t rec_words, const StreamState* state,
                                     uint32_t m_min, uint32_t* idx, uint32_t cap, uint32_t* m_out, uint32_t* err,
                                     cudaStream_t st) {
  stream_candidates_kernel<<<1, kFinThreads, 0, st>>>(rec, rec_words, state, m_min, idx, cap, m_out, err);
  return cudaGetLastError();
}

cudaError_t launch_stream_reset(StreamState* state, uint32_t* rec, uint32_t rec_words, cudaStream_t st) {
  stream_reset_kernel<<<1, 1024, 0, st>>>(state, rec, rec_words);
  return cudaGetLastError();
}

cudaError_t launch_gather(const uint8_t* frames, uint32_t n_frames, uint64_t frame_bytes, const uint32_t* idx, uint32_t m,
                          uint8_t* out, uint32_t* err, bool host_src, cudaStream_t st) {
  const bool vec = frame_bytes % 16 == 0 && reinterpret_cast<uintptr_t>(frames) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(out) % 16 == 0;
  const uint32_t gy = m < 65535u ? m : 65535u;
  if (vec) {
    const uint64_t per_block = static_cast<uint64_t>(kGatherThreads) * kGatherVecPerThread;
    dim3 grid(static_cast<uint32_t>((frame_bytes / 16 + per_block - 1) / per_block), gy);
    if (host_src)
      gather_kernel<true, true><<<grid, kGatherThreads, 0, st>>>(frames, n_frames, frame_bytes, idx, m, out, err);
    else
      gather_kernel<true, false><<<grid, kGatherThreads, 0, st>>>(frames, n_frames, frame_bytes, idx, m, out, err);
  } else {
    const uint64_t want = (frame_bytes + kGatherThreads - 1) / kGatherThreads;
    dim3 grid(static_cast<uint32_t>(want < 1024 ? want : 1024), gy);
    gather_kernel<false, false><<<grid, kGatherThreads, 0, st>>>(frames, n_frames, frame_bytes, idx, m, out, err);
  }
  return cudaGetLastError();
}

uint32_t take_bounds_errors_finalize() { return take_local_bounds_errors(); }

}  // namespace cofie
