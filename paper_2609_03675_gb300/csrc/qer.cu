// Query-specific evidence refinement (QER), CoFiE Sec. 3.3, Eqs. 6-8, on the
// GB300 tensor cores.
//
//   a_ij = (1/H) sum_h <q_i^h, k_j^h> / sqrt(d_h)            (Eq. 6)
//   w_f  = mean_{j in V_f} max_{i in Q} a_ij                  (Eq. 7)
//   S_e  = TopK_f(w_f, max(1, round(rho |S_c|))), in time order (Eq. 8)
//
// With grouped key/value heads (query head h reads key head h / G, G = H/H_kv)
// the head mean of Eq. 6 is one dot product over D = H_kv * d_h once the G
// query heads of each group are summed:
//   a_ij = <q~_i, k_j> / (H sqrt(d_h)),  q~_i[g, c] = sum_{h in group g} q_i^h[c].
// So Eq. 6 is a single bf16 GEMM-shaped contraction, Q~ [N x D] times K^T
// [D x n_visual], whose column maxima over text (Eq. 7, inner max) are all
// that is kept: the text-by-vision score matrix is never written to memory,
// which is the point of the paper's tiled computation.
//
// Kernels (one QER call launches four):
//   qer_prepare_q   q [n_text][H][d] -> q~ [N][D] bf16 (fp32 sums rounded to
//                   nearest even; rows n_text..N-1 zero, N = n_text rounded up to 16)
//   qer_score       persistent CTAs over tiles of 256 visual tokens: TMA
//                   (cp.async.bulk.tensor, 128-byte swizzle) streams 64-wide K
//                   chunks of the token tile and of q~ into a shared-memory
//                   ring; one thread issues tcgen05.mma (kind::f16, M = 128 per
//                   half tile, N, K = 16) into TMEM accumulators (128 lanes x N
//                   fp32 columns per half) and commits each stage back to the
//                   producer; four epilogue warps read the accumulators
//                   (tcgen05.ld) and keep each token's max over the n_text
//                   real columns;
//   qer_score_pair  the same over pairs of SMs (tcgen05 cta_group::2), for
//                   runs longer than one wave of qer_score;
//   qer_mean        w_f = (sum of the frame's token maxima) / (|V_f| H sqrt(d)),
//                   a warp per frame;
//   qer_rank        the k best frames by rank (ties to the lower index), a
//                   warp per frame; the last CTA writes them in time order.
// Every kernel after the first is a programmatic dependent of the one before
// it, so its launch and set-up overlap that kernel's tail.
// Every mbarrier wait is bounded by the global timer; a wait that runs out
// sets an error bit, stops issuing, lets the work already issued finish
// (bounded) and frees TMEM before the CTA exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "cofie_ngff.h"
#include "ngff_common.cuh"

namespace cofie {
namespace {

constexpr int kQerM = 128;          // visual tokens per MMA (M)
constexpr int kQerTile = 2 * kQerM; // visual tokens per tile: two MMAs share each q~ chunk
constexpr int kQerKChunk = 64;      // bf16 elements per 128-byte swizzled row
constexpr uint32_t kQerMaxStages = 8;
constexpr size_t kQerStageBudget = 200 * 1024;  // shared memory for the ring
constexpr int kQerUmmaK = 16;       // K of one tcgen05.mma for 16-bit inputs
constexpr int kQerEpiWarps = 4;    // epilogue warps: TMEM lanes 0..127
constexpr int kQerThreads = 32 * (2 + kQerEpiWarps);  // + TMA producer warp + MMA issuer warp
constexpr int kQerPairThreads = kQerThreads + 32;     // paired kernel: + a second producer warp (q~)
constexpr size_t kQerPairRingBudget = 224 * 1024;     // paired kernel: both rings (one CTA per SM)
constexpr uint32_t kQerPairQSlots = 3;                // q~ slots: enough to cover its L2 latency
constexpr uint32_t kQerMaxN = 256;      // text tokens (MMA N) per scoring pass
constexpr uint32_t kQerMaxText = 4096;  // text tokens per query: up to 16 passes
constexpr int kRankThreads = 256;  // 8 frames per CTA (a warp each): the O(m^2) ranking spreads over many SMs
constexpr uint32_t kRankTile = 2048;  // scores staged per pass of the ranking (8 KiB of shared memory)

constexpr uint32_t kQerErrProducer = 16u, kQerErrMma = 32u, kQerErrEpilogue = 64u, kQerErrDrain = 128u;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
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

__device__ __noinline__ bool mbar_wait_for(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try(bar, parity)) return true;
  const uint64_t t0 = gtimer();
  for (;;) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try(bar, parity)) return true;
    if (gtimer() - t0 > timeout_ns) return false;
  }
}

#if COFIE_DEBUG_CHECKS
// Bytes of dynamic shared memory this launch gave the CTA (checked build).
__device__ __forceinline__ uint32_t dynamic_smem_bytes() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(r));
  return r;
}
#endif

// The common case inline (the phase has already completed), the bounded
// wait loop out of line.
__device__ __forceinline__ bool mbar_wait_fast(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  return mbar_try(bar, parity) || mbar_wait_for(bar, parity, timeout_ns);
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int32_t x, int32_t y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major, 128-byte-swizzled tile whose
// rows are 128 bytes and whose 8-row swizzle atoms are 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr >> 4) & 0x3FFFu);  // start address
  d |= static_cast<uint64_t>(1u) << 16;                // leading byte offset (unused for swizzled K-major)
  d |= static_cast<uint64_t>(1024u >> 4) << 32;        // stride byte offset: 8 rows x 128 B
  d |= static_cast<uint64_t>(1u) << 46;                // descriptor version
  d |= static_cast<uint64_t>(2u) << 61;                // swizzle: 128 B
  return d;
}

// Instruction descriptor: bf16 x bf16 -> fp32, both operands K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(uint32_t m, uint32_t n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((n >> 3) << 17) | ((m >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// Programmatic dependent launch: let the next kernel in the stream be
// scheduled now / wait until the previous one has completed and its memory
// is visible (a no-op when the kernel was not launched as a dependent).
__device__ __forceinline__ void grid_dependents_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this thread's TMEM lane, without waiting.
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Max over the first n_text columns of this thread's TMEM lane (n_pad columns,
// a multiple of 16), reading 64 columns per wait.
__device__ __forceinline__ float tmem_row_max(uint32_t taddr, uint32_t n_pad, uint32_t n_text) {
  float best = -INFINITY;
  for (uint32_t c0 = 0; c0 < n_pad; c0 += 64) {
    uint32_t r0[32], r1[32];
    tmem_ld32_nowait(taddr + c0, r0);
    const bool two = c0 + 32 < n_pad;
    if (two) tmem_ld32_nowait(taddr + c0 + 32, r1);
    tmem_wait_ld();
    if (c0 + 64 <= n_text) {  // every column of the block is a real text token: no mask
      float m0 = __uint_as_float(r0[0]), m1 = __uint_as_float(r1[0]);
#pragma unroll
      for (uint32_t c = 1; c < 32; ++c) {
        m0 = fmaxf(m0, __uint_as_float(r0[c]));
        m1 = fmaxf(m1, __uint_as_float(r1[c]));
      }
      best = fmaxf(best, fmaxf(m0, m1));
      continue;
    }
#pragma unroll
    for (uint32_t c = 0; c < 32; ++c)
      if (c0 + c < n_text) best = fmaxf(best, __uint_as_float(r0[c]));
    if (two) {
#pragma unroll
      for (uint32_t c = 0; c < 32; ++c)
        if (c0 + 32 + c < n_text) best = fmaxf(best, __uint_as_float(r1[c]));
    }
  }
  return best;
}


// ---- paired-SM helpers (clusters of two CTAs) ----

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The address of the same shared variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}

__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

__device__ __forceinline__ bool mbar_try_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// A wait on a barrier that the peer CTA also arrives on (cluster-scope acquire).
__device__ __noinline__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try_cluster(bar, parity)) return true;
  const uint64_t t0 = gtimer();
  for (;;) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_cluster(bar, parity)) return true;
    if (gtimer() - t0 > timeout_ns) return false;
  }
}

// A tile load into this CTA's shared memory whose completion is counted on a
// barrier that may live in the peer CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int32_t x, int32_t y,
                                                 uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%2, %3}], "
      "[%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar_cluster)
      : "memory");
}

__device__ __forceinline__ void umma_pair_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

// Arrives on the barrier at this shared offset in both CTAs of the pair once
// every MMA this thread issued so far has completed.
__device__ __forceinline__ void umma_pair_commit_both(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// q~ row p of n_rows belongs to text block p / bp, row p % bp of it; block b
// holds text tokens [b per_blk, (b + 1) per_blk), the rest of its bp rows are
// zero. Returns the text token, or n_text for a zero row.
__device__ __forceinline__ uint32_t qer_text_of_row(uint32_t p, uint32_t bp, uint32_t per_blk, uint32_t n_text) {
  const uint32_t b = p / bp, r = p % bp, i = b * per_blk + r;
  return (r < per_blk && i < n_text) ? i : n_text;
}

__global__ void qer_prepare_q(const uint16_t* __restrict__ q, uint32_t n_text, uint32_t n_rows, uint32_t bp,
                              uint32_t per_blk, uint32_t H, uint32_t H_kv, uint32_t d,
                              __nv_bfloat16_raw* __restrict__ qg) {
  grid_dependents_launch();  // the scoring kernel may start; its q~ loads wait for this grid
  const uint32_t D = H_kv * d, G = H / H_kv;
  const uint64_t total = static_cast<uint64_t>(n_rows) * D;
  for (uint64_t e = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint32_t i = qer_text_of_row(static_cast<uint32_t>(e / D), bp, per_blk, n_text), r = static_cast<uint32_t>(e % D);
    const uint32_t g = r / d, c = r % d;
    float s = 0.f;
    if (i < n_text)
      for (uint32_t h = g * G; h < (g + 1) * G; ++h)
        s += __uint_as_float(static_cast<uint32_t>(q[(static_cast<uint64_t>(i) * H + h) * d + c]) << 16);
    qg[e] = static_cast<__nv_bfloat16_raw>(__float2bfloat16_rn(s));
  }
}

// The same with 8 consecutive channels per thread (d % 8 == 0, 16-byte aligned q).
__global__ void qer_prepare_q8(const uint4* __restrict__ q, uint32_t n_text, uint32_t n_rows, uint32_t bp,
                               uint32_t per_blk, uint32_t H, uint32_t H_kv, uint32_t d, uint4* __restrict__ qg) {
  grid_dependents_launch();  // the scoring kernel may start; its q~ loads wait for this grid
  const uint32_t d8 = d / 8, D8 = H_kv * d8, G = H / H_kv;
  const uint64_t total = static_cast<uint64_t>(n_rows) * D8;
  for (uint64_t e = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint32_t i = qer_text_of_row(static_cast<uint32_t>(e / D8), bp, per_blk, n_text), r = static_cast<uint32_t>(e % D8);
    const uint32_t g = r / d8, c8 = r % d8;
    float s[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (i < n_text)
      for (uint32_t h = g * G; h < (g + 1) * G; ++h) {
        const uint4 v = q[(static_cast<uint64_t>(i) * H + h) * d8 + c8];
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          s[2 * k] += __uint_as_float(w[k] << 16);
          s[2 * k + 1] += __uint_as_float(w[k] & 0xFFFF0000u);
        }
      }
    uint32_t out[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint32_t lo = static_cast<__nv_bfloat16_raw>(__float2bfloat16_rn(s[2 * k])).x;
      const uint32_t hi = static_cast<__nv_bfloat16_raw>(__float2bfloat16_rn(s[2 * k + 1])).x;
      out[k] = lo | (hi << 16);
    }
    qg[e] = make_uint4(out[0], out[1], out[2], out[3]);
  }
}

// Persistent, warp-specialised scoring kernel over tiles of 256 visual
// tokens (two M = 128 halves sharing every q~ chunk, which halves the q~
// traffic per token). Warp 0 (one thread) streams TMA chunks of the CTA's
// tiles into an n_stages ring (per stage: two 16 KiB key halves + the q~
// chunk); warp 1 (one thread) issues, per 16-wide K step, one MMA per half
// into accumulator pair t % n_buf (two blocks of acc_cols TMEM columns);
// warps 2..5 read the pair (warp w owns TMEM lanes 32 (w % 4) ..), so with
// two buffers the epilogue of tile t overlaps the MMAs of tile t + 1.
// Barriers: full/empty per ring stage (TMA bytes / MMA completion),
// tfull/tempty per accumulator pair (MMA completion / the epilogue warps).
__global__ void __launch_bounds__(kQerThreads) qer_score(const __grid_constant__ CUtensorMap map_k,
                                                         const __grid_constant__ CUtensorMap map_q,
                                                         uint32_t n_visual, uint32_t n_text, uint32_t n_pad,
                                                         uint32_t fold, uint32_t acc_cols, uint32_t n_buf,
                                                         uint32_t n_stages,
                                                         uint32_t n_chunks, uint32_t n_tiles,
                                                         float* __restrict__ colmax, uint32_t* __restrict__ err,
                                                         uint64_t timeout_ns) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kQerMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kQerMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile uint32_t abort_flag;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t half_bytes = kQerM * 128, a_bytes = 2 * half_bytes, b_bytes = n_pad * 128;
  const uint32_t stage_bytes = a_bytes + ((b_bytes + 1023) & ~1023u);
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t my_tiles = blockIdx.x < n_tiles ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
  const uint32_t tmem_total = 2 * acc_cols * n_buf;
  // checked build: the ring ends inside this launch's dynamic shared memory,
  // its slots fit the barrier arrays, and each accumulator's n_pad columns
  // lie inside its acc_cols (a failed check runs no tile: my_tiles = 0)
  const bool layout_ok = COFIE_BOUND(smem_u32(smem) + n_stages * stage_bytes <=
                                         smem_u32(smem_raw) + dynamic_smem_bytes() &&
                                     n_stages >= 1 && n_stages <= kQerMaxStages && n_pad <= acc_cols &&
                                     n_buf >= 1 && n_buf <= 2);

  if (warp == 0) {  // the whole warp allocates the accumulators
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(tmem_total)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (threadIdx.x == 32) {
    for (uint32_t s = 0; s < n_stages; ++s) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&full_bar[s])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&empty_bar[s])) : "memory");
    }
    for (int b = 0; b < 2; ++b) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&tfull_bar[b])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(&tempty_bar[b])), "r"(kQerEpiWarps)
                   : "memory");
    }
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&done_bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    abort_flag = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // --------------------------------------------------------- TMA producer
      grid_dependency_wait();  // q~ is written by the kernel before this one
      const uint32_t ring0 = smem_u32(smem), empty0 = smem_u32(&empty_bar[0]), full0 = smem_u32(&full_bar[0]);
      uint32_t g = 0, s = 0, ph = 0;  // chunk counter over all of this CTA's tiles; ring slot and phase
      bool stop = false;
      for (uint32_t t = 0; t < (layout_ok ? my_tiles : 0u) && !stop; ++t) {
        const int32_t row0 = static_cast<int32_t>((blockIdx.x + t * gridDim.x) * kQerTile);
        for (uint32_t kc = 0; kc < n_chunks; ++kc, ++g) {
          if (g >= n_stages && !mbar_wait_fast(empty0 + 8 * s, ph ^ 1, timeout_ns)) {
            atomicOr(err, kQerErrProducer);
            abort_flag = 1;
            stop = true;
            break;
          }
          const uint32_t fb = full0 + 8 * s;
          asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb), "r"(a_bytes + b_bytes)
                       : "memory");
          const uint32_t base = ring0 + s * stage_bytes;
          const int32_t x = static_cast<int32_t>(kc * kQerKChunk);
          tma_load_2d(base, &map_k, x, row0, fb);
          tma_load_2d(base + half_bytes, &map_k, x, row0 + kQerM, fb);
          tma_load_2d(base + a_bytes, &map_q, x, 0, fb);
          if (++s == n_stages) {
            s = 0;
            ph ^= 1;
          }
        }
      }
      // no copy may still be writing shared memory when the CTA exits
      for (uint32_t j = g > n_stages ? g - n_stages : 0; j < g; ++j)
        if (!mbar_wait_for(smem_u32(&full_bar[j % n_stages]), (j / n_stages) & 1, timeout_ns))
          atomicOr(err, kQerErrDrain);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ----------------------------------------------------------- MMA issuer
      // Per stage: one inline try of the full barrier, descriptors formed
      // once and stepped by the 32-byte K offset (the ring lies below 256
      // KiB, so the descriptor's 14-bit address field never carries).
      const uint32_t idesc = idesc_bf16_f32(kQerM, n_pad);
      const uint32_t ring0 = smem_u32(smem), empty0 = smem_u32(&empty_bar[0]), full0 = smem_u32(&full_bar[0]);
      uint32_t s = 0, ph = 0;
      bool stop = false;
      for (uint32_t t = 0; t < (layout_ok ? my_tiles : 0u) && !stop && !abort_flag; ++t) {
        const uint32_t b = t % n_buf, ub = t / n_buf;
        if (ub > 0 && !mbar_wait_fast(smem_u32(&tempty_bar[b]), (ub - 1) & 1, timeout_ns)) {
          atomicOr(err, kQerErrMma);
          abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t acc0 = tmem + b * 2 * acc_cols, acc1 = acc0 + acc_cols;
        for (uint32_t kc = 0; kc < n_chunks; ++kc) {
          if (!mbar_wait_fast(full0 + 8 * s, ph, timeout_ns)) {
            atomicOr(err, kQerErrMma);
            abort_flag = 1;
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = ring0 + s * stage_bytes;
          const uint64_t da0 = sw128_desc(a0), da1 = sw128_desc(a0 + half_bytes), db = sw128_desc(a0 + a_bytes);
          const uint32_t first = kc != 0;  // 0: the tile's first MMAs overwrite the accumulators
#pragma unroll
          for (uint32_t kk = 0; kk < kQerKChunk / kQerUmmaK; ++kk) {
            const uint64_t o = kk * (kQerUmmaK * 2 / 16);
            umma_bf16(acc0, da0 + o, db + o, idesc, kk ? 1u : first);
            umma_bf16(acc1, da1 + o, db + o, idesc, kk ? 1u : first);
          }
          umma_commit(empty0 + 8 * s);  // the stage is free once these MMAs have read it
          if (++s == n_stages) {
            s = 0;
            ph ^= 1;
          }
        }
        if (stop) break;
        umma_commit(smem_u32(&tfull_bar[b]));  // accumulator pair b holds tile t
      }
      umma_commit(smem_u32(&done_bar));  // every MMA this CTA issued is complete
    }
  } else {
    // --------------------------------------------------------------- epilogue
    const uint32_t quarter = warp & 3;  // TMEM lanes this warp may read
    for (uint32_t t = 0; t < (layout_ok ? my_tiles : 0u); ++t) {
      const uint32_t b = t % n_buf, ub = t / n_buf;
      bool ok = !abort_flag && mbar_wait_for(smem_u32(&tfull_bar[b]), ub & 1, timeout_ns);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) {
        if (lane == 0) atomicOr(err, kQerErrEpilogue);
        abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint32_t row0 = (blockIdx.x + t * gridDim.x) * kQerTile;
#pragma unroll 1
      for (uint32_t half = 0; half < 2; ++half) {
        const uint32_t taddr = tmem + (b * 2 + half) * acc_cols + ((quarter * 32u) << 16);
        const float best = tmem_row_max(taddr, n_pad, n_text);
        const uint32_t j = row0 + half * kQerM + quarter * 32 + lane;
        if (j < n_visual) colmax[j] = fold ? fmaxf(colmax[j], best) : best;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&tempty_bar[b])) : "memory");
    }
  }
  __syncwarp();
  // TMEM is freed only after every MMA this CTA issued has completed
  if (warp == 0) {
    const bool ok = mbar_wait_for(smem_u32(&done_bar), 0, timeout_ns);
    if (!ok && lane == 0) atomicOr(err, kQerErrDrain);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_total) : "memory");
  }
}

// Paired-SM scoring kernel (tcgen05 cta_group::2; clusters of two CTAs on two
// SMs). The pair covers a 256-token tile with one M = 256 MMA per 16-wide K
// step: CTA rank r stages key rows [128 r, 128 r + 128) of the tile (A) and
// q~ rows [r n_pad / 2, (r + 1) n_pad / 2) (half of B); the MMA, issued by
// rank 0, reads both CTAs' halves and writes each CTA's 128 token rows x
// n_pad text columns into that CTA's TMEM. Against the one-SM kernel this
// halves the shared-memory reads of q~ per SM (each half of B is read once
// for both SMs) and needs one accumulator of acc_cols columns per tile, so
// two of them overlap a tile's epilogue with the next tile's MMAs.
//
// Keys and q~ stream through two rings of kSub 64-wide K chunks per slot:
// keys come from DRAM and want as many bytes in flight as shared memory
// allows, q~ (the same for every tile) comes from L2 and needs only the few
// slots that cover its L2 latency, so the q~ chunks do not take key slots.
// Warp 0 streams keys, the last warp q~, warp 1 (rank 0) issues the MMAs,
// warps 2..5 are the epilogue.
//
// Synchronisation: each CTA's producers fill their own ring slots, and both
// CTAs' copies count their bytes on rank 0's full barriers (rank 1 through
// the paired form of the tensor copy), which rank 0's producers arm with the
// bytes of both; rank 0's MMA thread waits on them alone, and commits MMA
// completion to the empty barriers and accumulator barriers of both CTAs at
// once (multicast). The ring barriers are completed by the asynchronous
// proxy only (copy bytes, MMA commits), so their waits are CTA-scoped; the
// tempty barrier, on which the epilogue warps of both CTAs arrive, is waited
// on at cluster scope. Every wait is bounded, and both CTAs always meet at a
// final cluster barrier before TMEM is freed.
template <uint32_t kSub>
__global__ void __launch_bounds__(kQerPairThreads) qer_score_pair(
    const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_qh, uint32_t n_visual,
    uint32_t n_text, uint32_t n_pad, uint32_t fold, uint32_t acc_cols, uint32_t n_kst, uint32_t n_qst, uint32_t n_chunks,
    uint32_t n_tiles, float* __restrict__ colmax, uint32_t* __restrict__ err, uint64_t timeout_ns) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t kfull_bar[kQerMaxStages];
  __shared__ __align__(8) uint64_t kempty_bar[kQerMaxStages];
  __shared__ __align__(8) uint64_t qfull_bar[kQerMaxStages];
  __shared__ __align__(8) uint64_t qempty_bar[kQerMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ volatile uint32_t abort_flag;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t rank = cluster_ctarank();
  const uint32_t n_pairs = gridDim.x / 2, pair = blockIdx.x / 2;
  const uint32_t half_rows = n_pad / 2;
  const uint32_t a_chunk = kQerM * 128, b_chunk = half_rows * 128;  // one 64-wide K chunk of A / of half of B
  const uint32_t kslot = kSub * a_chunk, qslot = kSub * b_chunk;
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t my_tiles = pair < n_tiles ? (n_tiles - 1 - pair) / n_pairs + 1 : 0;
  const uint32_t tmem_total = 2 * acc_cols;  // two accumulators
  const uint32_t kring0 = smem_u32(smem), qring0 = kring0 + n_kst * kslot;
  // checked build: both rings end inside this launch's dynamic shared memory,
  // their slots fit the barrier arrays, the accumulators' n_pad columns lie
  // inside acc_cols, and the grid is whole clusters of two (a failed check
  // runs no tile: my_tiles = 0 in both CTAs, which see the same arguments)
  const bool layout_ok = COFIE_BOUND(qring0 + n_qst * qslot <= smem_u32(smem_raw) + dynamic_smem_bytes() &&
                                     n_kst >= 1 && n_kst <= kQerMaxStages && n_qst >= 1 && n_qst <= kQerMaxStages &&
                                     n_pad <= acc_cols && n_pad % 32 == 0 && gridDim.x % 2 == 0);
  const uint32_t run_tiles = layout_ok ? my_tiles : 0u;

  if (warp == 0) {  // one warp in each CTA of the pair allocates, together
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(tmem_total)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  if (threadIdx.x == 32) {
    for (uint32_t i = 0; i < n_kst; ++i) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&kfull_bar[i])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&kempty_bar[i])) : "memory");
    }
    for (uint32_t i = 0; i < n_qst; ++i) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&qfull_bar[i])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&qempty_bar[i])) : "memory");
    }
    for (int b = 0; b < 2; ++b) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&tfull_bar[b])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(&tempty_bar[b])), "r"(2 * kQerEpiWarps)
                   : "memory");
    }
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&done_bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    abort_flag = 0;
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers exist before any remote arrive or multicast commit
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  if (warp == 0 || warp == kQerPairThreads / 32 - 1) {
    if (lane == 0) {
      // ----------------------------- producers (both CTAs): warp 0 keys, last warp q~
      // Slot s and its phase ph advance incrementally; a wait that runs out
      // stops this thread (the other roles then run out on theirs).
      const bool keys = warp == 0;
      const uint32_t n_slots = keys ? n_kst : n_qst, slot_bytes = keys ? kslot : qslot;
      const uint32_t chunk = keys ? a_chunk : b_chunk, ring0 = keys ? kring0 : qring0;
      const uint32_t empty0 = smem_u32(keys ? &kempty_bar[0] : &qempty_bar[0]);
      const uint32_t full0 = smem_u32(keys ? &kfull_bar[0] : &qfull_bar[0]);
      const uint32_t full0_rank0 = map_to_rank(full0, 0);  // rank 0's full barriers count both CTAs' bytes
      const CUtensorMap* map = keys ? &map_k : &map_qh;
      const uint32_t tx = 2 * kSub * chunk;
      if (!keys) grid_dependency_wait();  // q~ is written by the kernel before this one; keys stream at once
      uint32_t g = 0, s = 0, ph = 0;
      bool stop = false;
      for (uint32_t t = 0; t < run_tiles && !stop; ++t) {
        const int32_t y = keys ? static_cast<int32_t>((pair + t * n_pairs) * kQerTile + rank * kQerM)
                               : static_cast<int32_t>(rank * half_rows);
        for (uint32_t kc = 0; kc < n_chunks; ++kc, ++g) {
          if (g >= n_slots && !mbar_wait_fast(empty0 + 8 * s, ph ^ 1, timeout_ns)) {
            atomicOr(err, kQerErrProducer);
            abort_flag = 1;
            stop = true;
            break;
          }
          if (rank == 0)
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(full0 + 8 * s), "r"(tx) : "memory");
          const uint32_t base = ring0 + s * slot_bytes, fb = full0_rank0 + 8 * s;
#pragma unroll
          for (uint32_t sub = 0; sub < kSub; ++sub)
            tma_load_2d_pair(base + sub * chunk, map, static_cast<int32_t>((kc * kSub + sub) * kQerKChunk), y, fb);
          if (++s == n_slots) {
            s = 0;
            ph ^= 1;
          }
        }
      }
      // no copy may still be writing shared memory when the CTA exits: the
      // last copies of every slot were read by MMAs whose completion reached
      // this CTA's empty barrier
      for (uint32_t j = g > n_slots ? g - n_slots : 0; j < g; ++j)
        if (!mbar_wait_cluster(empty0 + 8 * (j % n_slots), (j / n_slots) & 1, timeout_ns)) atomicOr(err, kQerErrDrain);
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ------------------------------------------------ MMA issuer (rank 0)
      // One thread issues every MMA of the pair, so its per-stage work is
      // kept small: slots and phases advance incrementally, the first try of
      // each wait is inline, and each stage's shared-memory descriptors are
      // formed once and stepped by the 32-byte K offset (2 in the
      // descriptor's 16-byte address units; the rings lie below 256 KiB, so
      // the 14-bit address field never carries).
      const uint32_t idesc = idesc_bf16_f32(2 * kQerM, n_pad);
      const uint32_t kfull0 = smem_u32(&kfull_bar[0]), kempty0 = smem_u32(&kempty_bar[0]);
      const uint32_t qfull0 = smem_u32(&qfull_bar[0]), qempty0 = smem_u32(&qempty_bar[0]);
      const uint64_t a16 = a_chunk >> 4, b16 = b_chunk >> 4;
      uint32_t ks = 0, kph = 0, qs = 0, qph = 0;
      bool stop = false;
      for (uint32_t t = 0; t < run_tiles && !stop && !abort_flag; ++t) {
        const uint32_t b = t & 1, ub = t >> 1;
        if (ub > 0 && !mbar_wait_cluster(smem_u32(&tempty_bar[b]), (ub - 1) & 1, timeout_ns)) {
          atomicOr(err, kQerErrMma);
          abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + b * acc_cols;
        for (uint32_t kc = 0; kc < n_chunks; ++kc) {
          if (!mbar_wait_fast(kfull0 + 8 * ks, kph, timeout_ns) || !mbar_wait_fast(qfull0 + 8 * qs, qph, timeout_ns)) {
            atomicOr(err, kQerErrMma);
            abort_flag = 1;
            stop = true;
            break;
          }
          tc_fence_after();
          const uint64_t da = sw128_desc(kring0 + ks * kslot), db = sw128_desc(qring0 + qs * qslot);
          const uint32_t first = kc != 0;  // 0: the tile's first MMA overwrites the accumulator
#pragma unroll
          for (uint32_t sub = 0; sub < kSub; ++sub)
#pragma unroll
            for (uint32_t kk = 0; kk < kQerKChunk / kQerUmmaK; ++kk) {
              const uint64_t o = kk * (kQerUmmaK * 2 / 16);
              umma_pair_bf16(acc, da + sub * a16 + o, db + sub * b16 + o, idesc, (sub | kk) ? 1u : first);
            }
          umma_pair_commit_both(kempty0 + 8 * ks);  // both CTAs' slots are free once read
          umma_pair_commit_both(qempty0 + 8 * qs);
          if (++ks == n_kst) {
            ks = 0;
            kph ^= 1;
          }
          if (++qs == n_qst) {
            qs = 0;
            qph ^= 1;
          }
        }
        if (stop) break;
        umma_pair_commit_both(smem_u32(&tfull_bar[b]));  // accumulator b holds tile t in both CTAs
      }
      umma_pair_commit_both(smem_u32(&done_bar));  // every MMA of the pair is complete
    }
  } else {
    // ------------------------------------------------------ epilogue (both CTAs)
    const uint32_t quarter = warp & 3;  // warps 2..5: TMEM lanes 32 (warp % 4) ..
    const uint32_t tempty0 = map_to_rank(smem_u32(&tempty_bar[0]), 0);
    const uint32_t tempty1 = map_to_rank(smem_u32(&tempty_bar[1]), 0);
    for (uint32_t t = 0; t < run_tiles; ++t) {
      const uint32_t b = t & 1, ub = t >> 1;
      bool ok = !abort_flag && mbar_wait_cluster(smem_u32(&tfull_bar[b]), ub & 1, timeout_ns);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) {
        if (lane == 0) atomicOr(err, kQerErrEpilogue);
        abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint32_t taddr = tmem + b * acc_cols + ((quarter * 32u) << 16);
      const float best = tmem_row_max(taddr, n_pad, n_text);
      const uint32_t j = (pair + t * n_pairs) * kQerTile + rank * kQerM + quarter * 32 + lane;
      if (j < n_visual) colmax[j] = fold ? fmaxf(colmax[j], best) : best;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(b ? tempty1 : tempty0);
    }
  }
  __syncwarp();
  // TMEM is freed only after every MMA of the pair has completed, and only
  // once both CTAs are past every remote arrive and multicast commit
  if (warp == 0) {
    const bool ok = mbar_wait_cluster(smem_u32(&done_bar), 0, timeout_ns);
    if (!ok && lane == 0) atomicOr(err, kQerErrDrain);
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_total) : "memory");
  }
}

// Eq. 7: w_f = mean over the frame's tokens of their max over text, times the
// 1/(H sqrt(d)) of Eq. 6. One warp per frame; a programmatic dependent of the
// scoring kernel, whose maxima it waits for.
__global__ void __launch_bounds__(256) qer_mean(const float* __restrict__ colmax, uint32_t n_frames, uint32_t tpf,
                                                float scale, float* __restrict__ w) {
  grid_dependency_wait();
  const uint32_t f = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (f >= n_frames) return;
  float s = 0.f;
  for (uint32_t t = lane; t < tpf; t += 32) s += colmax[static_cast<uint64_t>(f) * tpf + t];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) w[f] = s / static_cast<float>(tpf) * scale;
}

// Eq. 8: flag[f] = 1 when fewer than k frames rank above frame f (higher w,
// or equal w and lower index). A warp per frame: the CTA stages the m scores
// in shared memory, kRankTile at a time (one coalesced pass over the
// L2-resident w instead of a chain of dependent loads per lane), its lanes
// split each tile and one warp reduction counts them.
// The last CTA to finish (a ticket taken after a fence) then writes the flagged frames
// in time order (ballot, popcount and a scan of the warp totals per pass of
// kRankThreads frames), the count to k_out, and returns the ticket counter
// to zero. Launched as a programmatic dependent of the mean kernel, so every
// thread first waits for that grid's completion and memory.
__global__ void __launch_bounds__(kRankThreads) qer_rank(const float* __restrict__ w, uint32_t n_frames, uint32_t k,
                                                uint8_t* __restrict__ flag, uint32_t* __restrict__ done,
                                                uint32_t* __restrict__ sel,
                                                uint32_t* __restrict__ k_out) {
  constexpr uint32_t kWarps = kRankThreads / 32;
  __shared__ uint32_t wsum[kWarps];
  __shared__ uint32_t s_total, s_last;
  __shared__ float sw[kRankTile];
  grid_dependency_wait();
  const uint32_t tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t f = blockIdx.x * kWarps + warp;
  const bool mine = f < n_frames;  // uniform across the warp
  const float wf = mine ? w[f] : 0.f;
  uint32_t above = 0;
  for (uint32_t c0 = 0; c0 < n_frames; c0 += kRankTile) {
    const uint32_t cn = min(kRankTile, n_frames - c0);
    for (uint32_t i = tid; i < cn; i += kRankThreads) sw[i] = w[c0 + i];
    __syncthreads();
    if (mine)
      for (uint32_t j = lane; j < cn; j += 32) {
        const float wg = sw[j];
        above += (wg > wf) | ((wg == wf) & (c0 + j < f));
      }
    __syncthreads();  // the tile is read before the next one overwrites it
  }
  if (mine) {
    above = __reduce_add_sync(0xffffffffu, above);
    if (lane == 0) flag[f] = above < k;
  }
  __syncthreads();
  if (tid == 0) {
    __threadfence();  // this CTA's flags are visible before its ticket
    s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();  // every CTA's flags are visible to the last one
  uint32_t base = 0;
  for (uint32_t f0 = 0; f0 < n_frames; f0 += kRankThreads) {
    const uint32_t g = f0 + tid;
    const bool in = g < n_frames && __ldcg(flag + g) != 0;
    const uint32_t bal = __ballot_sync(0xffffffffu, in);
    const uint32_t before = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) wsum[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
      const uint32_t v = lane < kWarps ? wsum[lane] : 0u;
      uint32_t x = v;
#pragma unroll
      for (int dd = 1; dd < 32; dd <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, dd);
        if (lane >= static_cast<uint32_t>(dd)) x += y;
      }
      if (lane < kWarps) wsum[lane] = x - v;
      if (lane == 31) s_total = x;
    }
    __syncthreads();
    if (in) sel[base + wsum[warp] + before] = g;
    base += s_total;
    __syncthreads();
  }
  if (tid == 0) {
    *k_out = base;
    *done = 0;
  }
}

uint32_t qer_stage_bytes(uint32_t n_pad) { return 2 * kQerM * 128 + ((n_pad * 128 + 1023) & ~1023u); }

uint32_t qer_stages(uint32_t n_pad) {
  const size_t n = kQerStageBudget / qer_stage_bytes(n_pad);
  return static_cast<uint32_t>(n < kQerMaxStages ? n : kQerMaxStages);
}

// Key slots of the paired kernel: as many n_sub-chunk slots of 128 key rows
// as fit the ring budget beside kQerPairQSlots q~ slots (n_sub chunks of
// n_pad / 2 rows), at most kQerMaxStages.
uint32_t qer_pair_key_slots(uint32_t n_pad, uint32_t n_sub) {
  const size_t kslot = static_cast<size_t>(n_sub) * kQerM * 128, qslot = static_cast<size_t>(n_sub) * (n_pad / 2) * 128;
  const size_t n = (kQerPairRingBudget - kQerPairQSlots * qslot) / kslot;
  return static_cast<uint32_t>(n < kQerMaxStages ? n : kQerMaxStages);
}

size_t qer_pair_smem_bytes(uint32_t n_pad, uint32_t n_sub, uint32_t key_slots) {
  return static_cast<size_t>(n_sub) * (key_slots * kQerM * 128 + kQerPairQSlots * (n_pad / 2) * 128) + 1024;
}

size_t qer_smem_bytes(uint32_t n_pad) {
  return static_cast<size_t>(qer_stages(n_pad)) * qer_stage_bytes(n_pad) + 1024;  // + slack for 1024-B alignment
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor [rows][cols] (cols contiguous), boxes of 64 columns x box_rows.
bool make_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kQerKChunk), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace
}  // namespace cofie

using namespace cofie;

struct cofie_qer {
  cofie_qer_params p{};
  int device = 0;
  // the text is scored in n_blk passes of per_blk tokens (the last may have
  // fewer), each padded to n_pad q~ rows; q~ holds n_blk * n_pad rows
  uint32_t n_blk = 1, per_blk = 0;
  uint32_t n_pad = 0, D = 0, acc_cols = 0, n_buf = 1, n_stages = 0;
  int grid = 0;          // persistent CTAs
  size_t smem = 0;       // dynamic shared memory per CTA
  bool pair = false;     // the paired-SM kernel (clusters of two CTAs)
  uint32_t pair_key_slots = 0, pair_sub = 1;
  int pair_clusters = 0;  // co-resident clusters
  size_t pair_smem = 0;
  __nv_bfloat16_raw* d_qg = nullptr;
  float* d_colmax = nullptr;
  float* d_w = nullptr;
  uint8_t* d_flag = nullptr;
  uint32_t* d_k = nullptr;
  uint32_t* d_done = nullptr;  // CTAs of the ranking kernel that have finished
  uint32_t* d_err = nullptr;
  std::string err;
  // launch counter and optional event timing of the scoring kernel
  bool time_on = false;
  uint64_t launches = 0;
  double flops = 0.0, key_bytes = 0.0;
  std::vector<cudaEvent_t> ev;
  size_t ev_used = 0;
  int fail(int code, const std::string& m) {
    err = m;
    return code;
  }
};

namespace {

bool is_device(const void* p, int dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) && a.device == dev;
}

void qer_free(cofie_qer* h) {
  if (!h) return;
  int prev = -1;
  cudaGetDevice(&prev);
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  void* bufs[] = {h->d_qg, h->d_colmax, h->d_w, h->d_k, h->d_err, h->d_flag, h->d_done};
  for (void* b : bufs)
    if (b) cudaFree(b);
  for (cudaEvent_t e : h->ev) cudaEventDestroy(e);
  if (prev >= 0) cudaSetDevice(prev);
  delete h;
}

thread_local std::string g_qer_error;

}  // namespace

extern "C" {

int cofie_qer_create(const cofie_qer_params* p, cofie_qer_t** out) {
  if (!p || !out) return g_qer_error = "params or out is NULL", COFIE_EINVAL;
  if (p->n_text < 1 || p->n_text > kQerMaxText) return g_qer_error = "n_text must be in [1, 4096]", COFIE_EINVAL;
  if (p->n_heads < 1 || p->n_kv_heads < 1 || p->n_heads % p->n_kv_heads != 0)
    return g_qer_error = "n_kv_heads must divide n_heads", COFIE_EINVAL;
  const uint64_t D = static_cast<uint64_t>(p->n_kv_heads) * p->head_dim;
  if (p->head_dim < 1 || D % kQerKChunk != 0 || D > 16384)
    return g_qer_error = "n_kv_heads * head_dim must be a multiple of 64, at most 16384", COFIE_EINVAL;
  if (p->max_frames < 1 || p->tokens_per_frame < 1 ||
      static_cast<uint64_t>(p->max_frames) * p->tokens_per_frame > 0x7fffffffull)
    return g_qer_error = "max_frames and tokens_per_frame must be >= 1 (product < 2^31)", COFIE_EINVAL;
  if (!(p->rho >= 0.f && p->rho <= 1.f)) return g_qer_error = "rho must be in [0, 1]", COFIE_EINVAL;
  if (p->kernel > COFIE_QER_KERNEL_PAIR) return g_qer_error = "kernel must be one of COFIE_QER_KERNEL_*", COFIE_EINVAL;
  int dev = p->device;
  if (dev < 0 && cudaGetDevice(&dev) != cudaSuccess) return g_qer_error = "no CUDA device", COFIE_ECUDA;
  int prev = -1;
  cudaGetDevice(&prev);
  if (cudaSetDevice(dev) != cudaSuccess) return g_qer_error = "cannot select the device", COFIE_ECUDA;
  if (!tensor_map_encoder()) {
    if (prev >= 0) cudaSetDevice(prev);
    return g_qer_error = "cuTensorMapEncodeTiled is not available", COFIE_ECUDA;
  }
  cofie_qer* h = new (std::nothrow) cofie_qer();
  if (!h) return g_qer_error = "host allocation failed", COFIE_ENOMEM;
  h->p = *p;
  h->device = dev;
  h->D = static_cast<uint32_t>(D);
  h->n_blk = (p->n_text + kQerMaxN - 1) / kQerMaxN;  // balanced blocks of at most 256 tokens
  h->per_blk = (p->n_text + h->n_blk - 1) / h->n_blk;
  // rows of a block: a multiple of 16 (the MMA's N step), of 32 when there are
  // several blocks so that the paired kernel (half of q~ per CTA) stays open
  const uint32_t row_step = h->n_blk > 1 ? 32u : 16u;
  h->n_pad = (h->per_blk + row_step - 1) / row_step * row_step;
  h->acc_cols = 32;
  while (h->acc_cols < h->n_pad) h->acc_cols <<= 1;
  // Each tile needs two accumulators of acc_cols TMEM columns; double
  // buffering (overlapping a tile's epilogue with the next tile's MMAs)
  // doubles that when it still fits the SM's 512 columns.
  h->n_buf = (4 * h->acc_cols <= 512) ? 2 : 1;
  h->n_stages = qer_stages(h->n_pad);
  // The CTAs resident on one SM must never ask for more than its 512 TMEM
  // columns, or an allocation would wait for a CTA that only frees its
  // columns at exit; shared memory is requested large enough to keep the
  // residency within that limit.
  const int max_ctas_by_tmem = static_cast<int>(512 / (2 * h->acc_cols * h->n_buf));
  h->smem = qer_smem_bytes(h->n_pad);
  const size_t per_sm = 228 * 1024;
  while (max_ctas_by_tmem >= 1 && per_sm / (h->smem + 1024) > static_cast<size_t>(max_ctas_by_tmem))
    h->smem += 1024;
  const uint64_t nv = static_cast<uint64_t>(p->max_frames) * p->tokens_per_frame;
  cudaError_t e = cudaMalloc(&h->d_qg, static_cast<size_t>(h->n_blk) * h->n_pad * D * 2);
  if (e == cudaSuccess) e = cudaMalloc(&h->d_colmax, nv * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&h->d_w, static_cast<size_t>(p->max_frames) * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&h->d_k, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMalloc(&h->d_flag, p->max_frames);
  if (e == cudaSuccess) e = cudaMalloc(&h->d_done, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(h->d_done, 0, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMalloc(&h->d_err, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(h->d_err, 0, sizeof(uint32_t));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(qer_score, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(h->smem));
  int per_sm_ctas = 0, n_sms = 0;
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_ctas, qer_score, kQerThreads, h->smem);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess && (per_sm_ctas < 1 || per_sm_ctas > max_ctas_by_tmem)) e = cudaErrorInvalidConfiguration;
  h->grid = n_sms * (per_sm_ctas > 0 ? per_sm_ctas : 1);
  if (e == cudaSuccess && p->kernel != COFIE_QER_KERNEL_ONE_SM && h->n_pad % 32 == 0) {
    // the paired-SM kernel: one accumulator of acc_cols columns per buffer,
    // two buffers; the same TMEM residency rule through shared memory
    // two 64-wide K chunks per ring stage when D allows: every stage costs a
    // fixed synchronisation overhead, which more MMAs per stage amortise
    h->pair_sub = (h->D / kQerKChunk) % 2 == 0 ? 2 : 1;
    h->pair_key_slots = qer_pair_key_slots(h->n_pad, h->pair_sub);
    h->pair_smem = qer_pair_smem_bytes(h->n_pad, h->pair_sub, h->pair_key_slots);
    const int pair_ctas_by_tmem = static_cast<int>(512 / (2 * h->acc_cols));
    while (per_sm / (h->pair_smem + 1024) > static_cast<size_t>(pair_ctas_by_tmem)) h->pair_smem += 1024;
    const auto pair_fn = h->pair_sub == 2 ? qer_score_pair<2> : qer_score_pair<1>;  // the one launched
    cudaError_t pe = cudaFuncSetAttribute(pair_fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          static_cast<int>(h->pair_smem));
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * n_sms, 1, 1);
    cfg.blockDim = dim3(kQerPairThreads, 1, 1);
    cfg.dynamicSmemBytes = h->pair_smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (pe == cudaSuccess) pe = cudaOccupancyMaxActiveClusters(&clusters, pair_fn, &cfg);
    if (pe == cudaSuccess && clusters >= 1) {
      h->pair = true;
      h->pair_clusters = clusters;
    } else {
      cudaGetLastError();
      if (p->kernel == COFIE_QER_KERNEL_PAIR) e = pe != cudaSuccess ? pe : cudaErrorInvalidConfiguration;
    }
  } else if (e == cudaSuccess && p->kernel == COFIE_QER_KERNEL_PAIR) {
    if (prev >= 0) cudaSetDevice(prev);
    qer_free(h);
    return g_qer_error = "the paired-SM kernel needs the text block (n_text, or its blocks of at most 256) rounded up "
                         "to 16 to be a multiple of 32",
           COFIE_EINVAL;
  }
  if (prev >= 0) cudaSetDevice(prev);
  if (e != cudaSuccess) {
    g_qer_error = std::string("QER set-up failed: ") + cudaGetErrorString(e);
    cudaGetLastError();
    qer_free(h);
    return e == cudaErrorMemoryAllocation ? COFIE_ENOMEM : COFIE_ECUDA;
  }
  *out = h;
  return COFIE_OK;
}

void cofie_qer_destroy(cofie_qer_t* h) { qer_free(h); }

uint32_t cofie_qer_kernel_in_use(const cofie_qer_t* h) {
  return h ? (h->pair ? COFIE_QER_KERNEL_PAIR : COFIE_QER_KERNEL_ONE_SM) : 0u;
}

int cofie_qer_run(cofie_qer_t* h, const uint16_t* q, const uint16_t* k, uint32_t n_frames, float* w_out,
                  uint32_t* sel_out, uint32_t* k_out, void* cuda_stream) {
  if (!h) return COFIE_EINVAL;
  if (n_frames < 1 || n_frames > h->p.max_frames) return h->fail(COFIE_EINVAL, "n_frames must be in [1, max_frames]");
  if (!q || !k || !sel_out || !k_out) return h->fail(COFIE_EINVAL, "q, k, sel_out and k_out are required");
  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != h->device) cudaSetDevice(h->device);
  struct Restore {
    int prev, dev;
    ~Restore() {
      if (prev >= 0 && prev != dev) cudaSetDevice(prev);
    }
  } restore{prev, h->device};
  if (!is_device(q, h->device) || !is_device(k, h->device) || !is_device(sel_out, h->device) ||
      (w_out && !is_device(w_out, h->device)))
    return h->fail(COFIE_EINVAL, "q, k, w_out and sel_out must be device memory on the handle's device");
  if (reinterpret_cast<uintptr_t>(k) % 16 != 0) return h->fail(COFIE_EINVAL, "k must be 16-byte aligned");
  const cofie_qer_params& p = h->p;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  // Captured into a CUDA graph, the call's work is recorded, not run: every
  // buffer it writes is rewritten by each launch (the ranking kernel returns
  // its ticket to zero), so the graph can be launched again and again; a host
  // k_out would need a synchronisation and is refused, and timing is skipped.
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
    cudaGetLastError();
    return h->fail(COFIE_ECUDA, "cannot read the CUDA stream's capture state");
  }
  if (cs == cudaStreamCaptureStatusInvalidated) return h->fail(COFIE_ECUDA, "the stream's capture was invalidated");
  const bool capturing = cs == cudaStreamCaptureStatusActive;
  if (capturing && !is_device(k_out, h->device))
    return h->fail(COFIE_EINVAL, "k_out must be device memory while the stream captures a CUDA graph");
  const uint64_t nv = static_cast<uint64_t>(n_frames) * p.tokens_per_frame;
  CUtensorMap map_k, map_q;
  const uint32_t tiles = static_cast<uint32_t>((nv + kQerTile - 1) / kQerTile);
  // the paired kernel when asked for, or (automatic) when every tile gets a
  // pair of its own (each tile's MMAs split over two SMs: 14 us against 18 us
  // for up to 76 tiles) or the tiles exceed one wave of the one-SM kernel; in
  // between (one wave of that kernel, two of the pairs) the two run alike
  const bool pair_run = h->pair && (p.kernel == COFIE_QER_KERNEL_PAIR || tiles > static_cast<uint32_t>(h->grid) ||
                                    tiles <= static_cast<uint32_t>(h->pair_clusters));
  const uint32_t q_box = pair_run ? h->n_pad / 2 : h->n_pad;  // the pair's CTAs each stage half of q~
  if (!make_map(&map_k, k, nv, h->D, kQerM)) return h->fail(COFIE_ECUDA, "tensor map encoding failed");
  const uint32_t n_rows = h->n_blk * h->n_pad;
  if (p.head_dim % 8 == 0 && reinterpret_cast<uintptr_t>(q) % 16 == 0) {
    const uint64_t n8 = static_cast<uint64_t>(n_rows) * h->D / 8;
    const uint32_t blocks = static_cast<uint32_t>(std::min<uint64_t>((n8 + 255) / 256, 1024));
    qer_prepare_q8<<<blocks, 256, 0, st>>>(reinterpret_cast<const uint4*>(q), p.n_text, n_rows, h->n_pad, h->per_blk,
                                           p.n_heads, p.n_kv_heads, p.head_dim, reinterpret_cast<uint4*>(h->d_qg));
  } else {
    qer_prepare_q<<<256, 256, 0, st>>>(q, p.n_text, n_rows, h->n_pad, h->per_blk, p.n_heads, p.n_kv_heads,
                                       p.head_dim, h->d_qg);
  }
  const uint32_t grid = tiles < static_cast<uint32_t>(h->grid) ? tiles : static_cast<uint32_t>(h->grid);
  const uint32_t kk = static_cast<uint32_t>(std::max(1.0, std::nearbyint(static_cast<double>(p.rho) * n_frames)));
  const float scale = static_cast<float>(1.0 / (static_cast<double>(p.n_heads) * std::sqrt(static_cast<double>(p.head_dim))));
  float* w = w_out ? w_out : h->d_w;
  uint32_t* kdev = is_device(k_out, h->device) ? k_out : h->d_k;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (h->time_on && !capturing && h->ev_used + 2 <= (1u << 16)) {
    while (h->ev.size() < h->ev_used + 2) {
      cudaEvent_t x;
      if (cudaEventCreate(&x) != cudaSuccess) break;
      h->ev.push_back(x);
    }
    if (h->ev.size() >= h->ev_used + 2) {
      e0 = h->ev[h->ev_used];
      e1 = h->ev[h->ev_used + 1];
      h->ev_used += 2;
      cudaEventRecord(e0, st);
    }
  }
  // The scoring, mean and ranking kernels are programmatic dependents of the
  // kernel before them: each may be scheduled while its predecessor still
  // runs, and waits for it (griddepcontrol.wait) only where it reads that
  // kernel's output (the scoring kernel's q~ producer; every thread of the
  // mean and ranking kernels). With the timing events in between, the
  // scoring kernel's launch serialises as usual.
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = st;
  // One scoring pass per text block; passes after the first fold their
  // maxima into colmax (Eq. 7's max over all text tokens) and are ordered
  // after the pass before them as usual (no programmatic launch), so each
  // reads that pass's maxima complete.
  for (uint32_t blk = 0; blk < h->n_blk; ++blk) {
    if (!make_map(&map_q, h->d_qg + static_cast<size_t>(blk) * h->n_pad * h->D, h->n_pad, h->D, q_box))
      return h->fail(COFIE_ECUDA, "tensor map encoding failed");
    const uint32_t text_b = std::min(h->per_blk, p.n_text - blk * h->per_blk);  // real columns of this pass
    const uint32_t fold = blk > 0;
    if (pair_run) {
      const uint32_t clusters = std::min<uint32_t>(tiles, static_cast<uint32_t>(h->pair_clusters));
      cfg.gridDim = dim3(2 * clusters, 1, 1);
      cfg.blockDim = dim3(kQerPairThreads, 1, 1);
      cfg.dynamicSmemBytes = h->pair_smem;
      cfg.attrs = fold ? &attr[1] : attr;
      cfg.numAttrs = fold ? 1 : 2;
      const uint32_t n_chunks = h->D / kQerKChunk / h->pair_sub;
      cudaLaunchKernelEx(&cfg, h->pair_sub == 2 ? qer_score_pair<2> : qer_score_pair<1>, map_k, map_q,
                         static_cast<uint32_t>(nv), text_b, h->n_pad, fold, h->acc_cols, h->pair_key_slots,
                         kQerPairQSlots, n_chunks, tiles, h->d_colmax, h->d_err, 2000000000ull);
    } else {
      cfg.gridDim = dim3(grid, 1, 1);
      cfg.blockDim = dim3(kQerThreads, 1, 1);
      cfg.dynamicSmemBytes = h->smem;
      cfg.attrs = attr;
      cfg.numAttrs = fold ? 0 : 1;
      cudaLaunchKernelEx(&cfg, qer_score, map_k, map_q, static_cast<uint32_t>(nv), text_b, h->n_pad, fold,
                         h->acc_cols, h->n_buf, h->n_stages, h->D / kQerKChunk, tiles, h->d_colmax, h->d_err,
                         2000000000ull);
    }
  }
  if (e1) cudaEventRecord(e1, st);
  if (!capturing) {
    h->launches += 1;
    h->flops += 2.0 * n_rows * static_cast<double>(nv) * h->D;
    h->key_bytes += 2.0 * static_cast<double>(nv) * h->D * h->n_blk;  // each pass reads the keys
  }
  cfg.gridDim = dim3((n_frames + 7) / 8, 1, 1);
  cfg.blockDim = dim3(256, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, qer_mean, static_cast<const float*>(h->d_colmax), n_frames, p.tokens_per_frame, scale, w);
  cfg.gridDim = dim3((n_frames + kRankThreads / 32 - 1) / (kRankThreads / 32), 1, 1);
  cfg.blockDim = dim3(kRankThreads, 1, 1);
  cudaLaunchKernelEx(&cfg, qer_rank, static_cast<const float*>(w), n_frames, kk, h->d_flag, h->d_done, sel_out, kdev);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess && kdev != k_out) {
    e = cudaMemcpyAsync(k_out, kdev, sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  }
  if (e != cudaSuccess) return h->fail(COFIE_ECUDA, std::string("QER launch: ") + cudaGetErrorString(e));
  return COFIE_OK;
}

int cofie_qer_status(cofie_qer_t* h, void* cuda_stream) {
  if (!h) return COFIE_EINVAL;
  int prev = -1;
  cudaGetDevice(&prev);
  cudaSetDevice(h->device);
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(cuda_stream));
  uint32_t word = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&word, h->d_err, sizeof word, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && word) cudaMemset(h->d_err, 0, sizeof word);
  if (prev >= 0) cudaSetDevice(prev);
  const uint32_t bounds = take_local_bounds_errors();  // checked build only; 0 otherwise
  if (e != cudaSuccess) return h->fail(COFIE_ECUDA, cudaGetErrorString(e));
  if (bounds) return h->fail(COFIE_EDEVICE, "a layout check of the QER kernels failed (checked build)");
  if (word) return h->fail(COFIE_ETIMEOUT, "a device-side wait of the QER kernels ran out");
  return COFIE_OK;
}

int cofie_qer_profile_reset(cofie_qer_t* h, int time_kernels) {
  if (!h) return COFIE_EINVAL;
  h->time_on = time_kernels != 0;
  h->launches = 0;
  h->flops = h->key_bytes = 0.0;
  h->ev_used = 0;
  return COFIE_OK;
}

int cofie_qer_profile_read(cofie_qer_t* h, uint64_t* launches, uint64_t* timed, double* score_ms, double* flops,
                           double* key_bytes) {
  if (!h || !launches || !timed || !score_ms || !flops || !key_bytes) return COFIE_EINVAL;
  double ms = 0.0;
  for (size_t i = 0; i + 1 < h->ev_used; i += 2) {
    float t = 0.f;
    cudaError_t e = cudaEventSynchronize(h->ev[i + 1]);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t, h->ev[i], h->ev[i + 1]);
    if (e != cudaSuccess) return h->fail(COFIE_ECUDA, cudaGetErrorString(e));
    ms += t;
  }
  *launches = h->launches;
  *timed = h->ev_used / 2;
  *score_ms = ms;
  *flops = h->flops;
  *key_bytes = h->key_bytes;
  return COFIE_OK;
}

const char* cofie_qer_last_error(const cofie_qer_t* h) { return h ? h->err.c_str() : g_qer_error.c_str(); }

}  // extern "C"
