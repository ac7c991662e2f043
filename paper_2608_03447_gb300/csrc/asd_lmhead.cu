// libasd: fused LM-head + verify for GB300 (sm_103a).
//
// z = h W^T (h: [T, H] bf16 hidden states of the T = B(K+1) target rows,
// W: [V, H] bf16 LM-head weight) is computed on the 5th-generation tensor cores
// with fp32 accumulation in tensor memory, and reduced in the epilogue to what
// the verifier needs (Sec. 3.3: the top token, the top logit and the draft
// token's logit, with no [T, V] logit buffer); the selection of Alg. 1 then
// runs as in asd_verify. The logits never reach global memory.
//
// Tiling: two CTAs on a pair of SMs (a cluster of 2) share 2-SM MMAs
// (tcgen05 cta_group::2). An MMA's M is 256 vocabulary rows (128 per SM: the
// TMEM lanes), its N is 192 token rows (the TMEM columns), and the 576 rows of
// a B = 64, K = 8 step are exactly three token tiles (no padded rows). A pair
// works in units of two vocabulary tiles (512 rows) against one token tile:
// per 64-deep K step each SM loads 256 rows of W and half (96) of the token
// rows, 44 KB, and issues two MMAs over the same token slab, so the token rows
// cross from L2 once per two vocabulary tiles. A pair owns one token tile and
// walks the units with a stride; the pairs of the three token tiles that share
// a unit run at the same time, so each W tile comes from HBM once and from L2
// for the other two. Per CTA: warp 0 issues TMA loads (128B-swizzled 64-wide K
// slabs) into a kStages-deep ring, whose completion is counted on the first
// CTA's barrier; warp 1 allocates tensor memory, and in the first CTA one of
// its threads issues the MMAs; warps 2-9 read the two accumulators (192 of the
// 512 TMEM columns each) with tcgen05.ld, one warp per lane quarter and tile.
// The epilogue turns each 32 x 32 block (vocabulary rows x token columns) of a
// warp around through shared memory, so that a lane holds one token column and
// reduces it with plain register arithmetic, and keeps a running (value, index)
// key per token. The MMAs of the next unit wait for the epilogue: two
// accumulators fill the tensor memory, and this costs less than the extra L2
// traffic of one vocabulary tile per unit with double-buffered accumulators.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "asd.h"
#include "asd_device.cuh"

namespace {

using namespace asd_detail;

constexpr int kPairM = 256;               // vocabulary rows per CTA pair in one MMA (MMA M)
constexpr int kHalfM = 128;               // vocabulary rows per CTA in one MMA (TMEM lanes)
constexpr int kTN = 192;                  // token rows per tile (MMA N)
constexpr int kHalfN = kTN / 2;           // token rows each CTA of the pair loads
constexpr int kBK = 64;                   // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int kUmmaK = 16;                // K per tcgen05.mma (kind::f16)
constexpr int kW = 2;                     // vocabulary tiles per unit (MMAs per token slab)
constexpr int kUnitM = kW * kPairM;       // vocabulary rows per pair per unit
constexpr int kStages = 4;
constexpr int kStageB = kHalfN * kBK * 2;  // 12 KB of token rows
constexpr int kSlabA = kHalfM * kBK * 2;   // 16 KB of vocabulary rows per tile
constexpr int kStageA = kW * kSlabA;
constexpr uint32_t kStageTx = 2u * (kStageA + kStageB);  // both CTAs' bytes, counted on the first CTA
constexpr int kEpiWarps = 4 * kW;         // one per TMEM lane quarter and vocabulary tile
constexpr int kLmThreads = (2 + kEpiWarps) * 32;  // producer, MMA, epilogue warps
constexpr int kTmemCols = 512;            // accumulator j at column j * 256
constexpr int kAccStride = 256;
constexpr int kChunks = kTN / 32;         // 32-column TMEM loads per accumulator
constexpr int kPitch = 36;                // floats per row of an epilogue transpose block (conflict-free)
static_assert(kTN % 32 == 0 && kHalfN % 8 == 0, "token tile: whole 32-column loads, whole 8-row swizzle groups");
static_assert((kW - 1) * kAccStride + kTN <= kTmemCols, "accumulators fit in tensor memory");

struct LmShared {
  unsigned long long full[kStages];   // first CTA: both CTAs' loads of a stage have landed
  unsigned long long empty[kStages];  // each CTA: the MMAs have read its part of a stage
  unsigned long long acc_full;        // each CTA: the unit's accumulators are complete
  unsigned long long acc_empty;       // first CTA: both CTAs' epilogues have read them
  unsigned long long drain;
  uint32_t tmem_base;
  int abort;
  int draft[kTN];                     // x of the tile's token rows (-1: no draft / out of range)
  alignas(16) float xpose[kEpiWarps][32 * kPitch];  // per epilogue warp: a 32 x 32 block turned around
};
// dynamic shared memory: [1 KB alignment slack][stages x B][stages x A][LmShared]
constexpr size_t kLmSmemBytes = 1024 + static_cast<size_t>(kStages) * (kStageA + kStageB) + sizeof(LmShared);
static_assert(kLmSmemBytes <= 232448, "shared memory per CTA");

// ---------------------------------------------------------------- tcgen05 / TMA / cluster helpers

// Shared-memory matrix descriptor of a K-major operand tile written by TMA with
// 128-byte swizzling: rows of 128 bytes, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);          // start address
  d |= static_cast<uint64_t>(1u) << 16;                         // leading byte offset (unused when swizzled)
  d |= static_cast<uint64_t>((1024u >> 4) & 0x3FFFu) << 32;     // stride byte offset: 8 rows x 128 B
  d |= static_cast<uint64_t>(1u) << 46;                         // descriptor version
  d |= static_cast<uint64_t>(2u) << 61;                         // 128-byte swizzle
  return d;
}

// Instruction descriptor: kind::f16 with bf16 A and B, fp32 D, both K-major,
// M = kPairM (across the pair), N = kTN.
constexpr uint32_t kIdesc = (1u << 4)                               // D format: f32
                            | (1u << 7)                             // A format: bf16
                            | (1u << 10)                            // B format: bf16
                            | (static_cast<uint32_t>(kTN >> 3) << 17)     // N / 8
                            | (static_cast<uint32_t>(kPairM >> 4) << 24); // M / 16

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The shared::cluster address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_rank(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// One bounded wait on the phase with the given parity. The thread may sleep
// until the phase completes (at most kSuspendNs per call), so the warps that
// wait -- most of them, most of the time -- take no issue slots from the MMA
// and TMA threads (polling them cost this kernel about 7 %).
constexpr uint32_t kSuspendNs = 1000000;
__device__ __forceinline__ bool mbar_try_wait_cluster(unsigned long long* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity), "r"(kSuspendNs)
      : "memory");
  return done != 0;
}
// mbar_wait for barriers that the other CTA of the pair also signals; the
// abort flag and the clock are checked every 16 sleeps.
__device__ inline bool mbar_wait_cluster(unsigned long long* bar, uint32_t parity, volatile int* abort) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (unsigned it = 1;; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 15u) == 0) {
      if (*abort) return false;
      if (global_ns() - t0 > kWaitLimitNs) return false;
    }
  }
}

// TMA tile load into this CTA's shared memory whose completion is counted on
// an mbarrier of either CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar_cluster, int x,
                                                 int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%3, %4}], [%2];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void umma_pair_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

// The mbarrier at this offset in both CTAs of the pair arrives once every
// tcgen05 operation this thread issued so far has completed.
__device__ __forceinline__ void umma_commit_pair(unsigned long long* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
      ::"r"(smem_u32(bar)), "h"(static_cast<uint16_t>(0x3)) : "memory");
}
// Same, for this CTA's barrier only.
__device__ __forceinline__ void umma_commit_local(unsigned long long* bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];"
               ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// The sticky error word, when the call has a workspace (asd_lmhead_logits has none).
__device__ __forceinline__ void report_timeout(const VerifyParams& p) {
  if (p.error) atomicExch(p.error, static_cast<unsigned>(ASD_ERR_TIMEOUT));
}

// Sets the abort flag of both CTAs of the pair.
__device__ __forceinline__ void abort_pair(LmShared& sh, uint32_t peer) {
  sh.abort = 1;
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(map_rank(smem_u32(&sh.abort), peer)), "r"(1) : "memory");
}

// Order-preserving bits of a column maximum; NaN is mapped above +inf
// whatever its sign bit, so a NaN anywhere in a row reaches the row's key.
__device__ __forceinline__ uint32_t max_bits(float v) { return v != v ? 0xffc00000u : ordered_bits(v); }

struct LmParams {
  int T, H, V;
  int token_tiles;     // ceil(T / kTN)
  int pairs_per_tile;  // CTA pairs that share one token tile
  int vocab_units;     // ceil(V / kUnitM)
  int k_steps;         // ceil(H / kBK)
  float* logits_out;   // [T, V] when writing logits instead of verifying
};

// One CTA pair (cluster of 2): token tile m = pair % token_tiles, vocabulary
// units n = pair / token_tiles + i * pairs_per_tile (rows n * kUnitM on).
template <bool kStrict, bool kWriteLogits>
__global__ void __launch_bounds__(kLmThreads, 1)
    lmhead_verify_kernel(const __grid_constant__ CUtensorMap map_h, const __grid_constant__ CUtensorMap map_w,
                         const __grid_constant__ VerifyParams p, const LmParams q) {
  extern __shared__ __align__(1024) unsigned char lm_smem_raw[];
  const uint32_t raw = smem_u32(lm_smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // 1024-byte aligned for the 128-byte swizzle
  unsigned char* gbase = lm_smem_raw + (base - raw);
  const uint32_t sB = base;                                        // kStages x kStageB
  const uint32_t sA = base + kStages * kStageB;                    // kStages x kStageA
  LmShared& sh = *reinterpret_cast<LmShared*>(gbase + kStages * (kStageA + kStageB));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank() & 1u;
  const uint32_t peer = rank ^ 1u;
  const bool leader = rank == 0;
  const int pair = static_cast<int>(blockIdx.x >> 1);
  const int m = pair % q.token_tiles;
  const int n_first = pair / q.token_tiles;
  const int n_tiles =
      n_first < q.vocab_units ? (q.vocab_units - n_first + q.pairs_per_tile - 1) / q.pairs_per_tile : 0;
  const int K1 = p.K + 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], 1);
    }
    mbar_init(&sh.acc_full, 1);
    mbar_init(&sh.acc_empty, 2 * kEpiWarps);  // the epilogue warps of both CTAs
    mbar_init(&sh.drain, 1);
    sh.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (!kWriteLogits) {
    for (int c = threadIdx.x; c < kTN; c += kLmThreads) {
      const int tok = m * kTN + c;
      int x = -1;
      if (tok < q.T && (tok % K1) < p.K) {
        // the row of this CTA's weight that holds the draft token (a vocabulary
        // shard starts at global index v_offset), if any
        x = __ldg(p.draft + static_cast<long long>(tok / K1) * p.K + (tok % K1)) - p.v_offset;
        if (x < 0 || x >= p.V) x = -1;
      }
      sh.draft[c] = x;
    }
  }
  if (warp == 1) {  // tensor memory of both SMs, allocated together by one warp of each CTA
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&sh.tmem_base)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers exist before either signals the other's
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;

  int it_issued = 0;
  if (warp == 0) {
    // ---------------- TMA producer (both CTAs; completion counted on the first CTA's barrier)
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_h)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_w)) : "memory");
      const uint32_t full0 = map_rank(smem_u32(&sh.full[0]), 0);
      int it = 0;
      for (int t = 0; t < n_tiles && !sh.abort; ++t) {
        const int n = n_first + t * q.pairs_per_tile;
        for (int k = 0; k < q.k_steps; ++k, ++it) {
          const int s = it % kStages;
          if (!mbar_wait_cluster(&sh.empty[s], ((it / kStages) & 1) ^ 1, &sh.abort)) {
            abort_pair(sh, peer);
            report_timeout(p);
            break;
          }
          if (leader) mbar_expect_tx(&sh.full[s], kStageTx);
          const uint32_t bar = full0 + static_cast<uint32_t>(s * sizeof(unsigned long long));
          tma_load_2d_pair(sB + s * kStageB, &map_h, bar, k * kBK, m * kTN + static_cast<int>(rank) * kHalfN);
          // this CTA's 128 rows of both vocabulary tiles of the unit: rows n * 512 + rank * 256 on
          tma_load_2d_pair(sA + s * kStageA, &map_w, bar, k * kBK, n * kUnitM + static_cast<int>(rank) * kW * kHalfM);
          it_issued = it + 1;
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (one thread of the first CTA, for both SMs)
    if (leader && lane == 0) {
      int it = 0;
      for (int t = 0; t < n_tiles && !sh.abort; ++t) {
        // the epilogues of both CTAs have read the previous unit's accumulators
        if (!mbar_wait_cluster(&sh.acc_empty, (t & 1) ^ 1, &sh.abort)) {
          abort_pair(sh, peer);
          report_timeout(p);
          break;
        }
        tc_fence_after();
        bool ok = true;
        for (int k = 0; k < q.k_steps; ++k, ++it) {
          const int s = it % kStages;
          if (!mbar_wait_cluster(&sh.full[s], (it / kStages) & 1, &sh.abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t bd = smem_desc_sw128(sB + s * kStageB);
#pragma unroll
          for (int j = 0; j < kW; ++j) {  // both vocabulary tiles of the unit read the same token slab
            const uint32_t d = tmem + static_cast<uint32_t>(j * kAccStride);
            const uint64_t ad = smem_desc_sw128(sA + s * kStageA + j * kSlabA);
#pragma unroll
            for (int kk = 0; kk < kBK / kUmmaK; ++kk) {
              // advance 16 elements (32 bytes, encoded 2) along K inside the swizzle row
              umma_pair_bf16(d, ad + 2u * kk, bd + 2u * kk, (k > 0 || kk > 0) ? 1u : 0u);
            }
          }
          umma_commit_pair(&sh.empty[s]);  // frees the stage in both CTAs when these MMAs have read it
        }
        if (!ok) {
          abort_pair(sh, peer);
          report_timeout(p);
          break;
        }
        umma_commit_pair(&sh.acc_full);  // the accumulators are complete in both CTAs
      }
      umma_commit_local(&sh.drain);  // arrives once every MMA issued above has finished
      const unsigned long long t0 = global_ns();
      while (!mbar_try_wait(&sh.drain, 0) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ---------------- epilogue: warps 2 .. 1 + kEpiWarps, one vocabulary row (TMEM lane) per thread;
    // warps 2-5 read the first vocabulary tile of a unit, warps 6-9 the second
    const int quarter = warp & 3;                     // TMEM lanes this warp may read
    const int jt = (warp - 2) >> 2;                   // the unit's vocabulary tile this warp reduces
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t acc_empty0 = map_rank(smem_u32(&sh.acc_empty), 0);
    float* xpose = sh.xpose[warp - 2];
    int xs[kChunks];  // lane l: draft of token column c * 32 + l
#pragma unroll
    for (int c = 0; c < kChunks; ++c) xs[c] = kWriteLogits ? -1 : sh.draft[c * 32 + lane];
    unsigned long long best[kChunks];  // lane l: running key of token column c * 32 + l
#pragma unroll
    for (int c = 0; c < kChunks; ++c) best[c] = 0ull;
    for (int t = 0; t < n_tiles; ++t) {
      const bool ok = __all_sync(kFull, mbar_wait_cluster(&sh.acc_full, t & 1, &sh.abort));
      if (!ok) {
        if (lane == 0) {
          abort_pair(sh, peer);
          report_timeout(p);
        }
        break;
      }
      tc_fence_after();
      const int v_warp = (n_first + t * q.pairs_per_tile) * kUnitM + static_cast<int>(rank) * kW * kHalfM +
                         jt * kHalfM + quarter * 32;
      const int v = v_warp + lane;  // this thread's vocabulary row
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_base + static_cast<uint32_t>(jt * kAccStride + c * 32), r);
        tmem_ld_wait();
        if (kWriteLogits) {
          if (v < q.V) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int tok = m * kTN + c * 32 + i;
              if (tok < q.T) q.logits_out[static_cast<long long>(tok) * q.V + v] = __uint_as_float(r[i]);
            }
          }
        } else {
          // draft logits: the lane holding row x of column i keeps z_i(x) (rare: at most one row per column)
          unsigned hit = __ballot_sync(kFull, static_cast<unsigned>(xs[c] - v_warp) < 32u);
          while (hit) {
            const int i = __ffs(hit) - 1;
            hit &= hit - 1;
            const int owner = __shfl_sync(kFull, xs[c], i) - v_warp;
            if (lane == owner) {
              float z = 0.0f;
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (j == i) z = __uint_as_float(r[j]);
              p.draft_logit[m * kTN + c * 32 + i] = z;
            }
          }
          // argmax of each column over the warp's 32 rows: the block is turned
          // around through shared memory (lane l writes its row, then reads
          // column l), the lane takes the column's maximum, and where that
          // raises the column's running key, the lowest row holding it.
          if (v_warp >= q.V) continue;  // rows past the vocabulary: nothing to reduce
          if (v_warp + 31 >= q.V && v >= q.V) {  // the last, partial tile: rows past V never win
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(-INFINITY);
          }
#pragma unroll
          for (int i = 0; i < 8; ++i)
            *reinterpret_cast<uint4*>(xpose + lane * kPitch + 4 * i) =
                make_uint4(r[4 * i], r[4 * i + 1], r[4 * i + 2], r[4 * i + 3]);
          __syncwarp();
          float col[32];  // column `lane` of the block: the logits of token c * 32 + lane in the warp's 32 rows
#pragma unroll
          for (int i = 0; i < 32; ++i) col[i] = xpose[i * kPitch + lane];
          __syncwarp();  // the block is read before the next chunk overwrites it
          float zmax = col[0];
#pragma unroll
          for (int i = 1; i < 32; ++i) zmax = fmax_nan(zmax, col[i]);
          const uint32_t hi = max_bits(zmax);
          if (hi > static_cast<uint32_t>(best[c] >> 32)) {
            int w = 0;  // NaN: no row compares equal; the key still says NaN
#pragma unroll
            for (int i = 31; i >= 0; --i)
              if (col[i] == zmax) w = i;
            best[c] = (static_cast<unsigned long long>(hi) << 32) | (0xffffffffu - static_cast<uint32_t>(v_warp + w));
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(acc_empty0);
    }
    if (!kWriteLogits && !sh.abort) {
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        const int tok = m * kTN + c * 32 + lane;
        const unsigned long long key = best[c];
        if (tok < q.T && key) {
          atomicMax(&p.row_key[tok], key);
          if ((key >> 32) == 0xffc00000ull) atomicOr(&p.flags[tok / K1], ASD_STATUS_NAN_LOGIT);
        }
      }
    }
    __threadfence();
  }

  tc_fence_before();
  __syncthreads();
  if (sh.abort && leader && warp == 0 && lane == 0) {
    // wait (bounded) for the loads still in flight before the pair exits
    for (int it = it_issued > kStages ? it_issued - kStages : 0; it < it_issued; ++it) {
      const int s = it % kStages;
      const unsigned long long t0 = global_ns();
      while (!mbar_try_wait_cluster(&sh.full[s], (it / kStages) & 1) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  }
  __syncthreads();
  cluster_sync_all();  // neither CTA frees tensor memory or exits while the other may still use the pair
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
  if (kWriteLogits || sh.abort) return;

  // Count this CTA's rows of each request of its token tile; the CTA that
  // completes a request (every CTA of the tile has counted) runs its selection.
  const int t0 = m * kTN, t1 = (m + 1) * kTN < q.T ? (m + 1) * kTN : q.T;
  if (t0 < t1) {
    const int b_first = t0 / K1, b_last = (t1 - 1) / K1;
    const unsigned long long total = static_cast<unsigned long long>(K1) * 2ull * q.pairs_per_tile;
    for (int b = b_first + warp; b <= b_last; b += kLmThreads / 32) {
      const int r0 = b * K1 > t0 ? b * K1 : t0;
      const int r1 = (b + 1) * K1 < t1 ? (b + 1) * K1 : t1;
      finish_request<float, kStrict>(p, b, static_cast<unsigned long long>(r1 - r0), total, lane);
    }
  }
}

// ---------------------------------------------------------------- host side

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult res;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &res) ==
            cudaSuccess &&
        res == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 2-D bf16 row-major [rows, cols] tensor, boxes of box_rows x kBK columns,
// 128-byte swizzle; out-of-range rows and columns read as zero.
bool make_map(CUtensorMap* map, const void* ptr, int rows, int cols, int box_rows) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct LmDevice {
  int sms = 0;
  int major = 0, minor = 0;
  // CTA pairs resident at once, per kernel instance (0: not set up yet); the
  // set-up is idempotent, so two threads racing to do it store the same value
  std::atomic<int> pairs[4] = {};
};

int lm_device(LmDevice** out) {
  constexpr int kMaxDevices = 64;
  static LmDevice info[kMaxDevices];
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return ASD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return ASD_ERR_DEVICE;
  std::lock_guard<std::mutex> g(mu);
  if (info[dev].sms == 0) {
    if (cudaDeviceGetAttribute(&info[dev].sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&info[dev].major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&info[dev].minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return ASD_ERR_CUDA;
  }
  *out = &info[dev];
  return ASD_OK;
}

cudaLaunchConfig_t pair_config(unsigned grid, cudaStream_t stream, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kLmThreads, 1, 1);
  cfg.dynamicSmemBytes = kLmSmemBytes;
  cfg.stream = stream;
  attr->id = cudaLaunchAttributeClusterDimension;
  attr->val.clusterDim.x = 2;
  attr->val.clusterDim.y = 1;
  attr->val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

template <bool kStrict, bool kWriteLogits>
int launch_lmhead(const void* hidden, const void* weight, int H, int T, VerifyParams& p, float* logits_out,
                  cudaStream_t stream) {
  LmDevice* dev = nullptr;
  int rc = lm_device(&dev);
  if (rc != ASD_OK) return rc;
  if (dev->major != 10) return ASD_ERR_DEVICE;  // tcgen05 needs a Blackwell (sm_10x) device
  auto kernel = lmhead_verify_kernel<kStrict, kWriteLogits>;
  const int slot = (kStrict ? 1 : 0) + (kWriteLogits ? 2 : 0);
  cudaLaunchAttribute attr;
  int pairs = dev->pairs[slot].load(std::memory_order_acquire);
  if (pairs == 0) {
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kLmSmemBytes)) !=
        cudaSuccess)
      return ASD_ERR_CUDA;
    cudaLaunchConfig_t probe = pair_config(static_cast<unsigned>(dev->sms & ~1), stream, &attr);
    if (cudaOccupancyMaxActiveClusters(&pairs, kernel, &probe) != cudaSuccess || pairs < 1) return ASD_ERR_CUDA;
    dev->pairs[slot].store(pairs, std::memory_order_release);
  }
  CUtensorMap map_h, map_w;
  if (!make_map(&map_h, hidden, T, H, kHalfN) || !make_map(&map_w, weight, p.V, H, kW * kHalfM)) return ASD_ERR_CUDA;
  LmParams q;
  q.T = T;
  q.H = H;
  q.V = p.V;
  q.token_tiles = (T + kTN - 1) / kTN;
  q.pairs_per_tile = pairs / q.token_tiles > 0 ? pairs / q.token_tiles : 1;
  q.vocab_units = (p.V + kUnitM - 1) / kUnitM;
  if (q.pairs_per_tile > q.vocab_units) q.pairs_per_tile = q.vocab_units;
  q.k_steps = (H + kBK - 1) / kBK;
  q.logits_out = logits_out;
  const unsigned grid = 2u * static_cast<unsigned>(q.token_tiles * q.pairs_per_tile);
  cudaLaunchConfig_t cfg = pair_config(grid, stream, &attr);
  return cudaLaunchKernelEx(&cfg, kernel, map_h, map_w, p, q) == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

int check_lm_inputs(const void* hidden, const void* weight, int H) {
  if (!hidden || !weight) return ASD_ERR_NULL;
  if (H < 8 || H % 8 != 0) return ASD_ERR_SHAPE;  // TMA: row pitch a multiple of 16 bytes
  if (reinterpret_cast<uintptr_t>(hidden) % 16 != 0 || reinterpret_cast<uintptr_t>(weight) % 16 != 0)
    return ASD_ERR_ALIGN;
  return ASD_OK;
}

}  // namespace

extern "C" {

int asd_lmhead_workspace_size(int B, int K, int V, int H, size_t* bytes) {
  if (!bytes) return ASD_ERR_NULL;
  int rc = check_shape(B, K, V, ASD_BF16);
  if (rc != ASD_OK) return rc;
  if (H < 8 || H % 8 != 0) return ASD_ERR_SHAPE;
  *bytes = layout_for(B, K).total;
  return ASD_OK;
}

int asd_lmhead_verify(const void* hidden, const void* weight, int H, int B, int K, int V, const int32_t* draft,
                      asd_ledger* ledger, float gate, int cap, int32_t* accepted_len, int32_t* committed,
                      int32_t* recovery, int32_t* row_argmax, float* row_regret, float* row_top, int32_t* status,
                      void* workspace, size_t workspace_bytes, asd_stream_t stream) {
  int rc = check_shape(B, K, V, ASD_BF16);
  if (rc != ASD_OK) return rc;
  if (B == 0) return ASD_OK;
  rc = check_lm_inputs(hidden, weight, H);
  if (rc != ASD_OK) return rc;
  if (!accepted_len || !committed || !recovery || !workspace || !ledger) return ASD_ERR_NULL;
  if (K > 0 && !draft) return ASD_ERR_NULL;
  if (gate != gate || gate < 0.0f || cap < 0) return ASD_ERR_CONTROL;
  const WorkspaceLayout l = layout_for(B, K);
  if (workspace_bytes < l.total) return ASD_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0) return ASD_ERR_ALIGN;
  char* ws = static_cast<char*>(workspace);
  VerifyParams p = {};
  p.logits = nullptr;
  p.B = B;
  p.K = K;
  p.V = V;
  p.total = static_cast<long long>(B) * (K + 1);
  p.draft = draft;
  p.ledger = ledger;
  p.gate = gate;
  p.cap = cap;
  p.accepted_len = accepted_len;
  p.committed = committed;
  p.recovery = recovery;
  p.row_argmax = row_argmax;
  p.row_regret = row_regret;
  p.status = status;
  p.row_key = reinterpret_cast<unsigned long long*>(ws + l.row_key);
  p.draft_logit = reinterpret_cast<float*>(ws + l.draft_logit);
  p.done = reinterpret_cast<unsigned long long*>(ws + l.done);
  p.flags = reinterpret_cast<unsigned int*>(ws + l.flags);
  p.error = reinterpret_cast<unsigned int*>(ws + l.error);
  p.row_top = row_top;
  p.nblk = 1;
  return launch_lmhead<false, false>(hidden, weight, H, B * (K + 1), p, nullptr,
                                     reinterpret_cast<cudaStream_t>(stream));
}

int asd_lmhead_partials(const void* hidden, const void* weight, int H, int B, int K, int Vs, int v_offset,
                        int V, const int32_t* draft, asd_partial* partials, void* workspace,
                        size_t workspace_bytes, asd_stream_t stream) {
  int rc = check_shape(B, K, Vs, ASD_BF16);
  if (rc != ASD_OK) return rc;
  if (v_offset < 0 || V < 1 || static_cast<long long>(v_offset) + Vs > V) return ASD_ERR_SHAPE;
  if (B == 0) return ASD_OK;
  rc = check_lm_inputs(hidden, weight, H);
  if (rc != ASD_OK) return rc;
  if (!partials || !workspace) return ASD_ERR_NULL;
  if (K > 0 && !draft) return ASD_ERR_NULL;
  const WorkspaceLayout l = layout_for(B, K);
  if (workspace_bytes < l.total) return ASD_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0) return ASD_ERR_ALIGN;
  char* ws = static_cast<char*>(workspace);
  VerifyParams p = {};
  p.logits = nullptr;
  p.B = B;
  p.K = K;
  p.V = Vs;
  p.total = static_cast<long long>(B) * (K + 1);
  p.draft = draft;
  p.row_key = reinterpret_cast<unsigned long long*>(ws + l.row_key);
  p.draft_logit = reinterpret_cast<float*>(ws + l.draft_logit);
  p.done = reinterpret_cast<unsigned long long*>(ws + l.done);
  p.flags = reinterpret_cast<unsigned int*>(ws + l.flags);
  p.error = reinterpret_cast<unsigned int*>(ws + l.error);
  p.nblk = 1;
  p.v_offset = v_offset;
  p.v_total = V;
  p.partials = partials;
  return launch_lmhead<true, false>(hidden, weight, H, B * (K + 1), p, nullptr,
                                    reinterpret_cast<cudaStream_t>(stream));
}

int asd_lmhead_logits(const void* hidden, const void* weight, int H, int T, int V, float* logits,
                      asd_stream_t stream) {
  if (T < 0 || V < 1) return ASD_ERR_SHAPE;
  if (T == 0) return ASD_OK;
  int rc = check_lm_inputs(hidden, weight, H);
  if (rc != ASD_OK) return rc;
  if (!logits) return ASD_ERR_NULL;
  VerifyParams p = {};
  p.V = V;
  p.K = 0;
  p.nblk = 1;
  return launch_lmhead<false, true>(hidden, weight, H, T, p, logits, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
