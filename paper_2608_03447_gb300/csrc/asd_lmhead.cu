// libasd: fused LM-head + verify for GB300 (sm_103a).
//
// z = h W^T (h: [T, H] bf16 hidden states of the T = B(K+1) target rows,
// W: [V, H] bf16 LM-head weight) is computed on the 5th-generation tensor cores
// with fp32 accumulation in tensor memory, and reduced in the epilogue to what
// the verifier needs (Sec. 3.3: the top token, the top logit and the draft
// token's logit, with no [T, V] logit buffer); the selection of Alg. 1 then
// runs as in asd_verify. The logits never reach global memory.
//
// Tiling: a CTA owns one 128-token tile (the MMA's M, TMEM lanes = tokens)
// and loops over 256-wide vocabulary tiles (the MMA's N, TMEM columns), so each
// epilogue thread owns one token and reduces its logits in registers. The grid
// is (token tiles) x (CTAs per token tile); the CTAs that share a vocabulary
// tile run at the same time, so each W tile comes from HBM once and from L2
// for the other token tiles. Per CTA: warp 0 issues TMA loads (128B-swizzled
// 64-wide K slabs) into a 4-stage ring, warp 1 allocates tensor memory and
// issues tcgen05.mma from one thread, warps 2-5 read the accumulator with
// tcgen05.ld; the 512 TMEM columns hold two 256-column accumulators so the
// epilogue of one vocabulary tile overlaps the MMAs of the next.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cstdlib>
#include <mutex>

#include "asd.h"
#include "asd_device.cuh"

namespace {

using namespace asd_detail;

constexpr int kBM = 128;                  // tokens per tile (MMA M)
constexpr int kBN = 256;                  // vocabulary entries per tile (MMA N)
constexpr int kBK = 64;                   // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int kUmmaK = 16;                // K per tcgen05.mma (kind::f16)
constexpr int kStages = 4;
constexpr int kStageA = kBM * kBK * 2;    // 16 KB
constexpr int kStageB = kBN * kBK * 2;    // 32 KB
constexpr int kLmThreads = 6 * 32;        // producer, MMA, 4 epilogue warps
constexpr int kTmemCols = 2 * kBN;        // two accumulators

struct LmShared {
  unsigned long long full[kStages];
  unsigned long long empty[kStages];
  unsigned long long acc_full[2];
  unsigned long long acc_empty[2];
  unsigned long long drain;
  uint32_t tmem_base;
  int abort;
};
// dynamic shared memory: [1 KB alignment slack][stages x (A, B)][LmShared]
constexpr size_t kLmSmemBytes = 1024 + static_cast<size_t>(kStages) * (kStageA + kStageB) + sizeof(LmShared);

// ---------------------------------------------------------------- tcgen05 / TMA helpers

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
// M = kBM, N = kBN.
constexpr uint32_t kIdesc = (1u << 4)                              // D format: f32
                            | (1u << 7)                            // A format: bf16
                            | (1u << 10)                           // B format: bf16
                            | (static_cast<uint32_t>(kBN >> 3) << 17)  // N / 8
                            | (static_cast<uint32_t>(kBM >> 4) << 24); // M / 16

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

// The mbarrier arrives once every tcgen05 operation this thread issued so far has completed.
__device__ __forceinline__ void umma_commit(unsigned long long* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
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

struct LmParams {
  int T, H, V;
  int token_tiles;     // ceil(T / kBM)
  int ctas_per_tile;   // CTAs that share one token tile
  int vocab_tiles;     // ceil(V / kBN)
  int k_steps;         // ceil(H / kBK)
  float* logits_out;   // [T, V] when writing logits instead of verifying
};

// One CTA: token tile m = blockIdx.x % token_tiles, vocabulary tiles
// n = blockIdx.x / token_tiles + i * ctas_per_tile.
template <bool kStrict, bool kWriteLogits>
__global__ void __launch_bounds__(kLmThreads, 1)
    lmhead_verify_kernel(const __grid_constant__ CUtensorMap map_h, const __grid_constant__ CUtensorMap map_w,
                         const __grid_constant__ VerifyParams p, const LmParams q) {
  extern __shared__ __align__(1024) unsigned char lm_smem_raw[];
  const uint32_t raw = smem_u32(lm_smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // 1024-byte aligned for the 128-byte swizzle
  unsigned char* gbase = lm_smem_raw + (base - raw);
  const uint32_t sA = base;                                        // kStages x kStageA
  const uint32_t sB = base + kStages * kStageA;                    // kStages x kStageB
  LmShared& sh = *reinterpret_cast<LmShared*>(gbase + kStages * (kStageA + kStageB));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m = static_cast<int>(blockIdx.x) % q.token_tiles;
  const int n_first = static_cast<int>(blockIdx.x) / q.token_tiles;
  const int n_tiles = n_first < q.vocab_tiles ? (q.vocab_tiles - n_first + q.ctas_per_tile - 1) / q.ctas_per_tile : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sh.acc_full[a], 1);
      mbar_init(&sh.acc_empty[a], 4);
    }
    mbar_init(&sh.drain, 1);
    sh.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {  // tensor memory: 512 columns (this CTA is alone on its SM: see kLmSmemBytes)
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&sh.tmem_base)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;

  int it_issued = 0;
  if (warp == 0) {
    // ---------------- TMA producer
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_h)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_w)) : "memory");
      int it = 0;
      for (int t = 0; t < n_tiles && !sh.abort; ++t) {
        const int n = n_first + t * q.ctas_per_tile;
        for (int k = 0; k < q.k_steps; ++k, ++it) {
          const int s = it % kStages;
          if (!mbar_wait(&sh.empty[s], ((it / kStages) & 1) ^ 1, &sh.abort)) {
            sh.abort = 1;
            report_timeout(p);
            break;
          }
          mbar_expect_tx(&sh.full[s], kStageA + kStageB);
          tma_load_2d(sA + s * kStageA, &map_h, smem_u32(&sh.full[s]), k * kBK, m * kBM);
          tma_load_2d(sB + s * kStageB, &map_w, smem_u32(&sh.full[s]), k * kBK, n * kBN);
          it_issued = it + 1;
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (one thread)
    if (lane == 0) {
      int it = 0;
      for (int t = 0; t < n_tiles && !sh.abort; ++t) {
        const int a = t & 1;
        if (!mbar_wait(&sh.acc_empty[a], ((t >> 1) & 1) ^ 1, &sh.abort)) {
          sh.abort = 1;
          report_timeout(p);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(a * kBN);
        bool ok = true;
        for (int k = 0; k < q.k_steps; ++k, ++it) {
          const int s = it % kStages;
          if (!mbar_wait(&sh.full[s], (it / kStages) & 1, &sh.abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc_sw128(sA + s * kStageA);
          const uint64_t bd = smem_desc_sw128(sB + s * kStageB);
#pragma unroll
          for (int kk = 0; kk < kBK / kUmmaK; ++kk) {
            // advance 16 elements (32 bytes, encoded 2) along K inside the swizzle row
            umma_bf16(d, ad + 2u * kk, bd + 2u * kk, (k > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(&sh.empty[s]);  // frees the stage when these MMAs have read it
        }
        if (!ok) {
          sh.abort = 1;
          report_timeout(p);
          break;
        }
        umma_commit(&sh.acc_full[a]);  // the accumulator is complete
      }
      umma_commit(&sh.drain);  // arrives once every MMA issued above has finished
      const unsigned long long t0 = global_ns();
      while (!mbar_try_wait(&sh.drain, 0) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ---------------- epilogue: warps 2-5, one token row per thread
    const int quarter = warp & 3;                     // TMEM lanes this warp may read
    const int row = quarter * 32 + lane;              // row of the token tile
    const int tok = m * kBM + row;                    // global token row
    const bool valid = tok < q.T;
    const int K1 = p.K + 1;
    int x = -1;
    if (!kWriteLogits && valid && (tok % K1) < p.K) {
      x = __ldg(p.draft + static_cast<long long>(tok / K1) * p.K + (tok % K1));
      if (x < 0 || x >= p.V) x = -1;
    }
    float best = -INFINITY, zx = 0.0f, nan_acc = 0.0f;
    int best_i = -1;
    bool has_zx = false;
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    for (int t = 0; t < n_tiles; ++t) {
      const int a = t & 1;
      const bool ok = __all_sync(kFull, mbar_wait(&sh.acc_full[a], (t >> 1) & 1, &sh.abort));
      if (!ok) {
        sh.abort = 1;
        if (lane == 0) report_timeout(p);
        break;
      }
      tc_fence_after();
      const int n0 = (n_first + t * q.ctas_per_tile) * kBN;
#pragma unroll 1
      for (int c = 0; c < kBN; c += 32) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_base + static_cast<uint32_t>(a * kBN + c), r);
        tmem_ld_wait();
        if (kWriteLogits) {
          if (valid) {
            float* out = q.logits_out + static_cast<long long>(tok) * q.V + n0 + c;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (n0 + c + i < q.V) out[i] = __uint_as_float(r[i]);
          }
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int col = n0 + c + i;
            const float v = __uint_as_float(r[i]);
            if (col < q.V) {
              nan_acc = fmax_nan(nan_acc, v);
              if (v > best || best_i < 0) {  // columns arrive in increasing order: first maximum kept
                best = v;
                best_i = col;
              }
              if (col == x) {
                zx = v;
                has_zx = true;
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.acc_empty[a]);
    }
    if (!kWriteLogits && valid && !sh.abort) {
      const unsigned long long key = best_i < 0 ? 0ull : make_key(best, static_cast<uint32_t>(best_i));
      if (key) atomicMax(&p.row_key[tok], key);
      if (has_zx) p.draft_logit[tok] = zx;
      if (nan_acc != nan_acc) atomicOr(&p.flags[tok / K1], ASD_STATUS_NAN_LOGIT);
    }
    __threadfence();
  }

  tc_fence_before();
  __syncthreads();
  if (sh.abort && warp == 0 && lane == 0) {
    // wait (bounded) for the loads still in flight before the CTA exits
    for (int it = it_issued > kStages ? it_issued - kStages : 0; it < it_issued; ++it) {
      const int s = it % kStages;
      const unsigned long long t0 = global_ns();
      while (!mbar_try_wait(&sh.full[s], (it / kStages) & 1) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
  if (kWriteLogits || sh.abort) return;

  // Count this CTA's rows of each request of its token tile; the CTA that
  // completes a request (every CTA of the tile has counted) runs its selection.
  const int K1 = p.K + 1;
  const int t0 = m * kBM, t1 = (m + 1) * kBM < q.T ? (m + 1) * kBM : q.T;
  if (t0 < t1) {
    const int b_first = t0 / K1, b_last = (t1 - 1) / K1;
    const unsigned long long total = static_cast<unsigned long long>(K1) * q.ctas_per_tile;
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

// 2-D bf16 row-major [rows, cols] tensor, boxes of box_rows x 64 columns,
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
  bool ready[4] = {false, false, false, false};
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

template <bool kStrict, bool kWriteLogits>
int launch_lmhead(const void* hidden, const void* weight, int H, int T, VerifyParams& p, float* logits_out,
                  cudaStream_t stream) {
  LmDevice* dev = nullptr;
  int rc = lm_device(&dev);
  if (rc != ASD_OK) return rc;
  if (dev->major != 10) return ASD_ERR_DEVICE;  // tcgen05 needs a Blackwell (sm_10x) device
  auto kernel = lmhead_verify_kernel<kStrict, kWriteLogits>;
  const int slot = (kStrict ? 1 : 0) + (kWriteLogits ? 2 : 0);
  if (!dev->ready[slot]) {
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kLmSmemBytes)) !=
        cudaSuccess)
      return ASD_ERR_CUDA;
    dev->ready[slot] = true;
  }
  CUtensorMap map_h, map_w;
  if (!make_map(&map_h, hidden, T, H, kBM) || !make_map(&map_w, weight, p.V, H, kBN)) return ASD_ERR_CUDA;
  LmParams q;
  q.T = T;
  q.H = H;
  q.V = p.V;
  q.token_tiles = (T + kBM - 1) / kBM;
  q.ctas_per_tile = dev->sms / q.token_tiles > 0 ? dev->sms / q.token_tiles : 1;
  q.vocab_tiles = (p.V + kBN - 1) / kBN;
  if (q.ctas_per_tile > q.vocab_tiles) q.ctas_per_tile = q.vocab_tiles;
  q.k_steps = (H + kBK - 1) / kBK;
  q.logits_out = logits_out;
  const unsigned grid = static_cast<unsigned>(q.token_tiles * q.ctas_per_tile);
  kernel<<<grid, kLmThreads, kLmSmemBytes, stream>>>(map_h, map_w, p, q);
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
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
