// libasd: verifier of Approximate Speculative Decoding (arXiv 2608.03447) for
// GB300 (sm_103a). Logit-streaming path: asd_verify, asd_verify_strict,
// asd_verify_blocks, asd_shard_partials and asd_verify_noalloc.
//
// A step is two stages over the [B, K+1, V] logits, treated as one flat array:
//   row stage  (Eq. 1, Eq. 3) the flat array is cut into equal, 16-byte
//              aligned ranges; each range is streamed with 128-bit loads (or
//              TMA bulk copies into a shared-memory ring), every lane keeps a
//              NaN-propagating running maximum, and each row segment reduces
//              to one 64-bit key (order-preserving fp32 bits, then the
//              inverted vocabulary index) merged into the row's slot by
//              atomicMax: the largest key is the largest logit at the lowest
//              index, whatever order the segments finish in. The segment that
//              holds the draft token also records z_j(x_j).
//   selection  (Eq. 5-13, Alg. 1) one warp per request, lane j owning target
//              row j, resets the request's workspace slots to zero as it reads
//              them, so the workspace is zero again after every call (whatever
//              shape the next call has).
// Three row-stage kernels cover the input sizes: verify_small_kernel (one CTA
// per request, selection in the same CTA) below 1 MB when a request fits one
// round of loads, verify_kernel (register streaming; the warp that completes a
// request selects it) for other small inputs, and verify_tma_kernel from 1 MB,
// followed by select_kernel (or, as a launch option, selecting in the CTA that
// completes each request).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "asd.h"
#include "asd_device.cuh"

namespace {

using namespace asd_detail;

// Tuning constants (overridable at build time for launch-shape sweeps).
#ifndef ASD_VERIFY_THREADS
#define ASD_VERIFY_THREADS 256
#endif
#ifndef ASD_VERIFY_UNROLL
#define ASD_VERIFY_UNROLL 4
#endif
#ifndef ASD_VERIFY_MIN_BLOCKS
#define ASD_VERIFY_MIN_BLOCKS 0  // 0: no residency hint to the register allocator
#endif
#ifndef ASD_VERIFY_MIN_ELEMS_PER_WARP
#define ASD_VERIFY_MIN_ELEMS_PER_WARP 2048
#endif
constexpr int kThreads = ASD_VERIFY_THREADS;
constexpr int kWarpsPerBlock = kThreads / 32;
constexpr int kUnroll = ASD_VERIFY_UNROLL;  // 128-bit loads in flight per lane
constexpr long long kMinElemsPerWarp = ASD_VERIFY_MIN_ELEMS_PER_WARP;
__device__ __forceinline__ uint4 load_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float vec_max(const uint4& v, float) {
  return fmax_nan(fmax_nan(__uint_as_float(v.x), __uint_as_float(v.y)),
                  fmax_nan(__uint_as_float(v.z), __uint_as_float(v.w)));
}

__device__ __forceinline__ float vec_max(const uint4& v, __nv_bfloat16) {
  uint32_t m;
  asm("{\n\t.reg .b32 t0, t1;\n\t"
      "max.NaN.bf16x2 t0, %1, %2;\n\t"
      "max.NaN.bf16x2 t1, %3, %4;\n\t"
      "max.NaN.bf16x2 %0, t0, t1;\n\t}"
      : "=r"(m)
      : "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w));
  return fmax_nan(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
}

// ---------------------------------------------------------------- stage 1: one row segment

// Reduces elements [s0, s1) of one row (which starts at flat index row0) to a
// key; every lane returns the warp's key. Sets *nan when a NaN was seen.
template <typename T, int kU = kUnroll>
__device__ __forceinline__ unsigned long long segment_key(const T* z, long long s0, long long s1,
                                                          long long row0, long long head,
                                                          int lane, bool* nan) {
  constexpr int VN = Elem<T>::kVec;
  // the vector grid starts at `head`, the first 16-byte aligned element
  const long long rel0 = s0 - head, rel1 = s1 - head;
  long long bs = rel0 <= 0 ? head : head + ((rel0 + VN - 1) / VN) * VN;
  bs = bs < s1 ? bs : s1;
  long long be = rel1 <= 0 ? head : head + (rel1 / VN) * VN;
  be = be < bs ? bs : (be > s1 ? s1 : be);

  float best = -INFINITY;
  long long best_i = -1;
  bool saw_nan = false;

  // body: whole vectors, lane l takes vectors l, l+32, ... in increasing order,
  // so a strictly greater test keeps each lane's first occurrence
  const long long nvec = (be - bs) / VN;
  if (nvec > 0) {
    const uint4* vp = reinterpret_cast<const uint4*>(z + bs);
    float vbest = -INFINITY;
    int bvec = -1;
    uint4 saved = make_uint4(0, 0, 0, 0);
    long long k = lane;
    for (; k + 32 * (kU - 1) < nvec; k += 32 * kU) {
      uint4 v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) v[u] = load_stream(vp + k + 32 * u);
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const float m = vec_max(v[u], T());
        const bool gt = m > vbest;
        vbest = fmax_nan(vbest, m);
        if (gt) {
          saved = v[u];
          bvec = static_cast<int>(k + 32 * u);
        }
      }
    }
    for (; k < nvec; k += 32) {
      const uint4 v = load_stream(vp + k);
      const float m = vec_max(v, T());
      const bool gt = m > vbest;
      vbest = fmax_nan(vbest, m);
      if (gt) {
        saved = v;
        bvec = static_cast<int>(k);
      }
    }
    if (vbest != vbest) saw_nan = true;
    if (lane < nvec) {
      if (bvec >= 0) {
        int t_first = VN - 1;
#pragma unroll
        for (int t = VN - 1; t >= 0; --t)
          if (Elem<T>::lane(saved, t) == vbest) t_first = t;
        best = vbest;
        best_i = bs + static_cast<long long>(bvec) * VN + t_first;
      } else {
        // every value this lane saw is -inf (or NaN, flagged): its first element stands
        best = -INFINITY;
        best_i = bs + static_cast<long long>(lane) * VN;
      }
    }
  }

  // ragged ends: fewer than one vector on each side, one element per lane
  const long long n_head = bs - s0, n_tail = s1 - be;
  if (lane < n_head || lane < n_tail) {
#pragma unroll
    for (int side = 0; side < 2; ++side) {
      const long long e = side == 0 ? s0 + lane : be + lane;
      if (e >= (side == 0 ? bs : s1)) continue;
      const float v = Elem<T>::load(z, e);
      if (v != v) {
        saw_nan = true;
        continue;
      }
      if (best_i < 0 || v > best || (v == best && e < best_i)) {
        best = v;
        best_i = e;
      }
    }
  }

  *nan = __any_sync(kFull, saw_nan);
  const unsigned long long key =
      best_i < 0 ? 0ull : make_key(best, static_cast<uint32_t>(best_i - row0));
  return warp_max_key(key);
}

// ---------------------------------------------------------------- the fused kernel

#if ASD_VERIFY_MIN_BLOCKS > 0
#define ASD_VERIFY_BOUNDS __launch_bounds__(kThreads, ASD_VERIFY_MIN_BLOCKS)
#else
#define ASD_VERIFY_BOUNDS __launch_bounds__(kThreads)
#endif

template <typename T, bool kStrict>
__global__ void ASD_VERIFY_BOUNDS verify_kernel(const VerifyParams p) {
  const int lane = threadIdx.x & 31;
  const long long warp = static_cast<long long>(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  const long long lo = warp == 0 ? 0 : p.head + warp * p.per_warp;
  long long hi = p.head + (warp + 1) * p.per_warp;
  hi = hi < p.total ? hi : p.total;
  if (lo >= hi) return;

  const T* z = static_cast<const T*>(p.logits);
  const int V = p.V, K = p.K, K1 = p.K + 1;
  // counters are per request; a request is complete when all p.nblk of its blocks are
  const unsigned long long request_elems = static_cast<unsigned long long>(K1) * V * p.nblk;

  long long row = lo / V;
  int pending_b = static_cast<int>(row / K1);
  unsigned long long pending_n = 0;

  for (long long s0 = lo; s0 < hi; ++row) {
    const long long row0 = row * V;
    const long long s1 = hi < row0 + V ? hi : row0 + V;
    const int b = static_cast<int>(row / K1);
    const int j = static_cast<int>(row - static_cast<long long>(b) * K1);
    int x = -1;
    if (j < K) x = __ldg(p.draft + static_cast<long long>(b) * K + j) - p.v_offset;  // shard-local

    if (b != pending_b) {  // finished this warp's share of block-request pending_b
      bool last = false;
      if (lane == 0) {
        __threadfence();
        const unsigned long long old = atomicAdd(&p.done[pending_b % p.B], pending_n);
        last = old + pending_n == request_elems;
      }
      if (__shfl_sync(kFull, last, 0)) {
        __threadfence();
        select_request<T, kStrict>(p, pending_b % p.B, lane);
      }
      pending_b = b;
      pending_n = 0;
    }

    bool nan = false;
    const unsigned long long key = segment_key<T>(z, s0, s1, row0, p.head, lane, &nan);
    if (lane == 0) {
      atomicMax(&p.row_key[row], key);
      if (nan) atomicOr(&p.flags[b], ASD_STATUS_NAN_LOGIT);
      if (x >= 0 && x < V && row0 + x >= s0 && row0 + x < s1)
        p.draft_logit[row] = Elem<T>::load(z, row0 + x);
    }
    pending_n += static_cast<unsigned long long>(s1 - s0);
    s0 = s1;
  }

  bool last = false;
  if (lane == 0) {
    __threadfence();
    const unsigned long long old = atomicAdd(&p.done[pending_b % p.B], pending_n);
    last = old + pending_n == request_elems;
  }
  if (__shfl_sync(kFull, last, 0)) {
    __threadfence();
    select_request<T, kStrict>(p, pending_b % p.B, lane);
  }
}

// ---------------------------------------------------------------- one CTA per request (small inputs)
//
// When a request's K+1 rows are a few KB, what the streaming kernels pay for is
// their global round trips (row keys, counters, fences), not the bytes. Here a
// CTA takes one request: its warps split the request's rows flatly (one round
// of loads, every lane with up to kSmallUnroll vectors in flight), merge the
// row keys and the draft logits in shared memory, and warp 0 runs Alg. 1 from
// there. The workspace is not touched.

constexpr int kSmallThreads = 512;
constexpr int kSmallUnroll = 8;
constexpr long long kSmallMaxRequestBytes = 16LL * kSmallThreads * kSmallUnroll;  // 64 KB: one round of loads

template <typename T, bool kStrict>
__global__ void __launch_bounds__(kSmallThreads) verify_small_kernel(const __grid_constant__ VerifyParams p) {
  __shared__ unsigned long long s_key[32];
  __shared__ float s_zx[32];
  __shared__ unsigned int s_flags;
  constexpr int VN = Elem<T>::kVec;
  constexpr int kWarps = kSmallThreads / 32;
  const int b = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int V = p.V, K = p.K, K1 = p.K + 1;
  if (threadIdx.x < 32) {
    s_key[threadIdx.x] = 0ull;
    s_zx[threadIdx.x] = 0.0f;
  }
  if (threadIdx.x == 0) s_flags = 0u;
  // Programmatic dependent launch: the next call's CTAs may start now. With
  // resident inputs this call reads its logits and drafts before the previous
  // kernel on the stream has completed; the ledger and the outputs, which that
  // kernel may use, wait for it in every case.
  pdl_signal_dependents();
  if (!p.resident) pdl_wait_prerequisites();
  float budget = 0.0f, spent = 0.0f;
  if (!kStrict && !p.resident && threadIdx.x == 0) {  // in flight while the logits stream
    budget = p.ledger[b].budget;
    spent = p.ledger[b].spent;
  }
  __syncthreads();

  const T* z = static_cast<const T*>(p.logits);
  const long long n = static_cast<long long>(K1) * V;
  const long long base = static_cast<long long>(b) * n;
  long long per = (n + kWarps - 1) / kWarps;
  per = (per + VN - 1) / VN * VN;
  const long long lo = base + (warp * per < n ? warp * per : n);
  const long long hi = base + ((warp + 1) * per < n ? (warp + 1) * per : n);
  for (long long s0 = lo; s0 < hi;) {
    const long long row = s0 / V;
    const long long row0 = row * V;
    const long long s1 = hi < row0 + V ? hi : row0 + V;
    const int j = static_cast<int>(row - static_cast<long long>(b) * K1);
    bool nan = false;
    const unsigned long long key = segment_key<T, kSmallUnroll>(z, s0, s1, row0, p.head, lane, &nan);
    if (lane == 0) {
      atomicMax(&s_key[j], key);
      if (nan) atomicOr(&s_flags, ASD_STATUS_NAN_LOGIT);
      if (j < K) {
        const int x = __ldg(p.draft + static_cast<long long>(b) * K + j);
        if (x >= 0 && x < V && row0 + x >= s0 && row0 + x < s1) s_zx[j] = Elem<T>::load(z, row0 + x);
      }
    }
    s0 = s1;
  }
  __syncthreads();
  if (warp != 0) return;
  if (p.resident) {
    pdl_wait_prerequisites();
    if (!kStrict && lane == 0) {
      budget = p.ledger[b].budget;
      spent = p.ledger[b].spent;
    }
  }

  BlockInputs in;
  in.key = lane < K1 ? s_key[lane] : 0ull;
  in.x = lane < K ? __ldg(p.draft + static_cast<long long>(b) * K + lane) : -1;
  in.zx = lane < K ? s_zx[lane] : 0.0f;
  in.flags = s_flags | workspace_failed(p, lane);
  in.top = ordered_value(static_cast<uint32_t>(in.key >> 32));
  in.top_exact = false;
  budget = __shfl_sync(kFull, budget, 0);
  spent = __shfl_sync(kFull, spent, 0);
  bool wrote = false;
  select_block<T, kStrict>(p, b, in, budget, spent, wrote, lane);
  if (!kStrict && lane == 0 && wrote) p.ledger[b].spent = spent;
}

// ---------------------------------------------------------------- TMA pipeline kernel
//
// One CTA per SM per launch. The CTA owns an equal, 16-byte aligned slice of
// the flat logits and streams it through a ring of shared-memory stages with
// bulk copies (cp.async.bulk, completion counted on an mbarrier). A producer
// warp keeps every free stage in flight, so the bytes in flight per SM are set
// by the ring, not by registers. Each consumer warp takes a fixed sub-range of
// every chunk, so it visits its elements in increasing order and keeps one
// running (value, index) per lane for the row it is in; finished rows merge
// into a shared-memory row table (or straight into the workspace when a slice
// spans more rows than the table holds). Nothing touches the workspace before
// griddepcontrol.wait: every CTA signals its dependents at start, so the next
// launches on the stream stream their own logits while this one ends. The
// ring is small (4 x 16 KB) and registers are capped so that three CTAs --
// three consecutive launches -- share an SM: one ramping up, one streaming, one
// finishing. By default the selection then runs in select_kernel, launched
// right behind (split mode); otherwise the CTAs count their elements per
// request at the end and the last one to finish a request selects it.
// Every wait is bounded (about a second of %globaltimer); on a timeout the CTA
// records ASD_ERR_TIMEOUT in the workspace, stops, and drains its own copies.

#ifndef ASD_TMA_STAGES
#define ASD_TMA_STAGES 4  // 4 x 16 KB: three CTAs (three consecutive launches) fit on one SM
#endif
#ifndef ASD_TMA_CHUNK_BYTES
#define ASD_TMA_CHUNK_BYTES 16384
#endif
#ifndef ASD_TMA_CONSUMER_WARPS
#define ASD_TMA_CONSUMER_WARPS 8
#endif
#ifndef ASD_TMA_MIN_BLOCKS
#define ASD_TMA_MIN_BLOCKS 3  // CTAs per SM the register allocator must leave room for
#endif
#ifndef ASD_TMA_LONE_CTAS_PER_SM
#define ASD_TMA_LONE_CTAS_PER_SM 3  // CTAs per SM of a launch that cannot overlap the previous one
#endif
#ifndef ASD_TMA_L2_HINT
#define ASD_TMA_L2_HINT 1  // evict-first L2 policy on the streamed logits
#endif
constexpr int kTmaStages = ASD_TMA_STAGES;
constexpr int kTmaChunkBytes = ASD_TMA_CHUNK_BYTES;
constexpr int kTmaConsumers = ASD_TMA_CONSUMER_WARPS;
constexpr int kTmaThreads = (kTmaConsumers + 1) * 32;
static_assert(kTmaChunkBytes % (16 * 32 * kTmaConsumers) == 0,
              "every consumer warp takes whole 128-bit vectors of each chunk, one per lane per pass");

// Rows of one CTA's slice merged in shared memory until the end of the stream
// (then flushed to the workspace once); slices spanning more rows than this
// merge straight into the workspace.
constexpr int kRowTable = 256;

struct TmaShared {
  uint4 ring[kTmaStages][kTmaChunkBytes / 16];
  unsigned long long full[kTmaStages];
  unsigned long long empty[kTmaStages];
  unsigned long long row_key[kRowTable];  // merged (value, index) keys of the slice's rows
  float row_zx[kRowTable];                // the draft token's logit of each row, if seen here
  unsigned int row_bits[kRowTable];       // 1: a NaN was seen, 2: row_zx is valid
  int abort;
};

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          unsigned long long* bar, unsigned long long policy) {
#if ASD_TMA_L2_HINT
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
#else
  (void)policy;
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
#endif
}
__device__ __forceinline__ unsigned long long evict_first_policy() {
  unsigned long long pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint4 lds128(const uint4* p) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(smem_u32(p)));
  return v;
}

// Element `off` of a staged chunk, read with ld.shared (src is a shared-memory
// pointer: the global-only loads of Elem<T>::load must never see it).
__device__ __forceinline__ float smem_elem(const uint4* src, int off, float) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(smem_u32(src) + 4u * static_cast<uint32_t>(off)));
  return v;
}
__device__ __forceinline__ float smem_elem(const uint4* src, int off, __nv_bfloat16) {
  unsigned short bits;
  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(bits) : "r"(smem_u32(src) + 2u * static_cast<uint32_t>(off)));
  return __uint_as_float(static_cast<uint32_t>(bits) << 16);
}

// The first element of v equal to m, its maximum; VN - 1 if none (m is NaN).
template <typename T>
__device__ __forceinline__ int vec_first_equal(const uint4& v, float m) {
  int first = Elem<T>::kVec - 1;
#pragma unroll
  for (int t = Elem<T>::kVec - 1; t >= 0; --t)
    if (Elem<T>::lane(v, t) == m) first = t;
  return first;
}

// Merges one warp's partial result for a row into the workspace: the row's
// key, its NaN flag and (from the lane that holds it) the draft token's logit.
// The first global write of a warp: it waits for the previous launch first.
__device__ __noinline__ void flush_row_key(const VerifyParams& p, long long row, int b,
                                           unsigned long long key, bool nan, bool has_zx, float zx,
                                           int lane) {
  pdl_wait_prerequisites();
  key = warp_max_key(key);
  nan = __any_sync(kFull, nan);
  if (lane == 0) {
    if (key) atomicMax(&p.row_key[row], key);
    if (nan) atomicOr(&p.flags[b], ASD_STATUS_NAN_LOGIT);
  }
  if (has_zx) p.draft_logit[row] = zx;
}

// Per-warp cursor: the row and request the warp is in (warp-uniform) and each
// lane's running candidate for that row. Offsets are relative to the row start.
struct RowCursor {
  long long row;            // current row
  long long row0, row1;     // its flat element range [row0, row1)
  int b;                    // its request
  int x;                    // its draft id, -1 for the bonus row or an id outside [0, V)
  int next_x;               // prefetched draft id of row + 1
  float best;               // per lane: NaN-propagating maximum over whole vectors
  int saved_rel;            // per lane: offset of the vector that first reached best, -1 none
  uint4 saved;              // per lane: that vector
  int first_rel;            // per lane: offset of the lane's first vector in the row, -1 none
  float sbest;              // per lane: best single element seen at row boundaries
  int sidx;                 // per lane: its offset, -1 none
  bool snan;                // per lane: a single element was NaN
  float zx;                 // per lane: the draft token's logit, if this lane saw it
  bool has_zx;
};

__device__ __forceinline__ int draft_of_row(const VerifyParams& p, long long row) {
  const int K1 = p.K + 1;
  const long long b = row / K1;
  const int j = static_cast<int>(row - b * K1);
  if (j >= p.K || b >= static_cast<long long>(p.B) * p.nblk) return -1;  // b: block-request
  return __ldg(p.draft + b * p.K + j) - p.v_offset;  // shard-local (no shift without a shard)
}

__device__ __forceinline__ void cursor_enter(RowCursor& c, const VerifyParams& p, long long row) {
  c.row = row;
  c.row0 = row * p.V;
  c.row1 = c.row0 + p.V;
  c.b = static_cast<int>(row / (p.K + 1));
  c.x = (c.next_x >= 0 && c.next_x < p.V) ? c.next_x : -1;
  c.next_x = draft_of_row(p, row + 1);  // consumed at the next row change
  c.best = -INFINITY;
  c.saved_rel = -1;
  c.saved = make_uint4(0, 0, 0, 0);
  c.first_rel = -1;
  c.sbest = -INFINITY;
  c.sidx = -1;
  c.snan = false;
  c.zx = 0.0f;
  c.has_zx = false;
}

// Where a warp's finished rows go: the CTA's row table (rows table_row0 ..)
// or, when the slice spans too many rows, the workspace directly.
struct RowSink {
  TmaShared* sh;
  long long table_row0;
  bool table;
};

template <typename T>
__device__ __forceinline__ void cursor_flush_row(RowCursor& c, const VerifyParams& p, const RowSink& sink,
                                                 int lane) {
  float v = -INFINITY;
  int idx = -1;
  if (c.saved_rel >= 0) {
    v = c.best;
    idx = c.saved_rel + vec_first_equal<T>(c.saved, c.best);
  } else if (c.first_rel >= 0) {
    idx = c.first_rel;  // every whole-vector value this lane saw was -inf (or NaN, flagged)
  }
  if (c.sidx >= 0 && (idx < 0 || c.sbest > v || (c.sbest == v && c.sidx < idx))) {
    v = c.sbest;
    idx = c.sidx;
  }
  const unsigned long long key = idx < 0 ? 0ull : make_key(v, static_cast<uint32_t>(idx));
  const bool nan = c.snan || c.best != c.best;
  if (!sink.table) {
    flush_row_key(p, c.row, c.b, key, nan, c.has_zx, c.zx, lane);
    return;
  }
  const int t = static_cast<int>(c.row - sink.table_row0);
  const unsigned long long wkey = warp_max_key(key);
  const bool wnan = __any_sync(kFull, nan);
  if (lane == 0) {
    if (wkey) atomicMax(&sink.sh->row_key[t], wkey);
    if (wnan) atomicOr(&sink.sh->row_bits[t], 1u);
  }
  if (c.has_zx) {
    sink.sh->row_zx[t] = c.zx;
    atomicOr(&sink.sh->row_bits[t], 2u);
  }
}

// Moves the cursor to the row holding flat element e, flushing what it leaves.
template <typename T>
__device__ __forceinline__ void cursor_advance(RowCursor& c, const VerifyParams& p, const RowSink& sink,
                                               long long e, int lane) {
  cursor_flush_row<T>(c, p, sink, lane);
  const long long row = e / p.V;
  if (row != c.row + 1) c.next_x = draft_of_row(p, row);  // rows in between belong to other warps
  cursor_enter(c, p, row);
}

// One element at row offset rel (row boundaries, ragged head and tail).
__device__ __forceinline__ void lane_element(RowCursor& c, const VerifyParams& p, float v, int rel) {
  if (v != v) {
    c.snan = true;
  } else if (c.sidx < 0 || v > c.sbest) {
    c.sbest = v;
    c.sidx = rel;
  }
  if (rel == c.x) {
    c.zx = v;
    c.has_zx = true;
  }
}

// Elements [a, a + 32*VN*kPasses) of the flat array, staged at `src`, one
// vector per lane per pass (vector u*32 + lane); elements at or past `limit`
// are not data.
template <typename T, bool kStrict, int kPasses>
__device__ __forceinline__ void consume_span(RowCursor& c, const VerifyParams& p, const RowSink& sink,
                                             const uint4* src, long long a, long long limit, int lane) {
  constexpr int VN = Elem<T>::kVec;
  constexpr int kSpan = kPasses * 32 * VN;
  const long long span_end = a + kSpan;
  if (span_end <= c.row1 && span_end <= limit) {
    // fast path: the whole span lies in the current row; no branches per vector
    uint4 v[kPasses];
#pragma unroll
    for (int u = 0; u < kPasses; ++u) v[u] = lds128(src + u * 32 + lane);
    const int a_rel = static_cast<int>(a - c.row0);
    if (c.first_rel < 0) c.first_rel = a_rel + lane * VN;
#pragma unroll
    for (int u = 0; u < kPasses; ++u) {
      const float m = vec_max(v[u], T());
      const bool gt = m > c.best;
      c.best = fmax_nan(c.best, m);
      c.saved.x = gt ? v[u].x : c.saved.x;
      c.saved.y = gt ? v[u].y : c.saved.y;
      c.saved.z = gt ? v[u].z : c.saved.z;
      c.saved.w = gt ? v[u].w : c.saved.w;
      c.saved_rel = gt ? a_rel + (u * 32 + lane) * VN : c.saved_rel;
    }
    const int off = c.x - a_rel;  // the draft token's logit, if this span holds it
    if (static_cast<unsigned>(off) < static_cast<unsigned>(kSpan) && lane == 0) {
      c.zx = smem_elem(src, off, T());
      c.has_zx = true;
    }
    return;
  }
  // slow path: row boundaries (or the end of the data) inside the span
  const long long end = span_end < limit ? span_end : limit;
#pragma unroll 1
  for (int u = 0; u < kPasses; ++u) {
    const long long g0 = a + static_cast<long long>(u) * 32 * VN;  // this pass covers [g0, g0 + 32 VN)
    if (g0 >= end) break;
    const long long g1 = g0 + 32 * VN < end ? g0 + 32 * VN : end;
    const long long e0 = g0 + static_cast<long long>(lane) * VN;    // this lane's vector
    uint4 v = make_uint4(0, 0, 0, 0);
    if (e0 < g1) v = lds128(src + u * 32 + lane);
    long long pos = g0;
    while (pos < g1) {  // warp-uniform: one row of the pass at a time
      if (pos >= c.row1) cursor_advance<T>(c, p, sink, pos, lane);
      const long long seg_end = g1 < c.row1 ? g1 : c.row1;
#pragma unroll
      for (int t = 0; t < VN; ++t) {
        const long long e = e0 + t;
        if (e >= pos && e < seg_end) lane_element(c, p, Elem<T>::lane(v, t), static_cast<int>(e - c.row0));
      }
      pos = seg_end;
    }
  }
}

// Single elements [from, to) read from global memory (the ragged head and tail).
template <typename T, bool kStrict>
__device__ __forceinline__ void consume_loose(RowCursor& c, const VerifyParams& p, const RowSink& sink,
                                              long long from, long long to, int lane) {
  const T* z = static_cast<const T*>(p.logits);
  for (long long pos = from; pos < to;) {
    if (pos >= c.row1) cursor_advance<T>(c, p, sink, pos, lane);
    const long long seg_end = to < c.row1 ? to : c.row1;
    const long long e = pos + lane;
    if (e < seg_end) lane_element(c, p, Elem<T>::load(z, e), static_cast<int>(e - c.row0));
    pos = seg_end;
  }
}

template <typename T, bool kStrict, bool kSplit>
__global__ void __launch_bounds__(kTmaThreads, ASD_TMA_MIN_BLOCKS)
    verify_tma_kernel(const __grid_constant__ VerifyParams p, long long bulk_end, long long per_cta) {
  constexpr int VN = Elem<T>::kVec;
  constexpr int kChunkElems = kTmaChunkBytes / static_cast<int>(sizeof(T));
  constexpr int kWarpElems = kChunkElems / kTmaConsumers;  // one consumer's share of a chunk
  constexpr int kPasses = kWarpElems / (32 * VN);          // vectors per lane per chunk
  extern __shared__ __align__(128) unsigned char smem_raw[];
  TmaShared& sh = *reinterpret_cast<TmaShared*>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const T* z = static_cast<const T*>(p.logits);

  // this CTA's slice [lo, hi) of the bulk region [p.head, bulk_end)
  const long long lo = p.head + static_cast<long long>(blockIdx.x) * per_cta;
  long long hi = lo + per_cta;
  hi = hi < bulk_end ? hi : bulk_end;
  const int nchunks = lo < hi ? static_cast<int>((hi - lo + kChunkElems - 1) / kChunkElems) : 0;

  pdl_signal_dependents();

  // Shared-memory set-up first: it reads no input, so a launch that has to
  // wait for the previous kernel does it while waiting.
  // This CTA's rows, including the ragged head (CTA 0) and tail (last CTA).
  const long long cta_lo = blockIdx.x == 0 ? 0 : lo;
  const long long cta_hi = blockIdx.x == gridDim.x - 1 ? p.total : hi;
  RowSink sink;
  sink.sh = &sh;
  sink.table_row0 = cta_lo / p.V;
  const long long table_rows = cta_lo < cta_hi ? (cta_hi - 1) / p.V - sink.table_row0 + 1 : 0;
  sink.table = table_rows <= kRowTable;
  for (int t = threadIdx.x; t < kRowTable; t += blockDim.x) {
    sh.row_key[t] = 0ull;
    sh.row_bits[t] = 0u;
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kTmaStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], kTmaConsumers);
    }
    sh.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();

  // Unless the caller declared the inputs resident, the previous kernel on the
  // stream may be the one writing them: read nothing before it has completed.
  if (!p.resident) pdl_wait_prerequisites();

  // each consumer's first row is known now: start its draft-id load before the
  // first copy lands
  RowCursor c;
  c.next_x = -1;
  const long long first_a = lo + static_cast<long long>(warp) * kWarpElems;
  const bool head_here = blockIdx.x == 0 && warp == 0 && p.head > 0;
  if (warp < kTmaConsumers) c.next_x = draft_of_row(p, head_here ? 0 : (first_a < hi ? first_a : 0) / p.V);

  int issued = 0;  // producer: chunks issued
  if (warp == kTmaConsumers) {
    if (lane == 0) {
      const unsigned long long policy = evict_first_policy();
      for (int ch = 0; ch < nchunks; ++ch) {
        const int s = ch % kTmaStages;
        if (ch >= kTmaStages && !mbar_wait(&sh.empty[s], ((ch / kTmaStages) - 1) & 1, &sh.abort)) {
          sh.abort = 1;
          atomicExch(p.error, static_cast<unsigned>(ASD_ERR_TIMEOUT));
          break;
        }
        const long long e0 = lo + static_cast<long long>(ch) * kChunkElems;
        const long long n = hi - e0 < kChunkElems ? hi - e0 : kChunkElems;
        const uint32_t bytes = static_cast<uint32_t>(n * sizeof(T));
        mbar_expect_tx(&sh.full[s], bytes);
        bulk_load(sh.ring[s], z + e0, bytes, &sh.full[s], policy);
        issued = ch + 1;
      }
    }
  } else {
    bool started = false;

    // the ragged head [0, p.head) (fewer than VN elements) belongs to CTA 0, warp 0
    if (head_here) {
      cursor_enter(c, p, 0);
      started = true;
      consume_loose<T, kStrict>(c, p, sink, 0, p.head, lane);
    }

    for (int ch = 0; ch < nchunks; ++ch) {
      const int s = ch % kTmaStages;
      // every lane observes the phase itself (that makes the staged bytes visible
      // to it); the warp proceeds only if all lanes did
      const bool ok = __all_sync(kFull, mbar_wait(&sh.full[s], (ch / kTmaStages) & 1, &sh.abort));
      if (!ok) {
        sh.abort = 1;
        if (lane == 0) atomicExch(p.error, static_cast<unsigned>(ASD_ERR_TIMEOUT));
        break;
      }
      const long long a = lo + static_cast<long long>(ch) * kChunkElems + static_cast<long long>(warp) * kWarpElems;
      if (a < hi) {
        if (!started) {
          cursor_enter(c, p, a / p.V);  // its draft id was loaded at kernel start
          started = true;
        } else if (a >= c.row1) {
          cursor_advance<T>(c, p, sink, a, lane);
        }
        consume_span<T, kStrict, kPasses>(c, p, sink, sh.ring[s] + warp * (kWarpElems / VN), a, hi, lane);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.empty[s]);
    }

    // the ragged tail [bulk_end, total) (fewer than VN elements): last CTA, last consumer
    if (!sh.abort && blockIdx.x == gridDim.x - 1 && warp == kTmaConsumers - 1 && bulk_end < p.total) {
      if (!started) {
        c.next_x = draft_of_row(p, bulk_end / p.V);
        cursor_enter(c, p, bulk_end / p.V);
        started = true;
      }
      consume_loose<T, kStrict>(c, p, sink, bulk_end, p.total, lane);
    }
    if (started && !sh.abort) cursor_flush_row<T>(c, p, sink, lane);
    // this warp's direct key merges (slices spanning many rows) before the counts below
    if (!kSplit && !sink.table) __threadfence();
  }

  __syncthreads();
  if (sh.abort) {
    // after a timeout: wait (bounded) for this CTA's copies still in flight, then leave
    if (warp == kTmaConsumers && lane == 0) {
      for (int ch = issued > kTmaStages ? issued - kTmaStages : 0; ch < issued; ++ch) {
        const int s = ch % kTmaStages;
        const unsigned long long t0 = global_ns();
        while (!mbar_try_wait(&sh.full[s], (ch / kTmaStages) & 1) && global_ns() - t0 < kWaitLimitNs) {
        }
      }
    }
    return;
  }
  // The first touch of the workspace: wait for the previous launch, flush the
  // row table, then count this CTA's elements of each request it touched; the
  // CTA that completes a request runs its selection.
  pdl_wait_prerequisites();
  if (sink.table) {
    for (int t = threadIdx.x; t < table_rows; t += blockDim.x) {
      const long long row = sink.table_row0 + t;
      const unsigned long long key = sh.row_key[t];
      const unsigned bits = sh.row_bits[t];
      if (key) atomicMax(&p.row_key[row], key);
      if (bits & 1u) atomicOr(&p.flags[row / (p.K + 1)], ASD_STATUS_NAN_LOGIT);
      if (bits & 2u) p.draft_logit[row] = sh.row_zx[t];
    }
    // split mode: the selection runs in the next kernel, which the end of this
    // grid orders after every write above; nothing more to do here
    if (kSplit) return;
    __threadfence();
    __syncthreads();
  }
  if (kSplit) return;
  if (cta_lo < cta_hi) {
    const long long rv = static_cast<long long>(p.K + 1) * p.V;
    const long long b_first = cta_lo / rv, b_last = (cta_hi - 1) / rv;
    for (long long b = b_first + warp; b <= b_last; b += kTmaConsumers + 1) {
      const long long r0 = b * rv > cta_lo ? b * rv : cta_lo;
      const long long r1 = (b + 1) * rv < cta_hi ? (b + 1) * rv : cta_hi;
      finish_request<T, kStrict>(p, static_cast<int>(b % p.B), static_cast<unsigned long long>(r1 - r0),
                                 static_cast<unsigned long long>(rv) * p.nblk, lane);
    }
  }
}

// ---------------------------------------------------------------- split selection kernel
//
// With the row stage in verify_tma_kernel<..., kSplit = true>, the selection of
// every request runs here: one warp per request, launched right behind the row
// stage (programmatic dependent launch); griddepcontrol.wait returns once the
// row stage has completed and its writes are visible, so no counters and no
// fences are needed, and the streaming CTAs leave their SMs as soon as they
// have merged their rows.

constexpr int kSelectThreads = 128;  // small: fits beside the streaming CTAs on an SM

template <typename T, bool kStrict>
__global__ void __launch_bounds__(kSelectThreads) select_kernel(const __grid_constant__ VerifyParams p) {
  pdl_signal_dependents();
  pdl_wait_prerequisites();
  const int lane = threadIdx.x & 31;
  const int warps = kSelectThreads / 32;
  for (int b = blockIdx.x * warps + (threadIdx.x >> 5); b < p.B; b += gridDim.x * warps)
    select_request<T, kStrict>(p, b, lane);
}

// ---------------------------------------------------------------- host side

// Resident warps of a kernel on the current device, queried once per device.
template <typename T, bool kStrict>
int resident_warps(int* out) {
  constexpr int kMaxDevices = 64;
  static int cache[kMaxDevices] = {0};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return ASD_ERR_CUDA;
  if (dev >= 0 && dev < kMaxDevices) {
    std::lock_guard<std::mutex> g(mu);
    if (cache[dev] > 0) {
      *out = cache[dev];
      return ASD_OK;
    }
  }
  int sms = 0, blocks = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return ASD_ERR_CUDA;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, verify_kernel<T, kStrict>, kThreads, 0) !=
      cudaSuccess)
    return ASD_ERR_CUDA;
  const int w = sms * (blocks > 0 ? blocks : 1) * kWarpsPerBlock;
  if (dev >= 0 && dev < kMaxDevices) {
    std::lock_guard<std::mutex> g(mu);
    cache[dev] = w;
  }
  *out = w;
  return ASD_OK;
}

struct DeviceInfo {
  int sms = 0;
  // set once the TMA kernel instance has its shared-memory opt-in; the
  // opt-in is idempotent, so two threads racing to set it up is harmless
  std::atomic<bool> tma_ready[8] = {};
};

// Launch options (asd_set_launch_options): process-wide, read once per call,
// so a call (and a CUDA graph captured from it) sees one consistent set.
std::atomic<int> g_path{ASD_PATH_AUTO};
std::atomic<int> g_flags{0};  // bit 0: selection inside the row stage, bit 1: no PDL

struct LaunchOptions {
  int path;
  bool split;  // the TMA path's selection runs in select_kernel, right behind the row stage
  bool pdl;    // launches carry the programmatic-serialization attribute
};

LaunchOptions launch_options() {
  const int f = g_flags.load(std::memory_order_relaxed);
  LaunchOptions o;
  o.path = g_path.load(std::memory_order_relaxed);
  o.split = (f & 1) == 0;
  o.pdl = (f & 2) == 0;
  return o;
}

// SM count of the current device, and the one-time dynamic shared memory
// opt-in of the TMA kernels, cached per device.
int device_info(int* dev_out, DeviceInfo** info_out) {
  constexpr int kMaxDevices = 64;
  static DeviceInfo info[kMaxDevices];
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return ASD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return ASD_ERR_DEVICE;
  std::lock_guard<std::mutex> g(mu);
  if (info[dev].sms == 0) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return ASD_ERR_CUDA;
    info[dev].sms = sms;
  }
  *dev_out = dev;
  *info_out = &info[dev];
  return ASD_OK;
}

template <typename T, bool kStrict>
int launch_tma(VerifyParams& p, const LaunchOptions& opt, cudaStream_t stream) {
  constexpr int VN = Elem<T>::kVec;
  constexpr long long kMinPerCta = 2LL * kTmaChunkBytes / static_cast<long long>(sizeof(T));
  const uintptr_t addr = reinterpret_cast<uintptr_t>(p.logits);
  if (addr % sizeof(T) != 0) return ASD_ERR_ALIGN;
  long long head = static_cast<long long>(((16 - addr % 16) % 16) / sizeof(T));
  if (head > p.total) head = p.total;
  const long long bulk = (p.total - head) / VN * VN;
  int dev = 0;
  DeviceInfo* info = nullptr;
  int rc = device_info(&dev, &info);
  if (rc != ASD_OK) return rc;
  const bool split = opt.split;
  const int slot = (sizeof(T) == 2 ? 2 : 0) + (kStrict ? 1 : 0) + (split ? 4 : 0);
  if (!info->tma_ready[slot].load(std::memory_order_acquire)) {
    auto kernel = split ? verify_tma_kernel<T, kStrict, true> : verify_tma_kernel<T, kStrict, false>;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(sizeof(TmaShared))) != cudaSuccess)
      return ASD_ERR_CUDA;
    info->tma_ready[slot].store(true, std::memory_order_release);
  }
  // Resident inputs: one CTA per SM, so that three consecutive launches share
  // the SMs (one ramping up, one streaming, one finishing). Otherwise the
  // launch reads nothing before the previous kernel completes and runs alone,
  // so it fills every CTA slot of every SM itself.
  const long long max_cta =
      p.resident ? info->sms : static_cast<long long>(info->sms) * ASD_TMA_LONE_CTAS_PER_SM;
  long long ncta = (bulk + kMinPerCta - 1) / kMinPerCta;
  if (ncta > max_cta) ncta = max_cta;
  if (ncta < 1) ncta = 1;
  long long per_cta = (bulk + ncta - 1) / ncta;
  per_cta = (per_cta + VN - 1) / VN * VN;
  if (per_cta < VN) per_cta = VN;
  ncta = bulk > 0 ? (bulk + per_cta - 1) / per_cta : 1;
  p.head = head;
  p.per_warp = 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ncta));
  cfg.blockDim = dim3(kTmaThreads);
  cfg.dynamicSmemBytes = sizeof(TmaShared);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  if (opt.pdl) {
    cfg.attrs = attr;
    cfg.numAttrs = 1;
  }
  const long long bulk_end = head + bulk;
  if (!split) {
    if (cudaLaunchKernelEx(&cfg, verify_tma_kernel<T, kStrict, false>, p, bulk_end, per_cta) != cudaSuccess)
      return ASD_ERR_CUDA;
    return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
  }
  if (cudaLaunchKernelEx(&cfg, verify_tma_kernel<T, kStrict, true>, p, bulk_end, per_cta) != cudaSuccess)
    return ASD_ERR_CUDA;
  cudaLaunchConfig_t sel = cfg;
  constexpr int kWarps = kSelectThreads / 32;
  sel.gridDim = dim3(static_cast<unsigned>((p.B + kWarps - 1) / kWarps));
  sel.blockDim = dim3(kSelectThreads);
  sel.dynamicSmemBytes = 0;
  if (cudaLaunchKernelEx(&sel, select_kernel<T, kStrict>, p) != cudaSuccess) return ASD_ERR_CUDA;
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

// Which kernel streams the logits: the TMA pipeline for inputs of at least
// kTmaMinBytes; below that, one CTA per request when a request fits one round
// of loads of a CTA (single blocks, no vocabulary shard), else the
// register-streaming kernel (fewer, shorter warps start faster on small
// inputs). The launch options can force a kernel (the tests use that to cover
// every kernel); a forced `small` falls back to the default when the shape does
// not qualify.
constexpr long long kTmaMinBytes = 1LL << 20;

enum class Path { kSmall, kStream, kTma };

Path choose_path(int forced, long long bytes, long long request_bytes, int K, bool single_block) {
  const bool small_ok = single_block && K + 1 <= 32 && request_bytes <= kSmallMaxRequestBytes;
  if (forced == ASD_PATH_TMA) return Path::kTma;
  if (forced == ASD_PATH_STREAM) return Path::kStream;
  if (forced == ASD_PATH_SMALL && small_ok) return Path::kSmall;
  if (bytes >= kTmaMinBytes) return Path::kTma;
  return small_ok ? Path::kSmall : Path::kStream;
}

template <typename T, bool kStrict>
int launch(VerifyParams& p, cudaStream_t stream) {
  const long long request_bytes = static_cast<long long>(p.K + 1) * p.V * static_cast<long long>(sizeof(T));
  const LaunchOptions opt = launch_options();
  const Path path = choose_path(opt.path, p.total * static_cast<long long>(sizeof(T)), request_bytes, p.K,
                                p.nblk == 1 && !p.partials);
  if (path == Path::kTma) return launch_tma<T, kStrict>(p, opt, stream);
  constexpr int VN = Elem<T>::kVec;
  const uintptr_t addr = reinterpret_cast<uintptr_t>(p.logits);
  if (addr % sizeof(T) != 0) return ASD_ERR_ALIGN;
  long long head = static_cast<long long>(((16 - addr % 16) % 16) / sizeof(T));
  if (head > p.total) head = p.total;
  if (path == Path::kSmall) {
    p.head = head;
    p.per_warp = 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.B));
    cfg.blockDim = dim3(kSmallThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    if (opt.pdl) {
      cfg.attrs = attr;
      cfg.numAttrs = 1;
    }
    if (cudaLaunchKernelEx(&cfg, verify_small_kernel<T, kStrict>, p) != cudaSuccess) return ASD_ERR_CUDA;
    return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
  }
  const long long rest = p.total - head;
  int max_warps = 0;
  const int rc = resident_warps<T, kStrict>(&max_warps);
  if (rc != ASD_OK) return rc;
  long long nw = (rest + kMinElemsPerWarp - 1) / kMinElemsPerWarp;
  if (nw > max_warps) nw = max_warps;
  if (nw < 1) nw = 1;
  long long per_warp = (rest + nw - 1) / nw;
  per_warp = (per_warp + VN - 1) / VN * VN;
  if (per_warp < VN) per_warp = VN;
  nw = (rest + per_warp - 1) / per_warp;
  if (nw < 1) nw = 1;
  p.head = head;
  p.per_warp = per_warp;
  const long long blocks = (nw + kWarpsPerBlock - 1) / kWarpsPerBlock;
  verify_kernel<T, kStrict><<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(p);
  return cudaGetLastError() == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

int verify_common(bool strict, const void* logits, int dtype, int B, int K, int V,
                  const int32_t* draft, asd_ledger* ledger, float gate, int cap,
                  int32_t* accepted_len, int32_t* committed, int32_t* recovery,
                  int32_t* row_argmax, float* row_regret, int32_t* status, void* workspace,
                  size_t workspace_bytes, cudaStream_t stream, int nblk = 1, int v_offset = 0,
                  int v_total = 0, asd_partial* partials = nullptr) {
  const bool resident = (dtype & ASD_RESIDENT_INPUTS) != 0;
  dtype = dtype_code(dtype);
  int rc = check_shape(B, K, V, dtype);
  if (rc != ASD_OK) return rc;
  if (nblk < 0 || (nblk > 0 && B > INT32_MAX / nblk)) return ASD_ERR_SHAPE;
  if (B == 0 || nblk == 0) return ASD_OK;
  if (!logits || !workspace) return ASD_ERR_NULL;
  if (!partials && (!accepted_len || !committed || !recovery)) return ASD_ERR_NULL;
  if (K > 0 && !draft) return ASD_ERR_NULL;
  if (!strict && !partials) {
    if (!ledger) return ASD_ERR_NULL;
    if (gate != gate || gate < 0.0f || cap < 0) return ASD_ERR_CONTROL;
  }
  const WorkspaceLayout l = layout_for(nblk * B, K);
  if (workspace_bytes < l.total) return ASD_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0) return ASD_ERR_ALIGN;
  char* ws = static_cast<char*>(workspace);

  VerifyParams p = {};
  p.logits = logits;
  p.B = B;
  p.K = K;
  p.V = V;
  p.nblk = nblk;
  p.v_offset = v_offset;
  p.v_total = v_total > 0 ? v_total : V;
  p.partials = partials;
  p.total = static_cast<long long>(nblk) * B * (K + 1) * V;
  p.head = 0;
  p.per_warp = 0;
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
  p.row_top = nullptr;
  p.resident = resident ? 1 : 0;

  if (dtype == ASD_F32)
    return strict ? launch<float, true>(p, stream) : launch<float, false>(p, stream);
  return strict ? launch<__nv_bfloat16, true>(p, stream) : launch<__nv_bfloat16, false>(p, stream);
}

}  // namespace

extern "C" {

int asd_workspace_size(int B, int K, int V, int dtype, size_t* bytes) {
  if (!bytes) return ASD_ERR_NULL;
  const int rc = check_shape(B, K, V, dtype);
  if (rc != ASD_OK) return rc;
  *bytes = layout_for(B, K).total;
  return ASD_OK;
}

int asd_workspace_error(const void* workspace, int* error, asd_stream_t stream) {
  if (!workspace || !error) return ASD_ERR_NULL;
  unsigned int word = 0;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&word, workspace, sizeof word, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return ASD_ERR_CUDA;
  *error = static_cast<int>(word);
  return ASD_OK;
}

int asd_workspace_init(void* workspace, size_t bytes, asd_stream_t stream) {
  if (!workspace) return ASD_ERR_NULL;
  return cudaMemsetAsync(workspace, 0, bytes, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? ASD_OK
             : ASD_ERR_CUDA;
}

int asd_verify(const void* logits, int dtype, int B, int K, int V, const int32_t* draft,
               asd_ledger* ledger, float gate, int cap, int32_t* accepted_len,
               int32_t* committed, int32_t* recovery, int32_t* row_argmax, float* row_regret,
               int32_t* status, void* workspace, size_t workspace_bytes, asd_stream_t stream) {
  return verify_common(false, logits, dtype, B, K, V, draft, ledger, gate, cap, accepted_len,
                       committed, recovery, row_argmax, row_regret, status, workspace,
                       workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int asd_verify_strict(const void* logits, int dtype, int B, int K, int V, const int32_t* draft,
                      int32_t* accepted_len, int32_t* committed, int32_t* recovery,
                      int32_t* row_argmax, float* row_regret, int32_t* status, void* workspace,
                      size_t workspace_bytes, asd_stream_t stream) {
  return verify_common(true, logits, dtype, B, K, V, draft, nullptr, 0.0f, 0, accepted_len,
                       committed, recovery, row_argmax, row_regret, status, workspace,
                       workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int asd_host_alias(const void* host, void** device) {
  if (!host || !device) return ASD_ERR_NULL;
  void* alias = nullptr;
  if (cudaHostGetDevicePointer(&alias, const_cast<void*>(host), 0) != cudaSuccess || !alias) {
    cudaGetLastError();  // clear the sticky-free error this query leaves behind
    return ASD_ERR_ALIGN;
  }
  *device = alias;
  return ASD_OK;
}

int asd_verify_launches(int B, int K, int V, int dtype, int* launches) {
  if (!launches) return ASD_ERR_NULL;
  const int rc = check_shape(B, K, V, dtype);
  if (rc != ASD_OK) return rc;
  const long long request_bytes = static_cast<long long>(K + 1) * V * (dtype_code(dtype) == ASD_BF16 ? 2 : 4);
  const LaunchOptions opt = launch_options();
  const Path path = choose_path(opt.path, request_bytes * B, request_bytes, K, true);
  *launches = B == 0 ? 0 : (path == Path::kTma && opt.split ? 2 : 1);
  return ASD_OK;
}

int asd_set_launch_options(const asd_launch_options* options) {
  if (!options) {
    g_path.store(ASD_PATH_AUTO);
    g_flags.store(0);
    return ASD_OK;
  }
  if (options->path < ASD_PATH_AUTO || options->path > ASD_PATH_TMA) return ASD_ERR_CONTROL;
  g_path.store(options->path);
  g_flags.store((options->fused_select ? 1 : 0) | (options->no_pdl ? 2 : 0));
  return ASD_OK;
}

int asd_get_launch_options(asd_launch_options* options) {
  if (!options) return ASD_ERR_NULL;
  const LaunchOptions o = launch_options();
  options->path = o.path;
  options->fused_select = o.split ? 0 : 1;
  options->no_pdl = o.pdl ? 0 : 1;
  return ASD_OK;
}

int asd_blocks_workspace_size(int nblk, int B, int K, int V, int dtype, size_t* bytes) {
  if (!bytes) return ASD_ERR_NULL;
  const int rc = check_shape(B, K, V, dtype);
  if (rc != ASD_OK) return rc;
  if (nblk < 0 || (nblk > 0 && B > INT32_MAX / nblk)) return ASD_ERR_SHAPE;
  *bytes = layout_for(nblk * B, K).total;
  return ASD_OK;
}

int asd_verify_blocks(const void* logits, int dtype, int nblk, int B, int K, int V, const int32_t* draft,
                      asd_ledger* ledger, float gate, int cap, int32_t* accepted_len, int32_t* committed,
                      int32_t* recovery, int32_t* row_argmax, float* row_regret, int32_t* status,
                      void* workspace, size_t workspace_bytes, asd_stream_t stream) {
  return verify_common(false, logits, dtype, B, K, V, draft, ledger, gate, cap, accepted_len, committed,
                       recovery, row_argmax, row_regret, status, workspace, workspace_bytes,
                       reinterpret_cast<cudaStream_t>(stream), nblk);
}

int asd_shard_partials(const void* logits, int dtype, int B, int K, int Vs, int v_offset, int V,
                       const int32_t* draft, asd_partial* partials, void* workspace, size_t workspace_bytes,
                       asd_stream_t stream) {
  if (!partials) return ASD_ERR_NULL;
  if (v_offset < 0 || Vs < 1 || V < 1 || static_cast<long long>(v_offset) + Vs > V) return ASD_ERR_SHAPE;
  return verify_common(true, logits, dtype, B, K, Vs, draft, nullptr, 0.0f, 0, nullptr, nullptr, nullptr,
                       nullptr, nullptr, nullptr, workspace, workspace_bytes,
                       reinterpret_cast<cudaStream_t>(stream), 1, v_offset, V, partials);
}

const char* asd_status_string(int code) {
  switch (code) {
    case ASD_OK: return "ok";
    case ASD_ERR_NULL: return "a required pointer is NULL";
    case ASD_ERR_SHAPE: return "invalid shape (need B >= 0, 0 <= K <= 31, V >= 1, valid H)";
    case ASD_ERR_DTYPE: return "unknown dtype code";
    case ASD_ERR_CONTROL: return "invalid control (need gate >= 0 and not NaN, cap >= 0)";
    case ASD_ERR_WORKSPACE: return "workspace smaller than the size query requires";
    case ASD_ERR_ALIGN: return "pointer misaligned";
    case ASD_ERR_CUDA: return "CUDA call failed";
    case ASD_ERR_DEVICE: return "the current device cannot run this kernel";
    case ASD_ERR_TIMEOUT: return "a kernel gave up waiting on its own pipeline (outputs incomplete)";
    case ASD_ERR_SCRATCH_LIMIT:
      return "problem too large for the built-in scratch of asd_verify_noalloc (use asd_verify)";
    default: return "unknown status code";
  }
}

}  // extern "C"

// ---------------------------------------------------------------- allocation-free entry point
//
// asd_verify_noalloc: asd_verify for callers that may not allocate device
// memory at call time (a serving loop with a fixed device-memory budget, a
// plug-in whose host framework owns every device allocation, a latency-bound
// path where cudaMalloc/cudaFree could synchronise the device). Its workspace
// is this file's fixed device array instead of caller memory.

namespace {

// The scratch: every GPU that loads the library holds these bytes until exit.
static __device__ __align__(256) unsigned char g_noalloc_scratch[ASD_NOALLOC_SCRATCH_BYTES];

// Device address of g_noalloc_scratch on each device, looked up on the first
// call made with that device current. In host code the symbol itself is only a
// host-side stand-in: a kernel must be given the looked-up device address.
int noalloc_scratch(void** out) {
  constexpr int kMaxDevices = 64;
  static void* addr[kMaxDevices] = {nullptr};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return ASD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return ASD_ERR_DEVICE;
  std::lock_guard<std::mutex> g(mu);
  if (!addr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return ASD_ERR_CUDA;
    addr[dev] = ptr;
  }
  *out = addr[dev];
  return ASD_OK;
}

}  // namespace

extern "C" int asd_verify_noalloc(const void* logits, int dtype, int B, int K, int V,
                                  const int32_t* draft, asd_ledger* ledger, float gate, int cap,
                                  int32_t* accepted_len, int32_t* committed, int32_t* recovery,
                                  int32_t* row_argmax, float* row_regret, int32_t* status,
                                  asd_stream_t stream) {
  int rc = check_shape(B, K, V, dtype);
  if (rc != ASD_OK) return rc;
  const size_t need = layout_for(B, K).total;
  if (need > static_cast<size_t>(ASD_NOALLOC_SCRATCH_BYTES)) return ASD_ERR_SCRATCH_LIMIT;
  if (B == 0) return ASD_OK;
  void* scratch = nullptr;
  rc = noalloc_scratch(&scratch);
  if (rc != ASD_OK) return rc;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // The array keeps whatever the previous call left; the kernels need the part
  // they use to start at zero.
  if (cudaMemsetAsync(scratch, 0, need, s) != cudaSuccess) return ASD_ERR_CUDA;
  return verify_common(false, logits, dtype, B, K, V, draft, ledger, gate, cap, accepted_len,
                       committed, recovery, row_argmax, row_regret, status, scratch, need, s);
}
