// libasd: verifier of Approximate Speculative Decoding (arXiv 2608.03447) for
// GB300 (sm_103a). Logit-streaming path: asd_verify / asd_verify_strict.
//
// One launch does the whole step:
//   stage 1  row reduction (Eq. 1, Eq. 3). The [B, K+1, V] logits are treated
//            as one flat array and cut into equal, 16-byte aligned ranges, one
//            per warp, so every SM streams the same number of bytes whatever
//            B, K and V are. A warp walks its range row segment by row
//            segment with 128-bit streaming loads, keeps a per-lane running
//            maximum (NaN-propagating, so a NaN cannot hide), and reduces the
//            segment to one 64-bit key (order-preserving fp32 bits, then the
//            inverted vocabulary index) that one atomicMax merges into the
//            row's slot: the largest key is the largest logit at the lowest
//            index, whatever order the segments finish in. The segment that
//            holds the draft token also records z_j(x_j).
//   stage 2  selection (Eq. 5-13, Alg. 1). Each warp adds the element count
//            it finished to its request's counter; the warp that completes a
//            request runs the request's selection with lane j owning target
//            row j, and resets the request's workspace slots to zero, so that
//            the whole workspace is zero again after every call (whatever
//            shape the next call has).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "asd.h"

namespace {

constexpr int kThreads = 256;
constexpr int kWarpsPerBlock = kThreads / 32;
constexpr int kUnroll = 4;                  // 128-bit loads in flight per lane
constexpr long long kMinElemsPerWarp = 2048;
constexpr unsigned kFull = 0xffffffffu;

struct VerifyParams {
  const void* logits;
  int B, K, V;
  long long total;     // B * (K+1) * V elements
  long long head;      // elements before the first 16-byte boundary
  long long per_warp;  // elements per warp after the head (multiple of the vector width)
  const int32_t* draft;
  asd_ledger* ledger;
  float gate;
  int cap;
  int32_t* accepted_len;
  int32_t* committed;
  int32_t* recovery;
  int32_t* row_argmax;
  float* row_regret;
  int32_t* status;
  unsigned long long* row_key;  // [B*(K+1)] running (value, index) key, zero between calls
  float* draft_logit;           // [B*(K+1)] z_j(x_j), written by the segment holding x_j
  unsigned long long* done;     // [B] elements finished, zero between calls
  unsigned int* flags;          // [B] ASD_STATUS_NAN_LOGIT bits, zero between calls
};

// ---------------------------------------------------------------- element access

template <typename T> struct Elem;
template <> struct Elem<float> {
  static constexpr int kVec = 4;  // elements per 128-bit vector
  static __device__ __forceinline__ float load(const float* p, long long i) { return __ldg(p + i); }
  static __device__ __forceinline__ float lane(const uint4& v, int t) {
    const uint32_t w = t == 0 ? v.x : t == 1 ? v.y : t == 2 ? v.z : v.w;
    return __uint_as_float(w);
  }
};
template <> struct Elem<__nv_bfloat16> {
  static constexpr int kVec = 8;
  static __device__ __forceinline__ float load(const __nv_bfloat16* p, long long i) {
    const unsigned short bits = __ldg(reinterpret_cast<const unsigned short*>(p) + i);
    return __uint_as_float(static_cast<uint32_t>(bits) << 16);  // bf16 -> fp32 is exact
  }
  static __device__ __forceinline__ float lane(const uint4& v, int t) {
    const int q = t >> 1;
    const uint32_t w = q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w;
    return __uint_as_float((t & 1) ? (w & 0xffff0000u) : (w << 16));
  }
};

__device__ __forceinline__ uint4 load_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// max that returns NaN when either input is NaN
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float d;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
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

// ---------------------------------------------------------------- (value, index) keys

// Order-preserving map of fp32 onto uint32 with -0 folded onto +0, so that the
// two zeros compare equal as IEEE comparison has them.
__device__ __forceinline__ uint32_t ordered_bits(float v) {
  uint32_t u = __float_as_uint(v);
  if ((u << 1) == 0) u = 0;  // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float ordered_value(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}

// Larger key = larger value, then smaller index.
__device__ __forceinline__ unsigned long long make_key(float v, uint32_t index) {
  return (static_cast<unsigned long long>(ordered_bits(v)) << 32) | (0xffffffffu - index);
}

__device__ __forceinline__ unsigned long long warp_max_key(unsigned long long k) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const unsigned long long o = __shfl_xor_sync(kFull, k, off);
    k = o > k ? o : k;
  }
  return k;
}

// ---------------------------------------------------------------- stage 1: one row segment

// Reduces elements [s0, s1) of one row (which starts at flat index row0) to a
// key; every lane returns the warp's key. Sets *nan when a NaN was seen.
template <typename T>
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
    for (; k + 32 * (kUnroll - 1) < nvec; k += 32 * kUnroll) {
      uint4 v[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) v[u] = load_stream(vp + k + 32 * u);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
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

// ---------------------------------------------------------------- stage 2: selection

__device__ __forceinline__ bool ledger_invalid(float budget, float spent) {
  return budget != budget || spent != spent || budget < 0.0f || spent < 0.0f || spent > budget;
}

template <typename T, bool kStrict>
__device__ void select_request(const VerifyParams& p, int b, int lane) {
  const int K = p.K, K1 = p.K + 1;
  const long long row = static_cast<long long>(b) * K1 + lane;
  const T* z = static_cast<const T*>(p.logits);

  unsigned long long key = 0;
  int x = -1;
  float zx = 0.0f;
  if (lane < K1) key = atomicExch(&p.row_key[row], 0ull);
  if (lane < K) {
    x = p.draft[static_cast<long long>(b) * K + lane];
    zx = __ldcg(&p.draft_logit[row]);
    p.draft_logit[row] = 0.0f;  // the whole workspace is zero again after every call
  }
  unsigned flags = 0;
  float budget = 0.0f, spent = 0.0f;
  if (lane == 0) {
    flags = atomicExch(&p.flags[b], 0u);
    if (!kStrict) {
      budget = p.ledger[b].budget;
      spent = p.ledger[b].spent;
    }
  }
  flags = __shfl_sync(kFull, flags, 0);
  budget = __shfl_sync(kFull, budget, 0);
  spent = __shfl_sync(kFull, spent, 0);

  const int y = key == 0 ? 0 : static_cast<int>(0xffffffffu - static_cast<uint32_t>(key));
  const bool valid_x = lane < K && x >= 0 && x < p.V;
  if (__any_sync(kFull, lane < K && !valid_x)) flags |= ASD_STATUS_DRAFT_RANGE;

  // Eq. 3: r_j = z_j(y*_j) - z_j(x_j). The key holds the maximum exactly, except
  // that it folds -0 onto +0; a zero maximum is re-read to keep its sign.
  float r = 0.0f;
  if (lane < K) {
    if (valid_x) {
      float top = ordered_value(static_cast<uint32_t>(key >> 32));
      if (top == 0.0f) top = Elem<T>::load(z, row * p.V + y);
      r = __fsub_rn(top, zx);
    } else {
      r = __int_as_float(0x7fc00000);
    }
  }
  const bool d = lane < K && x != y;  // Eq. 5
  const unsigned dmask = __ballot_sync(kFull, d);
  if (!kStrict && ledger_invalid(budget, spent)) flags |= ASD_STATUS_BAD_LEDGER;

  int a;
  bool write_ledger = false;
  float new_spent = spent;
  if (flags) {
    a = 0;
  } else if (kStrict || budget == 0.0f) {
    a = dmask ? __ffs(dmask) - 1 : K;  // Eq. 2; Alg. 1's zero-budget dispatch
  } else {
    // Eq. 8-12 walked left to right; every lane runs the same loop
    float C = 0.0f;
    int N = 0;
    a = K;
    for (int j = 0; j < K; ++j) {
      const float rj = __shfl_sync(kFull, r, j);
      if (!((dmask >> j) & 1u)) continue;
      const float q = static_cast<float>(K - j);            // Eq. 6
      const float C_next = __fadd_rn(C, rj);                // Eq. 8
      const int N_next = N + 1;
      const bool ok = __fdiv_rn(rj, q) <= p.gate            // Eq. 7 / 11
                      && __fadd_rn(spent, C_next) <= budget  // Eq. 9 as fl(s + C) <= B
                      && N_next <= p.cap;                    // Eq. 10
      if (!ok) {
        a = j;
        break;
      }
      C = C_next;
      N = N_next;
    }
    new_spent = __fadd_rn(spent, C);  // Eq. 13
    write_ledger = true;
  }
  const int ya = __shfl_sync(kFull, y, a);

  if (lane < K1) {
    if (p.row_argmax) p.row_argmax[row] = y;
    p.committed[row] = lane < a ? x : (lane == a ? ya : -1);
  }
  if (lane < K && p.row_regret) p.row_regret[static_cast<long long>(b) * K + lane] = r;
  if (lane == 0) {
    p.accepted_len[b] = a;
    p.recovery[b] = ya;
    if (p.status) p.status[b] = static_cast<int32_t>(flags);
    if (write_ledger) p.ledger[b].spent = new_spent;
    p.done[b] = 0ull;
  }
}

// ---------------------------------------------------------------- the fused kernel

template <typename T, bool kStrict>
__global__ void __launch_bounds__(kThreads) verify_kernel(const VerifyParams p) {
  const int lane = threadIdx.x & 31;
  const long long warp = static_cast<long long>(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  const long long lo = warp == 0 ? 0 : p.head + warp * p.per_warp;
  long long hi = p.head + (warp + 1) * p.per_warp;
  hi = hi < p.total ? hi : p.total;
  if (lo >= hi) return;

  const T* z = static_cast<const T*>(p.logits);
  const int V = p.V, K = p.K, K1 = p.K + 1;
  const unsigned long long request_elems = static_cast<unsigned long long>(K1) * V;

  long long row = lo / V;
  int pending_b = static_cast<int>(row / K1);
  unsigned long long pending_n = 0;

  for (long long s0 = lo; s0 < hi; ++row) {
    const long long row0 = row * V;
    const long long s1 = hi < row0 + V ? hi : row0 + V;
    const int b = static_cast<int>(row / K1);
    const int j = static_cast<int>(row - static_cast<long long>(b) * K1);
    int x = -1;
    if (j < K) x = __ldg(p.draft + static_cast<long long>(b) * K + j);  // issued before the stream

    if (b != pending_b) {  // finished this warp's share of request pending_b
      bool last = false;
      if (lane == 0) {
        __threadfence();
        const unsigned long long old = atomicAdd(&p.done[pending_b], pending_n);
        last = old + pending_n == request_elems;
      }
      if (__shfl_sync(kFull, last, 0)) {
        __threadfence();
        select_request<T, kStrict>(p, pending_b, lane);
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
    const unsigned long long old = atomicAdd(&p.done[pending_b], pending_n);
    last = old + pending_n == request_elems;
  }
  if (__shfl_sync(kFull, last, 0)) {
    __threadfence();
    select_request<T, kStrict>(p, pending_b, lane);
  }
}

// ---------------------------------------------------------------- host side

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

struct WorkspaceLayout {
  size_t row_key, draft_logit, done, flags, total;
};

WorkspaceLayout layout_for(int B, int K) {
  const size_t R = static_cast<size_t>(B) * (K + 1);
  WorkspaceLayout l;
  l.row_key = 0;
  l.draft_logit = align_up(l.row_key + 8 * R, 256);
  l.done = align_up(l.draft_logit + 4 * R, 256);
  l.flags = align_up(l.done + 8 * static_cast<size_t>(B), 256);
  l.total = align_up(l.flags + 4 * static_cast<size_t>(B), 256);
  if (l.total == 0) l.total = 256;
  return l;
}

int check_shape(int B, int K, int V, int dtype) {
  if (dtype != ASD_F32 && dtype != ASD_BF16) return ASD_ERR_DTYPE;
  if (B < 0 || K < 0 || K > ASD_MAX_K || V < 1) return ASD_ERR_SHAPE;
  return ASD_OK;
}

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

template <typename T, bool kStrict>
int launch(VerifyParams& p, cudaStream_t stream) {
  constexpr int VN = Elem<T>::kVec;
  const uintptr_t addr = reinterpret_cast<uintptr_t>(p.logits);
  if (addr % sizeof(T) != 0) return ASD_ERR_ALIGN;
  long long head = static_cast<long long>(((16 - addr % 16) % 16) / sizeof(T));
  if (head > p.total) head = p.total;
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
                  size_t workspace_bytes, cudaStream_t stream) {
  int rc = check_shape(B, K, V, dtype);
  if (rc != ASD_OK) return rc;
  if (B == 0) return ASD_OK;
  if (!logits || !accepted_len || !committed || !recovery || !workspace) return ASD_ERR_NULL;
  if (K > 0 && !draft) return ASD_ERR_NULL;
  if (!strict) {
    if (!ledger) return ASD_ERR_NULL;
    if (gate != gate || gate < 0.0f || cap < 0) return ASD_ERR_CONTROL;
  }
  const WorkspaceLayout l = layout_for(B, K);
  if (workspace_bytes < l.total) return ASD_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0) return ASD_ERR_ALIGN;
  char* ws = static_cast<char*>(workspace);

  VerifyParams p;
  p.logits = logits;
  p.B = B;
  p.K = K;
  p.V = V;
  p.total = static_cast<long long>(B) * (K + 1) * V;
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
    default: return "unknown status code";
  }
}

}  // extern "C"
