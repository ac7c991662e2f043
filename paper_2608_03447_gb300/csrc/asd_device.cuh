// Device pieces shared by the verify kernels (asd_verify.cu) and the fused
// LM-head kernel (asd_lmhead.cu): parameters, element access, order-preserving
// (value, index) keys, the per-request selection (Alg. 1), the workspace
// layout, and the mbarrier / programmatic-dependent-launch helpers.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "asd.h"

namespace asd_detail {

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
  unsigned int* flags;          // [nblk*B] ASD_STATUS_NAN_LOGIT bits, zero between calls
  unsigned int* error;          // sticky: ASD_ERR_TIMEOUT when a pipeline wait gave up
  float* row_top;               // [B*(K+1)] z_j(y*_j), or NULL (written by the fused LM-head path)
  int nblk;                     // sequential blocks of the same B requests (block i = requests i*B ..)
  int v_offset;                 // vocabulary shard: global index of this shard's entry 0 (else 0)
  int v_total;                  // vocabulary shard: entries of the whole vocabulary (else V)
  asd_partial* partials;        // vocabulary shard: [B*(K+1)] outputs instead of the selection
  int resident;                 // ASD_RESIDENT_INPUTS: logits and drafts may be read before the
                                // previous launch on the stream has completed
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

// max that returns NaN when either input is NaN
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float d;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
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

// ---------------------------------------------------------------- stage 2: selection

__device__ __forceinline__ bool ledger_invalid(float budget, float spent) {
  return budget != budget || spent != spent || budget < 0.0f || spent < 0.0f || spent > budget;
}

// What one block's selection reads from the workspace for one request
// (lane j: target row j); loaded ahead of use.
struct BlockInputs {
  unsigned long long key;  // row j's (value, index) key
  int x;                   // draft token j (lanes < K)
  float zx;                // z_j(x_j) (lanes < K)
  unsigned flags;          // the block's status bits (every lane)
  float top;               // z_j(y*_j) as the key holds it (a zero may have lost its sign)
  bool top_exact;          // top is the stored value itself (sign of zero included)
};

// kWithError: also test the workspace's error word (ASD_STATUS_INCOMPLETE, see
// workspace_failed) in the same round trip as the block's loads.
template <bool kWithError = false>
__device__ __forceinline__ BlockInputs load_block(const VerifyParams& p, long long vb, int lane) {
  const int K = p.K, K1 = p.K + 1;
  const long long row = vb * K1 + lane;
  BlockInputs in;
  in.key = 0;
  in.x = -1;
  in.zx = 0.0f;
  in.flags = 0;
  if (lane < K1) {
    in.key = __ldcg(&p.row_key[row]);
    p.row_key[row] = 0ull;  // the whole workspace is zero again after every call
  }
  if (lane < K) {
    in.x = p.draft[vb * K + lane];
    in.zx = __ldcg(&p.draft_logit[row]);
    p.draft_logit[row] = 0.0f;
  }
  if (lane == 0) {
    const unsigned f = __ldcg(&p.flags[vb]);
    const unsigned e = (kWithError && p.error) ? __ldcg(p.error) : 0u;
    p.flags[vb] = 0u;
    in.flags = f | (e ? ASD_STATUS_INCOMPLETE : 0u);
  }
  in.flags = __shfl_sync(kFull, in.flags, 0);
  in.top = ordered_value(static_cast<uint32_t>(in.key >> 32));
  in.top_exact = false;
  return in;
}

// Alg. 1 for block vb of one request, given the request's ledger (budget,
// spent): writes the block's outputs and advances `spent` (Eq. 13) unless the
// block is strict, zero-budget or flagged.
template <typename T, bool kStrict>
__device__ __forceinline__ void select_block(const VerifyParams& p, long long vb, const BlockInputs& in,
                                             float budget, float& spent, bool& wrote, int lane) {
  const int K = p.K, K1 = p.K + 1;
  const long long row = vb * K1 + lane;
  const T* z = static_cast<const T*>(p.logits);
  unsigned flags = in.flags;
  const int x = in.x;

  const int y = in.key == 0 ? 0 : static_cast<int>(0xffffffffu - static_cast<uint32_t>(in.key));
  const bool valid_x = lane < K && x >= 0 && x < p.V;
  if (__any_sync(kFull, lane < K && !valid_x)) flags |= ASD_STATUS_DRAFT_RANGE;

  // Eq. 3: r_j = z_j(y*_j) - z_j(x_j). The key holds the maximum exactly, except
  // that it folds -0 onto +0; a zero maximum is re-read to keep its sign (when
  // the logits are in memory: the fused LM-head path passes none).
  const float top = in.top;
  float r = 0.0f;
  if (lane < K) {
    if (valid_x) {
      float t = top;
      if (t == 0.0f && !in.top_exact && z) t = Elem<T>::load(z, row * p.V + y);
      r = __fsub_rn(t, in.zx);
    } else {
      r = __int_as_float(0x7fc00000);
    }
  }
  const bool d = lane < K && x != y;  // Eq. 5
  const unsigned dmask = __ballot_sync(kFull, d);
  if (!kStrict && ledger_invalid(budget, spent)) flags |= ASD_STATUS_BAD_LEDGER;

  int a;
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
    spent = __fadd_rn(spent, C);  // Eq. 13
    wrote = true;
  }
  const int ya = __shfl_sync(kFull, y, a);

  if (lane < K1) {
    if (p.row_argmax) p.row_argmax[row] = y;
    p.committed[row] = lane < a ? x : (lane == a ? ya : -1);
    if (p.row_top) p.row_top[row] = top;
  }
  if (lane < K && p.row_regret) p.row_regret[vb * K + lane] = r;
  if (lane == 0) {
    p.accepted_len[vb] = a;
    p.recovery[vb] = ya;
    if (p.status) p.status[vb] = static_cast<int32_t>(flags);
  }
}

// The selection of request b over its p.nblk blocks in order (block i is the
// virtual request i * B + b): the ledger is read once, carried in registers
// from block to block, and written once. Runs in one warp.
// Vocabulary-shard mode: instead of selecting, hand each row's reduction of
// this shard to the combine step (global index, exact top, draft logit).
// ASD_STATUS_INCOMPLETE when the workspace's error word is set: a kernel that
// used this workspace gave up waiting on its copy pipeline, so row results may
// be missing (every lane gets the same answer). The partials pass folds the
// same test into its block's loads (load_block<true>: 0.5 us less per shard
// call); the selection keeps it separate, which measured 0.1 us faster there.
__device__ __forceinline__ unsigned workspace_failed(const VerifyParams& p, int lane) {
  unsigned err = 0;
  if (lane == 0 && p.error) err = __ldcg(p.error);
  return __shfl_sync(kFull, err, 0) ? ASD_STATUS_INCOMPLETE : 0u;
}

template <typename T>
__device__ void emit_partials(const VerifyParams& p, int b, int lane) {
  const int K = p.K, K1 = p.K + 1;
  const T* z = static_cast<const T*>(p.logits);
  BlockInputs in = load_block<true>(p, b, lane);
  if (lane < K1) {
    const long long row = static_cast<long long>(b) * K1 + lane;
    const uint32_t local = 0xffffffffu - static_cast<uint32_t>(in.key);
    float top = in.top;
    if (top == 0.0f && in.key && z) top = Elem<T>::load(z, row * p.V + local);  // keep the sign of a zero
    const int xl = lane < K ? in.x - p.v_offset : -1;
    asd_partial out;
    out.key = in.key ? ((in.key & 0xffffffff00000000ull) |
                        (0xffffffffu - (local + static_cast<uint32_t>(p.v_offset))))
                     : 0ull;
    out.top = top;
    out.draft_logit = (xl >= 0 && xl < p.V) ? in.zx : -INFINITY;
    out.flags = in.flags;
    out.reserved = 0u;
    p.partials[row] = out;
  }
  if (lane == 0) p.done[b] = 0ull;
}

template <typename T, bool kStrict>
__device__ void select_request(const VerifyParams& p, int b, int lane) {
  if (p.partials) {
    emit_partials<T>(p, b, lane);
    return;
  }
  float budget = 0.0f, spent = 0.0f;
  if (!kStrict && lane == 0) {
    budget = p.ledger[b].budget;
    spent = p.ledger[b].spent;
  }
  budget = __shfl_sync(kFull, budget, 0);
  spent = __shfl_sync(kFull, spent, 0);
  const unsigned incomplete = workspace_failed(p, lane);
  bool wrote = false;
  BlockInputs cur = load_block(p, b, lane);
  for (int i = 0; i < p.nblk; ++i) {
    const long long vb = static_cast<long long>(i) * p.B + b;
    BlockInputs next = cur;
    if (i + 1 < p.nblk) next = load_block(p, vb + p.B, lane);  // in flight while this block is selected
    cur.flags |= incomplete;
    select_block<T, kStrict>(p, vb, cur, budget, spent, wrote, lane);
    cur = next;
  }
  if (lane == 0) {
    if (wrote) p.ledger[b].spent = spent;
    p.done[b] = 0ull;
  }
}

// ---------------------------------------------------------------- request completion

// Adds `pend` to request b's counter; the warp whose addition reaches
// request_total runs the request's selection. Out of line: it runs a few times
// per launch.
template <typename T, bool kStrict>
__device__ __noinline__ void finish_request(const VerifyParams& p, int b, unsigned long long pend,
                                            unsigned long long request_total, int lane) {
  bool last = false;
  if (lane == 0) {
    __threadfence();
    const unsigned long long old = atomicAdd(&p.done[b], pend);
    last = old + pend == request_total;
  }
  if (__shfl_sync(kFull, last, 0)) {
    __threadfence();
    select_request<T, kStrict>(p, b, lane);
  }
}

// ---------------------------------------------------------------- mbarriers, programmatic dependent launch

#ifndef ASD_TMA_POLL
#define ASD_TMA_POLL 0  // 0: mbarrier.try_wait (may suspend), 1: mbarrier.test_wait spin
#endif

constexpr unsigned long long kWaitLimitNs = 1000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void* ptr) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(ptr));
}
__device__ __forceinline__ void mbar_init(unsigned long long* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(unsigned long long* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(unsigned long long* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(unsigned long long* bar, uint32_t parity) {
  uint32_t done;
#if ASD_TMA_POLL
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
#else
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
#endif
  return done != 0;
}
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Waits for the phase with the given parity; false on timeout or when another
// warp of the CTA has given up.
__device__ inline bool mbar_wait(unsigned long long* bar, uint32_t parity, volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (unsigned it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0) {  // the clock and the abort flag are checked now and then
      if (*abort) return false;
      if (global_ns() - t0 > kWaitLimitNs) return false;
    }
  }
}
// Programmatic dependent launch: the next launch on the stream may start once
// every CTA of this one has signalled; it waits for this launch to complete
// (and its writes to be visible) before its first access to the workspace,
// the ledger or the outputs. Its logits stream in the meantime.
__device__ __forceinline__ void pdl_signal_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait_prerequisites() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---------------------------------------------------------------- workspace layout (host)

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Workspace: the error word first (fixed offset for asd_workspace_error), then
// the per-row and per-request slots.
struct WorkspaceLayout {
  size_t error, row_key, draft_logit, done, flags, total;
};

inline WorkspaceLayout layout_for(int B, int K) {
  const size_t R = static_cast<size_t>(B) * (K + 1);
  WorkspaceLayout l;
  l.error = 0;
  l.row_key = 256;
  l.draft_logit = align_up(l.row_key + 8 * R, 256);
  l.done = align_up(l.draft_logit + 4 * R, 256);
  l.flags = align_up(l.done + 8 * static_cast<size_t>(B), 256);
  l.total = align_up(l.flags + 4 * static_cast<size_t>(B), 256);
  return l;
}

// The storage type of a dtype argument (without ASD_RESIDENT_INPUTS).
inline int dtype_code(int dtype) { return dtype & ~ASD_RESIDENT_INPUTS; }

inline int check_shape(int B, int K, int V, int dtype) {
  dtype = dtype_code(dtype);
  if (dtype != ASD_F32 && dtype != ASD_BF16) return ASD_ERR_DTYPE;
  if (B < 0 || K < 0 || K > ASD_MAX_K || V < 1) return ASD_ERR_SHAPE;
  return ASD_OK;
}

}  // namespace asd_detail
