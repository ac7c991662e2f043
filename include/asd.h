/*
 * asd.h - C ABI of libasd, the GB300 (sm_103a) verifier of Approximate
 * Speculative Decoding (ASD, arXiv 2608.03447).
 *
 * One verifier step takes the target model's teacher-forced logits for a batch
 * of draft blocks and, per request, returns the accepted prefix length, the
 * committed tokens, the recovery (or bonus) token and the updated regret
 * ledger (Sec. 3.2-3.3, Alg. 1).
 *
 * Conventions shared by every entry point
 *   - Every array argument is DEVICE memory owned by the caller, contiguous,
 *     row-major. The library allocates nothing and keeps no per-call state
 *     outside the caller's workspace.
 *   - Calls are asynchronous and ordered on `stream` (a cudaStream_t; NULL is
 *     the legacy default stream). Nothing synchronises with the host.
 *   - Indices are 0-based: request b in [0, B), draft position j in [0, K)
 *     (the paper's i = j + 1), target row j in [0, K] (row K is the bonus row).
 *   - A return value other than ASD_OK means that nothing was launched, except
 *     ASD_ERR_CUDA, which reports a failed launch.
 *   - Per-request data errors never abort the call: they set bits of
 *     status[b] (ASD_STATUS_*). Such a request accepts nothing (a = 0), emits
 *     y*_0 as its recovery token and keeps its ledger; for a NaN logit the
 *     argmax is deterministic but unspecified.
 *   - A workspace serves one call at a time: two calls that share a workspace
 *     must be ordered on one stream (or otherwise serialised).
 */
#ifndef ASD_H
#define ASD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;
typedef struct CUstream_st* asd_stream_t; /* == cudaStream_t */

/* The persistent per-request ledger (B, s) of Sec. 3.2: the request's total
 * regret budget and the regret already spent in earlier rounds. budget = 0
 * selects exact strict greedy verification (Alg. 1); budget = +INFINITY is
 * allowed. Valid ledgers have 0 <= spent <= budget and no NaN. */
typedef struct {
  float budget;
  float spent;
} asd_ledger;

/* One vocabulary shard's reduction of one target row (asd_shard_partials):
 * what the tensor-parallel remark of Sec. 3.3 says the verifier needs from
 * each shard, with no logit buffer. */
typedef struct {
  uint64_t key;        /* order-preserving (top logit, GLOBAL vocabulary index): larger wins */
  float top;           /* the shard's top logit, exactly as stored (sign of zero kept) */
  float draft_logit;   /* z(x) if the row's draft token is in this shard, else -INFINITY */
  uint32_t flags;      /* ASD_STATUS_NAN_LOGIT if the shard saw a NaN in the row's request */
  uint32_t reserved;
} asd_partial;

/* Logit storage types. */
enum { ASD_F32 = 0, ASD_BF16 = 1 };

/* Flag ORed into the dtype argument of the verify entry points: the logits and
 * draft tokens are resident, i.e. no kernel that is still running or queued
 * ahead of this call on the stream writes them (they were written by work that
 * has completed, by a copy, or by the host). The row stage then starts
 * streaming them while the previous kernel on the stream finishes (programmatic
 * dependent launch), which overlaps consecutive calls. Without the flag the row
 * stage still launches early but reads nothing before the previous kernel has
 * completed and its writes are visible, so a producer kernel (such as the
 * model's LM head) may write the logits right before the call. Results are the
 * same either way; only the overlap differs. */
#define ASD_RESIDENT_INPUTS 0x100

/* Return codes. */
enum {
  ASD_OK = 0,
  ASD_ERR_NULL = 1,      /* a required pointer is NULL */
  ASD_ERR_SHAPE = 2,     /* B < 0, K < 0, K > 31, V < 1, or H invalid */
  ASD_ERR_DTYPE = 3,     /* unknown dtype code */
  ASD_ERR_CONTROL = 4,   /* gate < 0 or NaN, cap < 0 */
  ASD_ERR_WORKSPACE = 5, /* workspace smaller than the size query returns */
  ASD_ERR_ALIGN = 6,     /* pointer not aligned as documented */
  ASD_ERR_CUDA = 7,      /* a CUDA call failed (launch or device query) */
  ASD_ERR_DEVICE = 8,    /* the current device cannot run the kernel (not sm_103) */
  ASD_ERR_TIMEOUT = 9,   /* reported by asd_workspace_error: a kernel gave up waiting */
  ASD_ERR_SCRATCH_LIMIT = 10 /* asd_verify_noalloc: the problem needs more than its scratch */
};

/* Per-request status bits (status[b]). */
#define ASD_STATUS_DRAFT_RANGE 1u /* a draft id outside [0, V) */
#define ASD_STATUS_NAN_LOGIT 2u   /* a NaN among the request's K+1 logit rows */
#define ASD_STATUS_BAD_LEDGER 4u  /* budget < 0 or NaN, spent < 0 or NaN, spent > budget */
#define ASD_STATUS_OVERFLOW 8u    /* asd_commit: the token history has no room for the block */
#define ASD_STATUS_INCOMPLETE 16u /* the workspace's error word was set when the request was
                                   * selected (asd_workspace_error): a kernel gave up waiting on
                                   * its copy pipeline, so row results may be missing. Set for
                                   * every request of such a call until asd_workspace_init. */

/* Largest draft length: one warp lane per target row of a block. */
#define ASD_MAX_K 31

/* Bytes of workspace that asd_verify / asd_verify_strict need for (B, K, V,
 * dtype). Writes *bytes; returns ASD_ERR_SHAPE / ASD_ERR_DTYPE / ASD_ERR_NULL
 * on bad arguments. */
int asd_workspace_size(int B, int K, int V, int dtype, size_t* bytes);

/* Zero a workspace (cudaMemsetAsync on `stream`). Required once before the
 * first call that uses it; every verify call leaves the workspace zeroed again
 * when it completes, so it can be reused for any shape (and captured in a CUDA
 * graph) with no further initialisation. */
int asd_workspace_init(void* workspace, size_t bytes, asd_stream_t stream);

/* Read the workspace's sticky error word (synchronises `stream`): 0, or
 * ASD_ERR_TIMEOUT if a kernel that used this workspace gave up waiting on its
 * own copy pipeline (a bounded wait of about one second; it does not happen in
 * normal operation). After a non-zero word the outputs of that call are
 * incomplete and the workspace must be re-initialised with asd_workspace_init. */
int asd_workspace_error(const void* workspace, int* error, asd_stream_t stream);

/* Self-test of the failure detection above (the paper has no counterpart):
 * launches one CTA whose thread waits, with the same bounded mbarrier wait as
 * the pipeline kernels, on a barrier that nothing signals. After about one
 * second the wait gives up, the kernel writes ASD_ERR_TIMEOUT to the
 * workspace's error word and returns; nothing faults and the context stays
 * usable. `workspace` is any workspace of at least 4 bytes (16-byte aligned);
 * read the result with asd_workspace_error and re-initialise the workspace
 * before its next verify call. Returns ASD_ERR_NULL / ASD_ERR_WORKSPACE /
 * ASD_ERR_ALIGN on bad arguments, ASD_ERR_CUDA if the launch fails. */
int asd_selftest_wait_timeout(void* workspace, size_t workspace_bytes, asd_stream_t stream);

/*
 * ASD verification of B draft blocks (Eq. 1, 3, 5-13; Alg. 1).
 *
 * logits        [B, K+1, V], dtype ASD_F32 or ASD_BF16; row b*(K+1)+j holds
 *               z_{j+1}. Aligned to its element size; any further alignment
 *               is handled.
 * draft         [B, K] int32 draft tokens x (may be NULL when K = 0)
 * ledger        [B] in/out. spent is updated to s' = fl(s + C_a) (Eq. 13);
 *               left untouched when budget == 0 or the request is flagged.
 * gate          g of Eq. 7 (>= 0; +INFINITY disables the gate)
 * cap           M of Eq. 10 (>= 0; INT32_MAX disables the cap)
 * accepted_len  [B]       a = longest feasible prefix (Eq. 12)
 * committed     [B, K+1]  x_0..x_{a-1}, y*_a, then -1 padding
 * recovery      [B]       y*_a: the recovery token (a < K) or the bonus (a = K)
 * row_argmax    [B, K+1]  y*_j (lowest index on ties); may be NULL
 * row_regret    [B, K]    r_j = fl32(z_j(y*_j) - z_j(x_j)), NaN for an
 *                         out-of-range draft; may be NULL
 * status        [B]       ASD_STATUS_* bits; may be NULL
 * workspace     >= asd_workspace_size(...) bytes, 16-byte aligned, zeroed
 *               by asd_workspace_init before first use
 * dtype         ASD_F32 or ASD_BF16, optionally | ASD_RESIDENT_INPUTS (above)
 *
 * Arithmetic (all fp32, round to nearest): argmax by IEEE comparison
 * (-0 == +0), then per request, left to right over the mismatches d_j = 1:
 * C' = C + r_j; accept while r_j / (K - j) <= g, fl(s + C') <= budget and
 * N' <= M; a is the first position that fails (else K). budget == 0
 * dispatches to the strict rule (Eq. 2) and keeps the ledger.
 */
int asd_verify(const void* logits, int dtype, int B, int K, int V, const int32_t* draft,
               asd_ledger* ledger, float gate, int cap, int32_t* accepted_len,
               int32_t* committed, int32_t* recovery, int32_t* row_argmax, float* row_regret,
               int32_t* status, void* workspace, size_t workspace_bytes, asd_stream_t stream);

/*
 * Strict greedy verification (Eq. 2): a = the first j with x_j != y*_j (else
 * K); committed and recovery as in asd_verify (the bonus y*_K is appended when
 * a = K). No ledger. Same arguments, layouts and workspace as asd_verify.
 */
int asd_verify_strict(const void* logits, int dtype, int B, int K, int V, const int32_t* draft,
                      int32_t* accepted_len, int32_t* committed, int32_t* recovery,
                      int32_t* row_argmax, float* row_regret, int32_t* status, void* workspace,
                      size_t workspace_bytes, asd_stream_t stream);

/*
 * Fused LM-head + verify (Sec. 3.1 Eq. 1 with Sec. 3.3's remark that the
 * verifier needs only the top token, the top logit and the draft token's logit,
 * so no [T, V] logit buffer is needed). The logits z = h W^T are computed on
 * the tensor cores (bf16 inputs, fp32 accumulation) and reduced on chip; they
 * are never written to memory. The selection is then the one of asd_verify.
 *
 * hidden        [B*(K+1), H] bf16 (as uint16 bits or __nv_bfloat16): the
 *               target's final hidden state of every row of every block,
 *               16-byte aligned
 * weight        [V, H] bf16 LM-head weight, 16-byte aligned
 * H             hidden size, a multiple of 8 (rows must be 16-byte pitched)
 * row_top       [B, K+1] the top logit z_j(y*_j) of each row; may be NULL
 * everything else as in asd_verify; the workspace size comes from
 * asd_lmhead_workspace_size. Requires a Blackwell (sm_10x) device: other
 * devices get ASD_ERR_DEVICE.
 * Precision: the logits are fp32 sums of bf16 products in the tensor core's
 * order, so ties and near-ties (within about 1e-5 of the row's scale) may
 * resolve differently from an exact (fp64) evaluation; exact ties between
 * equal fp32 logits go to the lowest index, as in asd_verify.
 * Launch: clusters of two CTAs, one per SM of a pair, each with about 214 KB
 * of shared memory and all 512 tensor-memory columns of its SM, so a call
 * occupies the GPU's SM pairs while it runs.
 */
int asd_lmhead_workspace_size(int B, int K, int V, int H, size_t* bytes);
int asd_lmhead_verify(const void* hidden, const void* weight, int H, int B, int K, int V,
                      const int32_t* draft, asd_ledger* ledger, float gate, int cap,
                      int32_t* accepted_len, int32_t* committed, int32_t* recovery,
                      int32_t* row_argmax, float* row_regret, float* row_top, int32_t* status,
                      void* workspace, size_t workspace_bytes, asd_stream_t stream);

/*
 * The same tensor-core LM-head GEMM writing its fp32 logits [T, V] (row-major,
 * device memory) instead of reducing them: for callers that need the logits
 * themselves, and to check the GEMM against an exact evaluation. No workspace.
 */
int asd_lmhead_logits(const void* hidden, const void* weight, int H, int T, int V, float* logits,
                      asd_stream_t stream);

/* Bytes of the fixed device scratch that asd_verify_noalloc uses. */
#define ASD_NOALLOC_SCRATCH_BYTES (1u << 20)

/*
 * asd_verify without a caller workspace and without allocating anything: for
 * callers that may not allocate device memory when they verify (a serving loop
 * with a fixed device-memory budget, a plug-in whose host framework owns every
 * device allocation, a latency-bound path where cudaMalloc / cudaFree could
 * synchronise the device). The paper has no counterpart; it is an interface
 * convenience around the same computation as asd_verify, with the same
 * arguments minus the workspace and the same results.
 *
 * Scratch: a fixed ASD_NOALLOC_SCRATCH_BYTES array of device memory inside the
 * library, held by every GPU that loads it until the process exits. A call
 * whose asd_workspace_size(B, K, V, dtype) exceeds it returns
 * ASD_ERR_SCRATCH_LIMIT and launches nothing.
 * Set-up: the first call made with a given device current looks up the
 * array's device address (cudaGetSymbolAddress); make that first call outside
 * any stream capture. The address is kept for the life of the process:
 * cudaDeviceReset unloads the library's device code, so after it this entry
 * point must not be called again in that process.
 * Each call clears the part of the array it uses (cudaMemsetAsync on
 * `stream`, which also clears the array's error word) and then launches the
 * verify kernels. Every call on every stream shares the one array: calls that
 * can overlap on the GPU (different streams, no ordering between them) race
 * and give wrong results. Order them on one stream. Allocates nothing: no
 * cudaMalloc, cudaFree or allocating library call.
 * Failure report: the array's error word is not readable by the caller, so a
 * call whose kernels gave up waiting on their copy pipeline (the bounded wait
 * of asd_workspace_error) flags every request ASD_STATUS_INCOMPLETE in
 * status[b] instead (a = 0, ledger kept); pass a status array to see it.
 */
int asd_verify_noalloc(const void* logits, int dtype, int B, int K, int V, const int32_t* draft,
                       asd_ledger* ledger, float gate, int cap, int32_t* accepted_len,
                       int32_t* committed, int32_t* recovery, int32_t* row_argmax,
                       float* row_regret, int32_t* status, asd_stream_t stream);

/*
 * Several sequential draft blocks of the same B requests in one call: block i
 * of request b is verified with the ledger left by block i-1 (Sec. 3.2: the
 * ledger (B, s) persists across decoding rounds). The result is bit for bit
 * that of nblk asd_verify calls made in order, block 0 first.
 *
 * logits        [nblk, B, K+1, V]; draft [nblk, B, K]; ledger [B] in/out
 * accepted_len, recovery, status  [nblk, B]; committed, row_argmax [nblk, B, K+1];
 * row_regret    [nblk, B, K]
 * workspace     asd_blocks_workspace_size(nblk, B, K, V, dtype) bytes
 * The logits of all blocks stream in one pass; only each request's selection
 * runs block after block, with the ledger in registers.
 */
int asd_blocks_workspace_size(int nblk, int B, int K, int V, int dtype, size_t* bytes);
int asd_verify_blocks(const void* logits, int dtype, int nblk, int B, int K, int V,
                      const int32_t* draft, asd_ledger* ledger, float gate, int cap,
                      int32_t* accepted_len, int32_t* committed, int32_t* recovery,
                      int32_t* row_argmax, float* row_regret, int32_t* status, void* workspace,
                      size_t workspace_bytes, asd_stream_t stream);

/*
 * The verifier-side opportunity rate of Eq. 4 (Sec. 3.1), as counts added to
 * `counts` (device, uint64, accumulated over calls; zero it to start):
 *   counts[t * np + u] += #{ mismatch positions (x, i) with r_i <= tau[t],
 *                            i + p[u] <= K and x_l = y*_l for l = i+1 .. i+p[u] }
 *   counts[ntau * np]  += |M|, the number of mismatch positions
 * so Omega(tau[t], p[u]) = counts[t * np + u] / counts[ntau * np].
 * row_argmax [n, K+1], draft [n, K], row_regret [n, K]: asd_verify's row
 * outputs for n block-requests (device); status [n] or NULL (block-requests
 * with a non-zero status are skipped). tau [ntau] and p [np] are HOST arrays,
 * 1 <= ntau, np <= ASD_OPPORTUNITY_MAX; tau not NaN, p >= 0.
 */
#define ASD_OPPORTUNITY_MAX 16
int asd_opportunity(const int32_t* row_argmax, const int32_t* draft, const float* row_regret,
                    const int32_t* status, int n, int K, const float* tau, int ntau, const int32_t* p,
                    int np, unsigned long long* counts, asd_stream_t stream);

/*
 * Vocabulary-sharded verify (Sec. 3.3: under tensor parallelism the verifier
 * needs only the top token, the top logit and the draft token's logit, which
 * each vocabulary shard can reduce locally). Step 1 on every shard:
 *   asd_shard_partials: logits [B, K+1, Vs] hold the shard's vocabulary entries
 *   v_offset .. v_offset+Vs-1 of a V-entry vocabulary; draft [B, K] holds
 *   GLOBAL token ids; writes partials [B*(K+1)]. Workspace and its rules as for
 *   asd_verify, sized with asd_workspace_size(B, K, Vs, dtype).
 * Step 2, once the S shards' partials sit side by side (an all-gather across
 * ranks, or S slices of one GPU):
 *   asd_shard_combine: partials [S, B*(K+1)] -> the outputs of asd_verify for
 *   the whole vocabulary, bit for bit (same keys, same fp32 arithmetic). No
 *   workspace. The ledger, gate, cap and outputs are as in asd_verify.
 */
int asd_shard_partials(const void* logits, int dtype, int B, int K, int Vs, int v_offset, int V,
                       const int32_t* draft, asd_partial* partials, void* workspace,
                       size_t workspace_bytes, asd_stream_t stream);
int asd_shard_combine(const asd_partial* partials, int S, int B, int K, int V, const int32_t* draft,
                      asd_ledger* ledger, float gate, int cap, int32_t* accepted_len,
                      int32_t* committed, int32_t* recovery, int32_t* row_argmax, float* row_regret,
                      int32_t* status, asd_stream_t stream);

/* Step 1 of the same scheme with the LM head fused (the remark of Sec. 3.3 as
 * a tensor-parallel rank would run it: no logit buffer anywhere):
 * weight [Vs, H] bf16 holds rows v_offset .. v_offset+Vs-1 of the LM-head
 * weight of a V-entry vocabulary; hidden [B*(K+1), H] bf16 and draft [B, K]
 * (GLOBAL ids) as in asd_lmhead_verify; writes partials [B*(K+1)] for
 * asd_shard_combine. The top logit in a partial is the value the key holds
 * (a zero maximum is +0). Workspace from asd_lmhead_workspace_size(B, K, Vs,
 * H). Same precision and launch notes as asd_lmhead_verify. */
int asd_lmhead_partials(const void* hidden, const void* weight, int H, int B, int K, int Vs, int v_offset,
                        int V, const int32_t* draft, asd_partial* partials, void* workspace,
                        size_t workspace_bytes, asd_stream_t stream);

/*
 * Advance along the emitted sequence (Sec. 3.3: the target cache, the draft
 * cache and the ledger advance only along the emitted tokens; proposal-only
 * state past the returned prefix is discarded). For each request b with
 * a = accepted_len[b]:
 *   tokens [B, max_tokens], token_len [B] (in/out): the a + 1 emitted tokens
 *     committed[b][0..a] are appended at token_len[b]; token_len[b] += a + 1
 *   kv_len [B] (in/out): kv_len[b] += pending + a -- the cache keeps the
 *     pending input token of the pass (pending = 1 when the verification pass
 *     consumed the previous round's recovery token before the drafts, else 0)
 *     and the a accepted drafts; positions from the new length on held
 *     proposal-only state and may be overwritten (call once per cache)
 *   status [B] (out, may be NULL): ASD_STATUS_OVERFLOW when the history has
 *     no room; such a request changes nothing.
 * tokens / token_len may be NULL together, kv_len may be NULL. Device arrays.
 * accepted_len values are those asd_verify writes (0..K); others are clamped.
 */
int asd_commit(int B, int K, const int32_t* accepted_len, const int32_t* committed, int pending,
               int32_t* kv_len, int32_t* tokens, int32_t* token_len, int max_tokens, int32_t* status,
               asd_stream_t stream);

/* The device address through which kernels read page-locked (pinned) host
 * memory, e.g. logits that stay in host memory and stream to the GPU over the
 * host link while asd_verify runs, with no separate copy. `host` should lie in
 * a pinned, mapped allocation (cudaHostAlloc / cudaHostRegister; runtime
 * contexts map pinned memory by default). On systems whose GPU reads pageable
 * memory through the host's page tables the runtime also accepts pageable
 * memory (slower to read); where neither applies the call returns
 * ASD_ERR_ALIGN. The alias is valid as long as the allocation is.
 * Synchronous, no allocation. */
int asd_host_alias(const void* host, void** device);

/* How many kernels one asd_verify / asd_verify_strict call launches for this
 * shape (1 or 2: the row stage, and for large inputs a separate selection
 * kernel launched right behind it); 0 for B = 0. For accounting only. */
int asd_verify_launches(int B, int K, int V, int dtype, int* launches);

/* Launch options of the logit-streaming entry points (asd_verify,
 * asd_verify_strict, asd_verify_blocks, asd_shard_partials, asd_verify_noalloc).
 * The paper has no counterpart: these choose among kernels that compute the
 * same results bit for bit, for tests that cover each kernel and for
 * measurements; the defaults (all fields 0) are what production calls want.
 *   path          ASD_PATH_AUTO picks the row-stage kernel by input size (the
 *                 one-CTA-per-request kernel below 1 MB when a request fits
 *                 it, the register-streaming kernel for other small inputs,
 *                 the TMA pipeline from 1 MB); the others force one (a forced
 *                 ASD_PATH_SMALL falls back to AUTO where the shape does not
 *                 fit it).
 *   fused_select  1: the TMA row stage runs the selection itself (the CTA that
 *                 completes a request selects it) instead of launching
 *                 select_kernel right behind it.
 *   no_pdl        1: launch without programmatic dependent launch.
 * Process-wide; each call reads the options once when it is issued, and a CUDA
 * graph keeps the kernels chosen at capture. asd_set_launch_options(NULL)
 * restores the defaults. Returns ASD_ERR_CONTROL for an unknown path. */
enum { ASD_PATH_AUTO = 0, ASD_PATH_SMALL = 1, ASD_PATH_STREAM = 2, ASD_PATH_TMA = 3 };
typedef struct {
  int path;
  int fused_select;
  int no_pdl;
} asd_launch_options;
int asd_set_launch_options(const asd_launch_options* options);
int asd_get_launch_options(asd_launch_options* options);

/* Human-readable text of a return code. Never NULL. */
const char* asd_status_string(int code);

#ifdef __cplusplus
}
#endif

#endif /* ASD_H */
