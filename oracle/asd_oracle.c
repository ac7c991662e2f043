/*
 * ASD verifier oracle: a plain, slow, obviously correct CPU implementation of
 * the verifier of "Approximate Speculative Decoding" (arXiv 2608.03447).
 *
 * THIS IS TEST INFRASTRUCTURE. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load it. It shares no code, header, table or
 * helper with the CUDA library: every constant below is written out here on
 * its own, from the paper's definitions.
 *
 * What it computes, per request b and draft block (paper notation, 1-based
 * i = j + 1 for our 0-based position j):
 *   Eq. 1   y*_i = argmax_v z_i(v)            (ties: the lowest index v)
 *   Eq. 3   r_i  = z_i(y*_i) - z_i(x_i)       (one fp32 subtraction)
 *   Eq. 5   d_i  = [x_i != y*_i]              (token ids)
 *   Eq. 6   q_i  = K - i + 1
 *   Eq. 7   r_i / q_i <= g                    (IEEE fp32 division)
 *   Eq. 8   C_t = sum_{i<=t} d_i r_i,  N_t = sum_{i<=t} d_i  (left to right)
 *   Eq. 9-11 feasibility; Eq. 12 longest feasible prefix a
 *   Alg. 1  zero budget dispatches to strict greedy (Eq. 2); the output is
 *           x_{1:a} followed by y*_{a+1} (recovery, a < K) or y*_{K+1} (bonus)
 *   Eq. 13  s' = s + C_a
 *
 * Readings where the paper leaves the arithmetic open (all fp32):
 *   - the budget test of Eq. 9, C_t <= B - s, is evaluated as
 *     fl(s + C_t) <= B; this is the same inequality over the reals and makes
 *     the updated ledger of Eq. 13 satisfy s' <= B exactly, because the
 *     compared value is the value stored;
 *   - C_t is summed left to right over the block, then added to s once;
 *   - argmax compares with IEEE float comparison, so -0 == +0 and the lower
 *     index wins;
 *   - the strict rule also appends the bonus y*_{K+1} when every draft token
 *     matches (Alg. 1's return value, "exact greedy verifier output");
 *   - a request whose block holds a NaN logit, a draft id outside [0, V) or an
 *     invalid ledger (budget < 0 or NaN, spent < 0 or NaN, spent > budget) is
 *     flagged in its status word; it accepts nothing (a = 0), emits y*_1 and
 *     keeps its ledger. The argmax of a row holding NaN is deterministic but
 *     unspecified.
 *
 * Fused LM-head variant (logits never stored on the GPU): the oracle forms
 * z = sum_k h_k W_vk in fp64 from the bf16 inputs and rounds it to fp32.
 *
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math -fPIC -shared
 * (no contraction into fused multiply-adds, no reassociation).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* dtype codes */
#define ORC_DTYPE_F32 0
#define ORC_DTYPE_BF16 1

/* per-request status bits */
#define ORC_STATUS_DRAFT_RANGE 1
#define ORC_STATUS_NAN_LOGIT 2
#define ORC_STATUS_BAD_LEDGER 4

/* bf16 -> fp32 is exact: the 16 bits become the high half of the fp32 word. */
static float bf16_bits_to_float(uint16_t bits) {
  uint32_t u = ((uint32_t)bits) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

static float logit_at(const void* logits, int dtype, int64_t index) {
  if (dtype == ORC_DTYPE_F32) return ((const float*)logits)[index];
  return bf16_bits_to_float(((const uint16_t*)logits)[index]);
}

/* Eq. 1: the lowest index v whose logit equals the row maximum. */
static int32_t row_argmax(const void* logits, int dtype, int64_t row_start, int V,
                          int* saw_nan) {
  int32_t best = 0;
  float best_value = logit_at(logits, dtype, row_start);
  if (best_value != best_value) *saw_nan = 1;
  for (int v = 1; v < V; v++) {
    float z = logit_at(logits, dtype, row_start + v);
    if (z != z) {
      *saw_nan = 1;
      continue;
    }
    if (z > best_value) { /* strictly greater: an equal later value never wins */
      best_value = z;
      best = v;
    }
  }
  return best;
}

/* Eq. 2: the longest prefix whose draft tokens equal the target argmax. */
static int strict_prefix(int K, const int32_t* x, const int32_t* y) {
  for (int j = 0; j < K; j++)
    if (x[j] != y[j]) return j;
  return K;
}

/*
 * Eq. 5-12 (Alg. 1 after the zero-budget test): walk the block once; a
 * matching token is always feasible (Eq. 14's first term, Proposition 1); a
 * mismatch is feasible when the gate, the cap and the budget all hold for the
 * prefix that ends at it. The first infeasible position ends the prefix
 * (contiguity: no infeasible token is ever skipped).
 * Returns a and writes C_a (the regret spent by the accepted mismatches).
 */
static int asd_prefix(int K, const int32_t* x, const int32_t* y, const float* r,
                      float budget, float spent, float gate, int cap, float* spent_regret) {
  float C = 0.0f; /* C_t, Eq. 8 */
  int N = 0;      /* N_t, Eq. 8 */
  for (int j = 0; j < K; j++) {
    if (x[j] == y[j]) continue; /* d = 0 */
    float q = (float)(K - j);   /* Eq. 6: q_i = K - i + 1 with i = j + 1 */
    float C_next = C + r[j];
    int N_next = N + 1;
    int gate_ok = (r[j] / q) <= gate;             /* Eq. 7 / Eq. 11 */
    int budget_ok = (spent + C_next) <= budget;   /* Eq. 9, read as fl(s + C_t) <= B */
    int cap_ok = N_next <= cap;                   /* Eq. 10 */
    if (!(gate_ok && budget_ok && cap_ok)) {
      *spent_regret = C;
      return j;
    }
    C = C_next;
    N = N_next;
  }
  *spent_regret = C;
  return K;
}

static int ledger_invalid(float budget, float spent) {
  if (budget != budget || spent != spent) return 1;
  if (budget < 0.0f || spent < 0.0f) return 1;
  if (spent > budget) return 1;
  return 0;
}

/*
 * Alg. 1 for one request, given its row-stage results: y*_0..y*_K, the
 * regrets r_0..r_{K-1} and the row-stage status bits (NaN logit, draft range).
 * Writes a, the committed tokens, the recovery token and the status word, and
 * updates the ledger (budget, spent) unless strict, zero-budget or flagged.
 */
static void select_block(int K, const int32_t* x, const int32_t* y, const float* r, int flags,
                         float* ledger_b, float gate, int cap, int strict, int32_t* accepted_len_b,
                         int32_t* committed_b, int32_t* recovery_b, int32_t* status_b) {
  float budget = ledger_b[0];
  float spent = ledger_b[1];
  if (!strict && ledger_invalid(budget, spent)) flags |= ORC_STATUS_BAD_LEDGER;

  int a;
  if (flags) {
    a = 0; /* a flagged request accepts nothing and keeps its ledger */
  } else if (strict || budget == 0.0f) {
    a = strict_prefix(K, x, y); /* Alg. 1: B = 0 -> exact greedy output, state kept */
  } else {
    float C = 0.0f;
    a = asd_prefix(K, x, y, r, budget, spent, gate, cap, &C);
    ledger_b[1] = spent + C; /* Eq. 13 */
  }
  *accepted_len_b = a;
  *recovery_b = y[a]; /* y*_{a+1}: recovery if a < K, bonus if a = K */
  for (int j = 0; j <= K; j++) {
    int32_t token = -1;
    if (j < a) token = x[j];
    else if (j == a) token = y[a];
    committed_b[j] = token;
  }
  *status_b = flags;
}

/*
 * Verify B draft blocks.
 *   logits       [B, K+1, V] fp32 or bf16 bits, row-major
 *   draft        [B, K] int32
 *   ledger       [B, 2] fp32 (budget, spent), updated in place unless strict
 *   strict       1: Eq. 2 for every request (ledger, gate, cap ignored)
 *   outputs      accepted_len [B], committed [B, K+1] (-1 padded),
 *                recovery [B], row_argmax [B, K+1], row_regret [B, K] (NaN
 *                where the draft id is out of range), status [B]
 * Returns 0, or -1 on an argument that the oracle cannot evaluate.
 */
int oracle_verify(const void* logits, int dtype, int B, int K, int V, const int32_t* draft,
                  float* ledger, float gate, int cap, int strict, int32_t* accepted_len,
                  int32_t* committed, int32_t* recovery, int32_t* row_argmax_out,
                  float* row_regret, int32_t* status) {
  if (B < 0 || K < 0 || K > 31 || V < 1) return -1;
  if (dtype != ORC_DTYPE_F32 && dtype != ORC_DTYPE_BF16) return -1;
  int32_t y[32];
  float r[32];
  for (int b = 0; b < B; b++) {
    int flags = 0;
    const int32_t* x = draft + (int64_t)b * K;
    /* Eq. 1 for the K + 1 rows of this block */
    for (int j = 0; j <= K; j++) {
      int saw_nan = 0;
      int64_t row = (int64_t)b * (K + 1) + j;
      y[j] = row_argmax(logits, dtype, row * V, V, &saw_nan);
      if (saw_nan) flags |= ORC_STATUS_NAN_LOGIT;
      row_argmax_out[row] = y[j];
    }
    /* Eq. 3 for the K draft positions */
    for (int j = 0; j < K; j++) {
      int64_t row = (int64_t)b * (K + 1) + j;
      if (x[j] < 0 || x[j] >= V) {
        flags |= ORC_STATUS_DRAFT_RANGE;
        r[j] = NAN;
      } else {
        float z_top = logit_at(logits, dtype, row * V + y[j]);
        float z_draft = logit_at(logits, dtype, row * V + x[j]);
        r[j] = z_top - z_draft;
      }
      row_regret[(int64_t)b * K + j] = r[j];
    }
    select_block(K, x, y, r, flags, ledger + 2 * b, gate, cap, strict, accepted_len + b,
                 committed + (int64_t)b * (K + 1), recovery + b, status + b);
  }
  return 0;
}

/*
 * The selection stage alone (Alg. 1 after Eq. 1 and Eq. 3), for callers that
 * already hold the row-stage results of a block (row_argmax [B, K+1],
 * row_regret [B, K], row_status [B] = the status bits of a strict run) and
 * want to replay the selection under other controls.
 */
int oracle_select(int B, int K, const int32_t* draft, const int32_t* row_argmax_in,
                  const float* row_regret_in, const int32_t* row_status, float* ledger,
                  float gate, int cap, int strict, int32_t* accepted_len, int32_t* committed,
                  int32_t* recovery, int32_t* status) {
  if (B < 0 || K < 0 || K > 31) return -1;
  for (int b = 0; b < B; b++) {
    select_block(K, draft + (int64_t)b * K, row_argmax_in + (int64_t)b * (K + 1),
                 row_regret_in + (int64_t)b * K, row_status[b], ledger + 2 * b, gate, cap, strict,
                 accepted_len + b, committed + (int64_t)b * (K + 1), recovery + b, status + b);
  }
  return 0;
}

/*
 * Fused LM-head oracle: logits of the selected token rows,
 *   z[t, v] = sum_k h[tokens[t], k] * W[v, k]
 * with bf16 inputs widened exactly and every product and sum in fp64.
 *   h [T_all, H], W [V, H] bf16 bits; tokens [T] indices into h
 *   out64 [T, V] fp64 (may be NULL), out32 [T, V] fp32 = fp64 rounded (may be NULL)
 */
void oracle_lmhead_logits(const uint16_t* h, const uint16_t* W, int H, int V,
                          const int32_t* tokens, int T, double* out64, float* out32) {
  for (int t = 0; t < T; t++) {
    const uint16_t* ht = h + (int64_t)tokens[t] * H;
    for (int v = 0; v < V; v++) {
      const uint16_t* wv = W + (int64_t)v * H;
      double acc = 0.0;
      for (int k = 0; k < H; k++)
        acc += (double)bf16_bits_to_float(ht[k]) * (double)bf16_bits_to_float(wv[k]);
      if (out64) out64[(int64_t)t * V + v] = acc;
      if (out32) out32[(int64_t)t * V + v] = (float)acc;
    }
  }
}

/*
 * Eq. 4, the verifier-side opportunity rate, as counts: over every mismatch
 * position (x, i) of the given blocks (1-based i with x_i != y*_i, i <= K),
 *   num[t][u] = #{ (x, i) : r_i <= tau[t], i + p[u] <= K, x_l = y*_l for l = i+1 .. i+p[u] }
 *   *den      = |M|, the number of mismatch positions.
 * Omega(tau, p) = num / den. Blocks with a non-zero status word (when given)
 * are skipped. Counts are added to num / den (accumulated over calls).
 *   row_argmax [n, K+1], draft [n, K], row_regret [n, K], status [n] or NULL
 */
void oracle_opportunity(const int32_t* row_argmax, const int32_t* draft, const float* row_regret,
                        const int32_t* status, int n, int K, const float* tau, int ntau,
                        const int32_t* p, int np, long long* num, long long* den) {
  for (int b = 0; b < n; b++) {
    if (status && status[b] != 0) continue;
    const int32_t* y = row_argmax + (int64_t)b * (K + 1);
    const int32_t* x = draft + (int64_t)b * K;
    const float* r = row_regret + (int64_t)b * K;
    for (int i = 1; i <= K; i++) {           /* 1-based position, as in Eq. 4 */
      if (x[i - 1] == y[i - 1]) continue;    /* only mismatches belong to M */
      *den += 1;
      for (int u = 0; u < np; u++) {
        int reusable = i + p[u] <= K;
        for (int l = i + 1; reusable && l <= i + p[u]; l++)
          if (x[l - 1] != y[l - 1]) reusable = 0;
        if (!reusable) continue;
        for (int t = 0; t < ntau; t++)
          if (r[i - 1] <= tau[t]) num[t * np + u] += 1;
      }
    }
  }
}

/*
 * Sec. 3.3, cache semantics: after a block is verified the caches and the
 * history advance along the emitted sequence only. The emitted sequence of
 * request b is committed[b][0..a] (x_1..x_a, then the recovery or bonus token).
 *   tokens [B][max_tokens], token_len [B]: the history gets the a + 1 emitted
 *     tokens appended at token_len[b]; token_len[b] += a + 1
 *   kv_len [B]: the target cache keeps the pending input token (pending = 1 if
 *     the verification pass consumed one before the drafts, else 0) and the a
 *     accepted drafts: kv_len[b] += pending + a; positions from the new length
 *     on held proposal-only state and are free
 *   a request whose history has no room for a + 1 more tokens changes nothing
 *     and gets status bit 8 (overflow)
 * tokens / token_len / kv_len / status may be NULL (that part is skipped).
 */
void oracle_commit(int B, int K, const int32_t* accepted_len, const int32_t* committed, int pending,
                   int32_t* kv_len, int32_t* tokens, int32_t* token_len, int max_tokens, int32_t* status) {
  for (int b = 0; b < B; b++) {
    int a = accepted_len[b];
    const int32_t* emitted = committed + (int64_t)b * (K + 1);
    if (tokens && token_len[b] + a + 1 > max_tokens) {
      if (status) status[b] = 8;
      continue;
    }
    if (status) status[b] = 0;
    if (tokens) {
      for (int j = 0; j <= a; j++) tokens[(int64_t)b * max_tokens + token_len[b] + j] = emitted[j];
      token_len[b] += a + 1;
    }
    if (kv_len) kv_len[b] += pending + a;
  }
}
