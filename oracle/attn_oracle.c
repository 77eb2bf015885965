/*
 * attn_oracle.c -- plain fp64 CPU oracle for causal / document-masked
 * multi-head self-attention, forward and backward.
 *
 * TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py load this library. It shares no code, header
 * or constant with the CUDA path in paper_2405_13226_gb300/csrc.
 *
 * What it computes (the plain definition; no blocking, no fusion):
 *   A sequence of L tokens is split into documents. Under the concat-and-chunk
 *   baseline with document masking (Sec. 1, "document-masking ... cross-document
 *   attention", and Sec. 3.5 where DM means avoiding cross-document attention)
 *   a token may only attend to earlier tokens of its own document; under
 *   dataset decomposition every sequence is cut from one document (Sec. 2.1,
 *   property (2)), so the mask is plain causal. Next-token training sees the
 *   contexts 0..l-1 of a length-l sequence (Appendix "Average sequence length
 *   vs average context length"), i.e. query i attends to keys j <= i.
 *
 *   live set   A(i) = { j <= i : doc(j) == doc(i) }
 *   scores     s_ij = scale * <q_i, k_j>
 *   LSE_i      = ln sum_{j in A(i)} exp(s_ij)          (natural log, max-shifted)
 *   P_ij       = exp(s_ij - LSE_i)
 *   o_i        = sum_j P_ij v_j
 *   backward, for a loss whose gradient w.r.t. o is dO:
 *   D_i        = <dO_i, o_i>
 *   dP_ij      = <dO_i, v_j>
 *   dS_ij      = P_ij (dP_ij - D_i)
 *   dq_i       = scale * sum_j dS_ij k_j
 *   dk_j       = scale * sum_i dS_ij q_i     (gathered per key j)
 *   dv_j       = sum_i P_ij dO_i             (gathered per key j)
 *   An empty live set (impossible under causal/DM, since j = i is always
 *   live) would give o_i = 0 and LSE_i = -inf.
 *
 * Layout: n independent (sequence, head) slices, each [L, d] row-major in
 * double; doc[n*L] holds the document id of every token of each slice.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Document id of every token of sequence b (tokens b*L .. b*L+L-1 of the
 * flattened stream), from cu_doc_offsets (non-decreasing, first 0, last B*L):
 * doc(t) = largest k with offsets[k] <= t. Sequence boundaries always cut
 * documents; ids only need to be compared within one sequence.
 * offsets == NULL means one document per sequence (plain causal). */
void oracle_doc_ids(int L, int b, const int32_t* offsets, int n_offsets, int32_t* doc_out) {
  for (int i = 0; i < L; i++) {
    long t = (long)b * L + i;
    int id = 0;
    if (offsets) {
      for (int k = 0; k < n_offsets; k++)
        if (offsets[k] <= t) id = k;
    }
    doc_out[i] = id;
  }
}

static double dot(const double* a, const double* b, int d) {
  double s = 0.0;
  for (int c = 0; c < d; c++) s += a[c] * b[c];
  return s;
}

/* Row pass for query i of one slice: LSE_i and o_i. */
static void row_forward(int L, int d, double scale, const int32_t* doc, const double* q, const double* k,
                        const double* v, int i, double* o_i, double* lse_i) {
  (void)L;
  double mx = -INFINITY;
  for (int j = 0; j <= i; j++)
    if (doc[j] == doc[i]) {
      double s = scale * dot(q + (long)i * d, k + (long)j * d, d);
      if (s > mx) mx = s;
    }
  for (int c = 0; c < d; c++) o_i[c] = 0.0;
  if (mx == -INFINITY) {
    *lse_i = -INFINITY;
    return;
  }
  double sum = 0.0;
  for (int j = 0; j <= i; j++)
    if (doc[j] == doc[i]) sum += exp(scale * dot(q + (long)i * d, k + (long)j * d, d) - mx);
  double lse = mx + log(sum);
  for (int j = 0; j <= i; j++)
    if (doc[j] == doc[i]) {
      double p = exp(scale * dot(q + (long)i * d, k + (long)j * d, d) - lse);
      for (int c = 0; c < d; c++) o_i[c] += p * v[(long)j * d + c];
    }
  *lse_i = lse;
}

void oracle_attn_fwd(int n, int L, int d, double scale, const int32_t* doc, const double* q, const double* k,
                     const double* v, double* o, double* lse) {
  long total = (long)n * L;
#pragma omp parallel for schedule(dynamic, 16)
  for (long t = 0; t < total; t++) {
    long s = t / L;
    int i = (int)(t % L);
    long base = s * (long)L * d;
    row_forward(L, d, scale, doc + s * L, q + base, k + base, v + base, i, o + base + (long)i * d, lse + t);
  }
}

/* Forward for selected query rows of one slice (sampled parity at full size). */
void oracle_attn_fwd_rows(int L, int d, double scale, const int32_t* doc, const double* q, const double* k,
                          const double* v, int nr, const int32_t* rows, double* o, double* lse) {
#pragma omp parallel for schedule(dynamic, 1)
  for (int r = 0; r < nr; r++)
    row_forward(L, d, scale, doc, q, k, v, rows[r], o + (long)r * d, lse + r);
}

/* Backward of one slice restricted to query rows `qrows` (dq) and key rows
 * `krows` (dk, dv); nq = L / nk = L with NULL lists means all rows. lse and
 * D of every query row a requested output depends on come from this
 * oracle's own fp64 forward. */
static void slice_backward(int L, int d, double scale, const int32_t* doc, const double* q, const double* k,
                           const double* v, const double* dO, int nq, const int32_t* qrows, double* dq, int nk,
                           const int32_t* krows, double* dk, double* dv, int parallel) {
  /* Which query rows need LSE_i and D_i: requested dq rows, and every row
   * that attends to a requested key (i >= j, same document). */
  char* need = (char*)calloc((size_t)L, 1);
  for (int r = 0; r < nq; r++) need[qrows ? qrows[r] : r] = 1;
  for (int r = 0; r < nk; r++) {
    int j = krows ? krows[r] : r;
    for (int i = j; i < L; i++)
      if (doc[i] == doc[j]) need[i] = 1;
  }
  double* lse = (double*)malloc(sizeof(double) * (size_t)L);
  double* D = (double*)malloc(sizeof(double) * (size_t)L);
  double* orow = (double*)malloc(sizeof(double) * (size_t)L * d);
#pragma omp parallel for schedule(dynamic, 8) if (parallel)
  for (int i = 0; i < L; i++) {
    if (!need[i]) continue;
    row_forward(L, d, scale, doc, q, k, v, i, orow + (long)i * d, &lse[i]);
    D[i] = dot(dO + (long)i * d, orow + (long)i * d, d);
  }
  /* dq_i = scale * sum_{j in A(i)} P_ij (dP_ij - D_i) k_j */
#pragma omp parallel for schedule(dynamic, 8) if (parallel)
  for (int r = 0; r < nq; r++) {
    int i = qrows ? qrows[r] : r;
    double* out = dq + (long)r * d;
    for (int c = 0; c < d; c++) out[c] = 0.0;
    for (int j = 0; j <= i; j++) {
      if (doc[j] != doc[i]) continue;
      double p = exp(scale * dot(q + (long)i * d, k + (long)j * d, d) - lse[i]);
      double ds = p * (dot(dO + (long)i * d, v + (long)j * d, d) - D[i]);
      for (int c = 0; c < d; c++) out[c] += scale * ds * k[(long)j * d + c];
    }
  }
  /* dk_j = scale * sum_{i : j in A(i)} dS_ij q_i ;  dv_j = sum_i P_ij dO_i */
#pragma omp parallel for schedule(dynamic, 8) if (parallel)
  for (int r = 0; r < nk; r++) {
    int j = krows ? krows[r] : r;
    double* ok = dk + (long)r * d;
    double* ov = dv + (long)r * d;
    for (int c = 0; c < d; c++) ok[c] = ov[c] = 0.0;
    for (int i = j; i < L; i++) {
      if (doc[i] != doc[j]) continue;
      double p = exp(scale * dot(q + (long)i * d, k + (long)j * d, d) - lse[i]);
      double ds = p * (dot(dO + (long)i * d, v + (long)j * d, d) - D[i]);
      for (int c = 0; c < d; c++) {
        ok[c] += scale * ds * q[(long)i * d + c];
        ov[c] += p * dO[(long)i * d + c];
      }
    }
  }
  free(need);
  free(lse);
  free(D);
  free(orow);
}

void oracle_attn_bwd(int n, int L, int d, double scale, const int32_t* doc, const double* q, const double* k,
                     const double* v, const double* dO, double* dq, double* dk, double* dv) {
  if (n == 1) {
    slice_backward(L, d, scale, doc, q, k, v, dO, L, NULL, dq, L, NULL, dk, dv, 1);
    return;
  }
#pragma omp parallel for schedule(dynamic, 1)
  for (int s = 0; s < n; s++) {
    long base = (long)s * L * d;
    slice_backward(L, d, scale, doc + (long)s * L, q + base, k + base, v + base, dO + base, L, NULL, dq + base, L,
                   NULL, dk + base, dv + base, 0);
  }
}

/* Backward of one slice for selected query rows (dq) and key rows (dk, dv). */
void oracle_attn_bwd_rows(int L, int d, double scale, const int32_t* doc, const double* q, const double* k,
                          const double* v, const double* dO, int nq, const int32_t* qrows, double* dq, int nk,
                          const int32_t* krows, double* dk, double* dv) {
  slice_backward(L, d, scale, doc, q, k, v, dO, nq, qrows, dq, nk, krows, dk, dv, 1);
}

/* Number of live (query, key) pairs of one sequence, by enumerating the mask. */
long long oracle_live_pairs(int L, const int32_t* doc) {
  long long n = 0;
  for (int i = 0; i < L; i++)
    for (int j = 0; j <= i; j++)
      if (doc[j] == doc[i]) n++;
  return n;
}
