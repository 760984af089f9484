/*
 * sva_oracle.c -- plain, slow, fp64 CPU oracle for policy-indexed
 * chunk-causal attention ("Rethinking Streaming Video Diffusion Model:
 * Context, Execution, and Training", Section 3).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library calls, links or
 * loads this file; only the tests, the package's smoke check and the
 * benchmark's CPU-baseline leg do.  It shares no code, header, table or
 * helper with the CUDA path.
 *
 * Every function states the passage it follows.  Readings of points the
 * paper leaves open (the full offset window, 3D RoPE, the bf16 cache store,
 * the fully-masked row) are stated where they are used.
 *
 * Parity pins: selection, pipeline rounds and availability are pinned by the
 * paper's worked example (Section 3.3, K = 3) and its counting facts; RoPE by
 * closed forms (identity at position zero, norm preservation, composition,
 * relative-position dot products, axis partition); attention by a dense-mask
 * brute force over the whole (chunk, level) grid, by softmax invariants and
 * by a library SDPA for the clean single-node case.  No function here is
 * "parity unpinned".
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORACLE_POLICY_CLEAN = 0, ORACLE_POLICY_SAME = 1, ORACLE_POLICY_PROG = 2 };

/* Eq. 3 (Section 3.2): the three position-independent policies.
 *   clean:       phi(j, r) = 0
 *   same-level:  phi(j, r) = j
 *   progressive: phi(j, r) = max(j - r, 0)
 * Returns -1 for an unknown policy id. */
int oracle_phi(int policy, int j, int r) {
  switch (policy) {
    case ORACLE_POLICY_CLEAN:
      return 0;
    case ORACLE_POLICY_SAME:
      return j;
    case ORACLE_POLICY_PROG:
      return (j - r > 0) ? (j - r) : 0;
    default:
      return -1;
  }
}

/* Eq. 2 (Section 3.2): the selected history of node (b, j) is
 * { x_{b-r}^{phi(j, r)} : r in R_{b,j} } with R_{b,j} a subset of
 * {1, ..., min(W, b-1)}.  Reading: R is the whole window.  Chunks are
 * numbered from 1 as in the paper, so chunk b has b-1 predecessors.
 * Writes the states in order of increasing offset r; returns their count,
 * or -1 for an unknown policy. */
int oracle_select(int policy, int W, int b, int j, int* chunks, int* levels) {
  int rmax = (W < b - 1) ? W : b - 1;
  int n = 0;
  for (int r = 1; r <= rmax; ++r) {
    int level = oracle_phi(policy, j, r);
    if (level < 0) return -1;
    chunks[n] = b - r;
    levels[n] = level;
    ++n;
  }
  return n;
}

/* Eq. 6 (Section 3.3): at the start of round n a pipeline that admits one
 * new chunk per round holds [x_n^K, x_{n-1}^{K-1}, ..., x_{n-K+1}^1]; chunk
 * indices outside 1..B are left out while the pipeline fills and drains.
 * Writes (chunk, level) pairs for levels K down to 1; returns the count. */
int oracle_pipeline_round(int K, int B, int n, int* chunks, int* levels) {
  int count = 0;
  for (int i = 0; i < K; ++i) {
    int level = K - i;
    int chunk = n - i;
    if (chunk >= 1 && chunk <= B) {
      chunks[count] = chunk;
      levels[count] = level;
      ++count;
    }
  }
  return count;
}

/* Eq. 7 (Section 3.3): in the pipeline of Eq. 6, when chunk b is at level j
 * the chunk b - r has reached level max(j - r, 0), so a read of level
 * `level` at offset r is available iff level >= max(j - r, 0). */
int oracle_available(int j, int r, int level) {
  int reached = (j - r > 0) ? (j - r) : 0;
  return level >= reached;
}

/* Round-to-nearest-even of a double to the bfloat16 grid (8 significant
 * bits, exponent range of binary32), returned as a double.  Reading: the KV
 * cache stores bf16, so the keys the attention sees are the rotated keys
 * rounded once to bf16. */
double oracle_bf16(double x) {
  if (x == 0.0 || !isfinite(x)) return x;
  int e = ilogb(x); /* |x| in [2^e, 2^(e+1)) */
  if (e < -126) e = -126;
  double q = ldexp(x, 7 - e); /* ulp of the result becomes 1 */
  double r = nearbyint(q);    /* default rounding mode: ties to even */
  return ldexp(r, e - 7);
}

void oracle_bf16_array(const double* x, double* y, long n) {
  for (long i = 0; i < n; ++i) y[i] = oracle_bf16(x[i]);
}

/* 3D rotary position embedding of one head's rows x[T][d] of a chunk
 * (reading; the paper does not name a positional encoding).  Token u of the
 * chunk is u = (f * Hp + h) * Wp + w with f the latent frame inside the
 * chunk; its absolute position on the three axes is (F * b + f, h, w).
 * Head dimension pairs (2p, 2p+1) are split into three consecutive groups
 * of pairs[0], pairs[1], pairs[2] pairs for the t, h and w axes.  Pair i of
 * axis a turns by the angle pos_a * theta^(-i / pairs[a]):
 *   (x, y) -> (x cos A - y sin A, x sin A + y cos A).
 * fp64 throughout; y is not rounded. */
void oracle_rope_head(const double* x, double* y, int T, int d, int F, int Hp, int Wp, long b,
                      const int* pairs, double theta) {
  for (int u = 0; u < T; ++u) {
    int f = u / (Hp * Wp);
    int hh = (u / Wp) % Hp;
    int ww = u % Wp;
    double pos[3];
    pos[0] = (double)F * (double)b + (double)f;
    pos[1] = (double)hh;
    pos[2] = (double)ww;
    int p = 0;
    for (int a = 0; a < 3; ++a) {
      for (int i = 0; i < pairs[a]; ++i, ++p) {
        double omega = pow(theta, -(double)i / (double)pairs[a]);
        double angle = pos[a] * omega;
        double c = cos(angle), s = sin(angle);
        double x0 = x[(long)u * d + 2 * p];
        double x1 = x[(long)u * d + 2 * p + 1];
        y[(long)u * d + 2 * p] = x0 * c - x1 * s;
        y[(long)u * d + 2 * p + 1] = x0 * s + x1 * c;
      }
    }
    /* any head-dimension elements beyond the pairs are copied unchanged */
    for (int c = 2 * p; c < d; ++c) y[(long)u * d + c] = x[(long)u * d + c];
  }
}

/* RMS normalisation of each row of x[T][n] (reading: the paper names no
 * normalisation; a token's whole query or key vector of n = H*d elements is
 * normalised before RoPE): y = x * gamma / sqrt(mean(x^2) + eps), fp64. */
void oracle_rms_norm(const double* x, const double* gamma, double* y, long T, int n, double eps) {
  for (long t = 0; t < T; ++t) {
    const double* xr = x + t * n;
    double ss = 0.0;
    for (int i = 0; i < n; ++i) ss += xr[i] * xr[i];
    const double r = 1.0 / sqrt(ss / n + eps);
    for (int i = 0; i < n; ++i) y[t * n + i] = xr[i] * r * gamma[i];
  }
}

/* Eq. 4 (Section 3.2): masked softmax attention.  For each query row i the
 * logits are l_v = scale * <q_i, k_v> + mask[v], with mask[v] = 0 where the
 * query may attend to key v and -inf otherwise; the mask is added before
 * the softmax, so a -inf entry gets weight zero.  Two passes in fp64: the
 * logits and their maximum m, then p_v = exp(l_v - m), out_i = sum p_v v_v /
 * sum p_v and lse_i = m + log(sum p_v).  A row whose every key is masked
 * (cannot arise in the chunk-causal setting, where a chunk always sees
 * itself) gets out = 0 and lse = -inf.
 *   q: [nrows][d], k, v: [L][d], mask: [L] (NULL = all visible). */
void oracle_attend_rows(const double* q, const double* k, const double* v, const double* mask,
                        long L, int d, long nrows, double scale, double* out, double* lse) {
#pragma omp parallel for schedule(dynamic, 1)
  for (long i = 0; i < nrows; ++i) {
    double* logit = (double*)malloc((size_t)(L > 0 ? L : 1) * sizeof(double));
    const double* qi = q + i * d;
    double* oi = out + i * d;
    double m = -INFINITY;
    for (long j = 0; j < L; ++j) {
      const double* kj = k + j * d;
      double s = 0.0;
      for (int c = 0; c < d; ++c) s += qi[c] * kj[c];
      s = s * scale + (mask ? mask[j] : 0.0);
      logit[j] = s;
      if (s > m) m = s;
    }
    for (int c = 0; c < d; ++c) oi[c] = 0.0;
    if (m == -INFINITY) {
      lse[i] = -INFINITY;
      free(logit);
      continue;
    }
    double sum = 0.0;
    for (long j = 0; j < L; ++j) {
      double p = exp(logit[j] - m);
      if (p == 0.0) continue;
      sum += p;
      const double* vj = v + j * d;
      for (int c = 0; c < d; ++c) oi[c] += p * vj[c];
    }
    for (int c = 0; c < d; ++c) oi[c] /= sum;
    lse[i] = m + log(sum);
    free(logit);
  }
}

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
