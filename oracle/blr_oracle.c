/*
 * Float64 CPU oracle for the BD-LRU scan of RecBLR (arXiv 2406.12580).
 *
 * TEST INFRASTRUCTURE ONLY. This file is the slow, serial, obviously-correct
 * statement of what the GPU path computes. Only the test suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it. It shares no
 * code, header or constant with the CUDA library, and the library never calls
 * it.
 *
 * Definitions (Sec. 3.2, the BD-LRU update and its gates), per batch row b,
 * time step t = 1..L and channel d:
 *   r_t     = sigmoid(rho_t)                       recurrence gate
 *   i_t     = sigmoid(iota_t)                      input gate
 *   alpha_t = exp(-c * softplus(Lambda) * r_t)     decay (c = 1 in the paper)
 *   beta_t  = sqrt(1 - alpha_t^2) * i_t            input normalisation
 *   h_t     = alpha_t * h_{t-1} + beta_t * x_t     the linear recurrence
 * with h_0 the initial state (zero in the paper, where h_1 = beta'_1; Sec. 3.3).
 *
 * The gate projections W_r x + b_r and W_i x + b_i are outside this path: rho
 * and iota arrive as pre-activation logits.
 *
 * Layouts (row-major, contiguous):
 *   x, h, dh, dx          (B, L, D)
 *   gl, dgl               (B, L, 2D): [.., 0:D] = rho, [.., D:2D] = iota
 *   lambda, dlambda       (D)
 *   h0, h_last, dh0, ...  (B, D)
 *
 * The gradient is not printed in the paper; it is the chain rule applied to the
 * definitions above, written out term by term (see blr_oracle_bwd). Finite
 * differences pin it in the tests.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double sigmoid(double z) { return 1.0 / (1.0 + exp(-z)); }

/* softplus(z) = log(1 + e^z), evaluated without overflow for large z. */
static double softplus(double z) {
  if (z > 0.0) return z + log1p(exp(-z));
  return log1p(exp(z));
}

/* Per-step gates of Sec. 3.2 for one (b, t, d). */
typedef struct {
  double r, i, alpha, beta;
} gates_t;

static gates_t step_gates(double c, double s, double rho, double iota) {
  gates_t g;
  g.r = sigmoid(rho);
  g.i = sigmoid(iota);
  g.alpha = exp(-c * s * g.r);
  g.beta = sqrt(1.0 - g.alpha * g.alpha) * g.i;
  return g;
}

static void set_threads(int nthreads) {
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
}

int blr_oracle_has_openmp(void) {
#ifdef _OPENMP
  return 1;
#else
  return 0;
#endif
}

/* alpha_t and beta_t for every (b, t, d): the pair c_t = (alpha_t, beta_t x_t)
 * of the scan formulation (Sec. 3.3) is (alpha, beta * x). Outputs (B, L, D). */
void blr_oracle_gates(int64_t B, int64_t L, int64_t D, double c, const double* gl,
                      const double* lambda, double* alpha, double* beta) {
  for (int64_t d = 0; d < D; ++d) {
    const double s = softplus(lambda[d]);
    for (int64_t b = 0; b < B; ++b)
      for (int64_t t = 0; t < L; ++t) {
        const int64_t row = b * L + t;
        gates_t g = step_gates(c, s, gl[row * 2 * D + d], gl[row * 2 * D + D + d]);
        alpha[row * D + d] = g.alpha;
        beta[row * D + d] = g.beta;
      }
  }
}

/* Forward scan (Sec. 3.2): serial recurrence per channel.
 * h0 may be NULL (zero initial state); h and h_last may be NULL. */
void blr_oracle_fwd(int64_t B, int64_t L, int64_t D, double c, const double* x, const double* gl,
                    const double* lambda, const double* h0, double* h, double* h_last,
                    int nthreads) {
  set_threads(nthreads);
  int64_t n = B * D;
#pragma omp parallel for schedule(static)
  for (int64_t bd = 0; bd < n; ++bd) {
    const int64_t b = bd / D, d = bd % D;
    const double s = softplus(lambda[d]);
    double state = h0 ? h0[b * D + d] : 0.0;
    for (int64_t t = 0; t < L; ++t) {
      const int64_t row = b * L + t;
      gates_t g = step_gates(c, s, gl[row * 2 * D + d], gl[row * 2 * D + D + d]);
      state = g.alpha * state + g.beta * x[row * D + d];
      if (h) h[row * D + d] = state;
    }
    if (h_last) h_last[b * D + d] = state;
  }
}

/* Backward of blr_oracle_fwd for the loss  sum_t <dh_t, h_t> + <dh_last, h_L>.
 *
 * With g_t the total derivative of the loss w.r.t. h_t,
 *   g_L = dh_L + dh_last,   g_t = dh_t + alpha_{t+1} g_{t+1},
 * and, from h_t = alpha_t h_{t-1} + sqrt(1 - alpha_t^2) i_t x_t,
 *   dh_t/dx_t      = beta_t
 *   dh_t/di_t      = sqrt(1 - alpha_t^2) x_t
 *   dh_t/dalpha_t  = h_{t-1} - alpha_t i_t x_t / sqrt(1 - alpha_t^2)
 *   dalpha_t/dr_t  = -c s alpha_t,   dalpha_t/ds = -c r_t alpha_t
 *   dr/drho = r (1 - r),  di/diota = i (1 - i),  ds/dLambda = sigmoid(Lambda)
 *   dh_t/dh_{t-1}  = alpha_t  (so dh0 = alpha_1 g_1).
 * Outputs: dx (B,L,D), dgl (B,L,2D), dlambda (D) and dh0 (B,D); h0, dh_last
 * and dh0 may be NULL. dlambda is written, not accumulated.
 *
 * The channel loop is parallel over d only, so each dlambda[d] is summed in a
 * fixed serial order (b outer, t inner, descending). */
void blr_oracle_bwd(int64_t B, int64_t L, int64_t D, double c, const double* dh,
                    const double* dh_last, const double* x, const double* gl,
                    const double* lambda, const double* h0, double* dx, double* dgl,
                    double* dlambda, double* dh0, int nthreads) {
  set_threads(nthreads);
#pragma omp parallel for schedule(static)
  for (int64_t d = 0; d < D; ++d) {
    const double s = softplus(lambda[d]);
    const double ds_dlambda = sigmoid(lambda[d]);
    double dlam = 0.0;
    for (int64_t b = 0; b < B; ++b) {
      /* Forward sweep: h_{t-1} for every t, parked in dx's slots (each slot is
       * overwritten with the real gradient by the reverse sweep below). */
      double state = h0 ? h0[b * D + d] : 0.0;
      for (int64_t t = 0; t < L; ++t) {
        const int64_t row = b * L + t;
        dx[row * D + d] = state; /* h_{t-1} */
        gates_t gt = step_gates(c, s, gl[row * 2 * D + d], gl[row * 2 * D + D + d]);
        state = gt.alpha * state + gt.beta * x[row * D + d];
      }
      /* Reverse sweep; g_next holds alpha_{t+1} g_{t+1} (dh_last at t = L). */
      double g_next = dh_last ? dh_last[b * D + d] : 0.0;
      for (int64_t t = L - 1; t >= 0; --t) {
        const int64_t row = b * L + t;
        const double hprev = dx[row * D + d];
        const double xt = x[row * D + d];
        gates_t gt = step_gates(c, s, gl[row * 2 * D + d], gl[row * 2 * D + D + d]);
        const double g = dh[row * D + d] + g_next;
        const double norm = sqrt(1.0 - gt.alpha * gt.alpha); /* sqrt(1 - alpha^2) */
        const double dh_dalpha = hprev - gt.alpha * gt.i * xt / norm;
        const double dL_dalpha = g * dh_dalpha;
        const double dL_dr = dL_dalpha * (-c * s * gt.alpha);
        const double dL_di = g * norm * xt;
        dx[row * D + d] = g * gt.beta;
        dgl[row * 2 * D + d] = dL_dr * gt.r * (1.0 - gt.r);
        dgl[row * 2 * D + D + d] = dL_di * gt.i * (1.0 - gt.i);
        dlam += dL_dalpha * (-c * gt.r * gt.alpha) * ds_dlambda;
        g_next = gt.alpha * g;
      }
      if (dh0) dh0[b * D + d] = g_next; /* alpha_1 g_1 */
    }
    dlambda[d] = dlam;
  }
}

/* The merge that follows the BD-LRU in the gated recurrent layer (Alg. 1,
 * H'_y = H_y (x) SiLU(H_z)): y = h * SiLU(z), SiLU(z) = z * sigmoid(z),
 * elementwise over n values. */
void blr_oracle_merge(int64_t n, const double* h, const double* z, double* y) {
  for (int64_t k = 0; k < n; ++k) y[k] = h[k] * (z[k] * sigmoid(z[k]));
}

/* Backward of blr_oracle_merge for the upstream gradient dy (chain rule):
 *   dh = dy * SiLU(z)
 *   dz = dy * h * SiLU'(z),  SiLU'(z) = sigmoid(z) * (1 + z * (1 - sigmoid(z))). */
void blr_oracle_merge_bwd(int64_t n, const double* dy, const double* h, const double* z,
                          double* dh, double* dz) {
  for (int64_t k = 0; k < n; ++k) {
    const double sg = sigmoid(z[k]);
    dh[k] = dy[k] * (z[k] * sg);
    dz[k] = dy[k] * h[k] * (sg * (1.0 + z[k] * (1.0 - sg)));
  }
}

/* One recurrent-inference step (low-cost inference, Sec. 1 and Sec. 4.3):
 * h_t = alpha_t h_prev + beta_t x_t for a batch of B states of width D.
 * x is (B, D), gl is (B, 2D). */
void blr_oracle_step(int64_t B, int64_t D, double c, const double* h_prev, const double* x,
                     const double* gl, const double* lambda, double* h_t) {
  for (int64_t b = 0; b < B; ++b)
    for (int64_t d = 0; d < D; ++d) {
      const double s = softplus(lambda[d]);
      gates_t g = step_gates(c, s, gl[b * 2 * D + d], gl[b * 2 * D + D + d]);
      h_t[b * D + d] = g.alpha * h_prev[b * D + d] + g.beta * x[b * D + d];
    }
}
