/*
 * CPU oracle for the schedule-parameterised tensor programs.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path (the CUDA library and
 * its Python binding) may call, link or load this file. Only the tests, the
 * smoke check and the bench's CPU-baseline leg use it.
 *
 * Every function is the plain definition of its operator, written as fp64
 * loop nests over inputs widened exactly from bf16 / fp32. The paper defines
 * every schedule transformation as semantics preserving (Sec. 2, Eq. 1), so
 * the output of any legal schedule must equal this definition up to floating
 * point reassociation and the storage precision of the outputs.
 *
 * Parallelism: OpenMP over the outermost output dimension only. Each output
 * element is reduced by one thread in a fixed order, so results do not
 * depend on the thread count.
 *
 * Conventions: row-major contiguous; bf16 tensors are uint16 bit patterns;
 * linear weights are [out][in].
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

#define EXPORT __attribute__((visibility("default")))

/* Thread count of the OpenMP loops (n > 0 sets it); returns the count now in
 * effect, 1 when built without OpenMP. Results do not depend on it. */
EXPORT int oracle_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
  return omp_get_max_threads();
#else
  (void)n;
  return 1;
#endif
}

static double bf(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* fp64 -> fp32 (round to nearest even) -> bf16 (round to nearest even).
 * Only used by the optional "round the intermediate to bf16" flag. */
static double round_bf16(double x) {
  float f = (float)x;
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) != 0x7F800000u) u = (u + 0x7FFFu + ((u >> 16) & 1u)) & 0xFFFF0000u;
  memcpy(&f, &u, 4);
  return (double)f;
}

static double silu(double x) { return x / (1.0 + exp(-x)); }

/* ------------------------------------------------------------------ K0 ---
 * fp32 GEMM with bias and ReLU. This is the loop nest of the paper's App. A
 * example (C[i,j] initialised to 0, then C[i,j] += A[i,k] * B[k,j]) with a
 * bias added along j and an optional ReLU:
 *   C[i,j] = max(0, bias[j] + sum_k A[i,k] B[k,j]).
 * A[M][K], B[K][N] (row-major, B indexed [k][j] as in App. A), bias[N] or NULL.
 */
EXPORT void oracle_gemm_bias_relu_f32(int64_t M, int64_t N, int64_t K, const float* A,
                                      const float* B, const float* bias, int relu, double* C) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < M; ++i) {
    for (int64_t j = 0; j < N; ++j) {
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k) acc += (double)A[i * K + k] * (double)B[k * N + j];
      if (bias) acc += (double)bias[j];
      if (relu && acc < 0.0) acc = 0.0;
      C[i * N + j] = acc;
    }
  }
}

/* ------------------------------------------------------------- linear ---
 * Y[r,n] = sum_k X[rows[r],k] W[n,k] for the requested rows (all rows when
 * rows == NULL, nrows = M). X[M][K], W[N][K] bf16; Y[nrows][N] fp64.
 */
EXPORT void oracle_linear_bf16(int64_t M, int64_t N, int64_t K, const uint16_t* X,
                               const uint16_t* W, const int64_t* rows, int64_t nrows, double* Y) {
  (void)M;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < nrows; ++r) {
    const int64_t i = rows ? rows[r] : r;
    const uint16_t* x = X + i * K;
    for (int64_t n = 0; n < N; ++n) {
      const uint16_t* w = W + n * K;
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k) acc += bf(x[k]) * bf(w[k]);
      Y[r * N + n] = acc;
    }
  }
}

/* --------------------------------------------------- K1a gate/up SwiGLU ---
 * h[r,n] = silu(g) * u with g = sum_k X[i,k] W1[n,k] (gate rows 0..I-1) and
 * u = sum_k X[i,k] W1[I+n,k] (up rows I..2I-1), silu(x) = x / (1 + e^-x).
 * X[M][K], W1[2I][K] bf16; h[nrows][I]. round_h: round h to bf16.
 */
EXPORT void oracle_swiglu_bf16(int64_t M, int64_t I, int64_t K, const uint16_t* X,
                               const uint16_t* W1, const int64_t* rows, int64_t nrows, int round_h,
                               double* h) {
  (void)M;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < nrows; ++r) {
    const int64_t i = rows ? rows[r] : r;
    const uint16_t* x = X + i * K;
    for (int64_t n = 0; n < I; ++n) {
      const uint16_t* wg = W1 + n * K;
      const uint16_t* wu = W1 + (I + n) * K;
      double g = 0.0, u = 0.0;
      for (int64_t k = 0; k < K; ++k) {
        g += bf(x[k]) * bf(wg[k]);
        u += bf(x[k]) * bf(wu[k]);
      }
      double v = silu(g) * u;
      h[r * I + n] = round_h ? round_bf16(v) : v;
    }
  }
}

/* ------------------------------------------------------- K1 MLP block ---
 * Y = (silu(X W_g^T) * (X W_u^T)) W2^T for the requested token rows.
 * X[T][H], W1[2I][H], W2[H][I] bf16; Y[nrows][H] fp64.
 * round_h = 0 keeps the intermediate in fp64; 1 rounds it to bf16 first.
 */
EXPORT void oracle_mlp_bf16(int64_t T, int64_t H, int64_t I, const uint16_t* X, const uint16_t* W1,
                            const uint16_t* W2, const int64_t* rows, int64_t nrows, int round_h,
                            double* Y) {
  (void)T;
  double* hbuf = (double*)malloc(sizeof(double) * (size_t)I * (size_t)(nrows > 0 ? nrows : 1));
  oracle_swiglu_bf16(T, I, H, X, W1, rows, nrows, round_h, hbuf);
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < nrows; ++r) {
    const double* hr = hbuf + r * I;
    for (int64_t n = 0; n < H; ++n) {
      const uint16_t* w = W2 + n * I;
      double acc = 0.0;
      for (int64_t k = 0; k < I; ++k) acc += hr[k] * bf(w[k]);
      Y[r * H + n] = acc;
    }
  }
  free(hbuf);
}

/* --------------------------------------------------- K2 GQA attention ---
 * For batch b, query position i and query head h, with KV head
 * g = h / (Hq / Hkv) (contiguous head groups):
 *   s_j = scale * sum_d Q[b,i,h,d] K[b,j,g,d]   for j <= i (causal) or all j,
 *   m = max_j s_j,  l = sum_j exp(s_j - m),
 *   O[b,i,h,:] = sum_j exp(s_j - m) V[b,j,g,:] / l,  LSE[b,h,i] = m + ln l.
 * Q[B][S][Hq][D], K/V[B][S][Hkv][D] bf16 (BSHD). Query positions: qpos[nq]
 * (all S when NULL). O[B][nq][Hq][D] fp64, lse[B][Hq][nq] fp64 (may be NULL).
 */
EXPORT void oracle_attention_bf16(int64_t B, int64_t S, int64_t Hq, int64_t Hkv, int64_t D,
                                  const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                                  int causal, double scale, const int64_t* qpos, int64_t nq,
                                  double* O, double* lse) {
  const int64_t group = Hq / Hkv;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
  for (int64_t b = 0; b < B; ++b) {
    for (int64_t r = 0; r < nq; ++r) {
      const int64_t i = qpos ? qpos[r] : r;
      const int64_t nkeys = causal ? i + 1 : S;
      double* s = (double*)malloc(sizeof(double) * (size_t)nkeys);
      for (int64_t h = 0; h < Hq; ++h) {
        const int64_t g = h / group;
        const uint16_t* q = Q + ((b * S + i) * Hq + h) * D;
        double m = -INFINITY;
        for (int64_t j = 0; j < nkeys; ++j) {
          const uint16_t* kr = K + ((b * S + j) * Hkv + g) * D;
          double acc = 0.0;
          for (int64_t d = 0; d < D; ++d) acc += bf(q[d]) * bf(kr[d]);
          s[j] = acc * scale;
          if (s[j] > m) m = s[j];
        }
        double l = 0.0;
        for (int64_t j = 0; j < nkeys; ++j) {
          s[j] = exp(s[j] - m);
          l += s[j];
        }
        double* o = O + ((b * nq + r) * Hq + h) * D;
        for (int64_t d = 0; d < D; ++d) {
          double acc = 0.0;
          for (int64_t j = 0; j < nkeys; ++j) acc += s[j] * bf(V[((b * S + j) * Hkv + g) * D + d]);
          o[d] = acc / l;
        }
        if (lse) lse[(b * Hq + h) * nq + r] = m + log(l);
      }
      free(s);
    }
  }
}

/* ------------------------------------------------------ K3 conv2d NHWC ---
 * y[n,p,q,co] = act(bias[co] + sum_{r,s,ci} x[n, p*st + r - pad, q*st + s - pad, ci] w[co,r,s,ci])
 * with zero padding outside the image. x[N][H][W][Cin] (NHWC), w[Cout][R][S][Cin]
 * (KRSC), bias[Cout] (may be NULL), act: 0 = identity, 1 = SiLU.
 * Output pixels: pix[npix] flat indices over (n, p, q) of the [N][P][Q] output
 * grid (all when NULL). y[npix][Cout] fp64.
 */
EXPORT void oracle_conv2d_nhwc_bf16(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                                    int64_t R, int64_t S, int64_t stride, int64_t pad,
                                    const uint16_t* x, const uint16_t* w, const uint16_t* bias,
                                    int act, const int64_t* pix, int64_t npix, double* y) {
  const int64_t P = (H + 2 * pad - R) / stride + 1;
  const int64_t Qo = (W + 2 * pad - S) / stride + 1;
  (void)N;
#pragma omp parallel for schedule(dynamic, 4)
  for (int64_t t = 0; t < npix; ++t) {
    const int64_t flat = pix ? pix[t] : t;
    const int64_t n = flat / (P * Qo);
    const int64_t p = (flat / Qo) % P;
    const int64_t q = flat % Qo;
    for (int64_t co = 0; co < Cout; ++co) {
      double acc = 0.0;
      for (int64_t r = 0; r < R; ++r) {
        const int64_t ih = p * stride + r - pad;
        if (ih < 0 || ih >= H) continue;
        for (int64_t s = 0; s < S; ++s) {
          const int64_t iw = q * stride + s - pad;
          if (iw < 0 || iw >= W) continue;
          const uint16_t* xr = x + ((n * H + ih) * W + iw) * Cin;
          const uint16_t* wr = w + ((co * R + r) * S + s) * Cin;
          for (int64_t ci = 0; ci < Cin; ++ci) acc += bf(xr[ci]) * bf(wr[ci]);
        }
      }
      if (bias) acc += bf(bias[co]);
      if (act == 1) acc = silu(acc);
      y[t * Cout + co] = acc;
    }
  }
}

/* -------------------------------------------------------- K4a routing ---
 * Per token t over E experts, with logits l (bf16 bits when logits_fp32 == 0,
 * float32 otherwise):
 *   p_e = exp(l_e - max l) / sum_e' exp(l_e' - max l)       (softmax over all E)
 *   ids[t,0..k-1] = the k experts ordered by (logit descending, id ascending)
 *   w[t,j] = p_{ids[t,j]} / sum_j' p_{ids[t,j']}   (renorm = 1) or p_{ids[t,j]}.
 * Selection compares logit values only. counts[e] = number of (t, j) routed
 * to e; offsets[E+1] is its exclusive scan; perm[T*k] lists the slots
 * s = t*k + j ordered by (expert, token, j).
 * A NaN logit has no place in that order; it is read as -inf, so it ranks
 * below every number (ties among such experts go to the lower id) and its
 * softmax probability is 0.
 */
EXPORT void oracle_moe_route(int64_t T, int64_t E, int64_t topk, const void* logits, int logits_fp32,
                             int renorm, int32_t* ids, double* w, int32_t* offsets, int32_t* perm) {
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    double* l = (double*)malloc(sizeof(double) * (size_t)E);
    char* taken = (char*)calloc((size_t)E, 1);
    for (int64_t e = 0; e < E; ++e) {
      l[e] = logits_fp32 ? (double)((const float*)logits)[t * E + e]
                         : bf(((const uint16_t*)logits)[t * E + e]);
      if (isnan(l[e])) l[e] = -INFINITY;
    }
    double mx = -INFINITY;
    for (int64_t e = 0; e < E; ++e)
      if (l[e] > mx) mx = l[e];
    double z = 0.0;
    for (int64_t e = 0; e < E; ++e) z += exp(l[e] - mx);
    double sel = 0.0;
    for (int64_t j = 0; j < topk; ++j) {
      int64_t best = -1;
      for (int64_t e = 0; e < E; ++e) {
        if (taken[e]) continue;
        if (best < 0 || l[e] > l[best]) best = e; /* strict >: equal logits keep the lower id */
      }
      taken[best] = 1;
      ids[t * topk + j] = (int32_t)best;
      w[t * topk + j] = exp(l[best] - mx) / z;
      sel += w[t * topk + j];
    }
    if (renorm)
      for (int64_t j = 0; j < topk; ++j) w[t * topk + j] /= sel;
    free(taken);
    free(l);
  }
  int64_t pos = 0;
  for (int64_t e = 0; e < E; ++e) {
    offsets[e] = (int32_t)pos;
    for (int64_t t = 0; t < T; ++t)
      for (int64_t j = 0; j < topk; ++j)
        if (ids[t * topk + j] == e) perm[pos++] = (int32_t)(t * topk + j);
  }
  offsets[E] = (int32_t)pos;
}

/* ---------------------------------------------------------- K4 MoE FFN ---
 * out[t] = sum_{j=0..k-1} w[t,j] * Y_{ids[t,j]}(x_t), summed in j order, with
 *   Y_e(x) = W2_e (silu(W1_e[0:I] x) * (W1_e[I:2I] x)).
 * X[T][H], W1[E][2I][H], W2[E][H][I] bf16; ids[T][k], w[T][k] from routing.
 * Tokens: tok[ntok] (all when NULL); out[ntok][H] fp64. round_h rounds the
 * SwiGLU intermediate to bf16.
 */
EXPORT void oracle_moe_ffn_bf16(int64_t T, int64_t H, int64_t E, int64_t I, int64_t topk,
                                const uint16_t* X, const uint16_t* W1, const uint16_t* W2,
                                const int32_t* ids, const double* w, const int64_t* tok,
                                int64_t ntok, int round_h, double* out) {
  (void)T;
  (void)E;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < ntok; ++r) {
    const int64_t t = tok ? tok[r] : r;
    const uint16_t* x = X + t * H;
    double* h = (double*)malloc(sizeof(double) * (size_t)I);
    double* o = out + r * H;
    for (int64_t n = 0; n < H; ++n) o[n] = 0.0;
    for (int64_t j = 0; j < topk; ++j) {
      const int64_t e = ids[t * topk + j];
      const uint16_t* w1 = W1 + e * 2 * I * H;
      const uint16_t* w2 = W2 + e * H * I;
      for (int64_t n = 0; n < I; ++n) {
        double g = 0.0, u = 0.0;
        for (int64_t k = 0; k < H; ++k) {
          g += bf(x[k]) * bf(w1[n * H + k]);
          u += bf(x[k]) * bf(w1[(I + n) * H + k]);
        }
        double v = silu(g) * u;
        h[n] = round_h ? round_bf16(v) : v;
      }
      const double wt = w[t * topk + j];
      for (int64_t n = 0; n < H; ++n) {
        double acc = 0.0;
        for (int64_t k = 0; k < I; ++k) acc += h[k] * bf(w2[n * I + k]);
        o[n] += wt * acc;
      }
    }
    free(h);
  }
}
