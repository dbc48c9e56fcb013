/*
 * P4Q oracle: a plain, slow CPU restatement of the pruned W4A4 hot path.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may link, load or call
 * this file; only the tests, the smoke check and the CPU-baseline leg of the
 * benchmark do. It shares no code, header or table with the CUDA library.
 *
 * What it computes (P4Q, Sec. 3.2 "Quantization-Aware Pre-LLM Selection",
 * Eq. 4, and App. A / App. B.3 for the W4A4 quantizer settings):
 *   - q4_quantize_rows: symmetric round-to-nearest 4-bit quantizer, one scale
 *     per row (per token for activations and selector copies, per output
 *     channel for weights), clip ratio 1.0, no groups.
 *   - q4_cosine: CosSim of two fake-quantized vectors s_a*c_a and s_b*c_b,
 *     evaluated on their integer codes (the positive scales cancel).
 *   - p4q_select_one: the three sequential selection stages of Eq. 4 (query
 *     relevance per concept, CLS saliency on the rest, greedy max-min
 *     diversity), then the retained indices in ascending order.
 *   - w4a4_gemm_s32 / w4a4_linear: the integer matmul of INT4 codes and the
 *     dequantization (acc * s_a) * s_w.
 *
 * Readings where the paper is silent (each is also listed in the design
 * notes):
 *   R1 quantizer arithmetic is IEEE fp32: a = max|x|, s = a / 7 (one rounded
 *      division), code = clamp(round_half_even(x / s), -8, 7) where x / s is
 *      one rounded fp32 division; a == 0 gives s = 0 and all codes 0.
 *   R2 the selector's fake quantizer is the deployment activation quantizer
 *      (4-bit, per token).
 *   R3 cosine := (float)dot / sqrtf((float)n_a * (float)n_b), every operation
 *      rounded to fp32 in that order, with n = sum of squared codes; 0 when
 *      n_a * n_b == 0.
 *   R4 budget split in integers: K_q = floor(alpha*K/1000),
 *      K_s = floor(beta*K/1000), K_d = K - K_q - K_s (alpha, beta in
 *      per mille); without concepts K_q moves to diversity, without CLS
 *      attention K_s moves to diversity.
 *   R5 query stage: concept j = 0..J-1 in order, quota
 *      floor(K_q/J) + (j < K_q mod J); each concept takes its best-scoring
 *      tokens not kept yet; ties go to the lower token index.
 *   R6 saliency stage: best A_cls among tokens not kept; ties to lower index.
 *   R7 diversity stage: m_i = max over kept r of cos(i, r), -inf when nothing
 *      is kept; pick argmin m_i (ties to lower index), keep it, repeat K_d
 *      times. Updating m_i with the newest pick equals recomputing the max
 *      over the whole kept set, because max is associative.
 *   R8 output indices are sorted ascending.
 *   R12 SwiGLU before down_proj (the decoder's MLP; the paper quantizes every
 *      linear's input per token): h = silu(gate) * up with silu(g) =
 *      g / (1 + e^-g), evaluated in float64 with the C library's exp and
 *      rounded once to fp32, then h quantized by R1. The paper fixes no
 *      SwiGLU arithmetic; this is the mathematical function, and a kernel
 *      that evaluates it in fp32 matches the codes except where the float64
 *      quotient h / s lies within its error bound of a .5 boundary.
 *   R13 RMSNorm before the quantized linears (the decoder's input norms feed
 *      q/k/v/gate/up; the paper quantizes every linear's input per token):
 *      S = sum x^2 exactly (fp16 squares are multiples of 2^-48; the sum is
 *      held as a 128-bit integer), rounded once to fp32; ms = S / d;
 *      r = 1 / sqrt(ms + eps) (r = 0 when ms + eps == 0); t = fp16(x * r);
 *      y = fp16(t * w) (every step one rounded fp32 or fp16 operation), then
 *      y quantized by R1.
 *   R14 attention on the pruned sequence (App. B: the key and value caches
 *      stay in FP16 while the linears run in W4A4): causal softmax attention
 *      of each of the m positions of a sample over positions 0..i, logits
 *      q . k / sqrt(d_h), heads sharing key/value heads in groups of H / H_kv
 *      (H_kv = H: one key/value head per head). Position encodings are
 *      applied by the caller. fp64 throughout.
 *   R15 calibration data path (Sec. 3.3, Eq. 5; App. A, Eq. 9): the block
 *      objective of a sample is the squared Frobenius distance of the W4A4 and
 *      full-precision block outputs over its m_n rows, divided by m_n d, and
 *      the batch objective their mean; the Top-K set of a score vector takes
 *      the K largest scores, ties to the lower index (as R8), and the
 *      replacement ratio is 1 - |T_ref & T_alt| / K, evaluated in fp32 from
 *      the integer intersection. fp64 sums.
 *   R11 CLS saliency (Sec. 3.2, Visual Saliency): in the vision tower's final
 *      self-attention, each crop's [CLS] token is the query; its attention
 *      row is the softmax, over the CLS key and the crop's patch keys, of
 *      q . k / sqrt(d_h); A_cls of a patch is that weight averaged over the
 *      heads. One CLS per crop (crops of N / C consecutive tokens). fp64.
 *
 * Build: plain C11, -O2 -ffp-contract=off (no fused multiply-add, no
 * fast-math), optional OpenMP over independent rows / images.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_BAD_ARG 1
#define ORACLE_OVERFLOW 2

int oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
  return omp_get_max_threads();
#else
  (void)n;
  return 1;
#endif
}

/* ------------------------------------------------------------------ */
/* Symmetric per-row 4-bit quantizer (App. A: symmetric round-to-nearest,  */
/* per-token activations / per-output-channel weights, group size -1,      */
/* clip ratio 1.0; App. B.3 repeats the settings). Reading R1.            */
/* ------------------------------------------------------------------ */
static void quantize_row(const float* x, int64_t cols, int8_t* code, float* scale) {
  float a = 0.0f;
  for (int64_t k = 0; k < cols; ++k) {
    float m = fabsf(x[k]);
    if (m > a) a = m;
  }
  if (a == 0.0f) {
    *scale = 0.0f;
    for (int64_t k = 0; k < cols; ++k) code[k] = 0;
    return;
  }
  float s = a / 7.0f;           /* one rounded fp32 division */
  for (int64_t k = 0; k < cols; ++k) {
    float q = x[k] / s;          /* one rounded fp32 division */
    float r = nearbyintf(q);     /* round half to even (default mode) */
    if (r < -8.0f) r = -8.0f;
    if (r > 7.0f) r = 7.0f;
    code[k] = (int8_t)r;
  }
  *scale = s;
}

int q4_quantize_rows(const float* x, int64_t rows, int64_t cols, int8_t* code, float* scale) {
  if (!x || !code || !scale || rows < 0 || cols <= 0) return ORACLE_BAD_ARG;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r)
    quantize_row(x + r * cols, cols, code + r * cols, scale + r);
  return ORACLE_OK;
}

/* Squared code norm n = sum c^2 (exact integer). */
static int64_t code_norm2(const int8_t* c, int64_t d) {
  int64_t n = 0;
  for (int64_t k = 0; k < d; ++k) n += (int64_t)c[k] * c[k];
  return n;
}

static int64_t code_dot(const int8_t* a, const int8_t* b, int64_t d) {
  int64_t g = 0;
  for (int64_t k = 0; k < d; ++k) g += (int64_t)a[k] * b[k];
  return g;
}

/* CosSim of fake-quantized vectors, Eq. 4; reading R3. */
static float cosine_from(int64_t dot, int64_t na, int64_t nb) {
  if (na == 0 || nb == 0) return 0.0f;
  float prod = (float)na * (float)nb;
  float den = sqrtf(prod);
  return (float)dot / den;
}

float q4_cosine(const int8_t* ca, const int8_t* cb, int64_t d) {
  return cosine_from(code_dot(ca, cb, d), code_norm2(ca, d), code_norm2(cb, d));
}

/* ------------------------------------------------------------------ */
/* Budget split (Sec. 3.2: alpha = 0.3, beta = 0.2, gamma = 0.5); R4.     */
/* ------------------------------------------------------------------ */
void p4q_budget(int K, int alpha_pm, int beta_pm, int have_q, int have_a, int* Kq, int* Ks, int* Kd) {
  int q = (int)(((int64_t)alpha_pm * K) / 1000);
  int s = (int)(((int64_t)beta_pm * K) / 1000);
  if (!have_q) q = 0;
  if (!have_a) s = 0;
  *Kq = q;
  *Ks = s;
  *Kd = K - q - s;
}

/* Pick the best not-kept token under score (higher better), lower index on ties. */
static int argbest_free(const float* score, const unsigned char* kept, int N) {
  int best = -1;
  for (int i = 0; i < N; ++i) {
    if (kept[i]) continue;
    if (best < 0 || score[i] > score[best]) best = i;
  }
  return best;
}

static int cmp_i32(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

/*
 * One image of the selector (Eq. 4 and the three stage paragraphs of
 * Sec. 3.2). V: [N, d] fp32 copies of fp16 features. Q: [J, d] or NULL.
 * A: [N] CLS saliency or NULL. Outputs:
 *   idx[K]          retained token indices, ascending (R8)
 *   order[K]        (optional) indices in the order they were kept
 *   stage[K]        (optional) 1 + concept j for query picks, -1 saliency,
 *                   -2 diversity, aligned with order[]
 */
int p4q_select_one(const float* V, int N, int d, const float* Q, int J, const float* A,
                   int K, int alpha_pm, int beta_pm, int32_t* idx, int32_t* order, int32_t* stage) {
  if (!V || N <= 0 || d <= 0 || K < 1 || K > N || !idx) return ORACLE_BAD_ARG;
  if (J < 0 || (J > 0 && !Q)) return ORACLE_BAD_ARG;
  int have_q = (Q != NULL && J > 0);
  int have_a = (A != NULL);
  int Kq, Ks, Kd;
  p4q_budget(K, alpha_pm, beta_pm, have_q, have_a, &Kq, &Ks, &Kd);
  if (Kq < 0 || Ks < 0 || Kd < 0) return ORACLE_BAD_ARG;

  /* Fake-quantized copies of the projector features and concept embeddings (R2). */
  int8_t* cv = (int8_t*)malloc((size_t)N * d);
  float* sv = (float*)malloc(sizeof(float) * N);
  int64_t* nv = (int64_t*)malloc(sizeof(int64_t) * N);
  unsigned char* kept = (unsigned char*)calloc(N, 1);
  float* score = (float*)malloc(sizeof(float) * N);
  int32_t* picks = (int32_t*)malloc(sizeof(int32_t) * K);
  int32_t* stg = (int32_t*)malloc(sizeof(int32_t) * K);
  if (!cv || !sv || !nv || !kept || !score || !picks || !stg) {
    free(cv); free(sv); free(nv); free(kept); free(score); free(picks); free(stg);
    return ORACLE_BAD_ARG;
  }
  for (int i = 0; i < N; ++i) {
    quantize_row(V + (int64_t)i * d, d, cv + (int64_t)i * d, sv + i);
    nv[i] = code_norm2(cv + (int64_t)i * d, d);
  }
  int nk = 0;

  /* Stage 1: query relevance, one ranking per concept (R5). */
  if (Kq > 0) {
    int8_t* cq = (int8_t*)malloc((size_t)d);
    float sq;
    for (int j = 0; j < J; ++j) {
      int quota = Kq / J + (j < Kq % J ? 1 : 0);
      quantize_row(Q + (int64_t)j * d, d, cq, &sq);
      int64_t nq = code_norm2(cq, d);
      for (int i = 0; i < N; ++i)
        score[i] = cosine_from(code_dot(cq, cv + (int64_t)i * d, d), nq, nv[i]);
      for (int t = 0; t < quota; ++t) {
        int b = argbest_free(score, kept, N);
        kept[b] = 1;
        picks[nk] = b;
        stg[nk] = 1 + j;
        ++nk;
      }
    }
    free(cq);
  }

  /* Stage 2: visual saliency on the tokens left by stage 1 (R6). */
  for (int t = 0; t < Ks; ++t) {
    int b = argbest_free(A, kept, N);
    kept[b] = 1;
    picks[nk] = b;
    stg[nk] = -1;
    ++nk;
  }

  /* Stage 3: greedy max-min diversity (R7). */
  if (Kd > 0) {
    float* m = score; /* reuse: m_i = max cosine to the kept set */
    for (int i = 0; i < N; ++i) {
      m[i] = -INFINITY;
      if (kept[i]) continue;
      for (int r = 0; r < nk; ++r) {
        int p = picks[r];
        float c = cosine_from(code_dot(cv + (int64_t)i * d, cv + (int64_t)p * d, d), nv[i], nv[p]);
        if (c > m[i]) m[i] = c;
      }
    }
    for (int t = 0; t < Kd; ++t) {
      int b = -1;
      for (int i = 0; i < N; ++i) {
        if (kept[i]) continue;
        if (b < 0 || m[i] < m[b]) b = i;
      }
      kept[b] = 1;
      picks[nk] = b;
      stg[nk] = -2;
      ++nk;
      for (int i = 0; i < N; ++i) {
        if (kept[i]) continue;
        float c = cosine_from(code_dot(cv + (int64_t)i * d, cv + (int64_t)b * d, d), nv[i], nv[b]);
        if (c > m[i]) m[i] = c;
      }
    }
  }

  for (int t = 0; t < K; ++t) {
    idx[t] = picks[t];
    if (order) order[t] = picks[t];
    if (stage) stage[t] = stg[t];
  }
  qsort(idx, (size_t)K, sizeof(int32_t), cmp_i32);
  free(cv); free(sv); free(nv); free(kept); free(score); free(picks); free(stg);
  return ORACLE_OK;
}

/* Batched selector: images are independent. */
int p4q_select_batch(const float* V, int B, int N, int d, const float* Q, int J, const float* A,
                     int K, int alpha_pm, int beta_pm, int32_t* idx) {
  if (B < 0) return ORACLE_BAD_ARG;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
  for (int b = 0; b < B; ++b) {
    const float* Qb = Q ? Q + (int64_t)b * J * d : NULL;
    const float* Ab = A ? A + (int64_t)b * N : NULL;
    bad |= p4q_select_one(V + (int64_t)b * N * d, N, d, Qb, J, Ab, K, alpha_pm, beta_pm,
                          idx + (int64_t)b * K, NULL, NULL);
  }
  return bad ? ORACLE_BAD_ARG : ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* W4A4 linear (App. B.3): integer matmul of the codes, then dequant.      */
/* ------------------------------------------------------------------ */
int w4a4_gemm_s32(const int8_t* a, const int8_t* w, int64_t M, int64_t N, int64_t K, int32_t* acc) {
  if (!a || !w || !acc || M < 0 || N < 0 || K <= 0) return ORACLE_BAD_ARG;
  int overflow = 0;
#pragma omp parallel for schedule(static) reduction(| : overflow)
  for (int64_t m = 0; m < M; ++m) {
    for (int64_t n = 0; n < N; ++n) {
      int64_t g = code_dot(a + m * K, w + n * K, K);
      if (g > INT32_MAX || g < INT32_MIN) overflow = 1;
      acc[m * N + n] = (int32_t)g;
    }
  }
  return overflow ? ORACLE_OVERFLOW : ORACLE_OK;
}

/* y[m, n] = ((float)acc * s_a[m]) * s_w[n], each product rounded to fp32. */
int w4a4_linear(const int8_t* a, const float* sa, const int8_t* w, const float* sw,
                int64_t M, int64_t N, int64_t K, float* y) {
  if (!sa || !sw || !y) return ORACLE_BAD_ARG;
  int32_t* acc = (int32_t*)malloc(sizeof(int32_t) * (size_t)(M * N > 0 ? M * N : 1));
  if (!acc) return ORACLE_BAD_ARG;
  int rc = w4a4_gemm_s32(a, w, M, N, K, acc);
  if (rc == ORACLE_OK) {
    for (int64_t m = 0; m < M; ++m)
      for (int64_t n = 0; n < N; ++n) {
        float t = (float)acc[m * N + n] * sa[m];
        y[m * N + n] = t * sw[n];
      }
  }
  free(acc);
  return rc;
}

/* Gather of the FP16 originals (Sec. 3.2: the originals, not the fake-quantized
 * copies, go to the language model): X = [V[idx]; text] per image. */
int p4q_gather(const float* V, int B, int N, int d, const int32_t* idx, int K, const float* text, int T,
               float* X) {
  if (!V || !idx || !X || B < 0 || K < 0 || T < 0 || (T > 0 && !text)) return ORACLE_BAD_ARG;
  for (int b = 0; b < B; ++b) {
    float* xb = X + (int64_t)b * (K + T) * d;
    for (int t = 0; t < K; ++t) {
      int i = idx[(int64_t)b * K + t];
      if (i < 0 || i >= N) return ORACLE_BAD_ARG;
      memcpy(xb + (int64_t)t * d, V + ((int64_t)b * N + i) * d, sizeof(float) * d);
    }
    for (int t = 0; t < T; ++t)
      memcpy(xb + (int64_t)(K + t) * d, text + ((int64_t)b * T + t) * d, sizeof(float) * d);
  }
  return ORACLE_OK;
}

/* CLS-to-patch saliency A_cls (Sec. 3.2, Visual Saliency; reading R11):
 *   q_cls, k_cls: [B, C, H, dh] (the final layer's CLS query and key of each
 *   crop, per head); k: [B, N, H, dh] (patch keys; crop c holds tokens
 *   [c * N / C, (c + 1) * N / C)); out A: [B, N]. For each image b, crop c,
 *   head h: logits l_0 = q . k_cls / sqrt(dh) and l_i = q . k_i / sqrt(dh)
 *   for the crop's patches, p = softmax over {l_0, l_i}, then
 *   A[b, i] = (1 / H) sum_h p_i. fp64 throughout. */
int p4q_cls_saliency(const float* q_cls, const float* k_cls, const float* k, int B, int N, int C, int H, int dh,
                     double* A) {
  if (!q_cls || !k_cls || !k || !A || B < 0 || N < 1 || C < 1 || N % C != 0 || H < 1 || dh < 1)
    return ORACLE_BAD_ARG;
  const int n = N / C;
  const double inv_sqrt = 1.0 / sqrt((double)dh);
  double* l = (double*)malloc(sizeof(double) * (size_t)(n + 1));
  if (!l) return ORACLE_BAD_ARG;
  for (int64_t i = 0; i < (int64_t)B * N; ++i) A[i] = 0.0;
  for (int b = 0; b < B; ++b) {
    for (int c = 0; c < C; ++c) {
      for (int h = 0; h < H; ++h) {
        const float* q = q_cls + (((int64_t)b * C + c) * H + h) * dh;
        const float* kc = k_cls + (((int64_t)b * C + c) * H + h) * dh;
        double dot = 0.0;
        for (int e = 0; e < dh; ++e) dot += (double)q[e] * (double)kc[e];
        l[0] = dot * inv_sqrt;
        for (int i = 0; i < n; ++i) {
          const float* ki = k + (((int64_t)b * N + (int64_t)c * n + i) * H + h) * dh;
          dot = 0.0;
          for (int e = 0; e < dh; ++e) dot += (double)q[e] * (double)ki[e];
          l[1 + i] = dot * inv_sqrt;
        }
        double mx = l[0];
        for (int i = 1; i <= n; ++i) mx = l[i] > mx ? l[i] : mx;
        double z = 0.0;
        for (int i = 0; i <= n; ++i) z += exp(l[i] - mx);
        for (int i = 0; i < n; ++i) A[(int64_t)b * N + (int64_t)c * n + i] += exp(l[1 + i] - mx) / z / (double)H;
      }
    }
  }
  free(l);
  return ORACLE_OK;
}

/* SwiGLU then the per-token quantizer (reading R12; the decoder MLP feeds
 * down_proj with silu(gate) * up, and App. A quantizes every linear input per
 * token): h = g / (1 + exp(-g)) * u in float64 with the C library's exp,
 * rounded once to fp32, then quantize_row (R1) on the fp32 row. gate, up:
 * [rows, cols] (fp16 values widened to fp32: exact). */
int p4q_swiglu_quantize_rows(const float* gate, const float* up, int64_t rows, int64_t cols, int8_t* code,
                             float* scale) {
  if (!gate || !up || !code || !scale || rows < 0 || cols <= 0) return ORACLE_BAD_ARG;
  int rc = ORACLE_OK;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    float* h = (float*)malloc(sizeof(float) * (size_t)cols);
    if (!h) {
      rc = ORACLE_BAD_ARG;
      continue;
    }
    for (int64_t k = 0; k < cols; ++k) {
      const double g = gate[r * cols + k];
      const double silu = g / (1.0 + exp(-g));
      h[k] = (float)(silu * (double)up[r * cols + k]);
    }
    quantize_row(h, cols, code + r * cols, scale + r);
    free(h);
  }
  return rc;
}

/* ------------------------------------------------------------------ */
/* RMSNorm then the per-token quantizer (reading R13).                   */
/* ------------------------------------------------------------------ */

/* fl32 of the exact sum of squares of fp16 values: |x| = k * 2^-24 with an
 * integer k < 2^40, so the sum is an integer count of 2^-48 held in 128 bits,
 * rounded once to 24 significant bits (to nearest, ties to even). Writes
 * ORACLE_BAD_ARG to *rc when some x is not an fp16 value. */
static float sumsq32(const float* x, int64_t n, int* rc) {
  unsigned __int128 S = 0;
  for (int64_t i = 0; i < n; ++i) {
    const double k = fabs((double)x[i]) * 16777216.0;
    if (!(k < 1099511627776.0) || k != floor(k)) {
      *rc = ORACLE_BAD_ARG;
      return 0.0f;
    }
    const uint64_t ki = (uint64_t)k;
    S += (unsigned __int128)ki * ki;
  }
  int L = 0;
  for (unsigned __int128 t = S; t != 0; t >>= 1) ++L;
  if (L <= 24) return ldexpf((float)(uint64_t)S, -48);
  const int sh = L - 24;
  uint64_t q = (uint64_t)(S >> sh);
  const unsigned __int128 rem = S - ((unsigned __int128)q << sh);
  const unsigned __int128 half = (unsigned __int128)1 << (sh - 1);
  if (rem > half || (rem == half && (q & 1u))) ++q;
  return ldexpf((float)q, sh - 48);
}

float oracle_sumsq32(const float* x, int64_t n) {
  int rc = ORACLE_OK;
  const float s = sumsq32(x, n, &rc);
  return rc == ORACLE_OK ? s : -1.0f;
}

static int rmsnorm_row(const float* x, const float* w, float eps, int64_t cols, float* y) {
  int rc = ORACLE_OK;
  const float S = sumsq32(x, cols, &rc);
  if (rc != ORACLE_OK) return rc;
  const float ms = S / (float)cols;
  const float den = ms + eps;
  const float r = den == 0.0f ? 0.0f : 1.0f / sqrtf(den);
  for (int64_t k = 0; k < cols; ++k) {
    const float t = (float)(_Float16)(x[k] * r);
    y[k] = (float)(_Float16)(t * w[k]);
  }
  return ORACLE_OK;
}

/* The normalized rows y (fp16 values, returned as fp32). x: [rows, cols] fp16
 * values, w: [cols] fp16 values (the norm's gain), eps >= 0. */
int p4q_rmsnorm_rows(const float* x, const float* w, float eps, int64_t rows, int64_t cols, float* y) {
  if (!x || !w || !y || rows < 0 || cols <= 0 || !(eps >= 0.0f)) return ORACLE_BAD_ARG;
  int rc = ORACLE_OK;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r)
    if (rmsnorm_row(x + r * cols, w, eps, cols, y + r * cols) != ORACLE_OK) rc = ORACLE_BAD_ARG;
  return rc;
}

/* RMSNorm then quantize_row on y: codes [rows, cols], scale [rows]. */
int p4q_rmsnorm_quantize_rows(const float* x, const float* w, float eps, int64_t rows, int64_t cols, int8_t* code,
                              float* scale) {
  if (!x || !w || !code || !scale || rows < 0 || cols <= 0 || !(eps >= 0.0f)) return ORACLE_BAD_ARG;
  int rc = ORACLE_OK;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    float* y = (float*)malloc(sizeof(float) * (size_t)cols);
    if (!y || rmsnorm_row(x + r * cols, w, eps, cols, y) != ORACLE_OK) {
      rc = ORACLE_BAD_ARG;
      free(y);
      continue;
    }
    quantize_row(y, cols, code + r * cols, scale + r);
    free(y);
  }
  return rc;
}

/* ------------------------------------------------------------------ */
/* Causal attention on the pruned sequence (reading R14).                 */
/* ------------------------------------------------------------------ */

/* q [B*m, H*dh], k and v [B*m, Hkv*dh] (rows of consecutive positions of one
 * sample, head h in columns h*dh .. h*dh + dh - 1), o [B*m, H*dh]:
 *   o_i = sum_{j <= i} p_ij v_j, p_i. = softmax_j(q_i . k_j / sqrt(dh)),
 * with key/value head h / (H / Hkv) for head h. fp64. */
int p4q_causal_attention(const float* q, const float* k, const float* v, int B, int m, int H, int Hkv, int dh,
                         double* o) {
  if (!q || !k || !v || !o || B < 0 || m < 1 || H < 1 || Hkv < 1 || H % Hkv != 0 || dh < 1) return ORACLE_BAD_ARG;
  const double inv_sqrt = 1.0 / sqrt((double)dh);
  const int64_t ldq = (int64_t)H * dh, ldk = (int64_t)Hkv * dh;
  int rc = ORACLE_OK;
#pragma omp parallel for collapse(2) schedule(static)
  for (int b = 0; b < B; ++b) {
    for (int h = 0; h < H; ++h) {
      const int hk = h / (H / Hkv);
      double* l = (double*)malloc(sizeof(double) * (size_t)m);
      if (!l) {
        rc = ORACLE_BAD_ARG;
        continue;
      }
      for (int i = 0; i < m; ++i) {
        const float* qi = q + ((int64_t)b * m + i) * ldq + (int64_t)h * dh;
        double mx = -INFINITY;
        for (int j = 0; j <= i; ++j) {
          const float* kj = k + ((int64_t)b * m + j) * ldk + (int64_t)hk * dh;
          double dot = 0.0;
          for (int e = 0; e < dh; ++e) dot += (double)qi[e] * (double)kj[e];
          l[j] = dot * inv_sqrt;
          if (l[j] > mx) mx = l[j];
        }
        double z = 0.0;
        for (int j = 0; j <= i; ++j) {
          l[j] = exp(l[j] - mx);
          z += l[j];
        }
        double* oi = o + ((int64_t)b * m + i) * ldq + (int64_t)h * dh;
        for (int e = 0; e < dh; ++e) oi[e] = 0.0;
        for (int j = 0; j <= i; ++j) {
          const float* vj = v + ((int64_t)b * m + j) * ldk + (int64_t)hk * dh;
          const double p = l[j] / z;
          for (int e = 0; e < dh; ++e) oi[e] += p * (double)vj[e];
        }
      }
      free(l);
    }
  }
  return rc;
}

/* ------------------------------------------------------------------ */
/* Pruning-aware calibration data path (reading R15).                   */
/* ------------------------------------------------------------------ */

/* Eq. 5's block objective: sample n owns rows off[n] .. off[n+1]-1 of the
 * W4A4 block output Yq and the full-precision output Yf (d columns each);
 * e[n] = sum (Yq - Yf)^2 / (m_n d), *L = (1/B) sum_n e[n]. fp64. */
int p4q_block_mse(const float* Yq, const float* Yf, const int32_t* off, int B, int d, double* e, double* L) {
  if (!Yq || !Yf || !off || !e || !L || B < 1 || d < 1 || off[0] != 0) return ORACLE_BAD_ARG;
  double tot = 0.0;
  for (int n = 0; n < B; ++n) {
    const int64_t r0 = off[n], r1 = off[n + 1];
    if (r1 <= r0) return ORACLE_BAD_ARG;
    double acc = 0.0;
    for (int64_t i = r0 * d; i < r1 * d; ++i) {
      const double diff = (double)Yq[i] - (double)Yf[i];
      acc += diff * diff;
    }
    e[n] = acc / ((double)(r1 - r0) * (double)d);
    tot += e[n];
  }
  *L = tot / (double)B;
  return ORACLE_OK;
}

/* Token i belongs to the Top-K set of s when fewer than K tokens rank above
 * it: a larger score, or an equal score at a lower index. */
static int in_topk(const float* s, int N, int K, int i) {
  int above = 0;
  for (int j = 0; j < N; ++j)
    if (s[j] > s[i] || (s[j] == s[i] && j < i)) ++above;
  return above < K;
}

/* Eq. 9's replacement ratio per sample: s_ref, s_alt [B, N] scores of the
 * same tokens under two precisions; inter[b] = |T_ref & T_alt|,
 * rho[b] = 1 - inter[b] / K (fp32 division and subtraction). */
int p4q_topk_replacement(const float* s_ref, const float* s_alt, int B, int N, int K, int32_t* inter, float* rho) {
  if (!s_ref || !s_alt || !inter || !rho || B < 0 || N < 1 || K < 1 || K > N) return ORACLE_BAD_ARG;
#pragma omp parallel for schedule(static)
  for (int b = 0; b < B; ++b) {
    const float* r = s_ref + (int64_t)b * N;
    const float* a = s_alt + (int64_t)b * N;
    int c = 0;
    for (int i = 0; i < N; ++i)
      if (in_topk(r, N, K, i) && in_topk(a, N, K, i)) ++c;
    inter[b] = c;
    rho[b] = 1.0f - (float)c / (float)K;
  }
  return ORACLE_OK;
}
