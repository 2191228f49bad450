/* A plain C (C11) client of the library: it uses only include/dard.h and the CUDA runtime's C
 * API, so it shows that the entry points are callable from C. It runs two cases whose
 * answers are known in closed form and returns 0 when every check passes.
 *
 * Scoring (Eq. 1, Eq. 8): four C rows whose shadow logits are 0 except one logit of 10.
 *   The confidence is e^10 / (e^10 + V - 1), the token is the planted one, and every row
 *   moves to U (the confidence is above tau_u).
 * Attention (Eq. 2, Sec. 3.2): one sequence of 8 rows with a block of 4 U positions and no
 *   shadow rows, so every query attends every row. With Q = 0 the softmax is uniform, and
 *   every output row is the mean of the V rows.
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include <cuda_runtime_api.h>

#include "dard.h"

static int failures = 0;

#define CHECK(cond, ...)                   \
  do {                                     \
    if (!(cond)) {                         \
      fprintf(stderr, "FAIL: " __VA_ARGS__); \
      fprintf(stderr, "\n");               \
      ++failures;                          \
    }                                      \
  } while (0)

#define CUDA(call)                                                          \
  do {                                                                      \
    cudaError_t e_ = (call);                                                \
    if (e_ != cudaSuccess) {                                                \
      fprintf(stderr, "CUDA error %s at %s\n", cudaGetErrorString(e_), #call); \
      return 2;                                                             \
    }                                                                       \
  } while (0)

static int score_case(void) {
  enum { B = 4, V = 1000 };
  const float big = 10.0f;
  float* h_logits = (float*)calloc((size_t)B * V, sizeof(float));
  uint8_t h_state[B] = {1, 1, 1, 1};
  for (int i = 0; i < B; ++i) h_logits[(size_t)i * V + 7 + i] = big;

  void *d_lx, *d_ls, *d_ws;
  uint8_t *d_state_in, *d_state_out;
  float* d_conf;
  int32_t *d_token, *d_counts;
  const size_t ws = dard_score_workspace_size(B, V, 1);
  CHECK(ws > 0, "workspace size %zu", ws);
  CUDA(cudaMalloc(&d_lx, (size_t)B * V * sizeof(float)));
  CUDA(cudaMalloc(&d_ls, (size_t)B * V * sizeof(float)));
  CUDA(cudaMalloc(&d_ws, ws));
  CUDA(cudaMemset(d_ws, 0, ws)); /* zero before the first use */
  CUDA(cudaMalloc((void**)&d_state_in, B));
  CUDA(cudaMalloc((void**)&d_state_out, B));
  CUDA(cudaMalloc((void**)&d_conf, B * sizeof(float)));
  CUDA(cudaMalloc((void**)&d_token, B * sizeof(int32_t)));
  CUDA(cudaMalloc((void**)&d_counts, 3 * sizeof(int32_t)));
  CUDA(cudaMemcpy(d_lx, h_logits, (size_t)B * V * sizeof(float), cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(d_ls, h_logits, (size_t)B * V * sizeof(float), cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(d_state_in, h_state, B, cudaMemcpyHostToDevice));

  const int32_t block_len[1] = {B};
  dard_score_args a = {0};
  a.logits_x = d_lx;
  a.logits_s = d_ls;
  a.dtype = DARD_F32;
  a.vocab = V;
  a.row_stride = V;
  a.num_seqs = 1;
  a.block_len = block_len;
  a.state_in = d_state_in;
  a.tau_c = 0.5f;
  a.tau_u = 0.8f;
  a.lambda = 0.917f;
  a.p0 = 0.1f;
  a.conf = d_conf;
  a.token = d_token;
  a.state_out = d_state_out;
  a.counts = d_counts;
  a.workspace = d_ws;
  a.workspace_bytes = ws;
  const dard_status st = dard_score_and_transition(&a, NULL);
  CHECK(st == DARD_OK, "dard_score_and_transition: %s (%s)", dard_status_string(st),
        dard_last_error());
  CUDA(cudaDeviceSynchronize());

  float conf[B];
  int32_t token[B], counts[3];
  uint8_t state_out[B];
  CUDA(cudaMemcpy(conf, d_conf, sizeof(conf), cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(token, d_token, sizeof(token), cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(state_out, d_state_out, sizeof(state_out), cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(counts, d_counts, sizeof(counts), cudaMemcpyDeviceToHost));
  const double want = exp((double)big) / (exp((double)big) + (V - 1));
  for (int i = 0; i < B; ++i) {
    CHECK(fabs(conf[i] - want) <= 1e-5, "row %d conf %.7f, want %.7f", i, conf[i], want);
    CHECK(token[i] == 7 + i, "row %d token %d, want %d", i, token[i], 7 + i);
    CHECK(state_out[i] == 2, "row %d state %d, want 2 (U)", i, state_out[i]);
  }
  CHECK(counts[0] == 0 && counts[1] == 0 && counts[2] == B, "counts %d %d %d", counts[0],
        counts[1], counts[2]);
  printf("score: conf %.7f (closed form %.7f), tokens %d..%d, counts %d/%d/%d\n", conf[0], want,
         token[0], token[B - 1], counts[0], counts[1], counts[2]);

  /* a NULL argument struct is rejected on the host, before any launch */
  CHECK(dard_score_and_transition(NULL, NULL) == DARD_ERR_NULL, "NULL args not rejected");

  cudaFree(d_lx);
  cudaFree(d_ls);
  cudaFree(d_ws);
  cudaFree(d_state_in);
  cudaFree(d_state_out);
  cudaFree(d_conf);
  cudaFree(d_token);
  cudaFree(d_counts);
  free(h_logits);
  return 0;
}

static int attention_case(void) {
  enum { N = 8, D = 64 };
  float h_q[N * D], h_v[N * D], h_o[N * D];
  for (int r = 0; r < N; ++r)
    for (int d = 0; d < D; ++d) {
      h_q[r * D + d] = 0.0f;
      h_v[r * D + d] = (float)((r * 7 + d * 3) % 11) - 5.0f;
    }
  const uint8_t h_state[4] = {2, 2, 2, 2};
  const float h_prev[4] = {0.9f, 0.9f, 0.9f, 0.9f};
  float *d_q, *d_k, *d_v, *d_o, *d_prev;
  uint8_t* d_state;
  int32_t* d_shadow;
  CUDA(cudaMalloc((void**)&d_q, sizeof(h_q)));
  CUDA(cudaMalloc((void**)&d_k, sizeof(h_q)));
  CUDA(cudaMalloc((void**)&d_v, sizeof(h_v)));
  CUDA(cudaMalloc((void**)&d_o, sizeof(h_o)));
  CUDA(cudaMalloc((void**)&d_prev, sizeof(h_prev)));
  CUDA(cudaMalloc((void**)&d_state, sizeof(h_state)));
  CUDA(cudaMalloc((void**)&d_shadow, sizeof(int32_t)));
  CUDA(cudaMemcpy(d_q, h_q, sizeof(h_q), cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(d_k, h_v, sizeof(h_v), cudaMemcpyHostToDevice));  /* any K: Q = 0 */
  CUDA(cudaMemcpy(d_v, h_v, sizeof(h_v), cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(d_prev, h_prev, sizeof(h_prev), cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(d_state, h_state, sizeof(h_state), cudaMemcpyHostToDevice));

  const int32_t n_orig[1] = {N}, block_start[1] = {4}, block_len[1] = {4}, shadow_len[1] = {0};
  dard_attn_args a = {0};
  a.q = d_q;
  a.k = d_k;
  a.v = d_v;
  a.o = d_o;
  a.dtype = DARD_F32;
  a.hq = 1;
  a.hkv = 1;
  a.head_dim = D;
  a.num_seqs = 1;
  a.n_orig = n_orig;
  a.block_start = block_start;
  a.block_len = block_len;
  a.shadow_len = shadow_len;
  a.state = d_state;
  a.prev_conf = d_prev;
  a.shadow_src = d_shadow;
  const dard_status st = dard_step_attention(&a, NULL);
  CHECK(st == DARD_OK, "dard_step_attention: %s (%s)", dard_status_string(st), dard_last_error());
  CUDA(cudaDeviceSynchronize());
  CUDA(cudaMemcpy(h_o, d_o, sizeof(h_o), cudaMemcpyDeviceToHost));
  double worst = 0.0;
  for (int d = 0; d < D; ++d) {
    double mean = 0.0;
    for (int r = 0; r < N; ++r) mean += h_v[r * D + d];
    mean /= N;
    for (int r = 0; r < N; ++r) {
      const double err = fabs(h_o[r * D + d] - mean);
      if (err > worst) worst = err;
    }
  }
  CHECK(worst <= 1e-5, "attention max |O - mean(V)| = %.3g", worst);
  printf("attention: max |O - mean(V)| = %.3g over %d rows\n", worst, N);

  /* head_dim outside {64, 128} is rejected on the host */
  a.head_dim = 96;
  CHECK(dard_step_attention(&a, NULL) == DARD_ERR_UNSUPPORTED, "head_dim 96 not rejected");

  cudaFree(d_q);
  cudaFree(d_k);
  cudaFree(d_v);
  cudaFree(d_o);
  cudaFree(d_prev);
  cudaFree(d_state);
  cudaFree(d_shadow);
  return 0;
}

int main(void) {
  printf("libdard version %d\n", (int)dard_version());
  if (score_case() != 0) return 2;
  if (attention_case() != 0) return 2;
  if (failures) {
    fprintf(stderr, "%d check(s) failed\n", failures);
    return 1;
  }
  printf("all checks passed\n");
  return 0;
}
