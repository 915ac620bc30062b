/* A plain C caller of the library (no Python, no torch): it includes only rl_loss.h and
 * links librl_loss.so. Argument "host" runs the host-side checks (argument checks and the host
 * prefix-tree builder on a worked example); argument "gpu" also runs
 * the advantages and the policy loss on a small batch whose result has a closed form:
 * uniform logits (all 0) give logp = -ln V for every token; with old_logp = logp the ratio
 * is 1, nothing is clipped, and the loss is -sum_i c_i L_i A_i, which is 0 for complete
 * groups under RL_AGG_SEQ_MEAN_TOKEN_MEAN; every trained gradient row is
 * -c_i A_i (onehot_a - 1/V); the fused head, the masked GAE and the value loss are checked
 * against closed forms too (gpu_checks_more). Exit status 0 on success. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "rl_loss.h"

/* The CUDA runtime calls this check needs, declared here so that the file needs no CUDA
 * header: they are resolved from libcudart at link time. */
typedef int cudaError_t;
extern cudaError_t cudaMalloc(void** p, size_t n);
extern cudaError_t cudaFree(void* p);
extern cudaError_t cudaMemcpy(void* dst, const void* src, size_t n, int kind);
extern cudaError_t cudaMemset(void* p, int v, size_t n);
enum { H2D = 1, D2H = 2 };

static int fails = 0;
#define CHECK(cond, ...)                      \
  do {                                        \
    if (!(cond)) {                            \
      fprintf(stderr, "FAIL: " __VA_ARGS__); \
      fprintf(stderr, "\n");                  \
      ++fails;                                \
    }                                         \
  } while (0)

static int host_checks(void) {
  CHECK(rl_version() >= 10000, "rl_version");
  CHECK(rl_workspace_size(0, 0, 0) == 256, "workspace header");
  CHECK(rl_workspace_size(16384, 151936, 0) == 256 + 16384 * 8, "workspace rows");
  rl_loss_params p;
  memset(&p, 0, sizeof p);
  p.clip_eps_low = 0.2f;
  p.clip_eps_high = 0.28f;
  p.adv_eps = 1e-6f;
  void* fake = (void*)(uintptr_t)0x10000;
  double* lacc = (double*)fake;
  /* a bad dtype, a misaligned gradient, a small workspace: errors before any launch */
  CHECK(rl_policy_loss_fwd_bwd(fake, (rl_dtype)7, 4, 8, 8, fake, fake, fake, 2, fake, fake, fake, NULL, NULL, &p,
                               fake, lacc, NULL, fake, 1 << 20, NULL) == RL_ERR_INVALID_ARG,
        "bad dtype");
  CHECK(rl_policy_loss_fwd_bwd(fake, RL_BF16, 4, 8, 8, fake, fake, fake, 2, fake, fake, fake, NULL, NULL, &p,
                               (char*)fake + 8, lacc, NULL, fake, 1 << 20, NULL) == RL_ERR_ALIGNMENT,
        "misaligned gradient");
  CHECK(rl_policy_loss_fwd_bwd(fake, RL_BF16, 4, 8, 8, fake, fake, fake, 2, fake, fake, fake, NULL, NULL, &p, fake,
                               lacc, NULL, fake, 100, NULL) == RL_ERR_WORKSPACE_TOO_SMALL,
        "small workspace");
  CHECK(strstr(rl_last_error_message(), "rl_policy_loss_fwd_bwd") != NULL, "error message");
  return fails;
}

/* The host prefix-tree builder on a worked example: prompt [1 2 3]; call 0 answers [10 11];
 * call 1 sees the tool output [20 21] after it and answers [30]; call 2 retries the first turn
 * (input [1 2 3]) with [12]. Call 0 and the retry form one segment; its longest leaf (call 1)
 * is kept, so the packed stream is [1 2 3 10 11 20 21 30] with mask 0 0 0 1 1 0 0 1, each token's
 * parent the previous position, 2 leaves in the tree and 1 kept. */
static int tree_checks(void) {
  const int64_t po[2] = {0, 3};
  const int32_t pt[3] = {1, 2, 3};
  const int32_t co[2] = {0, 3};
  const int64_t xo[4] = {0, 3, 10, 13};
  const int32_t xt[13] = {1, 2, 3, 1, 2, 3, 10, 11, 20, 21, 1, 2, 3};
  const int64_t yo[4] = {0, 2, 3, 4};
  const int32_t yt[4] = {10, 11, 30, 12};
  int64_t n = -1, ro[2], lo[2], parent[8], leaf_end[3];
  int32_t tokens[8], depth[8], owner[8], node_call[8], leaf_call[3];
  uint8_t mask[8];
  rl_tree_stats st;
  /* size query */
  CHECK(rl_prefix_tree_build_batch(1, po, pt, co, xo, xt, yo, yt, NULL, 0, 1, 0, NULL, NULL, NULL, NULL, NULL, NULL,
                                   NULL, NULL, NULL, NULL, NULL, &n) == RL_ERR_WORKSPACE_TOO_SMALL && n == 8,
        "tree size query: n = %lld", (long long)n);
  CHECK(rl_prefix_tree_build_batch(1, po, pt, co, xo, xt, yo, yt, NULL, 0, 1, 8, tokens, mask, parent, depth, owner,
                                   node_call, leaf_call, leaf_end, lo, &st, ro, &n) == RL_OK,
        "rl_prefix_tree_build_batch: %s", rl_last_error_message());
  const int32_t want_tok[8] = {1, 2, 3, 10, 11, 20, 21, 30};
  const uint8_t want_mask[8] = {0, 0, 0, 1, 1, 0, 0, 1};
  const int32_t want_call[8] = {-1, -1, -1, 0, 0, 1, 1, 1};
  for (int t = 0; t < 8; ++t) {
    CHECK(tokens[t] == want_tok[t] && mask[t] == want_mask[t], "tree token %d: %d/%d", t, tokens[t], mask[t]);
    CHECK(parent[t] == t - 1 && depth[t] == t && owner[t] == 0 && node_call[t] == want_call[t],
          "tree links of token %d: parent %lld depth %d owner %d call %d", t, (long long)parent[t], depth[t],
          owner[t], node_call[t]);
  }
  CHECK(st.valid == 1 && st.n_leaves == 2 && st.n_kept_leaves == 1 && st.n_unplaced == 0 && st.n_tokens == 8 &&
            st.n_trainable == 3,
        "tree stats: valid %d leaves %d kept %d unplaced %d tokens %lld trainable %lld", st.valid, st.n_leaves,
        st.n_kept_leaves, st.n_unplaced, (long long)st.n_tokens, (long long)st.n_trainable);
  CHECK(lo[0] == 0 && lo[1] == 1 && leaf_call[0] == 1 && leaf_end[0] == 7 && ro[0] == 0 && ro[1] == 8,
        "tree leaves: call %d end %lld", leaf_call[0], (long long)leaf_end[0]);
  return fails;
}

/* The advantages and the loss on uniform fp32 logits with old_logp = logp (-ln V), where the loss
 * is -sum_i c_i L_i A_i (0 for complete groups) and every trained gradient row is
 * -c_i A_i (onehot - 1/V); at V = 1,000 (rows of 4 KB: a warp per row) and V = 24,000 (rows of
 * 96 KB: clusters of CTAs). */
static int loss_checks(int V) {
  enum { G = 2, PER = 4, N = G * PER, LEN = 24, T = N * LEN };
  const int32_t go[G + 1] = {0, PER, 2 * PER};
  float rewards[N];
  int64_t offs[N + 1];
  uint8_t mask[T];
  int32_t ids[T];
  float old[T];
  int fails = 0;
  for (int i = 0; i < N; ++i) rewards[i] = (float)((i * 7) % 3);
  for (int i = 0; i <= N; ++i) offs[i] = (int64_t)i * LEN;
  for (int t = 0; t < T; ++t) {
    mask[t] = (uint8_t)((t % 5) != 0); /* every trajectory keeps trained tokens */
    ids[t] = (t * 37) % V;
    old[t] = (float)(-log((double)V));
  }
  rl_loss_params p;
  memset(&p, 0, sizeof p);
  p.clip_eps_low = 0.2f;
  p.clip_eps_high = 0.28f;
  p.adv_eps = 1e-6f;
  p.loss_agg = RL_AGG_SEQ_MEAN_TOKEN_MEAN;

  void *d_go, *d_rw, *d_offs, *d_mask, *d_ids, *d_old, *d_adv, *d_coef, *d_ntok, *d_tt, *d_logits, *d_grad, *d_loss,
      *d_ws;
  const size_t ws_bytes = rl_workspace_size(T, V, 0);
  int bad = 0;
  bad |= cudaMalloc(&d_go, sizeof go) | cudaMalloc(&d_rw, sizeof rewards) | cudaMalloc(&d_offs, sizeof offs);
  bad |= cudaMalloc(&d_mask, sizeof mask) | cudaMalloc(&d_ids, sizeof ids) | cudaMalloc(&d_old, sizeof old);
  bad |= cudaMalloc(&d_adv, N * 4) | cudaMalloc(&d_coef, N * 4) | cudaMalloc(&d_ntok, N * 4) | cudaMalloc(&d_tt, T * 4);
  bad |= cudaMalloc(&d_logits, (size_t)T * V * 4) | cudaMalloc(&d_grad, (size_t)T * V * 4);
  bad |= cudaMalloc(&d_loss, 8) | cudaMalloc(&d_ws, ws_bytes);
  if (bad) {
    fprintf(stderr, "FAIL: cudaMalloc\n");
    return 1;
  }
  cudaMemcpy(d_go, go, sizeof go, H2D);
  cudaMemcpy(d_rw, rewards, sizeof rewards, H2D);
  cudaMemcpy(d_offs, offs, sizeof offs, H2D);
  cudaMemcpy(d_mask, mask, sizeof mask, H2D);
  cudaMemcpy(d_ids, ids, sizeof ids, H2D);
  cudaMemcpy(d_old, old, sizeof old, H2D);
  cudaMemset(d_logits, 0, (size_t)T * V * 4); /* uniform rows */
  cudaMemset(d_loss, 0, 8);
  CHECK(rl_workspace_init(d_ws, ws_bytes, NULL) == RL_OK, "workspace init");
  CHECK(rl_group_advantages(N, G, d_go, d_rw, NULL, T, d_offs, d_mask, &p, d_adv, d_coef, d_ntok, d_tt, d_ws,
                            ws_bytes, NULL) == RL_OK,
        "rl_group_advantages: %s", rl_last_error_message());
  CHECK(rl_policy_loss_fwd_bwd(d_logits, RL_F32, T, V, V, d_ids, d_mask, d_tt, N, d_adv, d_coef, d_old, NULL, NULL,
                               &p, d_grad, d_loss, NULL, d_ws, ws_bytes, NULL) == RL_OK,
        "rl_policy_loss_fwd_bwd (V = %d): %s", V, rl_last_error_message());
  int32_t word = -1;
  CHECK(rl_query_status(d_ws, NULL, &word) == RL_OK && word == 0, "device status %d", word);

  float adv[N], coef[N];
  int32_t ntok[N];
  double loss = 0.0;
  cudaMemcpy(adv, d_adv, sizeof adv, D2H);
  cudaMemcpy(coef, d_coef, sizeof coef, D2H);
  cudaMemcpy(ntok, d_ntok, sizeof ntok, D2H);
  cudaMemcpy(&loss, d_loss, 8, D2H);
  double expect = 0.0, scale = 0.0;
  for (int i = 0; i < N; ++i) {
    expect -= (double)coef[i] * ntok[i] * adv[i];
    scale += fabs((double)coef[i] * ntok[i] * adv[i]);
  }
  CHECK(fabs(loss - expect) <= 1e-5 * scale + 1e-12, "V = %d: loss %.9g, closed form %.9g", V, loss, expect);
  CHECK(fabs(expect) <= 1e-6 * scale + 1e-12, "complete groups: the closed form is 0 (%.3g)", expect);
  /* gradient rows: -c A (onehot - 1/V) on trained tokens, zero elsewhere */
  float* row = (float*)malloc((size_t)V * sizeof(float));
  for (int t = 0; t < T; t += 7) {
    cudaMemcpy(row, (char*)d_grad + (size_t)t * V * 4, (size_t)V * sizeof(float), D2H);
    const int i = t / LEN;
    const double g = mask[t] ? -(double)coef[i] * adv[i] : 0.0;
    for (int v = 0; v < V; ++v) {
      const double ref = g * ((v == ids[t] ? 1.0 : 0.0) - 1.0 / V);
      if (fabs(row[v] - ref) > 1e-6 * fabs(g) + 1e-12) {
        fprintf(stderr, "FAIL: V = %d: grad[%d][%d] = %.9g, closed form %.9g\n", V, t, v, row[v], ref);
        ++fails;
        break;
      }
    }
  }
  free(row);
  void* all[] = {d_go, d_rw, d_offs, d_mask, d_ids, d_old, d_adv, d_coef, d_ntok, d_tt, d_logits, d_grad, d_loss, d_ws};
  for (size_t k = 0; k < sizeof all / sizeof all[0]; ++k) cudaFree(all[k]);
  return fails;
}

static int gpu_checks(void) { return loss_checks(1000) + loss_checks(24000); }

/* The fused head with all hidden states 0 (so every logits row is 0: uniform), the masked GAE at
 * gamma = lambda = 1 in the skip reading, and the value loss, each against its closed form:
 *   fused head: loss as above; dW = dZ^T H = 0 exactly; trained dH rows -c_i A_i (W[a] - mean_v W[v]);
 *   GAE: A_t = R_i - V_t and G_t = R_i on trainable tokens (Sec. 2.3.4), 0 on masked ones;
 *   value loss: sum_t c M (V_t - G_t)^2 and dV_t = 2 c M (V_t - G_t). */
static uint16_t bf16_bits(float x) { /* exact for the small multiples of 1/256 used here */
  uint32_t u;
  memcpy(&u, &x, 4);
  return (uint16_t)(u >> 16);
}

static int gpu_checks_more(void) {
  enum { G = 2, PER = 4, N = G * PER, LEN = 24, T = N * LEN, V = 1000, D = 64 };
  const int32_t go[G + 1] = {0, PER, 2 * PER};
  float rewards[N];
  int64_t offs[N + 1];
  uint8_t mask[T];
  int32_t ids[T];
  float old[T], values[T];
  for (int i = 0; i < N; ++i) rewards[i] = (float)((i * 7) % 3);
  for (int i = 0; i <= N; ++i) offs[i] = (int64_t)i * LEN;
  for (int t = 0; t < T; ++t) {
    mask[t] = (uint8_t)((t % 5) != 0);
    ids[t] = (t * 37) % V;
    old[t] = (float)(-log((double)V));
    values[t] = (float)((t * 13) % 29) / 32.0f;
  }
  uint16_t* w = (uint16_t*)malloc((size_t)V * D * 2);
  float* wf = (float*)malloc((size_t)V * D * 4);
  for (int v = 0; v < V; ++v)
    for (int d = 0; d < D; ++d) {
      wf[v * D + d] = (float)((v * 31 + d * 17) % 97 - 48) / 256.0f;
      w[v * D + d] = bf16_bits(wf[v * D + d]);
    }
  rl_loss_params p;
  memset(&p, 0, sizeof p);
  p.clip_eps_low = 0.2f;
  p.clip_eps_high = 0.28f;
  p.adv_eps = 1e-6f;
  p.loss_agg = RL_AGG_SEQ_MEAN_TOKEN_MEAN;

  void *d_go, *d_rw, *d_offs, *d_mask, *d_ids, *d_old, *d_adv, *d_coef, *d_ntok, *d_tt, *d_h, *d_w, *d_dh, *d_dw,
      *d_loss, *d_ws, *d_val, *d_gadv, *d_ret, *d_dv, *d_vloss;
  const size_t ws_bytes = rl_workspace_size(T, V, D);
  int bad = 0;
  bad |= cudaMalloc(&d_go, sizeof go) | cudaMalloc(&d_rw, sizeof rewards) | cudaMalloc(&d_offs, sizeof offs);
  bad |= cudaMalloc(&d_mask, sizeof mask) | cudaMalloc(&d_ids, sizeof ids) | cudaMalloc(&d_old, sizeof old);
  bad |= cudaMalloc(&d_adv, N * 4) | cudaMalloc(&d_coef, N * 4) | cudaMalloc(&d_ntok, N * 4) | cudaMalloc(&d_tt, T * 4);
  bad |= cudaMalloc(&d_h, (size_t)T * D * 2) | cudaMalloc(&d_w, (size_t)V * D * 2);
  bad |= cudaMalloc(&d_dh, (size_t)T * D * 4) | cudaMalloc(&d_dw, (size_t)V * D * 4);
  bad |= cudaMalloc(&d_loss, 8) | cudaMalloc(&d_ws, ws_bytes) | cudaMalloc(&d_val, T * 4);
  bad |= cudaMalloc(&d_gadv, T * 4) | cudaMalloc(&d_ret, T * 4) | cudaMalloc(&d_dv, T * 4) | cudaMalloc(&d_vloss, 8);
  if (bad) {
    fprintf(stderr, "FAIL: cudaMalloc\n");
    return 1;
  }
  cudaMemcpy(d_go, go, sizeof go, H2D);
  cudaMemcpy(d_rw, rewards, sizeof rewards, H2D);
  cudaMemcpy(d_offs, offs, sizeof offs, H2D);
  cudaMemcpy(d_mask, mask, sizeof mask, H2D);
  cudaMemcpy(d_ids, ids, sizeof ids, H2D);
  cudaMemcpy(d_old, old, sizeof old, H2D);
  cudaMemcpy(d_w, w, (size_t)V * D * 2, H2D);
  cudaMemcpy(d_val, values, sizeof values, H2D);
  cudaMemset(d_h, 0, (size_t)T * D * 2); /* zero hidden states: uniform logits */
  cudaMemset(d_dw, 0, (size_t)V * D * 4);
  cudaMemset(d_loss, 0, 8);
  cudaMemset(d_vloss, 0, 8);
  CHECK(rl_workspace_init(d_ws, ws_bytes, NULL) == RL_OK, "workspace init");
  CHECK(rl_group_advantages(N, G, d_go, d_rw, NULL, T, d_offs, d_mask, &p, d_adv, d_coef, d_ntok, d_tt, d_ws,
                            ws_bytes, NULL) == RL_OK,
        "rl_group_advantages: %s", rl_last_error_message());
  CHECK(rl_fused_head_loss_fwd_bwd(d_h, d_w, T, D, V, d_ids, d_mask, d_tt, N, d_adv, d_coef, d_old, NULL, NULL, &p,
                                   d_dh, RL_F32, d_dw, d_loss, NULL, d_ws, ws_bytes, NULL) == RL_OK,
        "rl_fused_head_loss_fwd_bwd: %s", rl_last_error_message());
  CHECK(rl_masked_gae(N, d_offs, T, d_mask, d_val, NULL, d_rw, 1.0f, 1.0f, 1, d_gadv, d_ret, d_ws, ws_bytes,
                      NULL) == RL_OK,
        "rl_masked_gae: %s", rl_last_error_message());
  CHECK(rl_value_loss_fwd_bwd(T, d_val, d_ret, d_mask, d_tt, N, d_coef, d_dv, d_vloss, d_ws, ws_bytes, NULL) == RL_OK,
        "rl_value_loss_fwd_bwd: %s", rl_last_error_message());
  int32_t word = -1;
  CHECK(rl_query_status(d_ws, NULL, &word) == RL_OK && word == 0, "device status %d", word);

  float adv[N], coef[N], gadv[T], ret[T], dv[T];
  int32_t ntok[N];
  double loss = 0.0, vloss = 0.0;
  float* dh = (float*)malloc((size_t)T * D * 4);
  float* dw = (float*)malloc((size_t)V * D * 4);
  cudaMemcpy(adv, d_adv, sizeof adv, D2H);
  cudaMemcpy(coef, d_coef, sizeof coef, D2H);
  cudaMemcpy(ntok, d_ntok, sizeof ntok, D2H);
  cudaMemcpy(&loss, d_loss, 8, D2H);
  cudaMemcpy(&vloss, d_vloss, 8, D2H);
  cudaMemcpy(dh, d_dh, (size_t)T * D * 4, D2H);
  cudaMemcpy(dw, d_dw, (size_t)V * D * 4, D2H);
  cudaMemcpy(gadv, d_gadv, sizeof gadv, D2H);
  cudaMemcpy(ret, d_ret, sizeof ret, D2H);
  cudaMemcpy(dv, d_dv, sizeof dv, D2H);

  /* fused head */
  double expect = 0.0, scale = 0.0;
  for (int i = 0; i < N; ++i) {
    expect -= (double)coef[i] * ntok[i] * adv[i];
    scale += fabs((double)coef[i] * ntok[i] * adv[i]);
  }
  CHECK(fabs(loss - expect) <= 1e-5 * scale + 1e-12, "fused head loss %.9g, closed form %.9g", loss, expect);
  int dw_nonzero = 0;
  for (size_t k = 0; k < (size_t)V * D; ++k) dw_nonzero += dw[k] != 0.0f;
  CHECK(dw_nonzero == 0, "dW must be exactly 0 with zero hidden states (%d nonzero)", dw_nonzero);
  double wmean[D], wabs = 0.0;
  for (int d = 0; d < D; ++d) {
    double m = 0.0;
    for (int v = 0; v < V; ++v) m += wf[v * D + d];
    wmean[d] = m / V;
  }
  for (size_t k = 0; k < (size_t)V * D; ++k) wabs += fabs(wf[k]);
  wabs /= (double)V * D;
  for (int t = 0; t < T; ++t) {
    const int i = t / LEN;
    const double g = mask[t] ? -(double)coef[i] * adv[i] : 0.0;
    for (int d = 0; d < D; ++d) {
      const double ref = g * (wf[ids[t] * D + d] - wmean[d]);
      /* dZ passes through two bf16 roundings (2^-8 each, relative) */
      const double tol = fabs(g) * (fabs(wf[ids[t] * D + d]) + wabs) * (1.0 / 64.0) + 1e-12;
      if (fabs(dh[t * D + d] - ref) > tol) {
        fprintf(stderr, "FAIL: dH[%d][%d] = %.9g, closed form %.9g (tol %.3g)\n", t, d, dh[t * D + d], ref, tol);
        ++fails;
        t = T;
        break;
      }
    }
  }
  /* GAE and value loss */
  double vexpect = 0.0, vscale = 0.0;
  for (int t = 0; t < T; ++t) {
    const int i = t / LEN;
    const double a_ref = mask[t] ? (double)rewards[i] - values[t] : 0.0;
    const double g_ref = mask[t] ? (double)rewards[i] : 0.0;
    if (fabs(gadv[t] - a_ref) > 1e-5 * (1.0 + fabs(a_ref)) || fabs(ret[t] - g_ref) > 1e-5 * (1.0 + fabs(g_ref))) {
      fprintf(stderr, "FAIL: GAE at %d: A %.9g (closed form %.9g), G %.9g (closed form %.9g)\n", t, gadv[t], a_ref,
              ret[t], g_ref);
      ++fails;
      break;
    }
    const double c = mask[t] ? coef[i] : 0.0, d = (double)values[t] - ret[t];
    vexpect += c * d * d;
    vscale += fabs(c * d * d);
    if (fabs(dv[t] - 2.0 * c * d) > 1e-6 * (fabs(2.0 * c * d) + 1e-6)) {
      fprintf(stderr, "FAIL: dV[%d] = %.9g, closed form %.9g\n", t, dv[t], 2.0 * c * d);
      ++fails;
      break;
    }
  }
  CHECK(fabs(vloss - vexpect) <= 1e-6 * vscale + 1e-12, "value loss %.9g, closed form %.9g", vloss, vexpect);

  free(dh);
  free(dw);
  free(w);
  free(wf);
  void* all[] = {d_go, d_rw, d_offs, d_mask, d_ids, d_old, d_adv, d_coef, d_ntok, d_tt, d_h, d_w, d_dh, d_dw,
                 d_loss, d_ws, d_val, d_gadv, d_ret, d_dv, d_vloss};
  for (size_t k = 0; k < sizeof all / sizeof all[0]; ++k) cudaFree(all[k]);
  return fails;
}

int main(int argc, char** argv) {
  int f = host_checks();
  f += tree_checks();
  if (argc > 1 && strcmp(argv[1], "gpu") == 0) f += gpu_checks() + gpu_checks_more();
  if (f == 0) printf("c_abi_check ok\n");
  return f == 0 ? 0 : 1;
}
