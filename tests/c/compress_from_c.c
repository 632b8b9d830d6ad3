/* The C ABI used from plain C (no Python, no PyTorch): one small stepkv_compress call.
 *
 *   compress_from_c host        argument checks and defaults only (no GPU needed)
 *   compress_from_c gpu DIR     a 2-layer problem with deterministic inputs; writes the inputs and the
 *                               outputs to DIR as raw little-endian arrays for the test to check
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "stepkv.h"

enum { L = 2, HKV = 2, HQ = 8, D = 64, T = 1000, W = 16, NSTEPS = 5, NSAL = 2 };

static uint32_t lcg_state = 12345u;
static float lcg_uniform(void) {
  lcg_state = lcg_state * 1664525u + 1013904223u;
  return (float)(lcg_state >> 8) * (1.0f / 16777216.0f);
}
/* bf16 bits of x (round to nearest even) */
static uint16_t to_bf16(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

static int write_file(const char* dir, const char* name, const void* p, size_t n) {
  char path[1024];
  snprintf(path, sizeof(path), "%s/%s", dir, name);
  FILE* f = fopen(path, "wb");
  if (!f) return 1;
  const size_t w = fwrite(p, 1, n, f);
  fclose(f);
  return w == n ? 0 : 1;
}

#define CK(x)                                                     \
  do {                                                            \
    cudaError_t e_ = (x);                                         \
    if (e_ != cudaSuccess) {                                      \
      fprintf(stderr, "CUDA error %d at line %d\n", (int)e_, __LINE__); \
      return 2;                                                   \
    }                                                             \
  } while (0)

static int host_mode(void) {
  stepkv_params_t p;
  stepkv_default_params(&p);
  printf("params %.3f %.3f %.3f %.3f %.3f %.3f %.3f %.3f %.3f %d\n", p.lambda, p.w_r, p.w_c, p.r_min,
         p.r_max, p.s_max, p.eta, p.alpha, p.beta, p.sal_norm);
  printf("status %s\n", stepkv_status_string(STEPKV_EINVAL));
  /* a null problem array is refused before anything is enqueued */
  printf("compress_null %d\n", (int)stepkv_compress(NULL, 1, &p, NULL, 0, NULL, NULL));
  stepkv_problem_t prob;
  memset(&prob, 0, sizeof(prob));
  printf("workspace_empty %zu\n", stepkv_compress_workspace_size(&prob, 1));
  return 0;
}

static int gpu_mode(const char* dir) {
  const size_t kv_elems = (size_t)HKV * T * D, q_elems = (size_t)HQ * W * D;
  uint16_t* hK = malloc(L * kv_elems * 2);
  uint16_t* hV = malloc(L * kv_elems * 2);
  uint16_t* hQ = malloc(NSAL * q_elems * 2);
  for (size_t i = 0; i < L * kv_elems; ++i) hK[i] = to_bf16(2.0f * lcg_uniform() - 1.0f);
  for (size_t i = 0; i < L * kv_elems; ++i) hV[i] = to_bf16(2.0f * lcg_uniform() - 1.0f);
  for (size_t i = 0; i < NSAL * q_elems; ++i) hQ[i] = to_bf16(2.0f * lcg_uniform() - 1.0f);
  int32_t step_id[T];
  uint8_t prot[T];
  for (int i = 0; i < T; ++i) {
    step_id[i] = i < 16 ? 0 : (int32_t)((int64_t)(i - 16) * NSTEPS / (T - 16));
    prot[i] = (uint8_t)(i < 16 || i >= T - W);
  }
  float sig[4][NSTEPS];
  for (int k = 0; k < NSTEPS; ++k) {
    sig[0][k] = lcg_uniform() < 0.8f ? 1.0f : 0.0f; /* valid */
    sig[1][k] = lcg_uniform();                      /* gain */
    sig[2][k] = lcg_uniform();                      /* red */
    sig[3][k] = lcg_uniform();                      /* obs_sim */
  }
  float reuse[NSTEPS] = {0};

  void *dK[L], *dV[L], *dKo[L], *dVo[L], *dQ[NSAL];
  for (int l = 0; l < L; ++l) {
    CK(cudaMalloc(&dK[l], kv_elems * 2));
    CK(cudaMalloc(&dV[l], kv_elems * 2));
    CK(cudaMalloc(&dKo[l], kv_elems * 2));
    CK(cudaMalloc(&dVo[l], kv_elems * 2));
    CK(cudaMemcpy(dK[l], hK + l * kv_elems, kv_elems * 2, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(dV[l], hV + l * kv_elems, kv_elems * 2, cudaMemcpyHostToDevice));
  }
  for (int i = 0; i < NSAL; ++i) {
    CK(cudaMalloc(&dQ[i], q_elems * 2));
    CK(cudaMemcpy(dQ[i], hQ + i * q_elems, q_elems * 2, cudaMemcpyHostToDevice));
  }
  int32_t *d_sid, *d_kept, *d_nkept, *d_status;
  uint8_t* d_prot;
  float* d_sig[4];
  float *d_reuse_in, *d_reuse_out;
  CK(cudaMalloc((void**)&d_sid, sizeof(step_id)));
  CK(cudaMalloc((void**)&d_prot, sizeof(prot)));
  CK(cudaMalloc((void**)&d_kept, T * 4));
  CK(cudaMalloc((void**)&d_nkept, 4));
  CK(cudaMalloc((void**)&d_status, 4));
  CK(cudaMalloc((void**)&d_reuse_in, sizeof(reuse)));
  CK(cudaMalloc((void**)&d_reuse_out, sizeof(reuse)));
  CK(cudaMemcpy(d_sid, step_id, sizeof(step_id), cudaMemcpyHostToDevice));
  CK(cudaMemcpy(d_prot, prot, sizeof(prot), cudaMemcpyHostToDevice));
  CK(cudaMemcpy(d_reuse_in, reuse, sizeof(reuse), cudaMemcpyHostToDevice));
  CK(cudaMemset(d_status, 0, 4));
  for (int s = 0; s < 4; ++s) {
    CK(cudaMalloc((void**)&d_sig[s], sizeof(sig[s])));
    CK(cudaMemcpy(d_sig[s], sig[s], sizeof(sig[s]), cudaMemcpyHostToDevice));
  }

  stepkv_problem_t prob;
  memset(&prob, 0, sizeof(prob));
  prob.L = L; prob.Hkv = HKV; prob.Hq = HQ; prob.d = D; prob.T = T; prob.W = W; prob.n_sal_layers = NSAL;
  prob.K = (const void* const*)dK;
  prob.V = (const void* const*)dV;
  prob.kv_head_stride = (int64_t)T * D;
  prob.Q = (const void* const*)dQ;
  prob.q_head_stride = (int64_t)W * D;
  prob.step_id = d_sid;
  prob.prot = d_prot;
  prob.steps.n_steps = NSTEPS;
  prob.steps.valid = d_sig[0];
  prob.steps.gain = d_sig[1];
  prob.steps.red = d_sig[2];
  prob.steps.obs_sim = d_sig[3];
  prob.steps.reuse_in = d_reuse_in;
  prob.steps.reuse_out = d_reuse_out;
  prob.budget.mode = STEPKV_BUDGET_RATIO;
  prob.budget.ratio_num = 1;
  prob.budget.ratio_den = 4;
  prob.K_out = dKo;
  prob.V_out = dVo;
  prob.out_head_stride = (int64_t)T * D;
  prob.sel.kept_idx = d_kept;
  prob.sel.kept_cap = T;
  prob.sel.n_kept = d_nkept;

  stepkv_params_t p;
  stepkv_default_params(&p);
  const size_t ws_bytes = stepkv_compress_workspace_size(&prob, 1);
  void* ws = NULL;
  CK(cudaMalloc(&ws, ws_bytes));
  const stepkv_status_t st = stepkv_compress(&prob, 1, &p, ws, ws_bytes, d_status, NULL);
  if (st != STEPKV_OK) {
    fprintf(stderr, "stepkv_compress: %s\n", stepkv_status_string(st));
    return 3;
  }
  CK(cudaDeviceSynchronize());
  int32_t dev_status = -1, n_kept = -1;
  CK(cudaMemcpy(&dev_status, d_status, 4, cudaMemcpyDeviceToHost));
  CK(cudaMemcpy(&n_kept, d_nkept, 4, cudaMemcpyDeviceToHost));
  if (dev_status != 0 || n_kept < 1 || n_kept > T) {
    fprintf(stderr, "device status %d, n_kept %d\n", dev_status, n_kept);
    return 4;
  }
  int32_t* kept = malloc((size_t)n_kept * 4);
  CK(cudaMemcpy(kept, d_kept, (size_t)n_kept * 4, cudaMemcpyDeviceToHost));
  uint16_t* kout = malloc((size_t)HKV * n_kept * D * 2);
  for (int h = 0; h < HKV; ++h)
    CK(cudaMemcpy(kout + (size_t)h * n_kept * D, (uint16_t*)dKo[1] + (size_t)h * T * D, (size_t)n_kept * D * 2,
                  cudaMemcpyDeviceToHost));
  int bad = write_file(dir, "K.bin", hK, L * kv_elems * 2) | write_file(dir, "V.bin", hV, L * kv_elems * 2) |
            write_file(dir, "Q.bin", hQ, NSAL * q_elems * 2) | write_file(dir, "step_id.bin", step_id, sizeof(step_id)) |
            write_file(dir, "prot.bin", prot, sizeof(prot)) | write_file(dir, "signals.bin", sig, sizeof(sig)) |
            write_file(dir, "kept.bin", kept, (size_t)n_kept * 4) |
            write_file(dir, "K_out_layer1.bin", kout, (size_t)HKV * n_kept * D * 2);
  printf("n_kept %d\n", n_kept);
  return bad ? 5 : 0;
}

int main(int argc, char** argv) {
  if (argc >= 2 && strcmp(argv[1], "host") == 0) return host_mode();
  if (argc >= 3 && strcmp(argv[1], "gpu") == 0) return gpu_mode(argv[2]);
  fprintf(stderr, "usage: %s host | gpu DIR\n", argv[0]);
  return 1;
}
