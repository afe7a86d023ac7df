/* One layer compressed by a plain C caller through the C ABI (no Python in the
 * call path): reads a problem and its bf16 inputs from a file, runs
 * tp_compress_layer on the device, and writes the kept indices, the int8 V
 * codes and the scales of the compressed cache to a second file.
 *
 * Input file (little-endian):  int32 H_q, H_kv, d, L_t, batch; double
 * keep_ratio; int64 doc_offsets[batch + 1]; then Q, K, V as uint16 bf16 bits
 * ([batch, H_q, L_t, d], [H_kv, N, d], [H_kv, N, d]).
 * Output file: int64 cap; int32 idx[batch * H_kv * cap];
 * int8 vqc[batch * H_kv * cap * d]; float gammac[batch * H_kv * cap]. */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "taskpress.h"

#define CUDA_OK(x)                                                         \
  do {                                                                     \
    cudaError_t e_ = (x);                                                  \
    if (e_ != cudaSuccess) {                                               \
      fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));             \
      return 2;                                                            \
    }                                                                      \
  } while (0)

static void* read_all(FILE* f, size_t bytes) {
  void* p = malloc(bytes ? bytes : 1);
  if (p && bytes && fread(p, 1, bytes, f) != bytes) {
    free(p);
    return NULL;
  }
  return p;
}

int main(int argc, char** argv) {
  if (argc != 3) {
    fprintf(stderr, "usage: %s input output\n", argv[0]);
    return 1;
  }
  FILE* in = fopen(argv[1], "rb");
  if (!in) return 1;
  int32_t hdr[5];
  double keep_ratio;
  if (fread(hdr, sizeof(int32_t), 5, in) != 5 || fread(&keep_ratio, sizeof(double), 1, in) != 1) return 1;
  const int hq = hdr[0], hkv = hdr[1], d = hdr[2], lt = hdr[3], batch = hdr[4];
  int64_t* offs = (int64_t*)read_all(in, sizeof(int64_t) * (size_t)(batch + 1));
  if (!offs) return 1;
  const int64_t n = offs[batch];
  const size_t qn = (size_t)batch * hq * lt * d, kn = (size_t)hkv * n * d;
  uint16_t* q = (uint16_t*)read_all(in, qn * 2);
  uint16_t* k = (uint16_t*)read_all(in, kn * 2);
  uint16_t* v = (uint16_t*)read_all(in, kn * 2);
  fclose(in);
  if (!q || !k || !v) return 1;

  tp_problem p;
  memset(&p, 0, sizeof(p));
  p.n_heads_q = hq;
  p.n_heads_kv = hkv;
  p.head_dim = d;
  p.guide_len = lt;
  p.batch = batch;
  p.pool_kernel = 5;
  p.quant_bits = 8;
  p.doc_offsets = offs;
  const int64_t cap = tp_kept_capacity(&p, keep_ratio, -1);
  const size_t ws_bytes = tp_workspace_bytes(&p, keep_ratio, -1);
  if (cap < 0 || ws_bytes == 0) return 3;
  const size_t m = (size_t)batch * hkv * (size_t)cap;

  void *dq, *dk, *dv, *dkc, *dvc, *dws;
  int32_t* didx;
  int8_t* dvqc;
  float* dgc;
  CUDA_OK(cudaMalloc(&dq, qn * 2));
  CUDA_OK(cudaMalloc(&dk, kn * 2));
  CUDA_OK(cudaMalloc(&dv, kn * 2));
  CUDA_OK(cudaMalloc((void**)&didx, m * sizeof(int32_t) + 4));
  CUDA_OK(cudaMalloc(&dkc, m * d * 2 + 16));
  CUDA_OK(cudaMalloc(&dvc, m * d * 2 + 16));
  CUDA_OK(cudaMalloc((void**)&dvqc, m * d + 16));
  CUDA_OK(cudaMalloc((void**)&dgc, m * sizeof(float) + 4));
  CUDA_OK(cudaMalloc(&dws, ws_bytes));
  CUDA_OK(cudaMemcpy(dq, q, qn * 2, cudaMemcpyHostToDevice));
  CUDA_OK(cudaMemcpy(dk, k, kn * 2, cudaMemcpyHostToDevice));
  CUDA_OK(cudaMemcpy(dv, v, kn * 2, cudaMemcpyHostToDevice));

  int st = tp_compress_layer(&p, dq, dk, dv, keep_ratio, -1, didx, dkc, dvc, dvqc, dgc, NULL, NULL,
                             dws, ws_bytes, NULL);
  if (st != TP_OK) {
    fprintf(stderr, "tp_compress_layer: %s\n", tp_status_string(st));
    return 4;
  }
  st = tp_check_status(dws, ws_bytes, NULL);  /* synchronises the stream */
  if (st != TP_OK) {
    fprintf(stderr, "device status: %s\n", tp_status_string(st));
    return 5;
  }
  int32_t* idx = (int32_t*)malloc(m * sizeof(int32_t) + 4);
  int8_t* vqc = (int8_t*)malloc(m * d + 1);
  float* gc = (float*)malloc(m * sizeof(float) + 4);
  if (!idx || !vqc || !gc) return 1;
  CUDA_OK(cudaMemcpy(idx, didx, m * sizeof(int32_t), cudaMemcpyDeviceToHost));
  CUDA_OK(cudaMemcpy(vqc, dvqc, m * d, cudaMemcpyDeviceToHost));
  CUDA_OK(cudaMemcpy(gc, dgc, m * sizeof(float), cudaMemcpyDeviceToHost));

  FILE* out = fopen(argv[2], "wb");
  if (!out) return 1;
  fwrite(&cap, sizeof(int64_t), 1, out);
  fwrite(idx, sizeof(int32_t), m, out);
  fwrite(vqc, 1, m * d, out);
  fwrite(gc, sizeof(float), m, out);
  fclose(out);
  cudaFree(dq);
  cudaFree(dk);
  cudaFree(dv);
  cudaFree(didx);
  cudaFree(dkc);
  cudaFree(dvc);
  cudaFree(dvqc);
  cudaFree(dgc);
  cudaFree(dws);
  printf("compress_layer ok: cap %lld\n", (long long)cap);
  return 0;
}
