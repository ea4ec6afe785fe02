/* A plain C99 caller of librefadapt.so: Algorithm 1 over a small block stack
 * through the C ABI alone (no Python anywhere on its path), for the test that
 * checks its results against the oracle.
 *
 * usage: algorithm1_client B H d n_text n_ref n_tgt blocks steps theta delta_max in.bin out.bin
 *
 * in.bin:  for t in steps, b in blocks: the joint bf16 tensor X[3][B][H][N][d]
 *          (q, k, v; rows text, reference, target; N = n_text + n_ref + n_tgt).
 * out.bin: for t in steps, b in blocks: mode[B] int32, gbar[B] f32, D[B][H] f32
 *          (0 at t = 0), M[B][H] f32 (the exposure the gate read, 0 at t = 0),
 *          O text, reference, target [B][H][n][d] bf16 each, a_b[B] int32.
 *
 * Per block and step: the gate (t = 0) or the Q change with the gate in one
 * call (t >= 1), then the joint attention, which reads this step's reference
 * rows for materialising samples and writes them into the block's cache
 * slot. Every call is on the default stream, in order. Returns 0 on success,
 * 2 on a library error (printed), 3 on a CUDA or file error. */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "refadapt.h"

#define CK(x)                                                               \
  do {                                                                      \
    cudaError_t e_ = (x);                                                   \
    if (e_ != cudaSuccess) {                                                \
      fprintf(stderr, "%s:%d %s\n", __FILE__, __LINE__, cudaGetErrorString(e_)); \
      return 3;                                                             \
    }                                                                       \
  } while (0)
#define RA(x)                                                               \
  do {                                                                      \
    ra_status s_ = (x);                                                     \
    if (s_ != RA_OK) {                                                      \
      fprintf(stderr, "%s:%d %s: %s\n", __FILE__, __LINE__, refadapt_status_string(s_), refadapt_last_error()); \
      return 2;                                                             \
    }                                                                       \
  } while (0)

/* A segment of rows [row0, row0 + n) of kind z (0 q, 1 k, 2 v) of a joint tensor. */
static ra_seg joint_seg(uint16_t* X, int z, int row0, int n, int B, int H, int N, int d) {
  ra_seg s;
  memset(&s, 0, sizeof(s));
  s.ptr = X + (size_t)z * B * H * N * d + (size_t)row0 * d;
  s.stride_b = (int64_t)H * N * d;
  s.stride_h = (int64_t)N * d;
  s.stride_n = d;
  s.n = n;
  return s;
}

static ra_seg plain_seg(void* p, int n, int H, int d) {
  ra_seg s;
  memset(&s, 0, sizeof(s));
  s.ptr = p;
  s.stride_b = (int64_t)H * n * d;
  s.stride_h = (int64_t)n * d;
  s.stride_n = d;
  s.n = n;
  return s;
}

int main(int argc, char** argv) {
  if (argc != 13) {
    fprintf(stderr, "usage: %s B H d n_text n_ref n_tgt blocks steps theta delta_max in.bin out.bin\n", argv[0]);
    return 3;
  }
  const int B = atoi(argv[1]), H = atoi(argv[2]), d = atoi(argv[3]);
  const int nt = atoi(argv[4]), nr = atoi(argv[5]), ng = atoi(argv[6]);
  const int nb = atoi(argv[7]), T = atoi(argv[8]);
  const double theta = atof(argv[9]);
  const int delta_max = atoi(argv[10]);
  const int N = nt + nr + ng;
  const size_t x_elems = (size_t)3 * B * H * N * d;
  const size_t bh = (size_t)B * H;

  FILE* fin = fopen(argv[11], "rb");
  FILE* fout = fopen(argv[12], "wb");
  if (!fin || !fout) return 3;
  uint16_t* hx = (uint16_t*)malloc(x_elems * 2);
  if (!hx) return 3;

  /* Device memory: every step's inputs of every block (read as q_{t-1} one
   * step later), the blocks' cache slots, mass partials, logs and outputs. */
  uint16_t** X = (uint16_t**)calloc((size_t)T * nb, sizeof(uint16_t*));
  for (int i = 0; i < T * nb; ++i) {
    if (fread(hx, 2, x_elems, fin) != x_elems) return 3;
    CK(cudaMalloc((void**)&X[i], x_elems * 2));
    CK(cudaMemcpy(X[i], hx, x_elems * 2, cudaMemcpyHostToDevice));
  }
  const int mpl = refadapt_mass_partial_len(nt, ng);
  const size_t cache_elems = (size_t)B * H * nr * d;
  void **cq = calloc(nb, sizeof(void*)), **ck = calloc(nb, sizeof(void*)), **cv = calloc(nb, sizeof(void*));
  float** mass = calloc(nb, sizeof(float*));
  int32_t** a_b = calloc(nb, sizeof(int32_t*));
  for (int b = 0; b < nb; ++b) {
    CK(cudaMalloc(&cq[b], cache_elems * 2));
    CK(cudaMalloc(&ck[b], cache_elems * 2));
    CK(cudaMalloc(&cv[b], cache_elems * 2));
    CK(cudaMemset(cq[b], 0, cache_elems * 2));
    CK(cudaMemset(ck[b], 0, cache_elems * 2));
    CK(cudaMemset(cv[b], 0, cache_elems * 2));
    CK(cudaMalloc((void**)&mass[b], bh * mpl * sizeof(float)));
    CK(cudaMalloc((void**)&a_b[b], B * sizeof(int32_t)));
    CK(cudaMemset(a_b[b], 0xff, B * sizeof(int32_t)));
  }
  const size_t ws_bytes = refadapt_q_delta_workspace_size(B, H);
  void* ws;
  CK(cudaMalloc(&ws, ws_bytes));
  CK(cudaMemset(ws, 0, ws_bytes));
  ra_state* state;
  CK(cudaMalloc((void**)&state, refadapt_state_size(B)));
  RA(refadapt_state_init(state, B, NULL));
  int32_t* mode;
  float *gbar, *D, *M;
  CK(cudaMalloc((void**)&mode, B * sizeof(int32_t)));
  CK(cudaMalloc((void**)&gbar, B * sizeof(float)));
  CK(cudaMalloc((void**)&D, bh * sizeof(float)));
  CK(cudaMalloc((void**)&M, bh * sizeof(float)));
  const int nrole[3] = {nt, nr, ng};
  void* O[3];
  uint16_t* ho[3];
  for (int r = 0; r < 3; ++r) {
    CK(cudaMalloc(&O[r], bh * nrole[r] * d * 2 + 16));
    ho[r] = (uint16_t*)malloc(bh * nrole[r] * d * 2 + 16);
  }
  int32_t* hmode = malloc(B * sizeof(int32_t));
  int32_t* hab = malloc(B * sizeof(int32_t));
  float* hg = malloc(B * sizeof(float));
  float* hd = malloc(bh * sizeof(float));
  float* hm = malloc(bh * sizeof(float));
  const int row0[3] = {0, nt, nt + nr};

  for (int t = 0; t < T; ++t) {
    for (int b = 0; b < nb; ++b) {
      uint16_t* x = X[t * nb + b];
      CK(cudaMemset(D, 0, bh * sizeof(float)));
      CK(cudaMemset(M, 0, bh * sizeof(float)));
      for (int r = 0; r < 3; ++r) CK(cudaMemset(O[r], 0, bh * nrole[r] * d * 2));
      ra_gate_args g;
      memset(&g, 0, sizeof(g));
      g.theta = theta;
      g.t = t;
      g.b = b;
      g.B = B;
      g.H = H;
      g.delta_max = delta_max;
      g.forced_boundary = -1;
      g.mass_partial_len = mpl;
      g.mass_row_count = ng;
      g.cue = RA_CUE_PRODUCT;
      g.state = state;
      g.mode_out = mode;
      g.gbar_out = gbar;
      g.m_out = M;
      if (t == 0) {
        RA(refadapt_gate(&g, NULL));
      } else {
        /* Eq. 1 on the target queries of steps t and t - 1, then the gate */
        g.mass_partial_prev = mass[b];
        ra_seg qc = joint_seg(x, 0, row0[2], ng, B, H, N, d);
        ra_seg qp = joint_seg(X[(t - 1) * nb + b], 0, row0[2], ng, B, H, N, d);
        RA(refadapt_q_delta_gate(&qc, &qp, B, H, d, 1e-6f, D, ws, ws_bytes, &g, NULL));
      }
      ra_attn_args a;
      memset(&a, 0, sizeof(a));
      a.B = B;
      a.H = H;
      a.d = d;
      for (int r = 0; r < 3; ++r) {
        if (r == RA_REF) {
          a.q[r] = plain_seg(cq[b], nr, H, d);
          a.k[r] = plain_seg(ck[b], nr, H, d);
          a.v[r] = plain_seg(cv[b], nr, H, d);
        } else {
          a.q[r] = joint_seg(x, 0, row0[r], nrole[r], B, H, N, d);
          a.k[r] = joint_seg(x, 1, row0[r], nrole[r], B, H, N, d);
          a.v[r] = joint_seg(x, 2, row0[r], nrole[r], B, H, N, d);
        }
        a.o[r] = plain_seg(O[r], nrole[r], H, d);
      }
      a.ref_fresh_q = joint_seg(x, 0, row0[1], nr, B, H, N, d);
      a.ref_fresh_k = joint_seg(x, 1, row0[1], nr, B, H, N, d);
      a.ref_fresh_v = joint_seg(x, 2, row0[1], nr, B, H, N, d);
      a.a_b = a_b[b];
      a.step = t;
      a.mode = mode;
      a.mass_partial = mass[b];
      RA(refadapt_joint_attn(&a, NULL));
      CK(cudaDeviceSynchronize());
      CK(cudaMemcpy(hmode, mode, B * sizeof(int32_t), cudaMemcpyDeviceToHost));
      CK(cudaMemcpy(hg, gbar, B * sizeof(float), cudaMemcpyDeviceToHost));
      CK(cudaMemcpy(hd, D, bh * sizeof(float), cudaMemcpyDeviceToHost));
      CK(cudaMemcpy(hm, M, bh * sizeof(float), cudaMemcpyDeviceToHost));
      CK(cudaMemcpy(hab, a_b[b], B * sizeof(int32_t), cudaMemcpyDeviceToHost));
      fwrite(hmode, sizeof(int32_t), B, fout);
      fwrite(hg, sizeof(float), B, fout);
      fwrite(hd, sizeof(float), bh, fout);
      fwrite(hm, sizeof(float), bh, fout);
      for (int r = 0; r < 3; ++r) {
        CK(cudaMemcpy(ho[r], O[r], bh * nrole[r] * d * 2, cudaMemcpyDeviceToHost));
        fwrite(ho[r], 2, bh * nrole[r] * d, fout);
      }
      fwrite(hab, sizeof(int32_t), B, fout);
    }
  }
  fclose(fout);
  fclose(fin);
  printf("client ok: %d steps x %d blocks\n", T, nb);
  return 0;
}
