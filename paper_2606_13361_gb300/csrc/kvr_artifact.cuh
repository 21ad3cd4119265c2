// kvr_artifact.cuh -- arguments of the artifact kernels (kvr_artifact.cu):
// one sequence's cache pages <-> an artifact, bf16 (Algorithm 1 store,
// Algorithm 2 deserialize) or per-tensor symmetric int8 (Sec. 5 "Quantizing
// the artifact"), through device-accessible pointers (device memory or pinned
// host memory seen through its device mapping).
#pragma once

#include "kvr_internal.h"

namespace kvr {

struct ArtifactArgs {
  char* pages;           // page area (cache rows of d bf16)
  const int32_t* table;  // device page-table row of the sequence
  int64_t n_pages;
  int layers, Hkv, d;
  int L;                 // positions 0..L-1 move (artifact stride)
  int n_tiles;           // tiles (pages) to move; 0: all of L
  char* art;             // bf16 artifact [layers][2][Hkv][L][d]
  int8_t* codes;         // int8 artifact codes [layers][2][Hkv][L][d]
  float* scales;         // int8 artifact scales [layers][2]
  uint32_t* amax;        // [layers][2] scratch: max |x| as bf16 magnitude bits (int8 export)
  int* err;
};

// bf16 artifact <-> pages, bit for bit.
cudaError_t launch_artifact_copy(const ArtifactArgs& a, bool to_pages, cudaStream_t st);
// int8 export: max |x| per tensor, then the codes and scales (a.amax zeroed by the caller).
cudaError_t launch_q8_export(const ArtifactArgs& a, cudaStream_t st);
// int8 load: bf16(code * s) into the pages.
cudaError_t launch_q8_load(const ArtifactArgs& a, cudaStream_t st);
// int8 codes into int8 pages (the first page_bytes / 2 of each page, rows of d
// bytes in the cache's row order), full tiles only.
cudaError_t launch_q8_codes_to_pages(const ArtifactArgs& a, cudaStream_t st);

}  // namespace kvr
