/* A plain C (C99) consumer of the library's ABI: compiled with gcc against include/ and linked
 * with libsoap.so, no CUDA headers and no PyTorch. It runs only host-side entry points (the
 * defaults, the layer-wise planner, host validation), so it needs no GPU. Exit code 0 = pass. */
#include <stdio.h>
#include <string.h>

#include "muon.h"
#include "soap.h"

int main(void) {
  soap_hparams hp;
  soap_default_hparams(&hp);
  if (hp.eig_every != 1 || hp.kl != 0 || hp.stale != 0 || hp.guard != 1) return 1;
  muon_hparams mh;
  muon_default_hparams(&mh);
  if (mh.ns_steps != 16 || mh.coeffs != NULL) return 2;

  /* the dense block on two ranks: every matrix gets exactly one owner */
  soap_shape block[7] = {{2048, 2048, 1, 1}, {2048, 2048, 1, 1}, {2048, 2048, 1, 1}, {2048, 2048, 1, 1},
                         {2048, 8192, 1, 1}, {2048, 8192, 1, 1}, {8192, 2048, 1, 1}};
  int32_t owner[7];
  double load[2];
  for (int policy = 0; policy < 2; ++policy) {
    memset(owner, 0xff, sizeof owner);
    if (soap_layerwise_assign(block, 7, 2, policy, owner, load) != SOAP_OK) return 3;
    for (int i = 0; i < 7; ++i)
      if (owner[i] != 0 && owner[i] != 1) return 4;
    if (!(load[0] > 0.0 && load[1] > 0.0)) return 5;
  }

  /* invalid arguments are refused on the host, before any device work */
  soap_handle h = NULL;
  soap_shape bad = {0, 4, 1, 1};
  if (soap_create(&bad, 1, &hp, 0, &h) != SOAP_ERR_INVALID_ARG || h != NULL) return 6;
  muon_handle mu = NULL;
  soap_shape odd = {12, 16, 0, 0};
  if (muon_create(&odd, 1, &mh, 0, &mu) != SOAP_ERR_INVALID_ARG || mu != NULL) return 7;
  if (strcmp(soap_last_error(NULL), "null handle") != 0) return 8;
  soap_destroy(NULL);
  muon_destroy(NULL);
  printf("c abi ok\n");
  return 0;
}
